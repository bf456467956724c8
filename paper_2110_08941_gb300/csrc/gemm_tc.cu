// Persistent, warp-specialised tcgen05 GEMM for sm_103a (bf16 operands, fp32 accumulation in
// tensor memory).  It evaluates every contraction of the per-worker forward and backward passes
// (Eq. 1 gradients g^m, Section 1):
//   forward       H_l   = act(H_{l-1} W_l^T + b_l)        A: K-major, B: K-major
//   input grad    dH    = (delta_l W_l) * 1[H_{l-1} > 0]   A: K-major, B: MN-major
//   weight grad   G_m   = delta_l[seg_m]^T H_{l-1}[seg_m]  A: MN-major, B: MN-major, one group per worker
//
// CTA layout (192 threads, one CTA per SM):
//   warp 0      one elected thread issues TMA tile loads into a 4-stage shared-memory ring
//   warp 1      owns the tensor-memory allocation; one elected thread issues tcgen05.mma
//   warps 2..5  epilogue: tcgen05.ld from tensor memory, fused bias/ReLU/mask, global stores
// Two 128x256 fp32 accumulators (512 TMEM columns) let the epilogue of one tile overlap the
// main loop of the next.  Every mbarrier wait is bounded; on expiry the kernel records
// kDevWaitTimeout in the status word, stops issuing work, frees its tensor memory and returns.
#include <cudaTypedefs.h>

#include "gemm_tc.cuh"

namespace hs {

namespace {

constexpr int BM = kTcBM, BN = kTcBN, BK = kTcBK, S = kTcStages;
constexpr int A_STAGE = BM * BK * 2;                 // 16 KB
constexpr int B_STAGE = BN * BK * 2;                 // 32 KB
constexpr uint32_t STAGE_TX = A_STAGE + B_STAGE;     // bytes landed per stage
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 2 * BN;               // two accumulator buffers
constexpr int MN_CHUNK = 64 * BK * 2;                // one 64-wide MN slab of an MN-major tile (8 KB)
constexpr uint64_t kWaitLimitNs = 2000000000ull;     // 2 s per wait

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with the given parity; false if the abort flag rises or the limit passes.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int c0, int c1,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* tm, uint32_t src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
               ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(src)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// At most one bulk group may still be reading shared memory.
__device__ __forceinline__ void bulk_wait_read_1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* tm) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
// 32 lanes x 32 consecutive fp32 columns: thread t receives row (quadrant base + t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
// The wait names the destination registers so no use of them is scheduled above it.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                 "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                 "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]),
                 "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]),
                 "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// Instruction descriptor, kind::f16: D fp32, A/B bf16, per-operand major-ness, N = BN, M = BM.
__host__ __device__ constexpr uint32_t make_idesc(bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

// Shared-memory matrix descriptor, 128-byte swizzle.  lbo/sbo in bytes.
//   K-major tile (rows x 64 K, 128 B per row, 8-row swizzle atoms of 1 KB): SBO = 1 KB between
//     8-row groups; LBO unused.  The K step of 16 elements advances the start by 32 B.
//   MN-major tile (64 K rows x 128 B per 64-wide MN slab): SBO = 1 KB between 8-row K groups,
//     LBO = 8 KB between 64-wide MN slabs.  The K step of 16 rows advances the start by 2 KB.
__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= 2ull << 61;
  return d;
}

__device__ __forceinline__ void record_error(DevStatus* st, int32_t code, int32_t info) {
  if (st && atomicCAS(&st->err, 0, code) == 0) st->err_info = info;
}

struct TileCoord {
  int g, tm, tn;
};

// Tiles are numbered group-major; within a group, bands of 16 M-tiles are walked N-tile by
// N-tile so that the CTAs running at the same time share A and B panels in L2.
__device__ __forceinline__ TileCoord decode_tile(int t, int tiles_m, int tiles_n) {
  const int per_group = tiles_m * tiles_n;
  TileCoord c;
  c.g = t / per_group;
  const int r = t - c.g * per_group;
  constexpr int GM = 16;
  const int band = r / (GM * tiles_n);
  const int within = r - band * GM * tiles_n;
  const int rows = min(GM, tiles_m - band * GM);
  c.tm = band * GM + within % rows;
  c.tn = within / rows;
  return c;
}

__device__ __forceinline__ float u2f(uint32_t u) { return __uint_as_float(u); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&v);
}

// One epilogue unit: a 128-byte column strip of one accumulator row (32 fp32 or 64 bf16 outputs),
// computed from `r` (columns n_base..n_base+31) and, for bf16 outputs, `r2` (n_base+32..+63), packed
// into eight 16-byte words.  Columns past n_store are computed but never stored (the TMA store
// clips them); only the bias and mask reads are guarded.
template <int EPI>
__device__ __forceinline__ void epilogue_unit(const TcGemmParams& p, int row, int n_base, const uint32_t (&r)[32],
                                              const uint32_t (&r2)[32], uint4 (&o)[8]) {
  if (EPI == kTcEpiStoreF32) {
#pragma unroll
    for (int j = 0; j < 8; ++j) o[j] = make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
  } else if (EPI == kTcEpiBiasF32) {
    float b[32];
    if (n_base + 32 <= p.Ndim) {
      const float4* b4 = reinterpret_cast<const float4*>(p.bias + n_base);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 t = __ldg(b4 + j);
        b[4 * j] = t.x; b[4 * j + 1] = t.y; b[4 * j + 2] = t.z; b[4 * j + 3] = t.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) b[j] = (n_base + j < p.Ndim) ? __ldg(p.bias + n_base + j) : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o[j] = make_uint4(__float_as_uint(u2f(r[4 * j]) + b[4 * j]), __float_as_uint(u2f(r[4 * j + 1]) + b[4 * j + 1]),
                        __float_as_uint(u2f(r[4 * j + 2]) + b[4 * j + 2]),
                        __float_as_uint(u2f(r[4 * j + 3]) + b[4 * j + 3]));
  } else {
    // bf16 outputs: 64 columns
    float v[64];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      v[j] = u2f(r[j]);
      v[32 + j] = u2f(r2[j]);
    }
    if (EPI == kTcEpiBiasReluBf16) {
      if (n_base + 64 <= p.Ndim) {
        const float4* b4 = reinterpret_cast<const float4*>(p.bias + n_base);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float4 t = __ldg(b4 + j);
          v[4 * j] = fmaxf(v[4 * j] + t.x, 0.f);
          v[4 * j + 1] = fmaxf(v[4 * j + 1] + t.y, 0.f);
          v[4 * j + 2] = fmaxf(v[4 * j + 2] + t.z, 0.f);
          v[4 * j + 3] = fmaxf(v[4 * j + 3] + t.w, 0.f);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 64; ++j)
          v[j] = fmaxf(v[j] + ((n_base + j < p.Ndim) ? __ldg(p.bias + n_base + j) : 0.f), 0.f);
      }
    } else {   // kTcEpiMaskBf16: ReLU' from the stored activation of the same row
      if (row < p.Mdim) {
        const __nv_bfloat16* z = p.Z + (int64_t)row * p.ldz + n_base;
        if (n_base + 64 <= p.n_store) {
          const uint4* z4 = reinterpret_cast<const uint4*>(z);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const uint4 zz = __ldg(z4 + j);
            const uint32_t w[4] = {zz.x, zz.y, zz.z, zz.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const __nv_bfloat162 pr = *reinterpret_cast<const __nv_bfloat162*>(&w[h]);
              const int k = 8 * j + 2 * h;
              v[k] = (__low2float(pr) > 0.f) ? v[k] : 0.f;
              v[k + 1] = (__high2float(pr) > 0.f) ? v[k + 1] : 0.f;
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < 64; ++j) v[j] = (n_base + j < p.n_store && __bfloat162float(z[j]) > 0.f) ? v[j] : 0.f;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o[j] = make_uint4(pack_bf16(v[8 * j], v[8 * j + 1]), pack_bf16(v[8 * j + 2], v[8 * j + 3]),
                        pack_bf16(v[8 * j + 4], v[8 * j + 5]), pack_bf16(v[8 * j + 6], v[8 * j + 7]));
  }
}

template <int EPI, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ TcGemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * A_STAGE;
  uint8_t* sStage = sB + S * B_STAGE;                 // epilogue staging, 1 KB aligned
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStage + kTcStagingBytes);
  uint64_t* full_bar = bars;
  uint64_t* empty_bar = bars + S;
  uint64_t* tfull_bar = bars + 2 * S;
  uint64_t* tempty_bar = bars + 2 * S + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&tfull_bar[b]), 1);
      mbar_init(smem_u32(&tempty_bar[b]), 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int total = p.groups * p.tiles_m * p.tiles_n;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int s = 0;
      uint32_t ph = 0;
      int last_g = -1;
      for (int t = blockIdx.x; t < total && !*abort_flag; t += gridDim.x) {
        const TileCoord c = decode_tile(t, p.tiles_m, p.tiles_n);
        const CUtensorMap* ta = &p.tmA[c.g];
        const CUtensorMap* tb = &p.tmB[c.g];
        if (c.g != last_g) {
          tma_prefetch_desc(ta);
          tma_prefetch_desc(tb);
          last_g = c.g;
        }
        const int nkb = p.num_kb[c.g];
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full_bar[s]);
          mbar_expect_tx(fb, STAGE_TX);
          const int k0 = kb * BK;
          const uint32_t a_dst = smem_u32(sA + s * A_STAGE);
          const uint32_t b_dst = smem_u32(sB + s * B_STAGE);
          if (A_MN) {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j) tma_load_2d(a_dst + j * MN_CHUNK, ta, c.tm * BM + 64 * j, k0, fb);
          } else {
            tma_load_2d(a_dst, ta, k0, c.tm * BM, fb);
          }
          if (B_MN) {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) tma_load_2d(b_dst + j * MN_CHUNK, tb, c.tn * BN + 64 * j, k0, fb);
          } else {
            tma_load_2d(b_dst, tb, k0, c.tn * BN, fb);
          }
          if (++s == S) { s = 0; ph ^= 1u; }
        }
        if (!ok) {
          record_error(p.st, kDevWaitTimeout, 1);
          *abort_flag = 1;
          break;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      constexpr uint32_t idesc = make_idesc(A_MN, B_MN);
      int s = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      for (int t = blockIdx.x; t < total && !*abort_flag; t += gridDim.x) {
        const TileCoord c = decode_tile(t, p.tiles_m, p.tiles_n);
        const int nkb = p.num_kb[c.g];
        if (!mbar_wait(smem_u32(&tempty_bar[ab]), aph ^ 1u, abort_flag)) {
          record_error(p.st, kDevWaitTimeout, 2);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + s * A_STAGE);
          const uint32_t b_base = smem_u32(sB + s * B_STAGE);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t ad = A_MN ? make_sdesc(a_base + kk * 2048, MN_CHUNK, 1024)
                                     : make_sdesc(a_base + kk * 32, 16, 1024);
            const uint64_t bd = B_MN ? make_sdesc(b_base + kk * 2048, MN_CHUNK, 1024)
                                     : make_sdesc(b_base + kk * 32, 16, 1024);
            umma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
          }
          umma_commit(smem_u32(&empty_bar[s]));
          if (++s == S) { s = 0; ph ^= 1u; }
        }
        if (!ok) {
          record_error(p.st, kDevWaitTimeout, 3);
          *abort_flag = 1;
          break;
        }
        umma_commit(smem_u32(&tfull_bar[ab]));
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue (warps 2..5)
    // Each warp owns 32 accumulator rows (its TMEM lane quadrant) and two 4 KB staging buffers.
    // Per unit: tcgen05.ld -> fused math -> 16-byte stores into a 128-byte-swizzled 32 x 128 B
    // box -> one TMA bulk store of the box (double-buffered: the store of one unit overlaps the
    // math of the next).
    constexpr bool kF32Out = (EPI == kTcEpiBiasF32 || EPI == kTcEpiStoreF32);
    constexpr int kUnitCols = kF32Out ? 32 : 64;
    constexpr int kUnits = BN / kUnitCols;
    const int q = warp & 3;   // the TMEM lane quadrant this warp may read
    const uint32_t stage_base = smem_u32(sStage) + (uint32_t)((warp - 2) * 8192);
    int sb = 0;
    int ab = 0;
    uint32_t aph = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      const TileCoord c = decode_tile(t, p.tiles_m, p.tiles_n);
      int ok = 1;
      if (lane == 0) ok = mbar_wait(smem_u32(&tfull_bar[ab]), aph, abort_flag) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          record_error(p.st, kDevWaitTimeout, 4);
          *abort_flag = 1;
        }
        break;
      }
      __syncwarp();
      tc_fence_after();
      const int row0 = c.tm * BM + q * 32;
      const int row = row0 + lane;
      const CUtensorMap* td = &p.tmD[c.g];
      const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN);
#pragma unroll 1
      for (int u = 0; u < kUnits; ++u) {
        const int n_base = c.tn * BN + u * kUnitCols;
        if (n_base >= p.n_store) break;
        uint32_t r[32], r2[32];
        tmem_ld32(t_row + (uint32_t)(u * kUnitCols), r);
        if (!kF32Out) tmem_ld32(t_row + (uint32_t)(u * kUnitCols + 32), r2);
        tmem_ld_wait(r);
        if (!kF32Out) tmem_ld_wait(r2);
        uint4 o[8];
        epilogue_unit<EPI>(p, row, n_base, r, r2, o);
        if (lane == 0) bulk_wait_read_1();   // the store that last used this buffer has read it
        __syncwarp();
        const uint32_t buf = stage_base + (uint32_t)(sb * 4096);
        const uint32_t rbase = buf + (uint32_t)(lane * 128);
#pragma unroll
        for (int j = 0; j < 8; ++j) st_shared_v4(rbase + (uint32_t)(((j ^ (lane & 7)) << 4)), o[j]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(td, buf, n_base, row0);
          bulk_commit();
        }
        sb ^= 1;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty_bar[ab]));
      if (++ab == 2) { ab = 0; aph ^= 1u; }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    // Give in-flight bulk copies and MMAs a bounded moment to land before the memory goes away.
    const uint64_t t0 = globaltimer();
    while (globaltimer() - t0 < 2000000ull) {
    }
  }
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

template <int EPI, bool A_MN, bool B_MN>
cudaError_t launch_variant(const TcGemmParams& p, int grid, cudaStream_t s) {
  static bool configured = false;
  auto kern = tc_gemm_kernel<EPI, A_MN, B_MN>;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  kern<<<grid, kThreads, kTcSmemBytes, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

bool tc_init_driver(const char** why) {
  if (g_encode) return true;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
    *why = "cuTensorMapEncodeTiled is not available from the driver";
    return false;
  }
  g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  return true;
}

static bool encode_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                      uint32_t box_inner, uint32_t box_outer, const char** why,
                      CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  if (!g_encode && !tc_init_driver(why)) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || (row_bytes & 15u) != 0) {
    *why = "TMA operand base or row stride is not 16-byte aligned";
    return false;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(tm, dtype, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the operand";
    return false;
  }
  return true;
}

bool tc_make_kmajor_map(CUtensorMap* tm, const TcOperand& op, int box_rows, const char** why) {
  return encode_2d(tm, op.base, (uint64_t)op.cols, (uint64_t)op.rows, (uint64_t)op.ld * 2, BK, (uint32_t)box_rows,
                   why);
}

bool tc_make_mnmajor_map(CUtensorMap* tm, const TcOperand& op, const char** why) {
  return encode_2d(tm, op.base, (uint64_t)op.cols, (uint64_t)op.rows, (uint64_t)op.ld * 2, 64, BK, why);
}

bool tc_make_store_map(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                       const char** why) {
  const uint64_t es = fp32 ? 4 : 2;
  return encode_2d(tm, base, (uint64_t)cols, (uint64_t)rows, (uint64_t)ld * es, (uint32_t)(128 / es), 32, why,
                   fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16);
}

cudaError_t launch_tc_gemm(const TcGemmParams& p, int num_sms, cudaStream_t s) {
  const int total = p.groups * p.tiles_m * p.tiles_n;
  if (total <= 0) return cudaSuccess;
  const int grid = total < num_sms ? total : num_sms;
  if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiBiasReluBf16, false, false>(p, grid, s);
  if (p.epi == kTcEpiBiasF32 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiBiasF32, false, false>(p, grid, s);
  if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn) return launch_variant<kTcEpiMaskBf16, false, true>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && p.a_mn && p.b_mn) return launch_variant<kTcEpiStoreF32, true, true>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiStoreF32, false, false>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && p.b_mn) return launch_variant<kTcEpiStoreF32, false, true>(p, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace hs
