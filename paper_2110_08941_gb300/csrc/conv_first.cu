// The first convolution of the CNN workload (3x3, padding 1, a few input channels) as one kernel:
// the input rows a tile reads staged by TMA, patch rows built from them in shared memory, the
// product with the resident bf16 weights on the tensor core, bias + ReLU, NHWC bf16 activations.
//
// The generic path materialised the patch rows with a separate kernel and ran them through the
// tiled GEMM, whose 256 x 128 tiles hold one 64-deep k-block each: per tile the epilogue (tensor-
// memory loads, bias, packing and stores for 256 x 64 outputs) was the bound, not memory traffic.
// Here a tile is 128 output pixels (whole output rows of one image).  One thread brings each
// tile's input rows (all channels, columns -4.., rows stride * ho0 - 1..; zero fill past the
// image is the padding) into a ring of shared-memory boxes several tiles ahead, so the producers
// never wait on global memory; 128 producer threads (one output pixel each) form the tile's patch
// rows (tap-major, the ones column at 9 C) from that box into the MMA operand layout and write them
// out for the weight-gradient product; the weights stay in shared memory for the whole launch;
// four accumulators in tensor memory let the epilogue drain one tile while the next ones are
// formed and multiplied.  The sums are the generic product's (same bf16 operands, same fp32
// accumulation; the zero columns past Kp add nothing), so the activations are the same bit for bit
// (tested).
//
// Roles (576 threads, one CTA per SM, persistent; the producers and the epilogue each run as two
// groups of four warps on alternate tiles):
//   warps 0..7   patch rows (group g = warp / 4 takes the CTA's tiles i with i % 2 == g; thread r
//                of a group: output pixel r of the tile) into a 4-stage ring
//   warps 8..15  epilogue (group (warp - 8) / 4): warp w drains tensor-memory lanes 32 * (w % 4)..
//                of a finished tile, bias + ReLU, bf16, 16-byte stores of its rows
//   warp 16      tensor-memory allocation; one thread loads the weights and issues the MMAs
//   warp 17      one thread issues the input boxes
// Every mbarrier wait is bounded and leaves through the error path (status word, abort flag).
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>

#include "ctx.cuh"
#include "tc_device.cuh"

namespace hs {

namespace {

using namespace tcdev;

constexpr int CF_BM = 128;                   // output pixels per tile (rows of the MMA)
constexpr int CF_S = 4;                      // patch-row stages
constexpr int CF_ACC = 4;                    // accumulators in tensor memory
constexpr int CF_IS = 8;                     // input-box stages
constexpr int CF_IN = 8192;                  // bytes per input-box stage
constexpr int CF_A = CF_BM * 128;            // one patch-row stage: 128 rows x 64 bf16 (K padded to 64), 16 KB
constexpr int CF_B = 128 * 128;              // the weights: up to 128 rows x 64 bf16
constexpr int kCfThreads = 576;
constexpr int kCfSmem = CF_S * CF_A + CF_B + CF_IS * CF_IN + 128 * 4 + 64 * 16 + 128 * 8 + 1024 + 512;
static_assert(kCfSmem <= 232448, "shared memory budget");
static_assert(CF_S % 2 == 0 && CF_ACC % 2 == 0 && CF_IS % 2 == 0, "alternate tiles of two groups");

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait16(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15])
               :
               : "memory");
}
__device__ __forceinline__ bool warp_wait_cf(uint32_t bar, uint32_t parity, volatile int* abort_flag, int lane) {
  int ok = 1;
  if (lane == 0) ok = mbar_wait(bar, parity, abort_flag) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  return ok != 0;
}

// KC: 16-byte chunks (8 patch columns) of a patch row that hold columns (Kp / 8).
template <int KC>
__global__ void __launch_bounds__(kCfThreads, 1) conv_first_fwd_kernel(const __grid_constant__ ConvFirstParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + CF_S * CF_A;
  uint8_t* sIn = sB + CF_B;
  float* sBias = reinterpret_cast<float*>(sIn + CF_IS * CF_IN);
  int4* sTab = reinterpret_cast<int4*>(sBias + 128);   // per patch column: offset in the input box, kind
  int2* sPix = reinterpret_cast<int2*>(sTab + 64);     // per tile row r: (output row in the tile, column)
  uint64_t* bars = reinterpret_cast<uint64_t*>(sPix + CF_BM);
  uint64_t* full_bar = bars;                           // [CF_S] patch rows written (the group's 4 warps)
  uint64_t* empty_bar = full_bar + CF_S;               // [CF_S] consumed by the MMAs
  uint64_t* tfull_bar = empty_bar + CF_S;              // [CF_ACC] accumulator holds a finished tile
  uint64_t* tempty_bar = tfull_bar + CF_ACC;           // [CF_ACC] drained (the group's 4 warps)
  uint64_t* in_full = tempty_bar + CF_ACC;             // [CF_IS] input box landed
  uint64_t* in_empty = in_full + CF_IS;                // [CF_IS] input box read (the group's 4 warps)
  uint64_t* w_bar = in_empty + CF_IS;                  // the weights landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(w_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t acc_cols = p.acc_cols;   // tensor-memory columns per accumulator (power of two >= npad)
  const int S = p.stride;

  if (threadIdx.x == 0) {
    for (int s = 0; s < CF_S; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 4);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int a = 0; a < CF_ACC; ++a) {
      mbar_init(smem_u32(&tfull_bar[a]), 1);
      mbar_init(smem_u32(&tempty_bar[a]), 4);
    }
    for (int s = 0; s < CF_IS; ++s) {
      mbar_init(smem_u32(&in_full[s]), 1);
      mbar_init(smem_u32(&in_empty[s]), 4);
    }
    mbar_init(smem_u32(w_bar), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  // patch column k < 9 C: tap = k / C (kh = tap / 3, kw = tap % 3), channel k % C; its value for
  // output pixel (rr, wo) of the tile sits at float (ci * box_h + S * rr + kh) * box_w + S * wo + kw + 3
  // of the input box; k = 9 C: the ones column
  if (threadIdx.x < 64) {
    const int k = threadIdx.x;
    int4 e = make_int4(0, 0, 0, 0);   // .x offset, .w kind: 0 zero, 1 input value, 2 one
    if (k < 9 * p.C) {
      const int tap = k / p.C, ci = k - tap * p.C;
      e = make_int4((ci * p.box_h + tap / 3) * p.box_w + tap % 3 + 3, 0, 0, 1);
    } else if (k == 9 * p.C) {
      e.w = 2;
    }
    sTab[k] = e;
  } else if (threadIdx.x >= 128 && threadIdx.x < 128 + CF_BM) {
    const int r = threadIdx.x - 128;
    const int rr = r / p.Wo;
    sPix[r] = make_int2(rr, r - rr * p.Wo);
  }
  if (warp < 8) {
    // the chunks past the patch columns stay zero in every stage (group g fills stages g, g + 2)
    const int r = threadIdx.x & 127;
    for (int s = threadIdx.x >> 7; s < CF_S; s += 2)
      for (int j = KC; j < 8; ++j)
        st_shared_v4(smem_u32(sA + s * CF_A + r * 128 + ((j ^ (r & 7)) << 4)), make_uint4(0u, 0u, 0u, 0u));
  }
  if (warp == 16) {
    tmem_alloc(smem_u32(tmem_slot), CF_ACC * acc_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dependency_wait();
  grid_dependents_launch();
  if (threadIdx.x < 128) sBias[threadIdx.x] = threadIdx.x < p.Cout ? __ldg(p.bias + threadIdx.x) : 0.f;
  __syncthreads();

  const int tiles = p.tiles;
  const int in_bytes = p.box_w * p.box_h * p.C * 4;

  if (warp < 8) {
    // ------------------------------------------------------------------ patch rows
    const int r = threadIdx.x & 127;
    const int grp = threadIdx.x >> 7;
    const int2 px = sPix[r];
    for (int i = grp, t = blockIdx.x + grp * gridDim.x; t < tiles && !*abort_flag; i += 2, t += 2 * gridDim.x) {
      const int s = i % CF_S, is = i % CF_IS;
      const uint32_t ph = (uint32_t)((i / CF_S) & 1), iph = (uint32_t)((i / CF_IS) & 1);
      if (!warp_wait_cf(smem_u32(&empty_bar[s]), ph ^ 1u, abort_flag, lane) ||
          !warp_wait_cf(smem_u32(&in_full[is]), iph, abort_flag, lane)) {
        if (lane == 0) {
          record_error(p.st, kDevWaitTimeout, 41);
          *abort_flag = 1;
        }
        break;
      }
      const int n = t / p.tpi;
      const int ho0 = (t - n * p.tpi) * p.R;
      const bool live = r < p.R * p.Wo && ho0 + px.x < p.Ho;
      const float* box = reinterpret_cast<const float*>(sIn + is * CF_IN);
      // rows past the tile's pixels read nothing (their (row, column) may lie beyond the box)
      const int base = live ? S * px.x * p.box_w + S * px.y : 0;
      float v[8 * KC];
#pragma unroll
      for (int k = 0; k < 8 * KC; ++k) {
        const int4 d = sTab[k];
        const float val = box[(live && d.w == 1) ? base + d.x : 0];
        v[k] = live ? (d.w == 1 ? val : (d.w == 2 ? 1.f : 0.f)) : 0.f;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&in_empty[is]));
      const uint32_t dst = smem_u32(sA + s * CF_A + r * 128);
      const int64_t row = ((int64_t)n * p.Ho + ho0) * p.Wo + r;
      uint4* gcol = reinterpret_cast<uint4*>(p.col + row * p.Kp);
#pragma unroll
      for (int j = 0; j < KC; ++j) {
        const uint4 q = make_uint4(pack_bf16(v[8 * j], v[8 * j + 1]), pack_bf16(v[8 * j + 2], v[8 * j + 3]),
                                   pack_bf16(v[8 * j + 4], v[8 * j + 5]), pack_bf16(v[8 * j + 6], v[8 * j + 7]));
        st_shared_v4(dst + ((j ^ (r & 7)) << 4), q);
        if (live) gcol[j] = q;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&full_bar[s]));
    }
  } else if (warp < 16) {
    // ------------------------------------------------------------------ epilogue
    const int q = warp & 3;                    // tensor-memory lane quadrant (warp % 4)
    const int grp = (warp - 8) >> 2;
    const int r = q * 32 + lane;               // this thread's row of the tile
    const int2 px = sPix[r];
    for (int i = grp, t = blockIdx.x + grp * gridDim.x; t < tiles; i += 2, t += 2 * gridDim.x) {
      const int a = i % CF_ACC;
      const uint32_t aph = (uint32_t)((i / CF_ACC) & 1);
      if (!warp_wait_cf(smem_u32(&tfull_bar[a]), aph, abort_flag, lane)) {
        if (lane == 0) {
          record_error(p.st, kDevWaitTimeout, 42);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const int n = t / p.tpi;
      const int ho0 = (t - n * p.tpi) * p.R;
      const bool live = r < p.R * p.Wo && ho0 + px.x < p.Ho;
      uint4* orow = reinterpret_cast<uint4*>(p.out + (((int64_t)n * p.Ho + ho0) * p.Wo + r) * p.Cout);
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(a * acc_cols);
      // 32 columns per round: two loads issued, one wait; with p.bits, the ReLU' of each 64 stored
      // values as one word
      uint64_t bits = 0;
      for (int cb = 0; cb < p.npad; cb += 32) {
        uint32_t v[2][16];
#pragma unroll
        for (int u = 0; u < 2; ++u)
          if (cb + 16 * u < p.npad) tmem_ld16(taddr + (uint32_t)(cb + 16 * u), v[u]);
#pragma unroll
        for (int u = 0; u < 2; ++u)
          if (cb + 16 * u < p.npad) tmem_ld_wait16(v[u]);
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int c0 = cb + 16 * u;
          if (c0 >= p.Cout) break;
          uint32_t o[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            o[e] = pack_bf16(fmaxf(__uint_as_float(v[u][2 * e]) + sBias[c0 + 2 * e], 0.f),
                             fmaxf(__uint_as_float(v[u][2 * e + 1]) + sBias[c0 + 2 * e + 1], 0.f));
          if (live) {
            orow[c0 >> 3] = make_uint4(o[0], o[1], o[2], o[3]);
            if (c0 + 8 < p.Cout) orow[(c0 >> 3) + 1] = make_uint4(o[4], o[5], o[6], o[7]);
          }
          if (p.bits) {
            // bf16 h > 0 exactly when 1 <= h <= 0x7fff as an unsigned half-word (sign clear, not
            // zero): the same decision as comparing the stored value, in integer operations
            uint32_t b16 = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              b16 |= (uint32_t)((o[e] & 0xffffu) - 1u < 0x7fffu) << (2 * e);
              b16 |= (uint32_t)((o[e] >> 16) - 1u < 0x7fffu) << (2 * e + 1);
            }
            bits |= (uint64_t)b16 << (c0 & 63);
            if (((c0 + 16) & 63) == 0) {
              if (live)
                p.bits[(int64_t)(c0 >> 6) * p.bits_ld + ((int64_t)n * p.Ho + ho0) * p.Wo + r] = bits;
              bits = 0;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty_bar[a]));
    }
  } else if (warp == 16) {
    if (lane == 0) {
      // ------------------------------------------------------------------ weights + MMA issuer
      tma_prefetch_desc(&p.tmW);
      mbar_expect_tx(smem_u32(w_bar), (uint32_t)(p.npad * 128));
      tma_load_2d(smem_u32(sB), &p.tmW, 0, 0, smem_u32(w_bar));
      bool ok = mbar_wait(smem_u32(w_bar), 0, abort_flag);
      const uint32_t idesc = make_idesc(false, false, CF_BM, p.npad);
      const uint64_t a_desc0 = make_sdesc(smem_u32(sA), 16, 1024);
      const uint64_t b_desc = make_sdesc(smem_u32(sB), 16, 1024);
      const int ksteps = (p.Kp + 15) >> 4;     // 16-column MMA steps holding patch columns
      int s = 0, a = 0;
      uint32_t ph = 0, aph = 0;
      for (int t = blockIdx.x; t < tiles && ok && !*abort_flag; t += gridDim.x) {
        if (!mbar_wait(smem_u32(&tempty_bar[a]), aph ^ 1u, abort_flag)) { ok = false; break; }
        tc_fence_after();
        if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(a * acc_cols);
        const uint64_t ad = a_desc0 + (uint64_t)((s * CF_A) >> 4);
        for (int kk = 0; kk < ksteps; ++kk) umma_bf16(d_tmem, ad + 2 * kk, b_desc + 2 * kk, idesc, kk ? 1u : 0u);
        umma_commit(smem_u32(&empty_bar[s]));
        umma_commit(smem_u32(&tfull_bar[a]));
        if (++s == CF_S) { s = 0; ph ^= 1u; }
        if (++a == CF_ACC) { a = 0; aph ^= 1u; }
      }
      if (!ok) {
        record_error(p.st, kDevWaitTimeout, 43);
        *abort_flag = 1;
      }
    }
  } else if (lane == 0) {
    // -------------------------------------------------------------------- input boxes
    tma_prefetch_desc(&p.tmX);
    int s = 0;
    uint32_t ph = 0;
    for (int t = blockIdx.x; t < tiles && !*abort_flag; t += gridDim.x) {
      if (!mbar_wait(smem_u32(&in_empty[s]), ph ^ 1u, abort_flag)) {
        record_error(p.st, kDevWaitTimeout, 44);
        *abort_flag = 1;
        break;
      }
      const int n = t / p.tpi;
      const int ho0 = (t - n * p.tpi) * p.R;
      const int c[4] = {-4, S * ho0 - 1, 0, n};
      mbar_expect_tx(smem_u32(&in_full[s]), (uint32_t)in_bytes);
      tma_load_4d(smem_u32(sIn + s * CF_IN), &p.tmX, c, smem_u32(&in_full[s]));
      if (++s == CF_IS) { s = 0; ph ^= 1u; }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    const uint64_t t0 = globaltimer();
    while (globaltimer() - t0 < 2000000ull) {
    }
  }
  if (warp == 16) {
    tc_fence_after();
    tmem_dealloc(tmem_base, CF_ACC * acc_cols);
  }
}

// Output rows per tile, input box columns and rows, for a first convolution of this shape.
void conv_first_geometry(const ConvLayer& L, int* R, int* box_w, int* box_h) {
  *R = std::min(L.hout, CF_BM / std::max(L.wout, 1));
  *box_w = (int)round_up((int64_t)L.stride * (L.wout - 1) + 6, 4);
  *box_h = L.stride * (*R - 1) + 3;
}

}  // namespace

bool conv_first_ok(const ConvLayer& L) {
  const char* v = getenv("HS_CONV_FIRST");
  if (v && !strcmp(v, "0")) return false;
  if (L.wout < 1 || L.wout > CF_BM || L.win % 4 || L.stride < 1 || L.stride > 2 || L.rows >= (1LL << 30)) return false;
  int R, bw, bh;
  conv_first_geometry(L, &R, &bw, &bh);
  return R >= 1 && bw <= 256 && bh <= 256 && (int64_t)bw * bh * L.cin * 4 <= CF_IN && L.Kp <= 64 && L.Kp >= 16 &&
         L.Kp % 8 == 0 && L.cout % 8 == 0 && L.cout >= 8 && L.cout <= 128;
}

hs_status conv_first_plan(hs_ctx* c, ConvFirstParams* p) {
  const ConvLayer& L = c->convs[0];
  const char* why = nullptr;
  std::memset(p, 0, sizeof(*p));
  p->npad = (L.cout + 15) / 16 * 16;
  p->acc_cols = p->npad <= 32 ? 32 : p->npad <= 64 ? 64 : 128;
  // the weights as a K-major [Cout][Kp] operand: one box of 64 columns x npad rows (zero fill past
  // Kp and Cout)
  if (!tc_make_kmajor_map(&p->tmW, TcOperand{c->d_wperm[0], L.cout, L.Kp, L.Kp}, p->npad, &why))
    return fail(c, HS_ERR_CUDA, why);
  p->C = L.cin;
  p->H = L.hin;
  p->W = L.win;
  p->Ho = L.hout;
  p->Wo = L.wout;
  p->stride = L.stride;
  p->Cout = L.cout;
  p->Kp = L.Kp;
  p->rows = L.rows;
  conv_first_geometry(L, &p->R, &p->box_w, &p->box_h);
  p->tpi = (L.hout + p->R - 1) / p->R;
  p->tiles = c->N * p->tpi;
  p->col = reinterpret_cast<__nv_bfloat16*>(c->d_col[0]);
  p->out = reinterpret_cast<__nv_bfloat16*>(c->d_cact[0]);
  p->st = c->d_status;
  p->x = nullptr;
  return HS_OK;
}

bool conv_first_bind_input(hs_ctx* c, const float* x) {
  ConvFirstParams& p = c->conv_first;
  if (p.x == x && x) return true;
  const char* why = nullptr;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) != 0 ||
      !tc_make_nchw_box_map(&p.tmX, x, c->N, p.C, p.H, p.W, p.box_w, p.box_h, &why)) {
    p.x = nullptr;
    return false;
  }
  p.x = x;
  return true;
}

namespace {
template <int KC>
cudaError_t launch_conv_first_kc(const ConvFirstParams& p, int grid, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(conv_first_fwd_kernel<KC>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCfSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_pdl(conv_first_fwd_kernel<KC>, dim3(grid), dim3(kCfThreads), (size_t)kCfSmem, s, p);
}
}  // namespace

cudaError_t launch_conv_first(const ConvFirstParams& p, int num_sms, cudaStream_t s) {
  int grid = p.tiles < num_sms ? p.tiles : num_sms;
  if (grid < 1) grid = 1;
  cudaError_t e;
  switch (p.Kp >> 3) {
    case 2: e = launch_conv_first_kc<2>(p, grid, s); break;
    case 3: e = launch_conv_first_kc<3>(p, grid, s); break;
    case 4: e = launch_conv_first_kc<4>(p, grid, s); break;
    case 5: e = launch_conv_first_kc<5>(p, grid, s); break;
    case 6: e = launch_conv_first_kc<6>(p, grid, s); break;
    case 7: e = launch_conv_first_kc<7>(p, grid, s); break;
    case 8: e = launch_conv_first_kc<8>(p, grid, s); break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace hs
