// Per-worker weight gradients averaged in tensor memory, with the SGD update applied in the epilogue.
//
// In the data-parallel step each worker m computes its layer weight gradient over its own rows,
// g^m = delta_m^T H_m (Eq. 1), and the exchange averages them, g = sum_m w_m g^m (Section 1: w_m =
// 1/M; Section 4.2: the normalised compute power), before theta <- theta - lr * g.  Here one SM pair
// owns a 256 x 256 tile of the layer's weight matrix and computes every worker's product for it in
// turn.  Worker m's k-blocks accumulate into one of two tensor-memory buffers, starting fresh at its
// first k-block, so the buffer holds g^m's tile exactly as the grouped per-worker launch stores it;
// while the tensor core runs worker m + 1 into the other buffer, the epilogue folds g^m into a
// running sum in registers, sum = fma(w_m, g^m, sum) from sum = 0, in worker order (the order of
// reduce_update_kernel).  After the last worker it applies theta = fma(-lr, sum, theta) and writes
// the bf16 copy of the new weights.  The per-worker gradients never leave the chip.
//
// Roles (320 threads per CTA, one CTA per SM, clusters of 2):
//   warp 0      (both CTAs) TMA loads of the CTA's A and B halves, completing on the leader's barrier
//   warp 1      (both CTAs) the collective allocation of all 512 tensor-memory columns (two 256-column
//               accumulators); in the leader CTA one thread issues the pair MMAs
//   warps 2..9  (both CTAs) epilogue: warp w reads tensor-memory lanes 32 * (w % 4).. (its row
//               quadrant) and columns 128 * ((w - 2) / 4).. of the buffer, 32 rows x 128 columns,
//               so each thread keeps 128 running sums; each warp reports the buffer free on the
//               leader's barrier, then updates its 32 x 128 block of theta through a 4 KB buffer
//               (fp32 boxes of 32 x 32 in, then out; bf16 boxes of 32 x 32 out)
// Every mbarrier wait is bounded (2 s of %globaltimer) and leaves through the error path.
#include <cudaTypedefs.h>

#include "tc_pair.cuh"

namespace hs {

namespace {

using namespace tcdev;
using namespace tcpair;

constexpr int kAvThreads = 320;
constexpr int kAvEpiWarps = 8;
constexpr int AV_PM = 256, AV_HM = 128;              // pair tile rows, per CTA
constexpr int AV_PN = 256, AV_HN = 128;              // pair tile columns, per CTA's B half / per epilogue warp
constexpr int AV_A_HALF = AV_HM * BK * 2;            // 16 KB
constexpr int AV_B_HALF = AV_HN * BK * 2;            // 16 KB
constexpr int AV_STAGE = AV_A_HALF + AV_B_HALF;      // 32 KB
constexpr int AV_S = 6;
constexpr uint32_t AV_TX = 2 * AV_STAGE;             // bytes landing per stage on the leader's barrier
constexpr uint32_t AV_TMEM_COLS = 2 * AV_PN;
constexpr int AV_BUF = 32 * 128;                     // per epilogue warp: one 32-row x 128-byte box
constexpr int kAvSmem = AV_S * AV_STAGE + kAvEpiWarps * AV_BUF + 1024 + 512;
static_assert(kAvSmem <= 232448, "shared memory budget");
constexpr int AV_GM = 8;                             // M-tiles per band of the tile order

__device__ __forceinline__ void tma_prefetch_l2_2d(const CUtensorMap* tm, int c0, int c1) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];"
               ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1)
               : "memory");
}
// No bulk group of this thread may still be reading shared memory.
__device__ __forceinline__ void bulk_wait_read_0() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// 32 lanes x 8 consecutive fp32 columns: thread t receives row (quadrant base + t).  (Narrow loads
// keep the 128 running sums of a thread in registers within the launch's 168.)
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait8(uint32_t (&r)[8]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7])
               :
               : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Tiles in bands of AV_GM M-tiles, walked N-tile by N-tile, so the pairs running at the same time
// share A and B panels in L2 (every pair streams all N rows of both for each tile).
__device__ __forceinline__ void av_decode(int t, int tiles_m, int tiles_n, int& tm, int& tn) {
  const int band = t / (AV_GM * tiles_n);
  const int within = t - band * AV_GM * tiles_n;
  const int rows = min(AV_GM, tiles_m - band * AV_GM);
  tm = band * AV_GM + within % rows;
  tn = within / rows;
}

// Lane 0 waits (bounded); the warp learns the outcome.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, int lane) {
  int ok = 1;
  if (lane == 0) ok = mbar_wait(bar, parity, abort_flag) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

// RECIPE: the update of the paper's experiments (Section 5): d = g + wd * theta, b = d (first step)
// or mu * b + d, theta <- theta - lr * b, with b read and written through tmM; theta, b and the
// bf16 copy then move in 16-column boxes (two fp32 boxes share the warp's 4 KB buffer).
template <bool RECIPE>
__global__ void __launch_bounds__(kAvThreads, 1) tc_wgrad_avg_pair_kernel(const __grid_constant__ TcGemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sBuf = smem + AV_S * AV_STAGE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sBuf + kAvEpiWarps * AV_BUF);
  uint64_t* full_bar = bars;                        // [AV_S] stage loaded (leader)
  uint64_t* empty_bar = bars + AV_S;                // [AV_S] stage consumed by the MMAs
  uint64_t* tfull_bar = bars + 2 * AV_S;            // [2] accumulator holds a finished group
  uint64_t* tempty_bar = bars + 2 * AV_S + 2;       // [2] accumulator drained (leader; 16 arrivals)
  uint64_t* tload_bar = bars + 2 * AV_S + 4;        // [8] theta box landed in epilogue warp e's buffer
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * AV_S + 4 + kAvEpiWarps);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // per group: k-blocks, MMA steps in the last one (a shared-memory copy: the producer and the
  // MMA issuer read it at every worker switch, where a parameter-space load would stall them)
  int2* kbinfo = reinterpret_cast<int2*>(bars + 32);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = (rank == 0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < AV_S; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&tfull_bar[b]), 1);
      mbar_init(smem_u32(&tempty_bar[b]), 2 * kAvEpiWarps);
    }
    for (int e = 0; e < kAvEpiWarps; ++e) mbar_init(smem_u32(&tload_bar[e]), 1);
    for (int g = 0; g < p.groups; ++g) kbinfo[g] = make_int2(p.num_kb[g], p.last_ksteps[g]);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), AV_TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dependency_wait();
  grid_dependents_launch();

  const int tiles_m = (p.Mdim + AV_PM - 1) / AV_PM;
  const int tiles_n = (p.n_store + AV_PN - 1) / AV_PN;
  const int total = tiles_m * tiles_n;
  const int G = p.groups;
  const int pair_id = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer (both CTAs)
      for (int g = 0; g < G; ++g) {
        tma_prefetch_desc(&p.tmA[g]);
        tma_prefetch_desc(&p.tmB[g]);
      }
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int t = pair_id; t < total && ok && !*abort_flag && !p.test_stall; t += n_pairs) {
        int tm, tn;
        av_decode(t, tiles_m, tiles_n, tm, tn);
        const int m0 = tm * AV_PM + (int)rank * AV_HM;
        const int n0 = tn * AV_PN + (int)rank * AV_HN;
        for (int g = 0; g < G && ok; ++g) {
          const CUtensorMap* ta = &p.tmA[g];
          const CUtensorMap* tb = &p.tmB[g];
          const int nkb = kbinfo[g].x;
          // the next worker's descriptors, ahead of its first load
          const int gn = g + 1 < G ? g + 1 : 0;
          tma_prefetch_desc(&p.tmA[gn]);
          tma_prefetch_desc(&p.tmB[gn]);
          for (int kb = 0; kb < nkb; ++kb) {
            if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, abort_flag)) { ok = false; break; }
            const uint32_t fb_local = smem_u32(&full_bar[s]);
            const uint32_t fb = map_to_rank(fb_local, 0);
            if (leader) mbar_expect_tx(fb_local, AV_TX);
            const int k0 = kb * BK;
            const uint32_t a_dst = smem_u32(smem + s * AV_STAGE);
            const uint32_t b_dst = a_dst + AV_A_HALF;
#pragma unroll
            for (int j = 0; j < AV_HM / 64; ++j) tma_load_2d_pair(a_dst + j * MN_CHUNK, ta, m0 + 64 * j, k0, fb);
#pragma unroll
            for (int j = 0; j < AV_HN / 64; ++j) tma_load_2d_pair(b_dst + j * MN_CHUNK, tb, n0 + 64 * j, k0, fb);
            if (++s == AV_S) { s = 0; ph ^= 1u; }
          }
        }
      }
      if (!ok) {
        record_error(p.st, kDevWaitTimeout, 21);
        *abort_flag = 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------------------ pair MMA issuer (leader)
      constexpr uint32_t idesc = make_idesc(true, true, AV_PM, AV_PN);
      constexpr uint64_t kStageDesc = AV_STAGE >> 4;   // one stage, in the descriptor's address field
      const uint64_t a_desc0 = make_sdesc(smem_u32(smem), MN_CHUNK, 1024);
      const uint64_t b_desc0 = make_sdesc(smem_u32(smem) + AV_A_HALF, MN_CHUNK, 1024);
      int s = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int t = pair_id; t < total && ok && !*abort_flag; t += n_pairs) {
        for (int g = 0; g < G; ++g) {
          if (!mbar_wait(smem_u32(&tempty_bar[ab]), aph ^ 1u, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)(ab * AV_PN);
          // full k-blocks, then the worker's partial last k-block
          const int2 ki = kbinfo[g];
          const int nkb = ki.x;
          LastKb lk;
          lk.kb_last = ki.y > 0 ? nkb - 1 : -1;
          lk.steps = ki.y;
          const int kb_full = lk.kb_last >= 0 ? lk.kb_last : nkb;
          int kb = 0;
          for (; kb < kb_full; ++kb) {
            if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) { ok = false; break; }
            tc_fence_after();
            const uint64_t off = kStageDesc * (uint64_t)s;
            mma_kblock_pair<true, true>(d_tmem, a_desc0 + off, b_desc0 + off, idesc, kb != 0 ? 1u : 0u);
            umma_commit_pair(smem_u32(&empty_bar[s]));
            if (++s == AV_S) { s = 0; ph ^= 1u; }
          }
          if (ok && kb < nkb) {
            if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) {
              ok = false;
            } else {
              tc_fence_after();
              const uint64_t off = kStageDesc * (uint64_t)s;
              mma_ksteps_pair<true, true>(d_tmem, a_desc0 + off, b_desc0 + off, idesc, kb != 0 ? 1u : 0u, lk.steps);
              umma_commit_pair(smem_u32(&empty_bar[s]));
              if (++s == AV_S) { s = 0; ph ^= 1u; }
            }
          }
          if (!ok) break;
          umma_commit_pair(smem_u32(&tfull_bar[ab]));
          if (++ab == 2) { ab = 0; aph ^= 1u; }
        }
      }
      if (!ok) {
        record_error(p.st, kDevWaitTimeout, 22);
        *abort_flag = 1;
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue (warps 2..9, both CTAs)
    const int e = warp - 2;
    const int q = warp & 3;
    const int h = e >> 2;
    const uint32_t buf = smem_u32(sBuf) + (uint32_t)(e * AV_BUF);
    const uint32_t rbase = buf + (uint32_t)(lane * 128);
    const uint32_t tbar = smem_u32(&tload_bar[e]);
    const float neg_lr = -(p.lr_dev ? *p.lr_dev : p.lr);
    int ab = 0;
    uint32_t aph = 0, tph = 0;
    bool ok = true;
#pragma unroll 1
    for (int t = pair_id; t < total && ok; t += n_pairs) {
      int tm, tn;
      av_decode(t, tiles_m, tiles_n, tm, tn);
      const int row0 = tm * AV_PM + (int)rank * AV_HM + q * 32;
      const int col0 = tn * AV_PN + h * AV_HN;
      const bool rows_live = row0 < p.Mdim;
      float sum[AV_HN];
#pragma unroll
      for (int i = 0; i < AV_HN; ++i) sum[i] = 0.f;
#pragma unroll 1
      for (int g = 0; g < G; ++g) {
        if (g == G - 1 && lane == 0 && rows_live) {
          // theta's block (and the momentum's) into L2 while the last group runs
          constexpr int kBox = RECIPE ? 16 : 32;
#pragma unroll
          for (int u = 0; u < AV_HN / kBox; ++u) {
            if (col0 + kBox * u >= p.n_store) break;
            tma_prefetch_l2_2d(&p.tmT, col0 + kBox * u, row0);
            if (RECIPE && !p.first) tma_prefetch_l2_2d(&p.tmM, col0 + kBox * u, row0);
          }
        }
        if (!warp_wait(smem_u32(&tfull_bar[ab]), aph, abort_flag, lane)) {
          if (lane == 0) {
            record_error(p.st, kDevWaitTimeout, 23);
            *abort_flag = 1;
          }
          ok = false;
          break;
        }
        tc_fence_after();
        const float wg = __ldg(p.wavg + g);
        const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * AV_PN + h * AV_HN);
#pragma unroll
        for (int u = 0; u < AV_HN / 8; ++u) {
          uint32_t r[8];
          tmem_ld8(taddr + (uint32_t)(u * 8), r);
          tmem_ld_wait8(r);
#pragma unroll
          for (int j = 0; j < 8; ++j) sum[u * 8 + j] = fmaf(wg, __uint_as_float(r[j]), sum[u * 8 + j]);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(map_to_rank(smem_u32(&tempty_bar[ab]), 0));
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
      if (!ok || !rows_live) continue;
      if (RECIPE) {
        // d = sum + wd * theta, b = d or mu * b + d, theta <- theta - lr * b: 16 columns at a time,
        // theta's 32 x 16 box at buf, the momentum's at buf + 2 KB (64-byte rows, no swizzle), then
        // the bf16 copy (32-byte rows) through the same buffer
        const float mu = p.mu, wd = p.wd;
        const bool first = p.first != 0;
#pragma unroll
        for (int u = 0; u < AV_HN / 16; ++u) {
          const int n_base = col0 + 16 * u;
          if (n_base >= p.n_store) break;
          if (lane == 0) {
            bulk_wait_read_0();
            mbar_expect_tx(tbar, first ? AV_BUF / 2 : AV_BUF);
            tma_load_2d(buf, &p.tmT, n_base, row0, tbar);
            if (!first) tma_load_2d(buf + AV_BUF / 2, &p.tmM, n_base, row0, tbar);
          }
          if (!warp_wait(tbar, tph, abort_flag, lane)) {
            if (lane == 0) {
              record_error(p.st, kDevWaitTimeout, 25);
              *abort_flag = 1;
            }
            ok = false;
            break;
          }
          tph ^= 1u;
          const uint32_t ta = buf + (uint32_t)(lane * 64);
          const uint32_t ma = ta + AV_BUF / 2;
          uint32_t sh[8];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 tv = ld_shared_v4(ta + 16u * j);
            const uint4 bv = first ? make_uint4(0u, 0u, 0u, 0u) : ld_shared_v4(ma + 16u * j);
            const float tin[4] = {__uint_as_float(tv.x), __uint_as_float(tv.y), __uint_as_float(tv.z),
                                  __uint_as_float(tv.w)};
            const float bin[4] = {__uint_as_float(bv.x), __uint_as_float(bv.y), __uint_as_float(bv.z),
                                  __uint_as_float(bv.w)};
            float tout[4], bout[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float d = fmaf(wd, tin[k], sum[u * 16 + 4 * j + k]);
              bout[k] = first ? d : fmaf(mu, bin[k], d);
              tout[k] = fmaf(neg_lr, bout[k], tin[k]);
            }
            st_shared_v4(ta + 16u * j, make_uint4(__float_as_uint(tout[0]), __float_as_uint(tout[1]),
                                                  __float_as_uint(tout[2]), __float_as_uint(tout[3])));
            st_shared_v4(ma + 16u * j, make_uint4(__float_as_uint(bout[0]), __float_as_uint(bout[1]),
                                                  __float_as_uint(bout[2]), __float_as_uint(bout[3])));
            sh[2 * j] = pack_bf16(tout[0], tout[1]);
            sh[2 * j + 1] = pack_bf16(tout[2], tout[3]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&p.tmT, buf, n_base, row0);
            tma_store_2d(&p.tmM, buf + AV_BUF / 2, n_base, row0);
            bulk_commit();
            bulk_wait_read_0();
          }
          __syncwarp();
          const uint32_t sbase = buf + (uint32_t)(lane * 32);
          st_shared_v4(sbase, make_uint4(sh[0], sh[1], sh[2], sh[3]));
          st_shared_v4(sbase + 16u, make_uint4(sh[4], sh[5], sh[6], sh[7]));
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&p.tmS, buf, n_base, row0);
            bulk_commit();
          }
        }
        continue;
      }
      // theta <- fma(-lr, sum, theta), 32 columns at a time through the warp's buffer (128-byte
      // swizzle: 16-byte chunk j of row r sits at chunk j ^ (r % 8)), then the same 32 columns of
      // the bf16 copy (64-byte rows, no swizzle).
#pragma unroll
      for (int u = 0; u < AV_HN / 32; ++u) {
        const int n_base = col0 + 32 * u;
        if (n_base >= p.n_store) break;
        if (lane == 0) {
          bulk_wait_read_0();
          mbar_expect_tx(tbar, AV_BUF);
          tma_load_2d(buf, &p.tmT, n_base, row0, tbar);
        }
        if (!warp_wait(tbar, tph, abort_flag, lane)) {
          if (lane == 0) {
            record_error(p.st, kDevWaitTimeout, 24);
            *abort_flag = 1;
          }
          ok = false;
          break;
        }
        tph ^= 1u;
        uint32_t sh[16];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint32_t a = rbase + (uint32_t)((j ^ (lane & 7)) << 4);
          const uint4 v = ld_shared_v4(a);
          const float t0 = fmaf(neg_lr, sum[u * 32 + 4 * j], __uint_as_float(v.x));
          const float t1 = fmaf(neg_lr, sum[u * 32 + 4 * j + 1], __uint_as_float(v.y));
          const float t2 = fmaf(neg_lr, sum[u * 32 + 4 * j + 2], __uint_as_float(v.z));
          const float t3 = fmaf(neg_lr, sum[u * 32 + 4 * j + 3], __uint_as_float(v.w));
          st_shared_v4(a, make_uint4(__float_as_uint(t0), __float_as_uint(t1), __float_as_uint(t2), __float_as_uint(t3)));
          sh[2 * j] = pack_bf16(t0, t1);
          sh[2 * j + 1] = pack_bf16(t2, t3);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&p.tmT, buf, n_base, row0);
          bulk_commit();
          bulk_wait_read_0();
        }
        __syncwarp();
        const uint32_t sbase = buf + (uint32_t)(lane * 64);
#pragma unroll
        for (int j = 0; j < 4; ++j) st_shared_v4(sbase + (uint32_t)(j * 16), make_uint4(sh[4 * j], sh[4 * j + 1], sh[4 * j + 2], sh[4 * j + 3]));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&p.tmS, buf, n_base, row0);
          bulk_commit();
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    const uint64_t t0 = globaltimer();
    while (globaltimer() - t0 < 2000000ull) {
    }
  }
  // Neither CTA may leave while the pair's MMAs, multicast commits or remote arrivals can still
  // touch its shared memory or tensor memory.
  cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, AV_TMEM_COLS);
  }
}

}  // namespace

namespace {
template <bool RECIPE>
cudaError_t launch_avg_variant(const TcGemmParams& p, int total, int num_sms, cudaStream_t s) {
  static bool configured = false;
  static int max_clusters = 0;
  auto kern = tc_wgrad_avg_pair_kernel<RECIPE>;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see grid_dependency_wait
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(kAvThreads, 1, 1);
  cfg.dynamicSmemBytes = kAvSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;   // the occupancy query takes the cluster shape only
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kAvSmem);
    if (e != cudaSuccess) return e;
    cfg.gridDim = dim3(num_sms & ~1, 1, 1);
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
    if (e != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    max_clusters = n;
    configured = true;
  }
  const int pairs = total < max_clusters ? total : max_clusters;
  cfg.gridDim = dim3(2 * (pairs < 1 ? 1 : pairs), 1, 1);
  cfg.numAttrs = 2;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_tc_wgrad_avg(const TcGemmParams& p, int num_sms, cudaStream_t s) {
  if (p.groups < 1 || p.groups > kTcMaxGroups || !p.a_mn || !p.b_mn || !p.wavg) return cudaErrorInvalidValue;
  for (int g = 0; g < p.groups; ++g)
    if (p.num_kb[g] < 1) return cudaErrorInvalidValue;
  const int total = ((p.Mdim + AV_PM - 1) / AV_PM) * ((p.n_store + AV_PN - 1) / AV_PN);
  if (total <= 0) return cudaSuccess;
  return p.recipe ? launch_avg_variant<true>(p, total, num_sms, s) : launch_avg_variant<false>(p, total, num_sms, s);
}

}  // namespace hs
