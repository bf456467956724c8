// SM-pair form of the tensor-core GEMM: a cluster of two CTAs computes one 256 x 256 output tile
// with tcgen05.mma.cta_group::2.  Each CTA of the pair stages 128 rows of A and half of B (128 of
// the 256 N columns) per k-block, so each SM reads 8 KB of operands from shared memory per
// 128-cycle MMA instead of the 12 KB of the one-SM 128 x 256 form; the freed shared-memory
// bandwidth is what the fp32 weight-gradient epilogue needs.  Same products and epilogues as
// gemm_tc.cu (forward, input gradient, per-worker grouped weight gradient of Eq. 1's g^m).
//
// Roles (64 + 32 x epilogue warps threads per CTA, one more warp for convolution products; one
// CTA per SM, clusters of 2):
//   warp 0      (both CTAs) TMA loads of the CTA's A and B halves; completion is signalled on the
//               leader CTA's stage barrier (the .cta_group::2 form of the bulk tensor copy); for
//               convolution products the warp after the epilogue warps issues every other box
//   warp 1      (both CTAs) the collective tensor-memory allocation; in the leader CTA one thread
//               issues the pair MMAs and commits them to both CTAs' barriers (multicast)
//   warps 2..5  (both CTAs) epilogue of the CTA's 128 accumulator rows; each warp reports the
//               accumulator free on the leader's barrier
// Every mbarrier wait is bounded as in the one-SM kernel.
#include <cudaTypedefs.h>

#include <cstdlib>

#include "tc_pair.cuh"

namespace hs {

namespace {

using namespace tcdev;
using namespace tcpair;

constexpr int PM = 256;                            // pair tile rows
constexpr int HM = PM / 2;                         // per-CTA half
constexpr int A_HALF = HM * BK * 2;                // 16 KB
// Pair tile of 256 x TN (TN = 256, or 128 for products at most 128 wide): per-CTA B half, stages
// (more of them when the B half is smaller), two TN-column accumulators in tensor memory.  EW
// epilogue warps: 4, or 8 for short-K products whose epilogue outlasts the main loop.  With
// 256-wide tiles the eight are two per tensor-memory lane quadrant, each on half of the tile's
// columns; with 128-wide tiles (kAlt) they are two groups of four, each draining every other tile
// (one accumulator buffer each), so two tiles' epilogues run at once even where the product is
// only 64 wide.  Eight epilogue warps cost stages to fit their staging buffers.
// KS k-blocks per pipeline stage: one barrier round trip (the producer's wait, expected-bytes
// arrive and box issues; the MMA issuer's wait and commit, each a few hundred cycles on one
// thread) then feeds KS k-blocks of MMAs.  A 256 x 128 tile's k-block is about 0.17 us of MMA,
// less than one round trip, so those products take KS = 2 (the same slots, paired).
template <int TN, int EW, int NP = 1, int KS = 1>
struct PairCfg {
  static constexpr int PN = TN;
  static constexpr int HN = TN / 2;
  static constexpr int B_HALF = HN * BK * 2;
  static constexpr int STAGE2 = A_HALF + B_HALF;
  static constexpr bool kAlt = (TN == 128 && EW == 8);
  static constexpr int S2 = TN == 256 ? (EW == 8 ? (KS == 2 ? 4 : 5) : 6) : (EW == 8 ? 6 : 8);   // slots
  static constexpr int kThreads = 64 + 32 * EW + 32 * (NP - 1);   // NP TMA producer warps
  static constexpr uint32_t PAIR_TX = 2 * STAGE2;   // bytes landing per stage on the leader's barrier
  static constexpr uint32_t kTmemCols2 = 2 * TN;
  static constexpr int kStaging = EW * 8192;         // two 32-row x 128-byte buffers per epilogue warp
  static constexpr int kSmem2 = S2 * STAGE2 + kStaging + 1024 + 256;
  // arrivals that free one accumulator buffer: the epilogue warps of both CTAs that drain it
  static constexpr uint32_t kFreeArrivals = 2 * (kAlt ? 4 : EW);
  static constexpr int NB = S2 / KS;                 // pipeline stages (barrier pairs) of KS slots each
  static_assert(kSmem2 <= 232448, "shared memory budget");
  static_assert(EW == 4 || EW == 8, "epilogue warps");
  static_assert((KS == 1 || KS == 2) && S2 % KS == 0, "k-blocks per stage");
};

// Convolution products keep two TMA producer warps busy: their operands come in 8 KB 4-D boxes
// (one output-pixel block of one tap each) whose issue, one thread at a time, took longer than the
// k-block's MMAs.  The producers split each k-block's boxes round-robin.
constexpr int kConvProducers = 2;

template <int EPI, bool A_MN, bool B_MN, bool CONV, int TN, int EW, int KS>
__global__ void __launch_bounds__(PairCfg<TN, EW, CONV ? kConvProducers : 1, KS>::kThreads, 1)
    tc_gemm_pair_kernel(const __grid_constant__ TcGemmParams p) {
  constexpr int NP = CONV ? kConvProducers : 1;
  using Cfg = PairCfg<TN, EW, NP, KS>;
  constexpr int PN = Cfg::PN, HN = Cfg::HN, S2 = Cfg::S2, STAGE2 = Cfg::STAGE2, NB = Cfg::NB;
  constexpr uint32_t PAIR_TX = Cfg::PAIR_TX, kTmemCols2 = Cfg::kTmemCols2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sStage = smem + S2 * STAGE2;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStage + Cfg::kStaging);
  uint64_t* full_bar = bars;
  uint64_t* empty_bar = bars + S2;
  uint64_t* tfull_bar = bars + 2 * S2;
  uint64_t* tempty_bar = bars + 2 * S2 + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S2 + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = (rank == 0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < NB; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&tfull_bar[b]), 1);
      mbar_init(smem_u32(&tempty_bar[b]), Cfg::kFreeArrivals);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), kTmemCols2);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dependency_wait();
  grid_dependents_launch();

  const int tiles_m = (p.Mdim + PM - 1) / PM;
  const int tiles_n = (p.n_store + PN - 1) / PN;
  const int total = p.groups * ksplit_of(p) * tiles_m * tiles_n;
  const int pair_id = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;

  // TMA producer warps: warp 0 and, for convolution products, the warps after the epilogue's
  const int prod = (warp == 0) ? 0 : (NP > 1 && warp >= 2 + EW) ? warp - (2 + EW) + 1 : -1;
  if (prod >= 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producers (both CTAs)
      // A k-block's boxes, A half then B half, numbered in order; producer `prod` issues those whose
      // number is prod mod NP (producer 0 also sets the leader's expected bytes).
      int s = 0;
      uint32_t ph = 0;
      int last_g = -1;
      for (int t = pair_id; t < total && !*abort_flag && !p.test_stall; t += n_pairs) {
        const TileWork w = tile_work(p, t, tiles_m, tiles_n);
        const TileCoord c = w.c;
        const CUtensorMap* ta = &p.tmA[w.g];
        const CUtensorMap* tb = &p.tmB[w.g];
        if (w.g != last_g) {
          tma_prefetch_desc(ta);
          tma_prefetch_desc(tb);
          last_g = w.g;
        }
        const int m0 = c.tm * PM + (int)rank * HM;
        const int n0 = c.tn * PN + (int)rank * HN;
        // implicit patch rows: the output-pixel part of the A boxes once per tile, the patch-column
        // part of the B boxes once per tile
        ConvRowPart arow[HM / 64];
        ConvColPart bcol[HN / 64];
        if (CONV && p.conv_a) {
#pragma unroll
          for (int j = 0; j < HM / 64; ++j)
            arow[j] = p.conv_a == 2 ? subpixel_row_part(p.conv, m0 + 64 * j) : conv_row_part(p.conv, m0 + 64 * j);
        }
        if (CONV && B_MN && p.conv_b) {
#pragma unroll
          for (int j = 0; j < HN / 64; ++j)
            if (n0 + 64 * j < p.conv.ones_col) bcol[j] = conv_col_part(p.conv, n0 + 64 * j);
        }
        // patch-column blocks of A and pixel blocks of B, stepped once per k-block
        ConvColIter a_it;
        ConvRowIter b_it;
        if (CONV && p.conv_a)
          a_it.init(p.conv, p.conv_a == 2 ? (p.conv.a_cls >= 0 ? p.conv.a_cls : w.g) : -1, w.kb_lo * BK);
        if (CONV && B_MN && p.conv_b) b_it.init(p.conv, w.kb_lo * BK);
        bool ok = true;
        for (int kb = w.kb_lo; kb < w.kb_hi; kb += KS) {
          // the stage's k-blocks: KS, or one where the tile's k-block count is odd
          const int nk = (KS == 1 || kb + 1 >= w.kb_hi) ? 1 : KS;
          if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t fb_local = smem_u32(&full_bar[s]);
          const uint32_t fb = map_to_rank(fb_local, 0);
          if (prod == 0 && leader) mbar_expect_tx(fb_local, PAIR_TX * (uint32_t)nk);
          int box = 0;
#pragma unroll
          for (int js = 0; js < KS; ++js) {
          if (js >= nk) break;
          const int k0 = (kb + js) * BK;
          const uint32_t a_dst = smem_u32(smem + (s * KS + js) * STAGE2);
          const uint32_t b_dst = a_dst + A_HALF;
          // the A half: two 64-column boxes (MN-major), two 64-pixel boxes (implicit patch rows) or
          // one 128-row box (K-major)
          if (A_MN) {
#pragma unroll
            for (int j = 0; j < HM / 64; ++j)
              if (box++ % NP == prod) tma_load_2d_pair(a_dst + j * MN_CHUNK, ta, m0 + 64 * j, k0, fb);
          } else if (CONV && p.conv_a) {
            const ConvColPart kc = a_it.part();
            if (p.conv.a_box == HM) {
              // one box of the half's 128 output pixels (lands as the two 64-row boxes would)
              if (box++ % NP == prod) {
                int cc[4];
                conv_coords(arow[0], kc, cc);
                tma_load_4d_pair(a_dst, ta, cc, fb);
              }
            } else {
#pragma unroll
              for (int j = 0; j < HM / 64; ++j)
                if (box++ % NP == prod) {
                  int cc[4];
                  conv_coords(arow[j], kc, cc);
                  tma_load_4d_pair(a_dst + j * MN_CHUNK, ta, cc, fb);
                }
            }
          } else {
            if (box++ % NP == prod) tma_load_2d_pair(a_dst, ta, k0, m0, fb);
          }
          if (B_MN) {
            ConvRowPart krow;
            if (CONV && p.conv_b) krow = b_it.part();
#pragma unroll
            for (int j = 0; j < HN / 64; ++j) {
              if (box++ % NP != prod) continue;
              const int col = n0 + 64 * j;
              if (!CONV || !p.conv_b) {
                tma_load_2d_pair(b_dst + j * MN_CHUNK, tb, col, k0, fb);
              } else if (col < p.conv.ones_col) {
                int cc[4];
                conv_coords(krow, bcol[j], cc);
                tma_load_4d_pair(b_dst + j * MN_CHUNK, tb, cc, fb);
              } else {
                tma_load_2d_pair(b_dst + j * MN_CHUNK, &p.tmOnes, col - p.conv.ones_col, 0, fb);
              }
            }
          } else {
            if (box++ % NP == prod) tma_load_2d_pair(b_dst, tb, k0, n0, fb);
          }
          if (CONV && p.conv_a) a_it.next();
          if (CONV && B_MN && p.conv_b) b_it.next();
          }
          if (++s == NB) { s = 0; ph ^= 1u; }
        }
        if (!ok) {
          record_error(p.st, kDevWaitTimeout, 11);
          *abort_flag = 1;
          break;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------------------ pair MMA issuer (leader)
      constexpr uint32_t idesc = make_idesc(A_MN, B_MN, PM, PN);
      constexpr uint64_t kStageDesc = STAGE2 >> 4;   // one slot, in the descriptor's address field
      const uint64_t a_desc0 = make_sdesc(smem_u32(smem), A_MN ? MN_CHUNK : 16, 1024);
      const uint64_t b_desc0 = make_sdesc(smem_u32(smem) + A_HALF, B_MN ? MN_CHUNK : 16, 1024);
      int s = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      for (int t = pair_id; t < total && !*abort_flag; t += n_pairs) {
        const TileWork w = tile_work(p, t, tiles_m, tiles_n);
        if (!mbar_wait(smem_u32(&tempty_bar[ab]), aph ^ 1u, abort_flag)) {
          record_error(p.st, kDevWaitTimeout, 12);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * PN);
        bool ok = true;
        // stages of KS full k-blocks; the group's partial last k-block (the tile's last, when the
        // tile holds it) takes only its steps that hold rows
        const LastKb lk = last_kb_of(p, w.g);
        const bool tail = lk.kb_last >= w.kb_lo && lk.kb_last < w.kb_hi;
        for (int kb = w.kb_lo; kb < w.kb_hi; kb += KS) {
          const int nk = (KS == 1 || kb + 1 >= w.kb_hi) ? 1 : KS;
          if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint64_t off = kStageDesc * (uint64_t)(s * KS);
          if (nk == KS && !(tail && kb + KS == w.kb_hi)) {
            mma_kblock_pair<A_MN, B_MN>(d_tmem, a_desc0 + off, b_desc0 + off, idesc, kb != w.kb_lo ? 1u : 0u);
            if (KS == 2) mma_kblock_pair<A_MN, B_MN>(d_tmem, a_desc0 + off + kStageDesc, b_desc0 + off + kStageDesc, idesc, 1u);
          } else {
            // the stage ends the tile: its k-blocks before the last are full, the last may be partial
            if (KS == 2 && nk == 2)
              mma_kblock_pair<A_MN, B_MN>(d_tmem, a_desc0 + off, b_desc0 + off, idesc, kb != w.kb_lo ? 1u : 0u);
            const uint64_t o2 = off + kStageDesc * (uint64_t)(nk - 1);
            const uint32_t acc = (kb + nk - 1) != w.kb_lo ? 1u : 0u;
            if (tail)
              mma_ksteps_pair<A_MN, B_MN>(d_tmem, a_desc0 + o2, b_desc0 + o2, idesc, acc, lk.steps);
            else
              mma_kblock_pair<A_MN, B_MN>(d_tmem, a_desc0 + o2, b_desc0 + o2, idesc, acc);
          }
          umma_commit_pair(smem_u32(&empty_bar[s]));
          if (++s == NB) { s = 0; ph ^= 1u; }
        }
        if (!ok) {
          record_error(p.st, kDevWaitTimeout, 13);
          *abort_flag = 1;
          break;
        }
        umma_commit_pair(smem_u32(&tfull_bar[ab]));
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue (warps 2..5, both CTAs)
    constexpr bool kF32Out = (EPI == kTcEpiBiasF32 || EPI == kTcEpiStoreF32);
    constexpr bool kAlt = Cfg::kAlt;
    constexpr int kUnitCols = kF32Out ? 32 : 64;
    constexpr int kUnits = kAlt ? PN / kUnitCols : PN / kUnitCols / (EW / 4);   // units of this warp's share
    const int q = warp & 3;
    const int second = (warp - 2) >> 2;                // 0, or 1 for the second warp of a quadrant
    const int col_share = kAlt ? 0 : second;           // 256-wide tiles: the second warp takes half the columns
    const uint32_t stage_base = smem_u32(sStage) + (uint32_t)((warp - 2) * 8192);
    int sb = 0;
    // kAlt: the MMA issuer fills buffer i % 2 for its i-th tile; group `second` drains buffer
    // `second`, i.e. every other tile starting at the group's first
    int ab = kAlt ? second : 0;
    uint32_t aph = 0;
    const int t_first = pair_id + (kAlt ? second * n_pairs : 0);
    const int t_step = kAlt ? 2 * n_pairs : n_pairs;
    for (int t = t_first; t < total; t += t_step) {
      const TileWork w = tile_work(p, t, tiles_m, tiles_n);
      const TileCoord c = w.c;
      uint4 zq[8];   // mask operand of the tile's first unit, loaded before the accumulator is ready
      const int n_warp = c.tn * PN + col_share * kUnits * kUnitCols;   // this warp's first column
      if (EPI == kTcEpiMaskBf16) load_mask_unit<CONV>(p, w.g, c.tm * PM + (int)rank * HM + q * 32 + lane, n_warp, zq);
      int ok = 1;
      if (lane == 0) ok = mbar_wait(smem_u32(&tfull_bar[ab]), aph, abort_flag) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          record_error(p.st, kDevWaitTimeout, 14);
          *abort_flag = 1;
        }
        break;
      }
      __syncwarp();
      tc_fence_after();
      const int row0 = c.tm * PM + (int)rank * HM + q * 32;
      const int row = row0 + lane;
      const CUtensorMap* td = &p.tmD[w.g];
      const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) +
                             (uint32_t)(ab * PN + col_share * kUnits * kUnitCols);
#pragma unroll 1
      for (int u = 0; u < kUnits; ++u) {
        const int n_base = n_warp + u * kUnitCols;
        if (n_base >= p.n_store) break;
        uint32_t r[32], r2[32];
        tmem_ld32(t_row + (uint32_t)(u * kUnitCols), r);
        if (!kF32Out) tmem_ld32(t_row + (uint32_t)(u * kUnitCols + 32), r2);
        tmem_ld_wait(r);
        if (!kF32Out) tmem_ld_wait(r2);
        uint4 o[8];
        epilogue_unit<EPI, CONV>(p, w.g, row, n_base, r, r2, zq, o);
        if (EPI == kTcEpiMaskBf16 && u + 1 < kUnits)   // the next unit's mask, behind this unit's stores
          load_mask_unit<CONV>(p, w.g, row, n_base + kUnitCols, zq);
        if (lane == 0) bulk_wait_read_1();
        __syncwarp();
        const uint32_t buf = stage_base + (uint32_t)(sb * 4096);
        const uint32_t rbase = buf + (uint32_t)(lane * 128);
#pragma unroll
        for (int j = 0; j < 8; ++j) st_shared_v4(rbase + (uint32_t)(((j ^ (lane & 7)) << 4)), o[j]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          store_strip<CONV>(p, td, buf, n_base, row0, w.part);
          bulk_commit();
        }
        sb ^= 1;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(map_to_rank(smem_u32(&tempty_bar[ab]), 0));
      if (kAlt) {
        aph ^= 1u;
      } else if (++ab == 2) {
        ab = 0;
        aph ^= 1u;
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
    tmem_dealloc_pair(tmem_base, kTmemCols2);
  }
}

template <int EPI, bool A_MN, bool B_MN, bool CONV, int TN = 256, int EW = 4, int KS = 1>
cudaError_t launch_pair_variant1(const TcGemmParams& p, int pairs_wanted, int num_sms, cudaStream_t s) {
  static bool configured = false;
  static int max_clusters = 0;
  using Cfg = PairCfg<TN, EW, CONV ? kConvProducers : 1, KS>;
  constexpr int kSmem2 = Cfg::kSmem2;
  auto kern = tc_gemm_pair_kernel<EPI, A_MN, B_MN, CONV, TN, EW, KS>;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see grid_dependency_wait
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(Cfg::kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmem2;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;   // the occupancy query takes the cluster shape only
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem2);
    if (e != cudaSuccess) return e;
    // Persistent grid: no more clusters than can be resident at once (SMs pair up within a GPC).
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
  int pairs = pairs_wanted < max_clusters ? pairs_wanted : max_clusters;
  if (pairs < 1) pairs = 1;
  const int grid = 2 * pairs;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.numAttrs = 2;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Two k-blocks per stage where a k-block's MMAs are shorter than, or about as long as, a barrier
// round trip: the 256 x 128 tiles, every convolution product (whose producers also form box
// coordinates) and the forward products (bias + ReLU, logits); measured, the 256 x 256 input- and
// weight-gradient products gained nothing.  HS_KSTAGE=1 keeps one, HS_KSTAGE=2 takes two
// everywhere (the same MMAs in the same order: identical results).
inline bool pair_two_kblocks(int tn, bool conv, int epi) {
  const char* v = getenv("HS_KSTAGE");   // read per launch: a step replayed from a graph launches nothing
  const int forced = v ? atoi(v) : 0;
  if (forced == 1) return false;
  if (forced == 2) return true;
  return tn == 128 || conv || epi == kTcEpiBiasReluBf16 || epi == kTcEpiBiasF32;
}

template <int EPI, bool A_MN, bool B_MN, bool CONV, int TN = 256, int EW = 4>
cudaError_t launch_pair_variant(const TcGemmParams& p, int pairs_wanted, int num_sms, cudaStream_t s) {
  if (pair_two_kblocks(TN, CONV, EPI)) return launch_pair_variant1<EPI, A_MN, B_MN, CONV, TN, EW, 2>(p, pairs_wanted, num_sms, s);
  return launch_pair_variant1<EPI, A_MN, B_MN, CONV, TN, EW, 1>(p, pairs_wanted, num_sms, s);
}

}  // namespace

cudaError_t launch_tc_gemm_pair(const TcGemmParams& p, int num_sms, cudaStream_t s) {
  const int tn = p.pn == 128 ? 128 : 256;
  const int tiles_m = (p.Mdim + PM - 1) / PM;
  const int tiles_n = (p.n_store + tn - 1) / tn;
  const int total = p.groups * (p.ksplit > 1 ? p.ksplit : 1) * tiles_m * tiles_n;
  if (total <= 0) return cudaSuccess;
  const int pairs = total;
  const int grid = num_sms;   // forwarded as the SM count for the residency query
  if (tn == 128) {
    // 256 x 128 tiles (K-major B maps with 64-row boxes): the narrow products of the convolutions,
    // with four epilogue warps or two groups of four on alternate tiles
    if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) {
      if (p.ew == 8)
        return (p.conv_a ? launch_pair_variant<kTcEpiBiasReluBf16, false, false, true, 128, 8>
                         : launch_pair_variant<kTcEpiBiasReluBf16, false, false, false, 128, 8>)(p, pairs, grid, s);
      return (p.conv_a ? launch_pair_variant<kTcEpiBiasReluBf16, false, false, true, 128>
                       : launch_pair_variant<kTcEpiBiasReluBf16, false, false, false, 128>)(p, pairs, grid, s);
    }
    if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn && (p.conv_a || p.conv_d))
      return p.ew == 8 ? launch_pair_variant<kTcEpiMaskBf16, false, true, true, 128, 8>(p, pairs, grid, s)
                       : launch_pair_variant<kTcEpiMaskBf16, false, true, true, 128>(p, pairs, grid, s);
    return cudaErrorInvalidValue;
  }
  // implicit convolution operands (forward, weight gradient, sub-pixel input gradient)
  if (p.conv_a || p.conv_b || p.conv_d) {
    if (p.ew == 8 && p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn)   // the one-product sub-pixel input gradient
      return launch_pair_variant<kTcEpiMaskBf16, false, true, true, 256, 8>(p, pairs, grid, s);
    if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) return launch_pair_variant<kTcEpiBiasReluBf16, false, false, true>(p, pairs, grid, s);
    if (p.epi == kTcEpiStoreF32 && p.a_mn && p.b_mn) return launch_pair_variant<kTcEpiStoreF32, true, true, true>(p, pairs, grid, s);
    if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn) return launch_pair_variant<kTcEpiMaskBf16, false, true, true>(p, pairs, grid, s);
    return cudaErrorInvalidValue;
  }
  if (p.ew == 8) {
    // short-K input gradients, whose epilogue (mask read, bf16 store) keeps up with the main loop
    // only with eight epilogue warps
    if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn)
      return launch_pair_variant<kTcEpiMaskBf16, false, true, false, 256, 8>(p, pairs, grid, s);
    return cudaErrorInvalidValue;
  }
  if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) return launch_pair_variant<kTcEpiBiasReluBf16, false, false, false>(p, pairs, grid, s);
  if (p.epi == kTcEpiBiasF32 && !p.a_mn && !p.b_mn) return launch_pair_variant<kTcEpiBiasF32, false, false, false>(p, pairs, grid, s);
  if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn) return launch_pair_variant<kTcEpiMaskBf16, false, true, false>(p, pairs, grid, s);
  if (p.epi == kTcEpiStoreF32 && p.a_mn && p.b_mn) return launch_pair_variant<kTcEpiStoreF32, true, true, false>(p, pairs, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && !p.b_mn) return launch_pair_variant<kTcEpiStoreF32, false, false, false>(p, pairs, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && p.b_mn) return launch_pair_variant<kTcEpiStoreF32, false, true, false>(p, pairs, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace hs
