// Persistent, warp-specialised tcgen05 GEMM for sm_103a (bf16 operands, fp32 accumulation in
// tensor memory).  It evaluates every contraction of the per-worker forward and backward passes
// (Eq. 1 gradients g^m, Section 1):
//   forward       H_l   = act(H_{l-1} W_l^T + b_l)        A: K-major, B: K-major
//   input grad    dH    = (delta_l W_l) * 1[H_{l-1} > 0]   A: K-major, B: MN-major
//   weight grad   G_m   = delta_l[seg_m]^T H_{l-1}[seg_m]  A: MN-major, B: MN-major, one group per worker
//
// CTA layout (192 threads, one CTA per SM; 224 for convolution products):
//   warp 0      one elected thread issues TMA tile loads into a 4-stage shared-memory ring (with
//               warp 6 for convolution products, each issuing every other box of a k-block)
//   warp 1      owns the tensor-memory allocation; one elected thread issues tcgen05.mma
//   warps 2..5  epilogue: tcgen05.ld from tensor memory, fused bias/ReLU/mask, global stores
// Two 128x256 fp32 accumulators (512 TMEM columns) let the epilogue of one tile overlap the
// main loop of the next.  Every mbarrier wait is bounded; on expiry the kernel records
// kDevWaitTimeout in the status word, stops issuing work, frees its tensor memory and returns.
#include <cudaTypedefs.h>

#include <cstdlib>
#include <cstring>

#include "tc_device.cuh"

namespace hs {

namespace {

using namespace tcdev;
constexpr int BM = kTcBM, BN = kTcBN, S = kTcStages;
constexpr int A_STAGE = BM * BK * 2;                 // 16 KB
constexpr int B_STAGE = BN * BK * 2;                 // 32 KB
constexpr uint32_t STAGE_TX = A_STAGE + B_STAGE;     // bytes landed per stage
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 2 * BN;               // two accumulator buffers
// Convolution products: a second TMA producer warp (warp 6) shares each k-block's boxes with warp 0
// (their implicit operands come in 8 KB 4-D boxes, slower to issue than the MMAs consume them).
constexpr int kConvProducers1 = 2;
template <bool CONV>
constexpr int threads_of() { return kThreads + (CONV ? 32 * (kConvProducers1 - 1) : 0); }

template <int EPI, bool A_MN, bool B_MN, bool CONV>
__global__ void __launch_bounds__(threads_of<CONV>(), 1) tc_gemm_kernel(const __grid_constant__ TcGemmParams p) {
  constexpr int NP = CONV ? kConvProducers1 : 1;
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
  grid_dependency_wait();
  grid_dependents_launch();

  const int total = p.groups * ksplit_of(p) * p.tiles_m * p.tiles_n;

  const int prod = (warp == 0) ? 0 : (NP > 1 && warp >= 6) ? warp - 6 + 1 : -1;
  if (prod >= 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producers
      // A k-block's boxes, A then B, numbered in order; producer `prod` issues those whose number is
      // prod mod NP (producer 0 also sets the stage's expected bytes).
      int s = 0;
      uint32_t ph = 0;
      int last_g = -1;
      for (int t = blockIdx.x; t < total && !*abort_flag && !p.test_stall; t += gridDim.x) {
        const TileWork w = tile_work(p, t, p.tiles_m, p.tiles_n);
        const TileCoord c = w.c;
        const CUtensorMap* ta = &p.tmA[w.g];
        const CUtensorMap* tb = &p.tmB[w.g];
        if (w.g != last_g) {
          tma_prefetch_desc(ta);
          tma_prefetch_desc(tb);
          last_g = w.g;
        }
        // implicit patch rows: the output-pixel part of the A boxes and the patch-column part of
        // the B boxes once per tile
        ConvRowPart arow[BM / 64];
        ConvColPart bcol[BN / 64];
        if (CONV && p.conv_a) {
#pragma unroll
          for (int j = 0; j < BM / 64; ++j)
            arow[j] = p.conv_a == 2 ? subpixel_row_part(p.conv, c.tm * BM + 64 * j)
                                    : conv_row_part(p.conv, c.tm * BM + 64 * j);
        }
        if (CONV && B_MN && p.conv_b) {
#pragma unroll
          for (int j = 0; j < BN / 64; ++j)
            if (c.tn * BN + 64 * j < p.conv.ones_col) bcol[j] = conv_col_part(p.conv, c.tn * BN + 64 * j);
        }
        // patch-column blocks of A and pixel blocks of B, stepped once per k-block
        ConvColIter a_it;
        ConvRowIter b_it;
        if (CONV && p.conv_a)
          a_it.init(p.conv, p.conv_a == 2 ? (p.conv.a_cls >= 0 ? p.conv.a_cls : w.g) : -1, w.kb_lo * BK);
        if (CONV && B_MN && p.conv_b) b_it.init(p.conv, w.kb_lo * BK);
        // 64-wide MN-major boxes wholly past the product's rows (A) or columns (B) are not loaded:
        // the tile's outputs in those rows and columns are never stored, and every stored output
        // reads only its own row of A and column of B, so whatever the skipped slots hold is
        // harmless (the one-SM tile is 128 x 256; the first convolution's weight gradient is 64 x 28)
        int a_live = BM / 64, b_live = BN / 64;
        if (A_MN) a_live = max(1, min(BM / 64, (p.Mdim - c.tm * BM + 63) / 64));
        if (B_MN) {
          const int ncols = (CONV && p.conv_b) ? p.conv.ones_col + 1 : p.Ndim;
          b_live = max(1, min(BN / 64, (ncols - c.tn * BN + 63) / 64));
        }
        const uint32_t tx = (uint32_t)((A_MN ? a_live * MN_CHUNK : A_STAGE) + (B_MN ? b_live * MN_CHUNK : B_STAGE));
        bool ok = true;
        for (int kb = w.kb_lo; kb < w.kb_hi; ++kb) {
          if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full_bar[s]);
          if (prod == 0) mbar_expect_tx(fb, tx);
          const int k0 = kb * BK;
          const uint32_t a_dst = smem_u32(sA + s * A_STAGE);
          const uint32_t b_dst = smem_u32(sB + s * B_STAGE);
          int box = 0;
          if (A_MN) {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j)
              if (j < a_live && box++ % NP == prod) tma_load_2d(a_dst + j * MN_CHUNK, ta, c.tm * BM + 64 * j, k0, fb);
          } else if (CONV && p.conv_a) {
            const ConvColPart kc = a_it.part();
            if (p.conv.a_box == BM) {
              // one box of the tile's 128 output pixels (lands as the two 64-row boxes would)
              if (box++ % NP == prod) {
                int cc[4];
                conv_coords(arow[0], kc, cc);
                tma_load_4d(a_dst, ta, cc, fb);
              }
            } else {
#pragma unroll
              for (int j = 0; j < BM / 64; ++j)
                if (box++ % NP == prod) {
                  int cc[4];
                  conv_coords(arow[j], kc, cc);
                  tma_load_4d(a_dst + j * MN_CHUNK, ta, cc, fb);
                }
            }
          } else {
            if (box++ % NP == prod) tma_load_2d(a_dst, ta, k0, c.tm * BM, fb);
          }
          if (B_MN) {
            ConvRowPart krow;
            if (CONV && p.conv_b) krow = b_it.part();
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) {
              if (j >= b_live || box++ % NP != prod) continue;
              const int col = c.tn * BN + 64 * j;
              if (!CONV || !p.conv_b) {
                tma_load_2d(b_dst + j * MN_CHUNK, tb, col, k0, fb);
              } else if (col < p.conv.ones_col) {
                int cc[4];
                conv_coords(krow, bcol[j], cc);
                tma_load_4d(b_dst + j * MN_CHUNK, tb, cc, fb);
              } else {
                tma_load_2d(b_dst + j * MN_CHUNK, &p.tmOnes, col - p.conv.ones_col, 0, fb);
              }
            }
          } else {
#pragma unroll
            for (int j = 0; j < BN / kTcBoxB; ++j)
              if (box++ % NP == prod) tma_load_2d(b_dst + j * (kTcBoxB * BK * 2), tb, k0, c.tn * BN + kTcBoxB * j, fb);
          }
          if (CONV && p.conv_a) a_it.next();
          if (CONV && B_MN && p.conv_b) b_it.next();
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
      constexpr uint32_t idesc_full = make_idesc(A_MN, B_MN, BM, BN);
      const uint64_t a_desc0 = make_sdesc(smem_u32(sA), A_MN ? MN_CHUNK : 16, 1024);
      const uint64_t b_desc0 = make_sdesc(smem_u32(sB), B_MN ? MN_CHUNK : 16, 1024);
      int s = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      for (int t = blockIdx.x; t < total && !*abort_flag; t += gridDim.x) {
        const TileWork w = tile_work(p, t, p.tiles_m, p.tiles_n);
        if (!mbar_wait(smem_u32(&tempty_bar[ab]), aph ^ 1u, abort_flag)) {
          record_error(p.st, kDevWaitTimeout, 2);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        // an MN-major B tile with 64-wide boxes past the product's columns runs narrower MMAs
        // (N = 64 x the live boxes): the stored columns get the same sums, the rest are never stored
        uint32_t idesc = idesc_full;
        if (B_MN) {
          const int ncols = (CONV && p.conv_b) ? p.conv.ones_col + 1 : p.Ndim;
          const int b_live = max(1, min(BN / 64, (ncols - w.c.tn * BN + 63) / 64));
          idesc = make_idesc(A_MN, B_MN, BM, 64 * b_live);
        }
        bool ok = true;
        const LastKb lk = last_kb_of(p, w.g);
        for (int kb = w.kb_lo; kb < w.kb_hi; ++kb) {
          if (!mbar_wait(smem_u32(&full_bar[s]), ph, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const int nks = kb == lk.kb_last ? lk.steps : BK / 16;
          mma_ksteps<A_MN, B_MN>(d_tmem, a_desc0 + (uint64_t)((s * A_STAGE) >> 4),
                                 b_desc0 + (uint64_t)((s * B_STAGE) >> 4), idesc, kb != w.kb_lo ? 1u : 0u, nks);
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
      const TileWork w = tile_work(p, t, p.tiles_m, p.tiles_n);
      const TileCoord c = w.c;
      uint4 zq[8];   // mask operand of the tile's first unit, loaded before the accumulator is ready
      if (EPI == kTcEpiMaskBf16) load_mask_unit<CONV>(p, w.g, c.tm * BM + q * 32 + lane, c.tn * BN, zq);
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
      const CUtensorMap* td = &p.tmD[w.g];
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
        epilogue_unit<EPI, CONV>(p, w.g, row, n_base, r, r2, zq, o);
        if (EPI == kTcEpiMaskBf16 && u + 1 < kUnits)   // the next unit's mask, behind this unit's stores
          load_mask_unit<CONV>(p, w.g, row, n_base + kUnitCols, zq);
        if (lane == 0) bulk_wait_read_1();   // the store that last used this buffer has read it
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

template <int EPI, bool A_MN, bool B_MN, bool CONV>
cudaError_t launch_variant(const TcGemmParams& p, int grid, cudaStream_t s) {
  static bool configured = false;
  auto kern = tc_gemm_kernel<EPI, A_MN, B_MN, CONV>;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see grid_dependency_wait
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(threads_of<CONV>(), 1, 1);
  cfg.dynamicSmemBytes = kTcSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
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
                      CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                      CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
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
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the operand";
    return false;
  }
  return true;
}

bool tc_make_kmajor_map(CUtensorMap* tm, const TcOperand& op, int box_rows, const char** why) {
  return encode_2d(tm, op.base, (uint64_t)op.cols, (uint64_t)op.rows, (uint64_t)op.ld * 2, kTcBK, (uint32_t)box_rows,
                   why);
}

bool tc_conv_implicit_ok(int C, int Ho, int Wo, int stride, int box_px) {
  if (box_px != 64 && box_px != 128) return false;
  if (C < 64 || C % 64 || Wo < 1 || Ho < 1 || box_px % Wo || stride < 1 || stride > 2) return false;
  const int hw = Ho * Wo;
  if (hw % box_px && box_px % hw) return false;
  const int hb = hw >= box_px ? box_px / Wo : Ho;   // output rows a box covers
  return stride * Wo <= 256 && stride * hb <= 256;
}

TcConvGeom tc_conv_geom(int C, int Ho, int Wo, int stride) {
  TcConvGeom g{};
  g.cblocks = C / 64;
  g.Wo = Wo;
  g.hw = Ho * Wo;
  g.stride = stride;
  g.ones_col = 9 * C;
  g.a_box = 64;
  g.a_cls = -1;
  g.cin_d = 0;
  return g;
}

bool tc_make_conv_map(CUtensorMap* tm, const __nv_bfloat16* base, int64_t images, int H, int W, int C, int Ho,
                      int Wo, int stride, const char** why, int box_px) {
  if (!g_encode && !tc_init_driver(why)) return false;
  if (!tc_conv_implicit_ok(C, Ho, Wo, stride, box_px) || images < 1) {
    *why = "convolution geometry not supported by the implicit patch rows";
    return false;
  }
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0) {
    *why = "TMA operand base is not 16-byte aligned";
    return false;
  }
  const int hw = Ho * Wo;
  const uint32_t hb = hw >= box_px ? (uint32_t)(box_px / Wo) : (uint32_t)Ho;
  const uint32_t nb = hw >= box_px ? 1u : (uint32_t)(box_px / hw);
  // dims innermost first: channels, input columns, input rows, images; a box traverses `stride`
  // input columns / rows per output pixel and loads ceil(extent / stride) of them
  cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)images};
  cuuint64_t strides[3] = {(cuuint64_t)C * 2, (cuuint64_t)W * C * 2, (cuuint64_t)H * W * C * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)(stride * Wo), (cuuint32_t)stride * hb, nb};
  cuuint32_t estr[4] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<__nv_bfloat16*>(base), dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the convolution operand";
    return false;
  }
  return true;
}

bool tc_grid_ok(int rows, int cols, int box_pixels) {
  if (rows < 1 || cols < 1 || box_pixels % cols) return false;
  const int hw = rows * cols;
  return hw % box_pixels == 0 || box_pixels % hw == 0;
}

bool tc_make_grid_map(CUtensorMap* tm, const void* base, int C, int cols, int rows, int64_t images,
                      int64_t col_stride, int64_t row_stride, int64_t img_stride, int box_pixels, const char** why) {
  if (!g_encode && !tc_init_driver(why)) return false;
  if (C < 64 || C % 64 || images < 1 || !tc_grid_ok(rows, cols, box_pixels)) {
    *why = "pixel grid not supported by the 4-D boxes";
    return false;
  }
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || (col_stride * 2) % 16 || (row_stride * 2) % 16 ||
      (img_stride * 2) % 16) {
    *why = "TMA grid base or stride is not 16-byte aligned";
    return false;
  }
  const int hw = rows * cols;
  const uint32_t hb = hw >= box_pixels ? (uint32_t)(box_pixels / cols) : (uint32_t)rows;
  const uint32_t nb = hw >= box_pixels ? 1u : (uint32_t)(box_pixels / hw);
  cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)images};
  cuuint64_t strides[3] = {(cuuint64_t)col_stride * 2, (cuuint64_t)row_stride * 2, (cuuint64_t)img_stride * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)cols, hb, nb};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the pixel grid";
    return false;
  }
  return true;
}

bool tc_make_nchw_box_map(CUtensorMap* tm, const float* x, int64_t images, int C, int H, int W, int box_w, int box_h,
                          const char** why) {
  if (!g_encode && !tc_init_driver(why)) return false;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) != 0 || (W * 4) % 16 || box_w % 4 || box_w > 256 || box_h > 256 ||
      C > 256 || images < 1) {
    *why = "NCHW input not addressable by TMA boxes";
    return false;
  }
  cuuint64_t dims[4] = {(cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)C, (cuuint64_t)images};
  cuuint64_t strides[3] = {(cuuint64_t)W * 4, (cuuint64_t)H * W * 4, (cuuint64_t)C * H * W * 4};
  cuuint32_t box[4] = {(cuuint32_t)box_w, (cuuint32_t)box_h, (cuuint32_t)C, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(x), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the NCHW input";
    return false;
  }
  return true;
}

bool tc_make_store_map_parts(CUtensorMap* tm, float* base, int64_t rows, int64_t cols, int64_t ld, int64_t parts,
                             int64_t part_stride, const char** why) {
  if (!g_encode && !tc_init_driver(why)) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || (ld * 4) % 16 || (part_stride * 4) % 16) {
    *why = "TMA store base or stride is not 16-byte aligned";
    return false;
  }
  cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)parts};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 4, (cuuint64_t)part_stride * 4};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the split-K output";
    return false;
  }
  return true;
}

bool tc_make_mnmajor_map(CUtensorMap* tm, const TcOperand& op, const char** why) {
  return encode_2d(tm, op.base, (uint64_t)op.cols, (uint64_t)op.rows, (uint64_t)op.ld * 2, 64, kTcBK, why);
}

bool tc_make_store_map(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                       const char** why) {
  const uint64_t es = fp32 ? 4 : 2;
  return encode_2d(tm, base, (uint64_t)cols, (uint64_t)rows, (uint64_t)ld * es, (uint32_t)(128 / es), 32, why,
                   fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16);
}

bool tc_make_store_map_bf16_32(CUtensorMap* tm, void* base, int64_t rows, int64_t cols, int64_t ld,
                               const char** why) {
  return encode_2d(tm, base, (uint64_t)cols, (uint64_t)rows, (uint64_t)ld * 2, 32, 32, why,
                   CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, CU_TENSOR_MAP_SWIZZLE_NONE);
}

bool tc_make_store_map_16(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                          const char** why) {
  return encode_2d(tm, base, (uint64_t)cols, (uint64_t)rows, (uint64_t)ld * (fp32 ? 4 : 2), 16, 32, why,
                   fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, CU_TENSOR_MAP_SWIZZLE_NONE);
}

namespace {
// Default form (SM pairs); HS_TC_FORM=single|pair in the environment overrides it at load time.
int initial_form() {
  const char* v = getenv("HS_TC_FORM");
  if (v && !strcmp(v, "pair")) return kTcFormPair;
  if (v && !strcmp(v, "single")) return kTcFormSingle;
  return kTcFormPair;
}
int g_form = initial_form();
}

void tc_set_form(int form) { g_form = (form == kTcFormPair) ? kTcFormPair : kTcFormSingle; }
int tc_get_form() { return g_form; }

cudaError_t launch_tc_gemm(const TcGemmParams& p, int num_sms, cudaStream_t s) {
  return launch_tc_gemm_form(p, num_sms, s, p.form ? p.form : g_form);
}

cudaError_t launch_tc_gemm_form(const TcGemmParams& p_in, int num_sms, cudaStream_t s, int form) {
  if (form == kTcFormPair) return launch_tc_gemm_pair(p_in, num_sms, s);
  TcGemmParams p = p_in;
  p.tiles_m = (p.Mdim + BM - 1) / BM;
  p.tiles_n = (p.n_store + BN - 1) / BN;
  const int total = p.groups * (p.ksplit > 1 ? p.ksplit : 1) * p.tiles_m * p.tiles_n;
  if (total <= 0) return cudaSuccess;
  const int grid = total < num_sms ? total : num_sms;
  // implicit convolution operands (forward, weight gradient, sub-pixel input gradient)
  if (p.conv_a || p.conv_b || p.conv_d) {
    if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiBiasReluBf16, false, false, true>(p, grid, s);
    if (p.epi == kTcEpiStoreF32 && p.a_mn && p.b_mn) return launch_variant<kTcEpiStoreF32, true, true, true>(p, grid, s);
    if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn) return launch_variant<kTcEpiMaskBf16, false, true, true>(p, grid, s);
    return cudaErrorInvalidValue;
  }
  if (p.epi == kTcEpiBiasReluBf16 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiBiasReluBf16, false, false, false>(p, grid, s);
  if (p.epi == kTcEpiBiasF32 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiBiasF32, false, false, false>(p, grid, s);
  if (p.epi == kTcEpiMaskBf16 && !p.a_mn && p.b_mn) return launch_variant<kTcEpiMaskBf16, false, true, false>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && p.a_mn && p.b_mn) return launch_variant<kTcEpiStoreF32, true, true, false>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && !p.b_mn) return launch_variant<kTcEpiStoreF32, false, false, false>(p, grid, s);
  if (p.epi == kTcEpiStoreF32 && !p.a_mn && p.b_mn) return launch_variant<kTcEpiStoreF32, false, true, false>(p, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace hs
