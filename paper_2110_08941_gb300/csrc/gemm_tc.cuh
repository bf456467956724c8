// Tensor-core (tcgen05) GEMM used by every bf16 contraction of the step.
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace hs {

constexpr int kTcMaxGroups = 32;   // groups (workers) per launch; more are split over launches

// Epilogue variants of the tensor-core GEMM.
enum TcEpi : int32_t {
  kTcEpiBiasReluBf16 = 0,   // D bf16 = bf16(max(acc + bias[n], 0))        (hidden-layer forward)
  kTcEpiBiasF32 = 1,        // D fp32 = acc + bias[n] (n < Ndim), 0 beyond   (logits)
  kTcEpiMaskBf16 = 2,       // D bf16 = bf16(acc * (Z(m, n) > 0))            (input gradient + ReLU')
  kTcEpiStoreF32 = 3,       // D fp32 = acc                                  (per-worker weight gradient)
};

// Implicit patch rows of a 3x3, padding-1 convolution over an NHWC bf16 input with C % 64 == 0:
// row r = (n, ho, wo) of the output grid, column tap * C + ci (tap = kh * 3 + kw), read straight
// from the input by 4-D TMA boxes of 64 output pixels x 64 channels (padding = the zero fill of
// out-of-range coordinates, the stride = the box's traversal stride).  Rows are grouped in blocks
// of 64, which must cover whole output rows (Wo divides 64) and whole images or parts of one
// (Ho * Wo a multiple or a divisor of 64).
struct TcConvGeom {
  int32_t cblocks;    // C / 64
  int32_t Wo, hw;     // output width, output pixels per image
  int32_t stride;
  int32_t ones_col;   // as the B operand: first column past the 9 * C patch columns, which holds
                      // ones (the bias gradient's column); columns past it read zeros
};

// D[Mdim x n_store] (row-major, leading dimension ldd) = A[Mdim x K] * B[K x Ndim] + epilogue.
// Operands are bf16 in global memory and are described by TMA tensor maps:
//   K-major   ("row-major with K contiguous"): A as [M rows][K], B as [N rows][K]
//   MN-major  ("K rows, M or N contiguous"):   A as [K rows][M], B as [K rows][N]
// Grouped launches run `groups` independent products that share Mdim/Ndim but each has its own
// A/B maps (a worker's row segment) and K extent; group g writes D + g * d_gstride.
// conv_a: A (K-major) is a convolution's implicit patch rows, tmA[g] a map from tc_make_conv_map.
// conv_b: B (MN-major) is the implicit patch rows of the group's samples (tmB[g] a conv map over
// them), and tmOnes supplies the ones column at conv.ones_col.
struct TcGemmParams {
  CUtensorMap tmA[kTcMaxGroups];
  CUtensorMap tmB[kTcMaxGroups];
  CUtensorMap tmD[kTcMaxGroups];   // output (store) maps: box of 32 rows x 128 bytes
  CUtensorMap tmOnes;              // MN-major [64][64] bf16, column 0 ones, the rest zero (conv_b)
  TcConvGeom conv;
  int32_t conv_a, conv_b;
  int32_t num_kb[kTcMaxGroups];
  int32_t groups;
  int32_t Mdim, Ndim, n_store;
  int32_t tiles_m, tiles_n;
  int32_t epi;
  int32_t a_mn, b_mn;
  void* D;
  int64_t ldd;
  int64_t d_gstride;
  const float* bias;
  const __nv_bfloat16* Z;
  int64_t ldz;
  DevStatus* st;
};

// Operand view for building tensor maps.  `rows` x `cols` bf16 matrix, row stride `ld` elements.
struct TcOperand {
  const __nv_bfloat16* base;
  int64_t rows, cols, ld;
};

// Host helpers.  Return false (and set *why) if the driver entry point or the encoding fails.
bool tc_init_driver(const char** why);
// K-major operand: matrix [rows][K] with K contiguous; box = 64 (K) x box_rows.
bool tc_make_kmajor_map(CUtensorMap* tm, const TcOperand& op, int box_rows, const char** why);
// MN-major operand: matrix [K rows][MN] with MN contiguous; box = 64 (MN) x 64 (K).
bool tc_make_mnmajor_map(CUtensorMap* tm, const TcOperand& op, const char** why);
// Implicit patch rows of a convolution (see TcConvGeom): input NHWC bf16 [images][H][W][C] at
// `base`, output grid Ho x Wo.  Box: 64 channels x 64 output pixels.
bool tc_conv_implicit_ok(int C, int Ho, int Wo, int stride);
bool tc_make_conv_map(CUtensorMap* tm, const __nv_bfloat16* base, int64_t images, int H, int W, int C, int Ho,
                      int Wo, int stride, const char** why);
TcConvGeom tc_conv_geom(int C, int Ho, int Wo, int stride);
// Output matrix [rows][cols] (row stride ld elements, fp32 or bf16) for TMA stores of 32-row x
// 128-byte boxes; rows >= `rows` and columns >= `cols` of a box are not written.
bool tc_make_store_map(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                       const char** why);

constexpr int kTcBM = 128, kTcBN = 256, kTcBK = 64, kTcStages = 4;
constexpr int kTcStagingBytes = 4 * 2 * 32 * 128;   // 4 epilogue warps x 2 buffers x (32 rows x 128 B)
constexpr int kTcSmemBytes =
    kTcStages * (kTcBM + kTcBN) * kTcBK * 2 + kTcStagingBytes + 1024 /*align*/ + 256 /*barriers*/;

constexpr int kTcBoxA = 64;    // rows of a K-major A box (a 128-row A tile is two boxes)
constexpr int kTcBoxB = 128;   // rows of a K-major B box (the 256-row B tile is two boxes)

// Kernel form: one SM per 128 x 256 tile, or an SM pair (cluster of 2, tcgen05 cta_group::2) per
// 256 x 256 tile.  Both read the same tensor maps; tiles_m / tiles_n are derived from the form.
enum TcForm : int32_t { kTcFormSingle = 1, kTcFormPair = 2 };
void tc_set_form(int form);
int tc_get_form();

// Launch on `num_sms` persistent CTAs (capped by the tile count) in the current form.
cudaError_t launch_tc_gemm(const TcGemmParams& p, int num_sms, cudaStream_t s);
cudaError_t launch_tc_gemm_form(const TcGemmParams& p, int num_sms, cudaStream_t s, int form);
cudaError_t launch_tc_gemm_pair(const TcGemmParams& p, int num_sms, cudaStream_t s);

}  // namespace hs
