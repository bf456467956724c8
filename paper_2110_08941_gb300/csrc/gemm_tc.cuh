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
  kTcEpiAvgUpdate = 4,      // theta -= lr * sum_g wavg[g] * acc_g, bf16 copy of the new theta
                            //   (per-worker weight gradients averaged in tensor memory; launch_tc_wgrad_avg)
};

// Implicit patch rows of a 3x3, padding-1 convolution over an NHWC bf16 input with C % 64 == 0:
// row r = (n, ho, wo) of the output grid, column tap * C + ci (tap = kh * 3 + kw), read straight
// from the input by 4-D TMA boxes of 64 output pixels x 64 channels (padding = the zero fill of
// out-of-range coordinates, the stride = the box's traversal stride).  Rows are grouped in blocks
// of 64, which must cover whole output rows (Wo divides 64) and whole images or parts of one
// (Ho * Wo a multiple or a divisor of 64).
//
// The input gradient of a stride-2 convolution (even H, W) splits the input pixels into four
// classes by the parity (ph, pw) of (hi, wi); class pixel (a, b) = input pixel (2a + ph, 2b + pw)
// receives kernel rows kh = 1 (ph = 0) or kh = 0, 2 (ph = 1), from output rows a, or a + 1 and a
// (likewise for columns).  Each class is then a product over an Ho x Wo grid: A = the output
// gradient at (a + dh, b + dw) per tap (4-D boxes, zero fill past the grid), K = taps x Cout,
// B = the class's weights, D = the class pixels of the input gradient (4-D store boxes), with the
// ReLU' of the input activation fused.  One grouped launch, group = class = 2 * ph + pw.
struct TcConvGeom {
  int32_t cblocks;    // (channels of the A grid) / 64
  int32_t Wo, hw;     // width of the A grid (output grid), its pixels per image
  int32_t stride;
  int32_t ones_col;   // as the B operand: first column past the 9 * C patch columns, which holds
                      // ones (the bias gradient's column); columns past it read zeros
  int32_t H, W;       // input grid (sub-pixel input gradient: where the ReLU' mask is read)
  int32_t a_box;      // output pixels per A box (conv_a): 64, or 128 (one box per 128 rows, whole
                      // output rows of one image or whole images; half the box issues per k-block)
  int32_t a_cls;      // sub-pixel A (conv_a = 2): -1 = the group's class, else this class's taps for
                      // every group (class 3: all four shifts (1,1), (1,0), (0,1), (0,0) in that order)
  int32_t cin_d;      // conv_d = 2: input-gradient channels per class block of D's columns
};

// D[Mdim x n_store] (row-major, leading dimension ldd) = A[Mdim x K] * B[K x Ndim] + epilogue.
// Operands are bf16 in global memory and are described by TMA tensor maps:
//   K-major   ("row-major with K contiguous"): A as [M rows][K], B as [N rows][K]
//   MN-major  ("K rows, M or N contiguous"):   A as [K rows][M], B as [K rows][N]
// Grouped launches run `groups` independent products that share Mdim/Ndim but each has its own
// A/B maps (a worker's row segment) and K extent; group g writes D + g * d_gstride.
// conv_a = 1: A (K-major) is a convolution's implicit patch rows, tmA[g] from tc_make_conv_map.
// conv_a = 2: A is the shifted output gradient of the sub-pixel input gradient (tc_make_grid_map,
//             64-pixel boxes), class = group; conv_d = 1: D rows are that class's input pixels
//             (tmD[g] from tc_make_grid_map with 32-pixel boxes) and the mask Z is read there.
//             conv_d = 2: one product for all four classes: D's columns are four blocks of
//             conv.cin_d channels, block c = class c (rows through tmD[c], mask at class c's pixels);
//             A walks the four shifts (conv.a_cls = 3) and B holds, per shift, each class's tap
//             with that shift or zeros.
// conv_b: B (MN-major) is the implicit patch rows of the group's samples (tmB[g] a conv map over
// them), and tmOnes supplies the ones column at conv.ones_col.
struct TcGemmParams {
  CUtensorMap tmA[kTcMaxGroups];
  CUtensorMap tmB[kTcMaxGroups];
  CUtensorMap tmD[kTcMaxGroups];   // output (store) maps: box of 32 rows x 128 bytes
  CUtensorMap tmOnes;              // MN-major [64][64] bf16, column 0 ones, the rest zero (conv_b)
  TcConvGeom conv;
  int32_t conv_a, conv_b, conv_d;
  int32_t form;                    // kernel form for this product (TcForm), 0 = the process default
  int32_t pn;                      // SM-pair tile width: 0 or 256, or 128 (then K-major B maps have
                                   // 64-row boxes and form must be kTcFormPair)
  int32_t test_stall;              // test hook only: the producer issues no loads (bounded waits expire)
  int32_t ew;                      // SM-pair form: 8 = eight epilogue warps (256-wide tiles: the MLP's
                                   // short-K input gradients, two warps per lane quadrant; 128-wide
                                   // tiles: two groups of four on alternate tiles); 0 or 4: four
  // kTcEpiAvgUpdate: the update's operands
  CUtensorMap tmT;                 // fp32 theta of the layer's weights [Mdim][n_store] (tc_make_store_map)
  CUtensorMap tmS;                 // bf16 copy of those weights, written beside theta (tc_make_store_map_bf16_32)
  const float* wavg;               // [groups] averaging weight of group (worker) g, on the device
  float lr;
  const float* lr_dev;             // non-null: the learning rate is read here (a step replayed from a graph)
  // recipe = 1: momentum mu and weight decay wd in the update, the momentum buffer through tmM
  // (first = 1: it starts as d); tmT, tmM and tmS then have 32-row x 16-column boxes
  // (tc_make_store_map_16)
  CUtensorMap tmM;
  int32_t recipe, first;
  float mu, wd;
  int32_t ksplit;                  // >= 2: each group's k-blocks split into ksplit contiguous parts, part j
                                   // a tile of its own writing part j of tmD[g], a 3-D map [parts][rows][cols]
                                   // (needs num_kb[g] >= ksplit); 0 or 1: no split
  int32_t num_kb[kTcMaxGroups];
  int32_t last_ksteps[kTcMaxGroups];   // 16-row MMA steps holding rows in group g's last k-block (1..4;
                                       // 0 = all 4): the zero-filled steps past the group's rows are skipped
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
  // ReLU' as bits, word [n / 64][row] (bits_ld rows per column unit): written by a
  // kTcEpiBiasReluBf16 launch (relu_bits_out), read by a kTcEpiMaskBf16 one in place of Z
  // (relu_bits_in); both null: Z as above
  uint64_t* relu_bits_out;
  const uint64_t* relu_bits_in;
  int64_t bits_ld;
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
// `base`, output grid Ho x Wo.  Box: 64 channels x `box_px` output pixels (64 or 128).
bool tc_conv_implicit_ok(int C, int Ho, int Wo, int stride, int box_px = 64);
bool tc_make_conv_map(CUtensorMap* tm, const __nv_bfloat16* base, int64_t images, int H, int W, int C, int Ho,
                      int Wo, int stride, const char** why, int box_px = 64);
TcConvGeom tc_conv_geom(int C, int Ho, int Wo, int stride);
// bf16 pixel grid [images][rows][cols][C] with arbitrary (16-byte multiple) strides, given in
// elements; box = 64 channels x `box_pixels` pixels (whole grid rows, or whole images).
bool tc_grid_ok(int rows, int cols, int box_pixels);
bool tc_make_grid_map(CUtensorMap* tm, const void* base, int C, int cols, int rows, int64_t images,
                      int64_t col_stride, int64_t row_stride, int64_t img_stride, int box_pixels, const char** why);
// Output matrix [rows][cols] (row stride ld elements, fp32 or bf16) for TMA stores of 32-row x
// 128-byte boxes; rows >= `rows` and columns >= `cols` of a box are not written.
bool tc_make_store_map(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                       const char** why);
// bf16 output matrix for TMA stores of 32-row x 32-column (64-byte) boxes, unswizzled (row r of a
// box at byte 64 * r of the staging buffer).
bool tc_make_store_map_bf16_32(CUtensorMap* tm, void* base, int64_t rows, int64_t cols, int64_t ld,
                               const char** why);
// fp32 or bf16 matrix for TMA loads and stores of 32-row x 16-column boxes, unswizzled (row r of a
// box at byte 64 * r, fp32, or 32 * r, bf16, of the staging buffer).
bool tc_make_store_map_16(CUtensorMap* tm, void* base, bool fp32, int64_t rows, int64_t cols, int64_t ld,
                          const char** why);
// NCHW fp32 tensor [images][C][H][W] (W a multiple of 4, 16-byte aligned base) for TMA loads of
// box_w columns x box_h rows x all C channels of one image, unswizzled (row r of channel c at float
// (c * box_h + r) * box_w of the box); out-of-range coordinates read zeros.
bool tc_make_nchw_box_map(CUtensorMap* tm, const float* x, int64_t images, int C, int H, int W, int box_w, int box_h,
                          const char** why);
// The same over `parts` such matrices `part_stride` elements apart (split-K partials, fp32).
bool tc_make_store_map_parts(CUtensorMap* tm, float* base, int64_t rows, int64_t cols, int64_t ld, int64_t parts,
                             int64_t part_stride, const char** why);

constexpr int kTcBM = 128, kTcBN = 256, kTcBK = 64, kTcStages = 4;
constexpr int kTcStagingBytes = 4 * 2 * 32 * 128;   // 4 epilogue warps x 2 buffers x (32 rows x 128 B)
constexpr int kTcSmemBytes =
    kTcStages * (kTcBM + kTcBN) * kTcBK * 2 + kTcStagingBytes + 1024 /*align*/ + 256 /*barriers*/;

constexpr int kTcBoxA = 128;   // rows of a K-major A box (one per 128-row A tile; implicit patch rows: two 64-pixel boxes)
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

// The per-worker weight gradients of one layer, averaged and applied (Eq. 1's g^m, the weighted
// average of Section 1 and Section 4.2, theta <- theta - lr * g).  Operands as for a kTcEpiStoreF32
// grouped launch with MN-major A and B (A_g = delta rows of worker g, B_g = input rows of worker g,
// groups <= kTcMaxGroups); no product is written out.  Each SM pair owns 256 x 256 tiles of the
// layer's weights and, per tile, runs the groups in order: group g's product accumulates in one of
// two tensor-memory buffers (fresh at its first k-block, exactly the per-worker gradient of the
// grouped launch) while the epilogue folds the previous group into a running sum in registers,
// sum = fma(wavg[g], acc_g, sum) from sum = 0 (the fixed worker order of reduce_update_kernel).
// After the last group: theta = fma(-lr, sum, theta) through tmT, the bf16 copy through tmS.
// The result equals the grouped launch followed by reduce_update_kernel bit for bit.
cudaError_t launch_tc_wgrad_avg(const TcGemmParams& p, int num_sms, cudaStream_t s);

}  // namespace hs
