// The CNN workload (stand-in for the paper's ResNet50 / VGG16 on CIFAR10, Section 5): three 3x3
// convolutions with padding 1 (strides 1, 2, 2, ReLU), global average pooling, one fully
// connected layer.  Activations are NHWC (channels last).  Every convolution is a product over
// its patch rows (tap-major columns) on the same GEMM kernels as the MLP:
//   forward: bias + ReLU fused; the patch rows are read straight from the input by 4-D TMA boxes
//     (implicit GEMM) where the input has a multiple of 64 channels, else materialised (im2col);
//   per-worker weight gradient G_m[W] = dA[seg_m]^T patches[seg_m] (Eq. 1's per-worker
//     gradient), its reduction over n_m * Ho * Wo rows split into k-block parts inside the kernel
//     so that the few output tiles still fill the GPU; the parts are added per worker in a fixed
//     order, and a ones column of the patch rows yields the bias gradient;
//   input gradient: for stride-2 convolutions four grouped sub-pixel products straight into the
//     input grid, else a product into patch space and a gather back, with ReLU' fused.
// The fp32 check path materialises everything and uses the SIMT products.
#include <algorithm>
#include <climits>
#include <cstring>

#include "ctx.cuh"

namespace hs {

namespace {

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// Patch rows of the first convolution from the NCHW fp32 input: col[r][ci*9 + kh*3 + kw] =
// x_pad[n][ci][s*ho + kh][s*wo + kw], r = (n*Ho + ho)*Wo + wo; columns K..Kp-1 are zero.
// Column of patch entry (ci, tap): tap-major (tap*C + ci: neighbouring channels adjacent, used by the
// bf16 path) or channel-major (ci*9 + tap: the order of theta's [Cout, Cin, 3, 3], used by the fp32
// check path).
template <bool kTapMajor>
__device__ __forceinline__ int patch_col(int ci, int tap, int C) {
  return kTapMajor ? tap * C + ci : ci * 9 + tap;
}

template <typename T, bool kTapMajor>
__global__ void im2col_nchw_kernel(const float* __restrict__ x, int N, int C, int H, int W, int Ho, int Wo, int s,
                                   T* __restrict__ col, int Kp) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t rows = (int64_t)N * Ho * Wo;
  if (idx >= rows * C) return;
  const int ci = (int)(idx % C);
  const int64_t r = idx / C;
  const int wo = (int)(r % Wo);
  const int ho = (int)((r / Wo) % Ho);
  const int n = (int)(r / ((int64_t)Wo * Ho));
  T* dst = col + r * Kp;
  const float* src = x + ((int64_t)n * C + ci) * H * W;
#pragma unroll
  for (int kh = 0; kh < 3; ++kh) {
    const int hi = s * ho + kh - 1;
#pragma unroll
    for (int kw = 0; kw < 3; ++kw) {
      const int wi = s * wo + kw - 1;
      const float v = (hi >= 0 && hi < H && wi >= 0 && wi < W) ? src[(int64_t)hi * W + wi] : 0.f;
      dst[patch_col<kTapMajor>(ci, kh * 3 + kw, C)] = from_f<T>(v);
    }
  }
  if (ci == 0)   // tail: the bf16 layout carries a ones column at 9*C (see cnn_build_wgrad_plan)
    for (int k = C * 9; k < Kp; ++k) col[r * Kp + k] = from_f<T>((kTapMajor && k == C * 9) ? 1.f : 0.f);
}

// bf16 patch rows of the first convolution from the NCHW fp32 input, one thread per row: the row's
// 9 * C tap-major values, the ones column and the zero tail are packed in registers and written
// as 16-byte stores (Kp a multiple of 8, at most 64 here).
template <int KP>
__global__ void im2col_nchw_row_kernel(const float* __restrict__ x, int N, int C, int H, int W, int Ho, int Wo,
                                       int s, __nv_bfloat16* __restrict__ col) {
  pdl_wait();
  pdl_trigger();
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= (int64_t)N * Ho * Wo) return;
  const int wo = (int)(r % Wo);
  const int ho = (int)((r / Wo) % Ho);
  const int n = (int)(r / ((int64_t)Wo * Ho));
  float v[KP];
#pragma unroll
  for (int k = 0; k < KP; ++k) {
    float val = 0.f;
    if (k < 9 * C) {
      const int tap = k / C, ci = k - tap * C;
      const int hi = s * ho + tap / 3 - 1, wi = s * wo + tap % 3 - 1;
      if (hi >= 0 && hi < H && wi >= 0 && wi < W) val = __ldg(x + (((int64_t)n * C + ci) * H + hi) * W + wi);
    } else if (k == 9 * C) {
      val = 1.f;
    }
    v[k] = val;
  }
  uint4* dst = reinterpret_cast<uint4*>(col + r * KP);
#pragma unroll
  for (int j = 0; j < KP / 8; ++j) {
    __nv_bfloat162 a = __floats2bfloat162_rn(v[8 * j], v[8 * j + 1]), b = __floats2bfloat162_rn(v[8 * j + 2], v[8 * j + 3]);
    __nv_bfloat162 c = __floats2bfloat162_rn(v[8 * j + 4], v[8 * j + 5]), d = __floats2bfloat162_rn(v[8 * j + 6], v[8 * j + 7]);
    uint4 o;
    o.x = *reinterpret_cast<uint32_t*>(&a);
    o.y = *reinterpret_cast<uint32_t*>(&b);
    o.z = *reinterpret_cast<uint32_t*>(&c);
    o.w = *reinterpret_cast<uint32_t*>(&d);
    dst[j] = o;
  }
}

// bf16 patch rows, tap-major, eight channels per thread (16-byte copies).  The tail of each row
// holds a ones column at 9*C (then zeros): the per-worker weight-gradient product then also
// yields the bias gradient, sum over the worker's rows of dA.
__global__ void im2col_nhwc_vec8_kernel(const __nv_bfloat16* __restrict__ h, int N, int C, int H, int W, int Ho,
                                        int Wo, int s, __nv_bfloat16* __restrict__ col, int Kp) {
  pdl_wait();
  pdl_trigger();
  const int C8 = C >> 3;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t rows = (int64_t)N * Ho * Wo;
  if (idx >= rows * 9 * C8) return;
  const int c8 = (int)(idx % C8);
  const int tap = (int)((idx / C8) % 9);
  const int64_t r = idx / ((int64_t)C8 * 9);
  const int wo = (int)(r % Wo);
  const int ho = (int)((r / Wo) % Ho);
  const int n = (int)(r / ((int64_t)Wo * Ho));
  const int hi = s * ho + tap / 3 - 1, wi = s * wo + tap % 3 - 1;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (hi >= 0 && hi < H && wi >= 0 && wi < W)
    v = *reinterpret_cast<const uint4*>(h + (((int64_t)n * H + hi) * W + wi) * C + c8 * 8);
  *reinterpret_cast<uint4*>(col + r * Kp + tap * C + c8 * 8) = v;
  if (tap == 0 && c8 == 0)
    for (int k = 9 * C; k < Kp; ++k) col[r * Kp + k] = __float2bfloat16_rn(k == 9 * C ? 1.f : 0.f);
}

// Input gradient of a convolution on its input grid (bf16 path): four channels per thread, float4
// reads of the tap-major patch-space gradient, ReLU' of the input activation fused.
__global__ void col2im_nhwc_vec4_kernel(const float* __restrict__ dcol, int ldc, const __nv_bfloat16* __restrict__ h,
                                        int N, int C, int H, int W, int Ho, int Wo, int s,
                                        __nv_bfloat16* __restrict__ dA) {
  pdl_wait();
  pdl_trigger();
  const int C4 = C >> 2;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)N * H * W * C4) return;
  const int c4 = (int)(idx % C4);
  const int64_t pix = idx / C4;
  const int wi = (int)(pix % W);
  const int hi = (int)((pix / W) % H);
  const int n = (int)(pix / ((int64_t)W * H));
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int kh = 0; kh < 3; ++kh) {
    const int th = hi + 1 - kh;
    if (th < 0 || th % s) continue;
    const int ho = th / s;
    if (ho >= Ho) continue;
#pragma unroll
    for (int kw = 0; kw < 3; ++kw) {
      const int tw = wi + 1 - kw;
      if (tw < 0 || tw % s) continue;
      const int wo = tw / s;
      if (wo >= Wo) continue;
      const float4 g = *reinterpret_cast<const float4*>(
          dcol + (((int64_t)n * Ho + ho) * Wo + wo) * ldc + (kh * 3 + kw) * C + c4 * 4);
      acc.x += g.x;
      acc.y += g.y;
      acc.z += g.z;
      acc.w += g.w;
    }
  }
  const int64_t o = pix * C + c4 * 4;
  const uint2 hv = *reinterpret_cast<const uint2*>(h + o);
  const __nv_bfloat162 h01 = *reinterpret_cast<const __nv_bfloat162*>(&hv.x);
  const __nv_bfloat162 h23 = *reinterpret_cast<const __nv_bfloat162*>(&hv.y);
  __nv_bfloat162 lo = __floats2bfloat162_rn(__low2float(h01) > 0.f ? acc.x : 0.f, __high2float(h01) > 0.f ? acc.y : 0.f);
  __nv_bfloat162 hi2 = __floats2bfloat162_rn(__low2float(h23) > 0.f ? acc.z : 0.f, __high2float(h23) > 0.f ? acc.w : 0.f);
  uint2 out;
  out.x = *reinterpret_cast<uint32_t*>(&lo);
  out.y = *reinterpret_cast<uint32_t*>(&hi2);
  *reinterpret_cast<uint2*>(dA + o) = out;
}

// fp32 check path: patch rows from an NHWC activation h[n][hi][wi][ci], channel-major columns.
__global__ void im2col_nhwc_f32_kernel(const float* __restrict__ h, int N, int C, int H, int W, int Ho, int Wo, int s,
                                       float* __restrict__ col, int Kp) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t rows = (int64_t)N * Ho * Wo;
  if (idx >= rows * C) return;
  const int ci = (int)(idx % C);
  const int64_t r = idx / C;
  const int wo = (int)(r % Wo);
  const int ho = (int)((r / Wo) % Ho);
  const int n = (int)(r / ((int64_t)Wo * Ho));
  float* dst = col + r * Kp;
#pragma unroll
  for (int kh = 0; kh < 3; ++kh) {
    const int hi = s * ho + kh - 1;
#pragma unroll
    for (int kw = 0; kw < 3; ++kw) {
      const int wi = s * wo + kw - 1;
      dst[patch_col<false>(ci, kh * 3 + kw, C)] =
          (hi >= 0 && hi < H && wi >= 0 && wi < W) ? h[(((int64_t)n * H + hi) * W + wi) * C + ci] : 0.f;
    }
  }
}

// pooled[n][c] = mean over the HW rows of sample n (global average pooling).
template <typename T>
__global__ void gap_forward_kernel(const T* __restrict__ h, int N, int HW, int C, T* __restrict__ pooled) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)N * C) return;
  const int c = (int)(idx % C);
  const int64_t n = idx / C;
  float acc = 0.f;
  for (int p = 0; p < HW; ++p) acc += to_f<T>(h[(n * HW + p) * C + c]);
  pooled[idx] = from_f<T>(acc / (float)HW);
}

constexpr int kGapThreads = 256;   // block of the bf16 pooling kernels: C / 8 channel groups x G pixel groups

// The same for bf16 activations (C % 8 == 0, C / 8 <= the block): one block per sample; thread
// (pixel group g, eight channels c8) sums pixels g, g + G, ... of its channels in fp32 from 16-byte
// loads, and each channel's G partial sums are then added in group order.  The activations come
// straight from the last convolution's epilogue (L2-resident); the loads of one thread are
// independent, so a sample's 64 pixels take one round of loads instead of 64.
// kFc: the fc layer in the same block (ncls <= 32 classes): logits[n][j] = sum_c p[c] W[j][c] + b[j]
// with p the stored (bf16) pooled row, W the fc weights' bf16 copy [ncls][C]; one warp per class,
// lanes on channels, an xor-shuffle tree, fp32.
template <bool kFc>
__global__ void gap_forward_vec8_kernel(const __nv_bfloat16* __restrict__ h, int HW, int C,
                                        __nv_bfloat16* __restrict__ pooled, const __nv_bfloat16* __restrict__ W,
                                        const float* __restrict__ bias, int ncls, float* __restrict__ logits,
                                        int ldl) {
  extern __shared__ float gap_part[];   // [G][C], then (kFc) the pooled row [C]
  pdl_wait();
  pdl_trigger();
  const int C8 = C >> 3;
  const int G = (int)blockDim.x / C8;
  const int n = blockIdx.x;
  const int c8 = (int)threadIdx.x % C8, g = (int)threadIdx.x / C8;
  if (g < G) {
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    const uint4* src = reinterpret_cast<const uint4*>(h + (int64_t)n * HW * C) + c8;
#pragma unroll 8
    for (int p = g; p < HW; p += G) {
      const uint4 v = __ldg(src + (int64_t)p * C8);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const __nv_bfloat162 pr = *reinterpret_cast<const __nv_bfloat162*>(&w[j]);
        acc[2 * j] += __low2float(pr);
        acc[2 * j + 1] += __high2float(pr);
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) gap_part[g * C + c8 * 8 + j] = acc[j];
  }
  __syncthreads();
  float* row = gap_part + G * C;
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    float sum = 0.f;
    for (int gg = 0; gg < G; ++gg) sum += gap_part[gg * C + c];
    const __nv_bfloat16 pb = __float2bfloat16_rn(sum / (float)HW);
    pooled[(int64_t)n * C + c] = pb;
    if (kFc) row[c] = __bfloat162float(pb);
  }
  if (kFc) {
    __syncthreads();
    const int warp = (int)threadIdx.x >> 5, lane = (int)threadIdx.x & 31;
    for (int j = warp; j < ncls; j += (int)blockDim.x >> 5) {
      const __nv_bfloat16* wj = W + (int64_t)j * C;
      float acc = 0.f;
      for (int c = lane; c < C; c += 32) acc = fmaf(row[c], __bfloat162float(wj[c]), acc);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0) logits[(int64_t)n * ldl + j] = acc + bias[j];
    }
  }
}

// dA[n][p][c] = dpooled[n][c] / HW * 1[h[n][p][c] > 0] (pooling backward with ReLU').
// The same for bf16 activations, eight channels per thread (16-byte loads and stores; C % 8 == 0,
// C / 8 <= the block): one block per sample, thread (pixel group g, channels c8) writing pixels
// g, g + G, ... from one load of its eight dpooled / HW.
// kFc: dpooled formed in the block from the fc layer's delta (bf16 [N][ldd], ncls classes) and
// weights (bf16 [ncls][C]): dpooled[c] = sum_j delta[n][j] W[j][c] in class order, fp32.
template <bool kFc>
__global__ void gap_backward_vec8_kernel(const float* __restrict__ dpooled, const __nv_bfloat16* __restrict__ h,
                                         int HW, int C, __nv_bfloat16* __restrict__ dA,
                                         const __nv_bfloat16* __restrict__ delta, int ldd,
                                         const __nv_bfloat16* __restrict__ W, int ncls) {
  extern __shared__ float gap_dp[];   // kFc: dpooled of the block's sample [C]
  pdl_wait();
  pdl_trigger();
  const int C8 = C >> 3;
  const int G = (int)blockDim.x / C8;
  const int n = blockIdx.x;
  const int c8 = (int)threadIdx.x % C8, g = (int)threadIdx.x / C8;
  const float* dp = dpooled + (int64_t)n * C;
  if (kFc) {
    const __nv_bfloat16* dn = delta + (int64_t)n * ldd;
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
      float acc = 0.f;
      for (int j = 0; j < ncls; ++j) acc = fmaf(__bfloat162float(dn[j]), __bfloat162float(W[(int64_t)j * C + c]), acc);
      gap_dp[c] = acc;
    }
    __syncthreads();
    dp = gap_dp;
  }
  if (g >= G) return;
  const float4 g0 = *reinterpret_cast<const float4*>(dp + c8 * 8);
  const float4 g1 = *reinterpret_cast<const float4*>(dp + c8 * 8 + 4);
  const float inv[8] = {g0.x / (float)HW, g0.y / (float)HW, g0.z / (float)HW, g0.w / (float)HW,
                        g1.x / (float)HW, g1.y / (float)HW, g1.z / (float)HW, g1.w / (float)HW};
  const int64_t base = (int64_t)n * HW * C8 + c8;
  const uint4* hs = reinterpret_cast<const uint4*>(h) + base;
  uint4* ds = reinterpret_cast<uint4*>(dA) + base;
#pragma unroll 8
  for (int p = g; p < HW; p += G) {
    const uint4 hv = __ldg(hs + (int64_t)p * C8);
    const uint32_t hw4[4] = {hv.x, hv.y, hv.z, hv.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const __nv_bfloat162 pr = *reinterpret_cast<const __nv_bfloat162*>(&hw4[j]);
      __nv_bfloat162 q = __floats2bfloat162_rn(__low2float(pr) > 0.f ? inv[2 * j] : 0.f,
                                               __high2float(pr) > 0.f ? inv[2 * j + 1] : 0.f);
      o[j] = *reinterpret_cast<uint32_t*>(&q);
    }
    ds[(int64_t)p * C8] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

template <typename T>
__global__ void gap_backward_kernel(const float* __restrict__ dpooled, const T* __restrict__ h, int N, int HW, int C,
                                    T* __restrict__ dA) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)N * HW * C) return;
  const int c = (int)(idx % C);
  const int64_t n = idx / ((int64_t)HW * C);
  const float g = dpooled[n * C + c] / (float)HW;
  dA[idx] = from_f<T>(to_f<T>(h[idx]) > 0.f ? g : 0.f);
}

// Input gradient on the input grid (fp32 check path): the adjoint of im2col (each input element
// sums the patch entries that read it), then ReLU' of that input: dA[n][hi][wi][ci].
__global__ void col2im_nhwc_f32_kernel(const float* __restrict__ dcol, int ldc, const float* __restrict__ h, int N,
                                       int C, int H, int W, int Ho, int Wo, int s, float* __restrict__ dA) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)N * H * W * C) return;
  const int ci = (int)(idx % C);
  const int wi = (int)((idx / C) % W);
  const int hi = (int)((idx / ((int64_t)C * W)) % H);
  const int n = (int)(idx / ((int64_t)C * W * H));
  float acc = 0.f;
#pragma unroll
  for (int kh = 0; kh < 3; ++kh) {
    const int th = hi + 1 - kh;
    if (th < 0 || th % s) continue;
    const int ho = th / s;
    if (ho >= Ho) continue;
#pragma unroll
    for (int kw = 0; kw < 3; ++kw) {
      const int tw = wi + 1 - kw;
      if (tw < 0 || tw % s) continue;
      const int wo = tw / s;
      if (wo >= Wo) continue;
      acc += dcol[(((int64_t)n * Ho + ho) * Wo + wo) * ldc + patch_col<false>(ci, kh * 3 + kw, C)];
    }
  }
  dA[idx] = h[idx] > 0.f ? acc : 0.f;
}

// bf16 copy of a convolution's weights in the tap-major column order of the bf16 patch rows:
// wp[co][tap*Cin + ci] = bf16(w[co][ci][tap]), rows padded from 9*Cin to Kp with zeros.
__global__ void permute_weights_kernel(const float* __restrict__ w, int cout, int cin, int Kp,
                                       __nv_bfloat16* __restrict__ wp) {
  pdl_wait();
  pdl_trigger();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= cout * Kp) return;
  const int k = idx % Kp, co = idx / Kp;
  float v = 0.f;
  if (k < 9 * cin) {
    const int tap = k / cin, ci = k % cin;
    v = w[((int64_t)co * cin + ci) * 9 + tap];
  }
  wp[idx] = __float2bfloat16_rn(v);
}

// bf16 weights of the four sub-pixel classes of a stride-2 convolution's input gradient (see
// TcConvGeom): class (ph, pw) = 2 * ph + pw holds [taps x Cout][Cin], row t * Cout + co, where the
// class's row taps are kh = 1 (ph = 0) or kh = 0, 2 (ph = 1) in that order, columns likewise, and
// t = th * (number of column taps) + tw.  Classes hold 1, 2, 2, 4 taps and sit back to back.
// comb: the combined layout of the one-product form instead: row T * Cout + co, column cls * Cin + ci,
// T = 2 (1 - dh) + (1 - dw) the tap's shift (dh = ph && kh == 0, dw = pw && kw == 0); the other
// blocks stay zero.
__device__ __forceinline__ int subpixel_comb_index(int co, int ci, int kh, int kw, int cout, int cin) {
  const int ph = kh != 1, pw = kw != 1;
  const int dh = ph && kh == 0, dw = pw && kw == 0;
  const int T = 2 * (1 - dh) + (1 - dw);
  return ((T * cout + co) * 4 + 2 * ph + pw) * cin + ci;   // < 16 Cout Cin, well inside 32 bits
}

__global__ void permute_weights_subpixel_kernel(const float* __restrict__ w, int cout, int cin,
                                                __nv_bfloat16* __restrict__ wc, int comb) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)cout * cin * 9) return;
  const int tap = (int)(idx % 9);
  const int ci = (int)((idx / 9) % cin);
  const int co = (int)(idx / (9 * (int64_t)cin));
  const int kh = tap / 3, kw = tap % 3;
  if (comb) {
    wc[subpixel_comb_index(co, ci, kh, kw, cout, cin)] = __float2bfloat16_rn(w[idx]);
    return;
  }
  const int ph = kh != 1, pw = kw != 1;
  const int th = (ph && kh == 2) ? 1 : 0, tw = (pw && kw == 2) ? 1 : 0;
  const int t = th * (pw ? 2 : 1) + tw;
  const int cls = 2 * ph + pw;
  const int64_t class_off = (cls == 0 ? 0 : cls == 1 ? 1 : cls == 2 ? 3 : 5) * (int64_t)cout * cin;
  wc[class_off + ((int64_t)t * cout + co) * cin + ci] = __float2bfloat16_rn(w[idx]);
}

// slabs[m][w_off + co*K + k] = sum over worker m's split-K parts (in order) of partial[part][co][k'], where
// k' = k for the fully connected layer (cin = 0) and, for a convolution, the tap-major column of
// theta's (ci, tap) entry k = ci*9 + tap (k' = tap*cin + ci).
// With cin != 0 the partial's column 9*cin is the ones column of the patch rows: its sums are the
// convolution's bias gradient, written at slabs[m][b_off + co].
__global__ void splitk_reduce_kernel(const float* __restrict__ partial, int rows, int K, int ldp,
                                     const int32_t* __restrict__ chunk_begin, float* __restrict__ slabs, int64_t Ps,
                                     int64_t w_off, int cin, int64_t b_off) {
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.y;
  const int cols = cin ? K + 1 : K;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * cols) return;
  const int k = idx % cols, co = idx / cols;
  const int kp = (cin && k < K) ? (k % 9) * cin + k / 9 : k;
  float acc = 0.f;
  for (int c = chunk_begin[m]; c < chunk_begin[m + 1]; ++c) acc += partial[((int64_t)c * rows + co) * ldp + kp];
  if (k < K)
    slabs[(int64_t)m * Ps + w_off + (int64_t)co * K + k] = acc;
  else
    slabs[(int64_t)m * Ps + b_off + co] = acc;
}

// The update of reduce_update_kernel (Section 1; Section 5's recipe with kRecipe), for the fused CNN update.
template <bool kRecipe>
__device__ __forceinline__ float apply_update_cnn(float t, float g, float lr, float* mb, float mu, float wd, int first) {
  if (!kRecipe) return fmaf(-lr, g, t);
  const float d = fmaf(wd, t, g);
  const float b = first ? d : fmaf(mu, *mb, d);
  *mb = b;
  return fmaf(-lr, b, t);
}

// The CNN step's synchronisation and update in one pass (Section 1; Section 4.2 for the weights;
// Section 5's momentum and weight decay with kRecipe): for every parameter, worker m's gradient is
// the sum of its split-K parts in part order (as splitk_reduce_kernel forms it), g = sum_m w_m g^m
// in worker order and theta's update as in reduce_update_kernel - the same fp32 operations in the
// same order, so the same bits - and the new value goes to theta, its bf16 shadow and the bf16
// copies the next step's products read: the tap-major rows of the forward (wperm) and the
// sub-pixel class matrices of the input gradient (wsub).  One work item per (output channel,
// column of the partials): columns are tap-major (tap * Cin + ci) as the products leave them, the
// ones column 9 * Cin holds the bias gradient; the fc layer's columns are its inputs, its bias
// gradients sit in the per-worker slabs.
struct CnnUpdLayer {
  const float* partial;       // [parts][rows][ldp]
  const int32_t* begin;       // [M + 1] worker m's parts are [begin[m], begin[m + 1])
  int rows, ldp, cols, cin;   // cols: weight columns (+ the ones column for a convolution); cin 0: fc
  int64_t w_off, b_off, first;   // theta offsets; first work item of the layer
  __nv_bfloat16* wperm;       // tap-major bf16 copy [rows][Kp] (convolutions)
  int Kp;
  __nv_bfloat16* wsub;        // sub-pixel copy (stride-2 convolutions whose input gradient is sub-pixel): class
                              // matrices, or the combined layout (kComb, subpixel_comb_index)
};
struct CnnUpdArgs {
  CnnUpdLayer layer[4];
  int block_first[5];         // first block of each layer's items, then of the fc bias
  int64_t items;              // work items of the four layers
  int64_t fc_b_off;           // the fc bias: C items after them, gradients from the slabs
  int C;
  const float* slabs;
  int64_t Ps;
};

// One layer's items for one block: the layer is the block's (blocks are assigned to layers in
// order), read into registers through a switch so the kernel never indexes its parameter array
// at run time.
template <bool kRecipe, bool kComb>
__device__ __forceinline__ void cnn_update_item(const CnnUpdLayer& L, int64_t it, float* __restrict__ theta, int M,
                                                const float* __restrict__ w, float lr,
                                                __nv_bfloat16* __restrict__ shadow, float* __restrict__ mbuf,
                                                float mu, float wd, int first) {
  const int co = (int)(it / L.cols);
  const int pc = (int)(it - (int64_t)co * L.cols);   // column of the partials
  int tap = 0, ci = 0;
  int64_t j;
  if (L.cin) {
    if (pc < 9 * L.cin) {
      tap = pc / L.cin;
      ci = pc - tap * L.cin;
      j = L.w_off + ((int64_t)co * L.cin + ci) * 9 + tap;
    } else {
      j = L.b_off + co;
    }
  } else {
    j = L.w_off + (int64_t)co * L.cols + pc;
  }
  const int64_t part_stride = (int64_t)L.rows * L.ldp;
  const float* col = L.partial + (int64_t)co * L.ldp + pc;
  float acc = 0.f;
  for (int m = 0; m < M; ++m) {
    // worker m's parts summed in part order; eight loads in flight, added in the same order
    float gm = 0.f;
    int c = __ldg(L.begin + m);
    const int ce = __ldg(L.begin + m + 1);
    for (; c + 8 <= ce; c += 8) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldcs(col + (int64_t)(c + u) * part_stride);
#pragma unroll
      for (int u = 0; u < 8; ++u) gm += v[u];
    }
    for (; c < ce; ++c) gm += __ldcs(col + (int64_t)c * part_stride);
    acc = fmaf(__ldg(w + m), gm, acc);
  }
  const float t = apply_update_cnn<kRecipe>(theta[j], acc, lr, kRecipe ? mbuf + j : nullptr, mu, wd, first);
  theta[j] = t;
  const __nv_bfloat16 tb = __float2bfloat16_rn(t);
  shadow[j] = tb;
  if (L.cin && pc < 9 * L.cin) {
    L.wperm[(int64_t)co * L.Kp + pc] = tb;
    if (kComb && L.wsub) {
      L.wsub[subpixel_comb_index(co, ci, tap / 3, tap % 3, L.rows, L.cin)] = tb;
    } else if (L.wsub) {
      const int kh = tap / 3, kw = tap % 3;
      const int ph = kh != 1, pw = kw != 1;
      const int th = (ph && kh == 2) ? 1 : 0, tw = (pw && kw == 2) ? 1 : 0;
      const int t2 = th * (pw ? 2 : 1) + tw;
      const int cls = 2 * ph + pw;
      const int64_t class_off = (cls == 0 ? 0 : cls == 1 ? 1 : cls == 2 ? 3 : 5) * (int64_t)L.rows * L.cin;
      L.wsub[class_off + ((int64_t)t2 * L.rows + co) * L.cin + ci] = tb;
    }
  }
}

// kComb: the sub-pixel weight copies in the combined layout (a compile-time choice: the run-time branch
// cost the kernel a third of its speed).
template <bool kRecipe, bool kComb>
__global__ void __launch_bounds__(256) cnn_update_kernel(const CnnUpdArgs a, float* __restrict__ theta, int M,
                                                         const float* __restrict__ w, float lr_arg,
                                                         const float* __restrict__ lr_dev,
                                                         __nv_bfloat16* __restrict__ shadow, float* __restrict__ mbuf,
                                                         float mu, float wd, int first) {
  pdl_wait();
  pdl_trigger();
  const float lr = lr_dev ? __ldg(lr_dev) : lr_arg;
  const int b = blockIdx.x;
  if (b >= a.block_first[4]) {
    // the fc bias: gradients from the per-worker slabs
    const int co = (b - a.block_first[4]) * blockDim.x + threadIdx.x;
    if (co >= a.C) return;
    const int64_t j = a.fc_b_off + co;
    float acc = 0.f;
    for (int m = 0; m < M; ++m) acc = fmaf(__ldg(w + m), a.slabs[(int64_t)m * a.Ps + j], acc);
    const float t = apply_update_cnn<kRecipe>(theta[j], acc, lr, kRecipe ? mbuf + j : nullptr, mu, wd, first);
    theta[j] = t;
    shadow[j] = __float2bfloat16_rn(t);
    return;
  }
  CnnUpdLayer L;
  int base;
  if (b >= a.block_first[3]) { L = a.layer[3]; base = a.block_first[3]; }
  else if (b >= a.block_first[2]) { L = a.layer[2]; base = a.block_first[2]; }
  else if (b >= a.block_first[1]) { L = a.layer[1]; base = a.block_first[1]; }
  else { L = a.layer[0]; base = 0; }
  const int64_t it = (int64_t)(b - base) * blockDim.x + threadIdx.x;
  if (it >= (int64_t)L.rows * L.cols) return;
  cnn_update_item<kRecipe, kComb>(L, it, theta, M, w, lr, shadow, mbuf, mu, wd, first);
}

inline int blocks_for(int64_t n, int threads) { return (int)((n + threads - 1) / threads); }

// bf16 step whose fc layer (at most 32 classes) runs inside the pooling kernels: the logits in the
// pooling forward's block of each sample, the fc input gradient in the pooling backward's
// (HS_CNN_FC_POOL=0 keeps the two tensor-core products).
inline bool cnn_fc_in_pooling(const hs_ctx* c) {
  const int c3 = c->convs[2].cout;
  return c->precision == HS_BF16 && c->cnn_fc_pool && c3 % 8 == 0 && c3 / 8 <= kGapThreads && c->C <= 32;
}

// bf16 patch rows of the first convolution: one thread per row where the row is short, else the
// per-channel kernel.
void launch_im2col_first(const float* x, int N, const ConvLayer& L, __nv_bfloat16* col, cudaStream_t s) {
  const int T = 256;
  const int64_t rows = L.rows;
#define HS_ROW_CASE(KP)                                                                                      \
  case KP:                                                                                                   \
    launch_pdl(im2col_nchw_row_kernel<KP>, blocks_for(rows, T), T, 0, s, x, N, L.cin, L.hin, L.win, L.hout, L.wout, \
                                                                 L.stride, col);                           \
    return;
  switch (L.Kp) {
    HS_ROW_CASE(16) HS_ROW_CASE(24) HS_ROW_CASE(32) HS_ROW_CASE(40) HS_ROW_CASE(48) HS_ROW_CASE(56) HS_ROW_CASE(64)
    default:
      launch_pdl(im2col_nchw_kernel<__nv_bfloat16, true>, blocks_for(rows * L.cin, T), T, 0, s,
          x, N, L.cin, L.hin, L.win, L.hout, L.wout, L.stride, col, L.Kp);
  }
#undef HS_ROW_CASE
}

}  // namespace

// ---------------------------------------------------------------------------------- plans
// Weight-gradient plan for one layer: one group per worker (up to 32 per launch), both operands
// MN-major [rows][cols] over the worker's rows, each worker's reduction split in the kernel into
// `ksplit` contiguous k-block ranges (parts) so that about 2 x 152 tiles run although the output
// is only Cout x (9 Cin + 1): part j of worker m lands at partial[m * ksplit + j].
hs_status cnn_build_wgrad_plan(hs_ctx* c, int layer, const __nv_bfloat16* a, int a_cols, int64_t lda,
                               const __nv_bfloat16* b, int b_cols, int64_t ldb, int64_t rows_per_sample) {
  const char* why = nullptr;
  CnnWgrad& wg = c->cnn_wgrad[layer];
  const ConvLayer* conv = layer < 3 ? &c->convs[layer] : nullptr;
  wg.plans.clear();
  wg.rows_out = a_cols;
  wg.K = b_cols;
  wg.ldp = (int)round_up(b_cols, 4);
  const int tiles = (int)(((a_cols + kTcBM - 1) / kTcBM) * ((b_cols + kTcBN - 1) / kTcBN));
  const int64_t part_elems = (int64_t)wg.rows_out * wg.ldp;
  int64_t min_kb = INT64_MAX;
  for (int m = 0; m < c->M; ++m)
    min_kb = std::min<int64_t>(min_kb, ((int64_t)c->counts[m] * rows_per_sample + kTcBK - 1) / kTcBK);
  const int per_launch = std::min(c->M, kTcMaxGroups);
  const int64_t want = (2LL * c->num_sms + (int64_t)per_launch * tiles - 1) / ((int64_t)per_launch * tiles);
  const int64_t fit = wg.partial_capacity / part_elems / c->M;   // parts the partial buffer holds per worker
  const int ksplit = (int)std::max<int64_t>(1, std::min<int64_t>(std::min<int64_t>(want, min_kb), fit));
  if ((int64_t)c->M * ksplit * part_elems > wg.partial_capacity)
    return fail(c, HS_ERR_OOM, "split-K partial buffer too small");
  std::vector<int32_t> begin;
  for (int m = 0; m <= c->M; ++m) begin.push_back(m * ksplit);
  for (int g0 = 0; g0 < c->M; g0 += kTcMaxGroups) {
    const int ng = std::min(kTcMaxGroups, c->M - g0);
    wg.plans.emplace_back();
    TcGemmParams& p = wg.plans.back();
    std::memset(&p, 0, sizeof(p));
    for (int g = 0; g < ng; ++g) {
      const int m = g0 + g;
      const int64_t r0 = (int64_t)c->offsets[m] * rows_per_sample;
      const int64_t rows = (int64_t)c->counts[m] * rows_per_sample;
      float* dg = wg.d_partial + (int64_t)m * ksplit * part_elems;
      bool ok = tc_make_mnmajor_map(&p.tmA[g], TcOperand{a + r0 * lda, rows, a_cols, lda}, &why) &&
                (ksplit > 1 ? tc_make_store_map_parts(&p.tmD[g], dg, a_cols, b_cols, wg.ldp, ksplit, part_elems, &why)
                            : tc_make_store_map(&p.tmD[g], dg, true, a_cols, b_cols, wg.ldp, &why));
      if (conv && conv->implicit) {
        // B = the implicit patch rows of the worker's samples, read from the layer's input
        const __nv_bfloat16* in = reinterpret_cast<const __nv_bfloat16*>(c->d_cact[layer - 1]) +
                                  (int64_t)c->offsets[m] * conv->hin * conv->win * conv->cin;
        ok = ok && tc_make_conv_map(&p.tmB[g], in, c->counts[m], conv->hin, conv->win, conv->cin, conv->hout,
                                    conv->wout, conv->stride, &why);
      } else {
        ok = ok && tc_make_mnmajor_map(&p.tmB[g], TcOperand{b + r0 * ldb, rows, b_cols, ldb}, &why);
      }
      if (!ok) return fail(c, HS_ERR_CUDA, why);
      p.num_kb[g] = (int32_t)((rows + kTcBK - 1) / kTcBK);
    }
    p.groups = ng;
    p.ksplit = ksplit;
    p.Mdim = a_cols;
    p.Ndim = b_cols;
    p.n_store = b_cols;
    p.tiles_m = (a_cols + kTcBM - 1) / kTcBM;
    p.tiles_n = (b_cols + kTcBN - 1) / kTcBN;
    p.epi = kTcEpiStoreF32;
    p.a_mn = 1;
    p.b_mn = 1;
    if (conv && conv->implicit) {
      p.conv_b = 1;
      p.conv = tc_conv_geom(conv->cin, conv->hout, conv->wout, conv->stride);
      if (!tc_make_mnmajor_map(&p.tmOnes, TcOperand{c->d_ones, 64, 64, 64}, &why)) return fail(c, HS_ERR_CUDA, why);
    }
    // outputs of at most 128 rows (Cout <= 128) fill the one-SM form's 128-row tile but only half
    // of an SM pair's 256 rows
    if (a_cols <= kTcBM) p.form = kTcFormSingle;
    p.D = wg.d_partial + (int64_t)g0 * ksplit * part_elems;
    p.ldd = wg.ldp;
    p.d_gstride = (int64_t)ksplit * part_elems;
    p.st = c->d_status;
  }
  cudaError_t e = cudaMemcpy(wg.d_chunk_begin, begin.data(), sizeof(int32_t) * begin.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "split-K part table");
  return HS_OK;
}

namespace {

// Epilogue warps of the 256 x 128 SM-pair tiles: two groups of four on alternate tiles (the
// default), or four (HS_NARROW_EW=4).
int narrow_epilogue_warps() {
  const char* v = getenv("HS_NARROW_EW");
  return (v && !strcmp(v, "4")) ? 4 : 8;
}

// Output pixels per A box of a convolution product: 128 where the output grid allows it (whole
// output rows of one image, or whole images), which halves the boxes a k-block issues; else 64.
// HS_CONV_ABOX=64 keeps 64.
int conv_a_box(int C, int Ho, int Wo, int stride) {
  const char* v = getenv("HS_CONV_ABOX");
  if (v && !strcmp(v, "64")) return 64;
  return tc_conv_implicit_ok(C, Ho, Wo, stride, 128) ? 128 : 64;
}
int grid_a_box(int rows, int cols) {
  const char* v = getenv("HS_CONV_ABOX");
  if (v && !strcmp(v, "64")) return 64;
  return tc_grid_ok(rows, cols, 128) ? 128 : 64;
}

// A is K-major [a_rows][a_cols], or (conv != nullptr) the implicit patch rows of that convolution.
// narrow = true: 256 x 128 SM-pair tiles for a product at most 128 wide (K-major B in 64-row boxes).
hs_status plan_dense(hs_ctx* c, TcGemmParams* p, int epi, const __nv_bfloat16* a, int64_t a_rows, int a_cols,
                     int64_t lda, const __nv_bfloat16* b, int64_t b_rows, int b_cols, int64_t ldb, bool b_mn,
                     void* d, bool d_f32, int Mdim, int Ndim, int n_store, int64_t ldd, const __nv_bfloat16* z,
                     int64_t ldz, const ConvLayer* conv = nullptr, bool narrow = false) {
  const char* why = nullptr;
  std::memset(p, 0, sizeof(*p));
  bool ok;
  if (conv) {
    const int abox = conv_a_box(conv->cin, conv->hout, conv->wout, conv->stride);
    ok = tc_make_conv_map(&p->tmA[0], a, c->N, conv->hin, conv->win, conv->cin, conv->hout, conv->wout,
                          conv->stride, &why, abox);
    p->conv_a = 1;
    p->conv = tc_conv_geom(conv->cin, conv->hout, conv->wout, conv->stride);
    p->conv.a_box = abox;
  } else {
    ok = tc_make_kmajor_map(&p->tmA[0], TcOperand{a, a_rows, a_cols, lda}, kTcBoxA, &why);
  }
  ok = ok && (b_mn ? tc_make_mnmajor_map(&p->tmB[0], TcOperand{b, b_rows, b_cols, ldb}, &why)
                   : tc_make_kmajor_map(&p->tmB[0], TcOperand{b, b_rows, b_cols, ldb}, narrow ? kTcBoxB / 2 : kTcBoxB,
                                        &why));
  if (narrow) {
    p->pn = 128;
    p->form = kTcFormPair;
    p->ew = narrow_epilogue_warps();
  }
  ok = ok && tc_make_store_map(&p->tmD[0], d, d_f32, Mdim, n_store, ldd, &why);
  if (!ok) return fail(c, HS_ERR_CUDA, why);
  const int K = b_mn ? (int)b_rows : b_cols;
  p->num_kb[0] = (K + kTcBK - 1) / kTcBK;
  p->groups = 1;
  p->Mdim = Mdim;
  p->Ndim = Ndim;
  p->n_store = n_store;
  p->tiles_m = (Mdim + kTcBM - 1) / kTcBM;
  p->tiles_n = (n_store + kTcBN - 1) / kTcBN;
  p->epi = epi;
  p->a_mn = 0;
  p->b_mn = b_mn ? 1 : 0;
  p->D = d;
  p->ldd = ldd;
  p->Z = z;
  p->ldz = ldz;
  p->st = c->d_status;
  return HS_OK;
}

// Input gradient of stride-2 convolution k as four grouped class products (see TcConvGeom):
// A = dA_k [N][Ho][Wo][Cout] (64-pixel boxes), B = the class weights (MN-major), D = the class
// pixels of dA_{k-1} [N][H][W][Cin] (32-pixel store boxes), ReLU' of h_{k-1} fused.
hs_status plan_subpixel_dgrad_comb(hs_ctx* c, int k);

hs_status plan_subpixel_dgrad(hs_ctx* c, int k) {
  if (c->convs[k].comb) return plan_subpixel_dgrad_comb(c, k);
  const ConvLayer& L = c->convs[k];
  const char* why = nullptr;
  TcGemmParams& p = c->tc_dgrad[k];
  std::memset(&p, 0, sizeof(p));
  const int64_t hw = (int64_t)L.hout * L.wout;
  const int taps[4] = {1, 2, 2, 4};
  int64_t off = 0;
  auto* dprev = reinterpret_cast<__nv_bfloat16*>(c->d_dA[k - 1]);
  const int abox = grid_a_box(L.hout, L.wout);
  for (int g = 0; g < 4; ++g) {
    const int ph = g >> 1, pw = g & 1;
    const int64_t kg = (int64_t)taps[g] * L.cout;
    bool ok = tc_make_grid_map(&p.tmA[g], c->d_dA[k], L.cout, L.wout, L.hout, c->N, L.cout, (int64_t)L.wout * L.cout,
                               hw * L.cout, abox, &why) &&
              tc_make_mnmajor_map(&p.tmB[g], TcOperand{c->d_wsub[k] + off, kg, L.cin, L.cin}, &why) &&
              tc_make_grid_map(&p.tmD[g], dprev + ((int64_t)ph * L.win + pw) * L.cin, L.cin, L.wout, L.hout, c->N,
                               2LL * L.cin, 2LL * L.win * L.cin, (int64_t)L.hin * L.win * L.cin, 32, &why);
    if (!ok) return fail(c, HS_ERR_CUDA, why);
    p.num_kb[g] = (int32_t)(kg / kTcBK);
    off += kg * L.cin;
  }
  p.groups = 4;
  p.Mdim = (int32_t)L.rows;
  p.Ndim = L.cin;
  p.n_store = L.cin;
  p.tiles_m = (p.Mdim + kTcBM - 1) / kTcBM;
  p.tiles_n = (p.n_store + kTcBN - 1) / kTcBN;
  p.epi = kTcEpiMaskBf16;
  p.a_mn = 0;
  p.b_mn = 1;
  p.conv_a = 2;
  p.conv_d = 1;
  if (L.cin <= 128) {   // 256 x 128 SM-pair tiles (the class weights are MN-major: 64-column boxes)
    p.pn = 128;
    p.form = kTcFormPair;
    p.ew = narrow_epilogue_warps();
  }
  p.conv = tc_conv_geom(L.cout, L.hout, L.wout, L.stride);
  p.conv.a_box = abox;
  p.conv.H = L.hin;
  p.conv.W = L.win;
  p.D = dprev;
  p.ldd = L.cin;
  p.Z = reinterpret_cast<const __nv_bfloat16*>(c->d_cact[k - 1]);
  p.ldz = L.cin;
  if (c->d_relu_bits.size() > (size_t)(k - 1) && c->d_relu_bits[k - 1]) {   // ReLU' of h_{k-1} as bits
    p.relu_bits_in = c->d_relu_bits[k - 1];
    p.bits_ld = c->convs[k - 1].rows;
  }
  p.st = c->d_status;
  return HS_OK;
}

// The same input gradient as one product over all four classes (conv_d = 2): rows = the Ho x Wo grid,
// K = the four shifts of A (the class-3 tap order (1,1), (1,0), (0,1), (0,0)) x Cout, columns = four
// blocks of Cin (class c = 2 ph + pw), B = the combined weights [4 x Cout][4 x Cin] whose block (shift,
// class) holds the class's tap with that shift, or zeros.  Each class sums the products of the
// grouped form over its taps in the same order, with exact zeros between: the same bits.  A k-block
// of A (one shift of the output gradient) now feeds the MMAs of every class that reads that shift
// (four, two, two and one of them) in one 256-wide product instead of one 64- or 128-wide product
// per class tap.
hs_status plan_subpixel_dgrad_comb(hs_ctx* c, int k) {
  const ConvLayer& L = c->convs[k];
  const char* why = nullptr;
  TcGemmParams& p = c->tc_dgrad[k];
  std::memset(&p, 0, sizeof(p));
  const int64_t hw = (int64_t)L.hout * L.wout;
  auto* dprev = reinterpret_cast<__nv_bfloat16*>(c->d_dA[k - 1]);
  const int abox = grid_a_box(L.hout, L.wout);
  bool ok = tc_make_grid_map(&p.tmA[0], c->d_dA[k], L.cout, L.wout, L.hout, c->N, L.cout, (int64_t)L.wout * L.cout,
                             hw * L.cout, abox, &why) &&
            tc_make_mnmajor_map(&p.tmB[0], TcOperand{c->d_wsub[k], 4LL * L.cout, 4 * L.cin, 4LL * L.cin}, &why);
  for (int g = 0; g < 4 && ok; ++g) {
    const int ph = g >> 1, pw = g & 1;
    ok = tc_make_grid_map(&p.tmD[g], dprev + ((int64_t)ph * L.win + pw) * L.cin, L.cin, L.wout, L.hout, c->N,
                          2LL * L.cin, 2LL * L.win * L.cin, (int64_t)L.hin * L.win * L.cin, 32, &why);
  }
  if (!ok) return fail(c, HS_ERR_CUDA, why);
  p.num_kb[0] = (int32_t)(4LL * L.cout / kTcBK);
  p.groups = 1;
  p.Mdim = (int32_t)L.rows;
  p.Ndim = 4 * L.cin;
  p.n_store = 4 * L.cin;
  p.tiles_m = (p.Mdim + kTcBM - 1) / kTcBM;
  p.tiles_n = (p.n_store + kTcBN - 1) / kTcBN;
  p.epi = kTcEpiMaskBf16;
  p.a_mn = 0;
  p.b_mn = 1;
  p.conv_a = 2;
  p.conv_d = 2;
  p.form = kTcFormPair;   // 256 x 256 SM-pair tiles
  // eight epilogue warps (two groups of four on alternate tiles) where the epilogue bounds it:
  // 64 channels per class block, four class blocks per tile (HS_SUBPIXEL_EW=4 or 8 forces either)
  const char* ew = getenv("HS_SUBPIXEL_EW");
  p.ew = (ew && !strcmp(ew, "8")) ? 8 : (ew && !strcmp(ew, "4")) ? 4 : (L.cin <= 64 ? 8 : 4);
  p.conv = tc_conv_geom(L.cout, L.hout, L.wout, L.stride);
  p.conv.a_box = abox;
  p.conv.a_cls = 3;
  p.conv.cin_d = L.cin;
  p.conv.H = L.hin;
  p.conv.W = L.win;
  p.D = dprev;
  p.ldd = L.cin;
  p.Z = reinterpret_cast<const __nv_bfloat16*>(c->d_cact[k - 1]);
  p.ldz = L.cin;
  if (c->d_relu_bits.size() > (size_t)(k - 1) && c->d_relu_bits[k - 1]) {   // ReLU' of h_{k-1} as bits
    p.relu_bits_in = c->d_relu_bits[k - 1];
    p.bits_ld = c->convs[k - 1].rows;
  }
  p.st = c->d_status;
  return HS_OK;
}

}  // namespace

hs_status cnn_build_static(hs_ctx* c) {
  const char* why = nullptr;
  if (!tc_init_driver(&why)) return fail(c, HS_ERR_CUDA, why);
  {
    // the ones column of the implicit patch rows: [64][64] bf16 with column 0 = 1
    std::vector<__nv_bfloat16> ones(64 * 64, __float2bfloat16(0.f));
    for (int r = 0; r < 64; ++r) ones[r * 64] = __float2bfloat16(1.f);
    cudaError_t e = cudaMemcpy(c->d_ones, ones.data(), sizeof(__nv_bfloat16) * ones.size(), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(c, e, "ones tile");
  }
  const int N = c->N;
  auto bf = [](void* p) { return reinterpret_cast<const __nv_bfloat16*>(p); };
  c->conv_first_on = c->precision == HS_BF16 && conv_first_ok(c->convs[0]);
  if (c->conv_first_on) {
    hs_status st = conv_first_plan(c, &c->conv_first);
    if (st != HS_OK) return st;
    if (c->d_relu_bits.size() > 0 && c->d_relu_bits[0]) {
      c->conv_first.bits = c->d_relu_bits[0];
      c->conv_first.bits_ld = c->convs[0].rows;
    }
  }
  c->tc_fwd.assign(4, TcGemmParams{});
  c->tc_dgrad.assign(4, TcGemmParams{});
  for (int k = 0; k < 3; ++k) {
    const ConvLayer& L = c->convs[k];
    const __nv_bfloat16* wb = c->d_wperm[k];
    const int64_t ldw = L.Kp;
    const __nv_bfloat16* a = L.implicit ? bf(c->d_cact[k - 1]) : bf(c->d_col[k]);
    hs_status st = plan_dense(c, &c->tc_fwd[k], kTcEpiBiasReluBf16, a, L.rows, L.K, L.Kp, wb, L.cout, L.K, ldw,
                              false, c->d_cact[k], false, (int)L.rows, L.cout, L.cout, L.cout, nullptr, 0,
                              L.implicit ? &L : nullptr, L.cout <= 128);
    if (st != HS_OK) return st;
    if (c->d_relu_bits.size() > (size_t)k && c->d_relu_bits[k]) {   // ReLU' bits for the next input gradient
      c->tc_fwd[k].relu_bits_out = c->d_relu_bits[k];
      c->tc_fwd[k].bits_ld = L.rows;
    }
  }
  // fully connected layer on the pooled features
  const int c3 = c->convs[2].cout;
  hs_status st = plan_dense(c, &c->tc_fwd[3], kTcEpiBiasF32, bf(c->d_pooled), N, c3, c3, c->d_shadow + c->fc_w_off,
                            c->C, c3, c3, false, c->d_logits, true, N, c->C, c->Cp, c->Cp, nullptr, 0);
  if (st != HS_OK) return st;
  // input gradients: fc -> pooled features (fp32), conv3 / conv2 -> patch space (fp32)
  st = plan_dense(c, &c->tc_dgrad[3], kTcEpiStoreF32, bf(c->d_delta[0]), N, c->C, c->Cp, c->d_shadow + c->fc_w_off,
                  c->C, c3, c3, true, c->d_dpooled, true, N, c3, c3, c3, nullptr, 0);
  if (st != HS_OK) return st;
  for (int k = 2; k >= 1; --k) {
    const ConvLayer& L = c->convs[k];
    if (L.subpixel) {
      st = plan_subpixel_dgrad(c, k);
    } else {
      st = plan_dense(c, &c->tc_dgrad[k], kTcEpiStoreF32, bf(c->d_dA[k]), L.rows, L.cout, L.cout,
                      c->d_wperm[k], L.cout, L.K, L.Kp, true, c->d_dcol, true, (int)L.rows, L.K, L.K, L.K,
                      nullptr, 0);
    }
    if (st != HS_OK) return st;
  }
  return HS_OK;
}

hs_status cnn_build_partition_plans(hs_ctx* c) {
  auto bf = [](void* p) { return reinterpret_cast<const __nv_bfloat16*>(p); };
  // fc: A^T = delta [N][C] (ld Cp), B = pooled [N][c3]
  const int c3 = c->convs[2].cout;
  hs_status st = cnn_build_wgrad_plan(c, 3, bf(c->d_delta[0]), c->C, c->Cp, bf(c->d_pooled), c3, c3, 1);
  for (int k = 2; k >= 0 && st == HS_OK; --k) {
    const ConvLayer& L = c->convs[k];
    st = cnn_build_wgrad_plan(c, k, bf(c->d_dA[k]), L.cout, L.cout, bf(c->d_col[k]), L.K + 1, L.Kp,
                              (int64_t)L.hout * L.wout);
  }
  return st;
}

// ---------------------------------------------------------------------------------- the step
hs_status cnn_step(hs_ctx* c, float* params, const float* x, const int32_t* y, cudaStream_t s) {
  const bool bf16 = (c->precision == HS_BF16);
  const int N = c->N, T = 256;
  const ConvLayer* L = c->convs.data();
  const int c3 = L[2].cout;
  const int hw3 = L[2].hout * L[2].wout;
  // (the bf16 weight copies the products read are current: cnn_refresh_weights or the fused update)
  {
    PhaseScope ph(c, HS_PHASE_FORWARD, s);
    for (int k = 0; k < 3; ++k) {
      const int64_t n_items = L[k].rows * L[k].cin;
      if (k == 0 && c->conv_first_on && conv_first_bind_input(c, x)) {
        // input boxes, patch rows, product, bias + ReLU in one kernel (the patch rows also written
        // for the weight gradient)
        ConvFirstParams& f = c->conv_first;
        f.bias = params + L[0].b_off;
        cudaError_t e = launch_conv_first(f, c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "first convolution launch");
        ph.launched();
        continue;
      }
      if (k == 0) {
        if (bf16)
          launch_im2col_first(x, N, L[0], reinterpret_cast<__nv_bfloat16*>(c->d_col[0]), s);
        else
          launch_pdl(im2col_nchw_kernel<float, false>, blocks_for(n_items, T), T, 0, s,
              x, N, L[0].cin, L[0].hin, L[0].win, L[0].hout, L[0].wout, L[0].stride,
              reinterpret_cast<float*>(c->d_col[0]), L[0].Kp);
      } else if (L[k].implicit) {
        // the forward product reads the patch rows straight from d_cact[k - 1]
      } else {
        if (bf16)
          launch_pdl(im2col_nhwc_vec8_kernel, blocks_for(L[k].rows * 9 * (L[k].cin / 8), T), T, 0, s,
              reinterpret_cast<const __nv_bfloat16*>(c->d_cact[k - 1]), N, L[k].cin, L[k].hin, L[k].win, L[k].hout,
              L[k].wout, L[k].stride, reinterpret_cast<__nv_bfloat16*>(c->d_col[k]), L[k].Kp);
        else
          launch_pdl(im2col_nhwc_f32_kernel, blocks_for(n_items, T), T, 0, s,
              reinterpret_cast<const float*>(c->d_cact[k - 1]), N, L[k].cin, L[k].hin, L[k].win, L[k].hout,
              L[k].wout, L[k].stride, reinterpret_cast<float*>(c->d_col[k]), L[k].Kp);
      }
      if (!L[k].implicit) ph.launched();
      if (bf16) {
        TcGemmParams& f = c->tc_fwd[k];
        f.bias = params + L[k].b_off;
        cudaError_t e = launch_tc_gemm(f, c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "conv forward GEMM launch");
      } else {
        GemmF32Args g{};
        g.A = reinterpret_cast<const float*>(c->d_col[k]); g.a_sm = L[k].Kp; g.a_sk = 1;
        g.B = params + L[k].w_off; g.b_sk = 1; g.b_sn = L[k].K;
        g.C = reinterpret_cast<float*>(c->d_cact[k]); g.ldc = L[k].cout;
        g.Mdim = (int)L[k].rows; g.Ndim = L[k].cout; g.Kdim = L[k].K;
        g.epi = kEpiBiasRelu; g.bias = params + L[k].b_off;
        launch_gemm_f32(g, s);
      }
      ph.launched();
    }
    const bool fc_pool = cnn_fc_in_pooling(c);
    const __nv_bfloat16* w_fc = c->d_shadow + c->fc_w_off;
    if (bf16 && c3 % 8 == 0 && c3 / 8 <= kGapThreads) {
      const size_t smem = ((size_t)(kGapThreads / (c3 / 8)) * c3 + (fc_pool ? c3 : 0)) * sizeof(float);
      if (fc_pool)   // the fc layer's logits in the same block
        launch_pdl(gap_forward_vec8_kernel<true>, N, kGapThreads, smem, s,
            reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), hw3, c3, reinterpret_cast<__nv_bfloat16*>(c->d_pooled),
            w_fc, params + c->fc_b_off, c->C, c->d_logits, c->Cp);
      else
        launch_pdl(gap_forward_vec8_kernel<false>, N, kGapThreads, smem, s,
            reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), hw3, c3, reinterpret_cast<__nv_bfloat16*>(c->d_pooled),
            (const __nv_bfloat16*)nullptr, (const float*)nullptr, 0, (float*)nullptr, 0);
    } else if (bf16) {
      launch_pdl(gap_forward_kernel<__nv_bfloat16>, blocks_for((int64_t)N * c3, T), T, 0, s,
          reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), N, hw3, c3, reinterpret_cast<__nv_bfloat16*>(c->d_pooled));
    } else {
      launch_pdl(gap_forward_kernel<float>, blocks_for((int64_t)N * c3, T), T, 0, s,
          reinterpret_cast<const float*>(c->d_cact[2]), N, hw3, c3, reinterpret_cast<float*>(c->d_pooled));
    }
    ph.launched();
    if (fc_pool) {
      // the logits came out of the pooling kernel
    } else if (bf16) {
      TcGemmParams& f = c->tc_fwd[3];
      f.bias = params + c->fc_b_off;
      cudaError_t e = launch_tc_gemm(f, c->num_sms, s);
      if (e != cudaSuccess) return cuda_fail(c, e, "fc forward GEMM launch");
      ph.launched();
    } else {
      GemmF32Args g{};
      g.A = reinterpret_cast<const float*>(c->d_pooled); g.a_sm = c3; g.a_sk = 1;
      g.B = params + c->fc_w_off; g.b_sk = 1; g.b_sn = c3;
      g.C = c->d_logits; g.ldc = c->Cp;
      g.Mdim = N; g.Ndim = c->C; g.Kdim = c3;
      g.epi = kEpiBias; g.bias = params + c->fc_b_off;
      launch_gemm_f32(g, s);
      ph.launched();
    }
  }
  {
    PhaseScope ph(c, HS_PHASE_LOSS, s);
    if (bf16 && softmax_loss_bias_ok(c->C, c->Cp, c->Cp)) {
      // softmax, loss reduction and the fc bias gradients in one launch
      launch_softmax_loss_bias(c->d_logits, c->Cp, y, c->d_scale, c->C, reinterpret_cast<__nv_bfloat16*>(c->d_delta[0]),
                               c->Cp, c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket,
                               c->d_slabs, c->Ps, c->fc_b_off, s);
      ph.launched();
    } else {
      launch_softmax_xent(c->d_logits, c->Cp, y, c->d_scale, N, c->C, c->d_delta[0], c->Cp, bf16, c->d_ce,
                          c->d_status, s);
      if (bf16 && c->C <= loss_bias_max_width())   // the fc bias gradients in the same launch
        launch_loss_bias_reduce(c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket,
                                reinterpret_cast<const __nv_bfloat16*>(c->d_delta[0]), c->Cp, c->C, c->d_slabs, c->Ps,
                                c->fc_b_off, s);
      else
        launch_loss_reduce(c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket, s);
      ph.launched(2);
    }
  }
  // ---- backward: layer index 3 = fc, 2..0 = conv3..conv1
  for (int k = 3; k >= 0; --k) {
    const bool fc = (k == 3);
    const int width = fc ? c->C : L[k].cout;
    void* delta = fc ? c->d_delta[0] : c->d_dA[k];
    const int ld_delta = fc ? c->Cp : L[k].cout;
    const int64_t w_off = fc ? c->fc_w_off : L[k].w_off;
    const int64_t b_off = fc ? c->fc_b_off : L[k].b_off;
    {
      PhaseScope ph(c, HS_PHASE_WGRAD, s);
      if (bf16) {
        CnnWgrad& wg = c->cnn_wgrad[k];
        for (const TcGemmParams& p : wg.plans) {
          cudaError_t e = launch_tc_gemm(p, c->num_sms, s);
          if (e != cudaSuccess) return cuda_fail(c, e, "conv weight-gradient GEMM launch");
          ph.launched();
        }
        if (!cnn_fused_update(c)) {   // else the fused update reads the split-K parts itself
          const int kw = fc ? wg.K : wg.K - 1;   // weight columns (the conv partials carry the bias column)
          dim3 grid2(blocks_for((int64_t)wg.rows_out * wg.K, T), c->M);
          launch_pdl(splitk_reduce_kernel, grid2, T, 0, s, wg.d_partial, wg.rows_out, kw, wg.ldp, wg.d_chunk_begin,
                     c->d_slabs, c->Ps, w_off, fc ? 0 : L[k].cin, b_off);
          ph.launched();
        }
      } else {
        GemmF32Args w{};
        w.A = reinterpret_cast<const float*>(delta); w.a_sm = 1; w.a_sk = ld_delta;
        if (fc) {
          w.B = reinterpret_cast<const float*>(c->d_pooled); w.b_sk = c3; w.b_sn = 1; w.Ndim = c3;
        } else {
          w.B = reinterpret_cast<const float*>(c->d_col[k]); w.b_sk = L[k].Kp; w.b_sn = 1; w.Ndim = L[k].K;
        }
        w.C = c->d_slabs + w_off; w.ldc = w.Ndim;
        w.Mdim = width; w.Kdim = 0;
        w.epi = kEpiStore;
        w.k_offsets = c->d_row_off[k]; w.groups = c->M; w.c_gstride = c->Ps;
        launch_gemm_f32(w, s);
        ph.launched();
      }
    }
    {
      PhaseScope ph(c, HS_PHASE_BIASGRAD, s);
      if (bf16 && !fc) {
        // the convolutions' bias gradients came out of the weight-gradient product (ones column)
      } else if (bf16 && c->C <= loss_bias_max_width()) {
        // the fc bias gradients came out of the loss reduction
      } else if (bf16) {
        const ChunkTable& ct = c->cnn_chunks[k];
        launch_bias_grad_bf16(reinterpret_cast<const __nv_bfloat16*>(delta), ld_delta, width, ct.d_chunks, ct.n,
                              ct.d_begin, c->M, c->d_bg_partial, c->d_slabs, c->Ps, b_off, s);
        ph.launched(2);
      } else {
        launch_bias_grad(delta, false, ld_delta, width, c->d_row_off[k], c->M, c->d_slabs, c->Ps, b_off, s);
        ph.launched();
      }
    }
    if (k == 0) break;
    PhaseScope ph(c, HS_PHASE_DGRAD, s);
    if (fc) {
      // dpooled = delta W_fc, then pooling backward with ReLU' into conv3's output gradient
      const bool fc_pool = cnn_fc_in_pooling(c);
      if (fc_pool) {
        // dpooled is formed inside the pooling backward
      } else if (bf16) {
        cudaError_t e = launch_tc_gemm(c->tc_dgrad[3], c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "fc input-gradient GEMM launch");
        ph.launched();
      } else {
        GemmF32Args d{};
        d.A = reinterpret_cast<const float*>(c->d_delta[0]); d.a_sm = c->Cp; d.a_sk = 1;
        d.B = params + c->fc_w_off; d.b_sk = c3; d.b_sn = 1;
        d.C = c->d_dpooled; d.ldc = c3;
        d.Mdim = N; d.Ndim = c3; d.Kdim = c->C; d.epi = kEpiStore;
        launch_gemm_f32(d, s);
        ph.launched();
      }
      if (fc_pool)
        launch_pdl(gap_backward_vec8_kernel<true>, N, kGapThreads, c3 * sizeof(float), s,
            (const float*)nullptr, reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), hw3, c3,
            reinterpret_cast<__nv_bfloat16*>(c->d_dA[2]), reinterpret_cast<const __nv_bfloat16*>(c->d_delta[0]), c->Cp,
            c->d_shadow + c->fc_w_off, c->C);
      else if (bf16 && c3 % 8 == 0 && c3 / 8 <= kGapThreads)
        launch_pdl(gap_backward_vec8_kernel<false>, N, kGapThreads, 0, s,
            c->d_dpooled, reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), hw3, c3,
            reinterpret_cast<__nv_bfloat16*>(c->d_dA[2]), (const __nv_bfloat16*)nullptr, 0,
            (const __nv_bfloat16*)nullptr, 0);
      else if (bf16)
        launch_pdl(gap_backward_kernel<__nv_bfloat16>, blocks_for((int64_t)N * hw3 * c3, T), T, 0, s,
            c->d_dpooled, reinterpret_cast<const __nv_bfloat16*>(c->d_cact[2]), N, hw3, c3,
            reinterpret_cast<__nv_bfloat16*>(c->d_dA[2]));
      else
        launch_pdl(gap_backward_kernel<float>, blocks_for((int64_t)N * hw3 * c3, T), T, 0, s,
            c->d_dpooled, reinterpret_cast<const float*>(c->d_cact[2]), N, hw3, c3, reinterpret_cast<float*>(c->d_dA[2]));
      ph.launched();
    } else {
      if (L[k].subpixel) {
        // the four class products write dA_{k-1} directly (ReLU' of h_{k-1} fused)
        cudaError_t e = launch_tc_gemm(c->tc_dgrad[k], c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "conv sub-pixel input-gradient GEMM launch");
        ph.launched();
        continue;
      }
      // dcol = dA_k W_k (patch space, fp32), then gather back to layer k's input grid with ReLU'
      if (bf16) {
        cudaError_t e = launch_tc_gemm(c->tc_dgrad[k], c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "conv input-gradient GEMM launch");
      } else {
        GemmF32Args d{};
        d.A = reinterpret_cast<const float*>(c->d_dA[k]); d.a_sm = L[k].cout; d.a_sk = 1;
        d.B = params + L[k].w_off; d.b_sk = L[k].K; d.b_sn = 1;
        d.C = c->d_dcol; d.ldc = L[k].K;
        d.Mdim = (int)L[k].rows; d.Ndim = L[k].K; d.Kdim = L[k].cout; d.epi = kEpiStore;
        launch_gemm_f32(d, s);
      }
      const int64_t n_in = (int64_t)N * L[k].hin * L[k].win * L[k].cin;
      if (bf16)
        launch_pdl(col2im_nhwc_vec4_kernel, blocks_for(n_in / 4, T), T, 0, s,
            c->d_dcol, L[k].K, reinterpret_cast<const __nv_bfloat16*>(c->d_cact[k - 1]), N, L[k].cin, L[k].hin,
            L[k].win, L[k].hout, L[k].wout, L[k].stride, reinterpret_cast<__nv_bfloat16*>(c->d_dA[k - 1]));
      else
        launch_pdl(col2im_nhwc_f32_kernel, blocks_for(n_in, T), T, 0, s,
            c->d_dcol, L[k].K, reinterpret_cast<const float*>(c->d_cact[k - 1]), N, L[k].cin, L[k].hin, L[k].win,
            L[k].hout, L[k].wout, L[k].stride, reinterpret_cast<float*>(c->d_dA[k - 1]));
      ph.launched(2);
    }
  }
  return HS_OK;
}

bool cnn_fused_update(const hs_ctx* c) {
  return c->arch == HS_CNN && c->precision == HS_BF16 && c->cnn_fuse_update && !c->debug;
}

// The bf16 copies of theta the CNN's products read: tap-major rows (forward, patch-space input
// gradient) and, for the sub-pixel input gradients, the class matrices.  The fused update writes
// them beside theta; this runs when they are stale (first step, external change of params, a
// step on the slab path).
hs_status cnn_refresh_weights(hs_ctx* c, const float* params, cudaStream_t s) {
  const int T = 256;
  PhaseScope ph(c, HS_PHASE_CAST, s);
  for (int k = 0; k < 3; ++k) {
    const ConvLayer& L = c->convs[k];
    launch_pdl(permute_weights_kernel, blocks_for((int64_t)L.cout * L.Kp, T), T, 0, s,
        params + L.w_off, L.cout, L.cin, L.Kp, c->d_wperm[k]);
    ph.launched();
    if (L.subpixel) {
      launch_pdl(permute_weights_subpixel_kernel, blocks_for(9LL * L.cout * L.cin, T), T, 0, s,
          params + L.w_off, L.cout, L.cin, c->d_wsub[k], L.comb ? 1 : 0);
      ph.launched();
    }
  }
  HS_CUDA(c, cudaGetLastError());
  return HS_OK;
}

hs_status launch_cnn_update(hs_ctx* c, float* params, float lr, const float* lr_dev, cudaStream_t s) {
  CnnUpdArgs a{};
  int64_t items = 0;
  const int T = 256;
  int blocks = 0;
  for (int k = 0; k < 4; ++k) {
    const bool fc = (k == 3);
    const CnnWgrad& wg = c->cnn_wgrad[k];
    CnnUpdLayer& u = a.layer[k];
    u.partial = wg.d_partial;
    u.begin = wg.d_chunk_begin;
    u.rows = wg.rows_out;
    u.ldp = wg.ldp;
    u.cols = wg.K;   // convolutions: 9 * Cin weight columns and the ones column; fc: its inputs
    u.cin = fc ? 0 : c->convs[k].cin;
    u.w_off = fc ? c->fc_w_off : c->convs[k].w_off;
    u.b_off = fc ? c->fc_b_off : c->convs[k].b_off;
    u.first = items;
    u.wperm = fc ? nullptr : c->d_wperm[k];
    u.Kp = fc ? 0 : c->convs[k].Kp;
    u.wsub = (!fc && c->convs[k].subpixel) ? c->d_wsub[k] : nullptr;
    a.block_first[k] = blocks;
    blocks += blocks_for((int64_t)u.rows * u.cols, T);
    items += (int64_t)u.rows * u.cols;
  }
  a.block_first[4] = blocks;
  blocks += blocks_for(c->C, T);
  a.items = items;
  a.fc_b_off = c->fc_b_off;
  a.C = c->C;
  a.slabs = c->d_slabs;
  a.Ps = c->Ps;
  if (items + c->C != c->P) return fail(c, HS_ERR_CUDA, "fused CNN update does not cover the parameters");
  PhaseScope ph(c, HS_PHASE_UPDATE, s);
  // the sub-pixel layers share the layout (a sub-pixel layer's input has a multiple of 64 channels)
  const bool comb = c->convs[1].comb || c->convs[2].comb;
  auto kern = c->opt_recipe ? (comb ? cnn_update_kernel<true, true> : cnn_update_kernel<true, false>)
                            : (comb ? cnn_update_kernel<false, true> : cnn_update_kernel<false, false>);
  if (c->opt_recipe)
    launch_pdl(kern, blocks, T, 0, s, a, params, c->M, static_cast<const float*>(c->d_w), lr, lr_dev, c->d_shadow,
               c->d_mom, c->opt_momentum, c->opt_weight_decay, c->mom_valid ? 0 : 1);
  else
    launch_pdl(kern, blocks, T, 0, s, a, params, c->M, static_cast<const float*>(c->d_w), lr, lr_dev, c->d_shadow,
               static_cast<float*>(nullptr), 0.f, 0.f, 0);
  ph.launched();
  HS_CUDA(c, cudaGetLastError());
  return HS_OK;
}

}  // namespace hs
