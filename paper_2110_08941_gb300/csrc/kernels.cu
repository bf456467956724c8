// Bandwidth-bound kernels of the step: input cast, partition scatter, fused softmax
// cross-entropy, per-worker loss and bias-gradient reductions, and the fused gradient
// reduction + SGD update.  All reductions run in a fixed order (deterministic results).
#include "common.cuh"

namespace hs {

// ------------------------------------------------------------------------------------ cast
__global__ void cast_f32_bf16_kernel(const float* __restrict__ x, __nv_bfloat16* __restrict__ y,
                                     int64_t n) {
  pdl_wait();
  pdl_trigger();
  const int64_t nvec = n / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const float4 a = __ldcs(reinterpret_cast<const float4*>(x) + v);
    __nv_bfloat162 lo = __floats2bfloat162_rn(a.x, a.y);
    __nv_bfloat162 hi = __floats2bfloat162_rn(a.z, a.w);
    uint2 packed;
    packed.x = *reinterpret_cast<uint32_t*>(&lo);
    packed.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(y)[v] = packed;
  }
  for (int64_t j = nvec * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride)
    y[j] = __float2bfloat16_rn(x[j]);
}

void launch_cast_f32_bf16(const float* x, __nv_bfloat16* y, int64_t n, cudaStream_t s) {
  if (n <= 0) return;
  int64_t blocks = (n / 4 + 255) / 256;
  if (blocks < 1) blocks = 1;
  if (blocks > 4096) blocks = 4096;
  launch_pdl(cast_f32_bf16_kernel, (int)blocks, 256, 0, s, x, y, n);
}

// ------------------------------------------------------------------------ partition scatter
// Algorithm 1 fixes the partition sizes; samples are laid out as contiguous worker segments:
// index_map[i] = m for offsets[m] <= i < offsets[m+1], scale[i] = 1 / n_m (Eq. 1's mean).
__global__ void partition_scatter_kernel(const int32_t* __restrict__ offsets, int M, int N,
                                         int32_t* __restrict__ index_map, float* __restrict__ scale,
                                         int32_t* __restrict__ index_map_out) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ int32_t s_off[];
  for (int k = threadIdx.x; k <= M; k += blockDim.x) s_off[k] = offsets[k];
  __syncthreads();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  int lo = 0, hi = M - 1;          // largest m with s_off[m] <= i
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_off[mid] <= i) lo = mid; else hi = mid - 1;
  }
  index_map[i] = lo;
  scale[i] = 1.0f / (float)(s_off[lo + 1] - s_off[lo]);
  if (index_map_out) index_map_out[i] = lo;
}

void launch_partition_scatter(const int32_t* d_offsets, int M, int N, int32_t* index_map,
                              float* scale, int32_t* index_map_out, cudaStream_t s) {
  const int threads = 256;
  const int blocks = (N + threads - 1) / threads;
  launch_pdl(partition_scatter_kernel, blocks, threads, (M + 1) * sizeof(int32_t), s,
      d_offsets, M, N, index_map, scale, index_map_out);
}

// out[i] = w[m(i)] * scale[i]: the loss-gradient scale of the slab-free formulation, where worker
// m's weight is folded into its samples (sum_m w_m G_m = one product over all rows).
__global__ void scale_by_weight_kernel(const int32_t* __restrict__ index_map, const float* __restrict__ scale,
                                       const float* __restrict__ w, int N, float* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < N) out[i] = w[index_map[i]] * scale[i];
}

void launch_scale_by_weight(const int32_t* index_map, const float* scale, const float* w, int N, float* out,
                            cudaStream_t s) {
  launch_pdl(scale_by_weight_kernel, (N + 255) / 256, 256, 0, s, index_map, scale, w, N, out);
}

// ------------------------------------------------------------------ softmax cross-entropy
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ void record_error(DevStatus* st, int32_t code, int32_t info) {
  if (atomicCAS(&st->err, 0, code) == 0) st->err_info = info;
}

// One warp per sample row i (Eq. 1 per-sample loss and its gradient):
//   ce_i = logsumexp(z_i) - z_{i,y_i},  delta_i = (softmax(z_i) - onehot(y_i)) * scale_i,
// scale_i = 1/n_{m(i)} (the derivative of worker m(i)'s mean loss).
template <bool kBf16>
__global__ void softmax_xent_kernel(const float* __restrict__ logits, int ldl,
                                    const int32_t* __restrict__ y, const float* __restrict__ scale,
                                    int N, int C, void* __restrict__ delta, int ldd,
                                    float* __restrict__ ce, DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  const int warps_per_block = blockDim.x >> 5;
  const int row = blockIdx.x * warps_per_block + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= N) return;
  const float* z = logits + (int64_t)row * ldl;
  int label = y[row];
  if (label < 0 || label >= C) {
    if (lane == 0) record_error(st, kDevBadLabel, row);
    label = label < 0 ? 0 : C - 1;
  }
  float mx = -INFINITY;
  for (int j = lane; j < C; j += 32) mx = fmaxf(mx, z[j]);
  mx = warp_max(mx);
  float se = 0.f;
  for (int j = lane; j < C; j += 32) se += expf(z[j] - mx);
  se = warp_sum(se);
  const float lse = mx + logf(se);
  if (lane == 0) ce[row] = lse - z[label];
  const float inv = 1.0f / se;
  const float sc = scale[row];
  for (int j = lane; j < ldd; j += 32) {
    float d = 0.f;
    if (j < C) d = (expf(z[j] - mx) * inv - (j == label ? 1.f : 0.f)) * sc;
    if (kBf16)
      reinterpret_cast<__nv_bfloat16*>(delta)[(int64_t)row * ldd + j] = __float2bfloat16_rn(d);
    else
      reinterpret_cast<float*>(delta)[(int64_t)row * ldd + j] = d;
  }
}

// The same with the row held in registers (C <= 32 * 4 * KV, ldl and ldd multiples of 4): one
// float4 read of the logits per chunk, exp evaluated once per entry, 8- or 16-byte stores of delta.
template <bool kBf16, int KV>
__global__ void softmax_xent_reg_kernel(const float* __restrict__ logits, int ldl,
                                        const int32_t* __restrict__ y, const float* __restrict__ scale,
                                        int N, int C, void* __restrict__ delta, int ldd,
                                        float* __restrict__ ce, DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  const int warps_per_block = blockDim.x >> 5;
  const int row = blockIdx.x * warps_per_block + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= N) return;
  const float* z = logits + (int64_t)row * ldl;
  int label = y[row];
  if (label < 0 || label >= C) {
    if (lane == 0) record_error(st, kDevBadLabel, row);
    label = label < 0 ? 0 : C - 1;
  }
  float v[KV][4];
  float mx = -INFINITY;
#pragma unroll
  for (int k = 0; k < KV; ++k) {
    const int j = 4 * (lane + 32 * k);
    float4 q = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    if (j < C) q = __ldg(reinterpret_cast<const float4*>(z + j));
    v[k][0] = q.x; v[k][1] = (j + 1 < C) ? q.y : -INFINITY;
    v[k][2] = (j + 2 < C) ? q.z : -INFINITY; v[k][3] = (j + 3 < C) ? q.w : -INFINITY;
#pragma unroll
    for (int e = 0; e < 4; ++e) mx = fmaxf(mx, v[k][e]);
  }
  mx = warp_max(mx);
  float se = 0.f;
#pragma unroll
  for (int k = 0; k < KV; ++k)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[k][e] = (4 * (lane + 32 * k) + e < C) ? expf(v[k][e] - mx) : 0.f;
      se += v[k][e];
    }
  se = warp_sum(se);
  const float lse = mx + logf(se);
  if (lane == 0) ce[row] = lse - z[label];
  const float inv = 1.0f / se;
  const float sc = scale[row];
#pragma unroll
  for (int k = 0; k < KV; ++k) {
    const int j = 4 * (lane + 32 * k);
    if (j >= ldd) break;
    float d[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) d[e] = (j + e < C) ? (v[k][e] * inv - (j + e == label ? 1.f : 0.f)) * sc : 0.f;
    if (kBf16) {
      __nv_bfloat162 a = __floats2bfloat162_rn(d[0], d[1]), b = __floats2bfloat162_rn(d[2], d[3]);
      uint2 o;
      o.x = *reinterpret_cast<uint32_t*>(&a);
      o.y = *reinterpret_cast<uint32_t*>(&b);
      *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(delta) + (int64_t)row * ldd + j) = o;
    } else {
      *reinterpret_cast<float4*>(reinterpret_cast<float*>(delta) + (int64_t)row * ldd + j) =
          make_float4(d[0], d[1], d[2], d[3]);
    }
  }
}

void launch_softmax_xent(const float* logits, int ldl, const int32_t* y, const float* scale, int N,
                         int C, void* delta, int ldd, bool delta_bf16, float* ce, DevStatus* st,
                         cudaStream_t s) {
  const int threads = 256;
  const int rows_per_block = threads / 32;
  const int blocks = (N + rows_per_block - 1) / rows_per_block;
  if (ldl % 4 == 0 && ldd % 4 == 0 && ldd <= 1024 && C <= ldd) {
    if (ldd <= 128) {
      if (delta_bf16) launch_pdl(softmax_xent_reg_kernel<true, 1>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
      else launch_pdl(softmax_xent_reg_kernel<false, 1>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
    } else {
      if (delta_bf16) launch_pdl(softmax_xent_reg_kernel<true, 8>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
      else launch_pdl(softmax_xent_reg_kernel<false, 8>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
    }
    return;
  }
  if (delta_bf16)
    launch_pdl(softmax_xent_kernel<true>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
  else
    launch_pdl(softmax_xent_kernel<false>, blocks, threads, 0, s, logits, ldl, y, scale, N, C, delta, ldd, ce, st);
}

// ------------------------------------------------------------------ per-worker loss reduction
// L_m = (1/n_m) sum_{i in seg_m} ce_i (Eq. 1); loss = sum_m w_m L_m.
// One block per worker: L_m = mean of its per-sample losses (strided partial sums, then a tree, in
// a fixed order); the last block to finish forms sum_m w_m L_m in worker order and resets the
// ticket for the next step.  With `delta`, the block also forms its worker's bias gradient of the
// output layer (width <= 32 columns, one lane per column): warp v sums rows b + v, b + v + 32, ...
// in row order, and the 32 warps' sums are added in warp order (deterministic); the two launches
// of the chunked bias-gradient reduction are then not needed for that layer.
constexpr int kLossThreads = 1024;

__global__ void __launch_bounds__(kLossThreads) loss_reduce_kernel(
    const float* __restrict__ ce, const int32_t* __restrict__ offsets, int M, const float* __restrict__ w,
    float* __restrict__ lm, DevStatus* st, unsigned int* ticket, const __nv_bfloat16* __restrict__ delta, int ld,
    int width, float* __restrict__ slabs, int64_t Ps, int64_t b_off) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[kLossThreads];
  __shared__ bool last;
  const int m = blockIdx.x;
  const int b = offsets[m], e = offsets[m + 1];
  float acc = 0.f;
  for (int i = b + threadIdx.x; i < e; i += blockDim.x) acc += ce[i];
  float bacc = 0.f;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (delta && lane < width) {
    int i = b + warp;
    for (; i + 96 < e; i += 128) {   // four rows in flight, added in row order
      const float v0 = __bfloat162float(delta[(int64_t)i * ld + lane]);
      const float v1 = __bfloat162float(delta[(int64_t)(i + 32) * ld + lane]);
      const float v2 = __bfloat162float(delta[(int64_t)(i + 64) * ld + lane]);
      const float v3 = __bfloat162float(delta[(int64_t)(i + 96) * ld + lane]);
      bacc += v0;
      bacc += v1;
      bacc += v2;
      bacc += v3;
    }
    for (; i < e; i += 32) bacc += __bfloat162float(delta[(int64_t)i * ld + lane]);
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int h = blockDim.x >> 1; h > 0; h >>= 1) {
    if (threadIdx.x < h) red[threadIdx.x] += red[threadIdx.x + h];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    lm[m] = red[0] / (float)(e - b);
    __threadfence();
    last = (atomicAdd(ticket, 1u) == (unsigned int)(M - 1));
  }
  __syncthreads();
  if (delta) {
    red[threadIdx.x] = bacc;   // [warp][lane]
    __syncthreads();
    if (threadIdx.x < width) {
      float t = 0.f;
      for (int v = 0; v < kLossThreads / 32; ++v) t += red[v * 32 + threadIdx.x];
      slabs[(int64_t)m * Ps + b_off + threadIdx.x] = t;
    }
  }
  if (last && threadIdx.x == 0) {
    __threadfence();
    const volatile float* lmv = lm;
    float loss = 0.f;
    for (int k = 0; k < M; ++k) loss += w[k] * lmv[k];
    st->loss = loss;
    *ticket = 0u;
  }
}

void launch_loss_reduce(const float* ce, const int32_t* d_offsets, int M, const float* d_w,
                        float* lm, DevStatus* st, unsigned int* ticket, cudaStream_t s) {
  launch_pdl(loss_reduce_kernel, M, kLossThreads, 0, s, ce, d_offsets, M, d_w, lm, st, ticket,
             (const __nv_bfloat16*)nullptr, 0, 0, (float*)nullptr, (int64_t)0, (int64_t)0);
}

int loss_bias_max_width() { return 32; }

void launch_loss_bias_reduce(const float* ce, const int32_t* d_offsets, int M, const float* d_w, float* lm,
                             DevStatus* st, unsigned int* ticket, const __nv_bfloat16* delta, int ld, int width,
                             float* slabs, int64_t Ps, int64_t b_off, cudaStream_t s) {
  launch_pdl(loss_reduce_kernel, M, kLossThreads, 0, s, ce, d_offsets, M, d_w, lm, st, ticket, delta, ld, width,
             slabs, Ps, b_off);
}

// Softmax cross-entropy, per-worker loss and the output layer's per-worker bias gradient in one
// launch, for at most 16 classes with bf16 delta (ldl % 4 == 0, ldd % 8 == 0, ldd <= 16): one block
// per worker, one thread per row of it (rows b + t, b + t + blockDim, ...).  Each row takes the
// arithmetic of softmax_xent (max, exp once per entry, ce = lse - z_y, delta_j = (e_j / se - [j = y])
// * scale_i, columns C..ldd-1 zero); then L_m = mean of the block's ce (per-thread sums, a tree) and
// the bias sums of the stored bf16 delta per class (each thread's rows in order, a warp xor tree,
// the warps' sums in warp order), deterministic; the last block forms sum_m w_m L_m as
// loss_reduce does.
constexpr int kSlbThreads = 512;
constexpr int kSlbMaxC = 16;

__global__ void __launch_bounds__(kSlbThreads) softmax_loss_bias_kernel(
    const float* __restrict__ logits, int ldl, const int32_t* __restrict__ y, const float* __restrict__ scale, int C,
    __nv_bfloat16* __restrict__ delta, int ldd, float* __restrict__ ce, const int32_t* __restrict__ offsets, int M,
    const float* __restrict__ w, float* __restrict__ lm, DevStatus* st, unsigned int* ticket,
    float* __restrict__ slabs, int64_t Ps, int64_t b_off) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[kSlbThreads];
  __shared__ float bred[kSlbThreads / 32][kSlbMaxC];
  __shared__ bool last;
  const int m = blockIdx.x;
  const int b = offsets[m], e = offsets[m + 1];
  float lacc = 0.f;
  float bsum[kSlbMaxC];
#pragma unroll
  for (int j = 0; j < kSlbMaxC; ++j) bsum[j] = 0.f;
  for (int i = b + (int)threadIdx.x; i < e; i += blockDim.x) {
    const float* zr = logits + (int64_t)i * ldl;
    float z[kSlbMaxC];
#pragma unroll
    for (int q = 0; q < kSlbMaxC / 4; ++q) {
      float4 v = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      if (4 * q < C) v = __ldg(reinterpret_cast<const float4*>(zr + 4 * q));
      z[4 * q] = v.x;
      z[4 * q + 1] = (4 * q + 1 < C) ? v.y : -INFINITY;
      z[4 * q + 2] = (4 * q + 2 < C) ? v.z : -INFINITY;
      z[4 * q + 3] = (4 * q + 3 < C) ? v.w : -INFINITY;
    }
    int label = y[i];
    if (label < 0 || label >= C) {
      record_error(st, kDevBadLabel, i);
      label = label < 0 ? 0 : C - 1;
    }
    float mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < kSlbMaxC; ++j) mx = fmaxf(mx, z[j]);
    float se = 0.f;
#pragma unroll
    for (int j = 0; j < kSlbMaxC; ++j) {
      z[j] = (j < C) ? expf(z[j] - mx) : 0.f;
      se += z[j];
    }
    const float cei = mx + logf(se) - __ldg(zr + label);
    ce[i] = cei;
    lacc += cei;
    const float inv = 1.0f / se;
    const float sc = scale[i];
    uint32_t pk[kSlbMaxC / 2];
#pragma unroll
    for (int j = 0; j < kSlbMaxC; j += 2) {
      const float d0 = (j < C) ? (z[j] * inv - (j == label ? 1.f : 0.f)) * sc : 0.f;
      const float d1 = (j + 1 < C) ? (z[j + 1] * inv - (j + 1 == label ? 1.f : 0.f)) * sc : 0.f;
      const __nv_bfloat162 q = __floats2bfloat162_rn(d0, d1);
      bsum[j] += __low2float(q);
      bsum[j + 1] += __high2float(q);
      pk[j / 2] = *reinterpret_cast<const uint32_t*>(&q);
    }
    uint4* drow = reinterpret_cast<uint4*>(delta + (int64_t)i * ldd);
    drow[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    if (ldd > 8) drow[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
  }
  red[threadIdx.x] = lacc;
  __syncthreads();
  for (int h = blockDim.x >> 1; h > 0; h >>= 1) {
    if (threadIdx.x < h) red[threadIdx.x] += red[threadIdx.x + h];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    lm[m] = red[0] / (float)(e - b);
    __threadfence();
    last = (atomicAdd(ticket, 1u) == (unsigned int)(M - 1));
  }
  const int warp = (int)threadIdx.x >> 5, lane = (int)threadIdx.x & 31;
#pragma unroll
  for (int j = 0; j < kSlbMaxC; ++j) {
    float v = bsum[j];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) bred[warp][j] = v;
  }
  __syncthreads();
  if ((int)threadIdx.x < C) {
    float t = 0.f;
    for (int v = 0; v < kSlbThreads / 32; ++v) t += bred[v][threadIdx.x];
    slabs[(int64_t)m * Ps + b_off + threadIdx.x] = t;
  }
  if (last && threadIdx.x == 0) {
    __threadfence();
    const volatile float* lmv = lm;
    float loss = 0.f;
    for (int k = 0; k < M; ++k) loss += w[k] * lmv[k];
    st->loss = loss;
    *ticket = 0u;
  }
}

bool softmax_loss_bias_ok(int C, int ldl, int ldd) {
  return C <= kSlbMaxC && ldd <= kSlbMaxC && ldd % 8 == 0 && ldl % 4 == 0 && C <= ldd && C <= ldl;
}

void launch_softmax_loss_bias(const float* logits, int ldl, const int32_t* y, const float* scale, int C,
                              __nv_bfloat16* delta, int ldd, float* ce, const int32_t* d_offsets, int M,
                              const float* d_w, float* lm, DevStatus* st, unsigned int* ticket, float* slabs,
                              int64_t Ps, int64_t b_off, cudaStream_t s) {
  launch_pdl(softmax_loss_bias_kernel, M, kSlbThreads, 0, s, logits, ldl, y, scale, C, delta, ldd, ce, d_offsets, M,
             d_w, lm, st, ticket, slabs, Ps, b_off);
}

// ------------------------------------------------------------------ per-worker bias gradient
// G_m[b_l][j] = sum_{i in seg_m} delta_l[i][j]: one thread per column, rows in order.
template <bool kBf16>
__global__ void bias_grad_kernel(const void* __restrict__ delta, int ld, int width,
                                 const int32_t* __restrict__ offsets, float* __restrict__ slabs,
                                 int64_t Ps, int64_t b_off) {
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.y;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= width) return;
  const int b = offsets[m], e = offsets[m + 1];
  // two-level sum (blocks of 256 rows) keeps the fp32 rounding of long segments small
  float tot = 0.f;
  for (int i0 = b; i0 < e; i0 += 256) {
    const int i1 = min(e, i0 + 256);
    float acc = 0.f;
#pragma unroll 8
    for (int i = i0; i < i1; ++i) {
      if (kBf16)
        acc += __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(delta)[(int64_t)i * ld + j]);
      else
        acc += reinterpret_cast<const float*>(delta)[(int64_t)i * ld + j];
    }
    tot += acc;
  }
  slabs[(int64_t)m * Ps + b_off + j] = tot;
}

// Two-stage form for bf16 delta (16-byte rows).  Stage 1: each block sums a chunk of <= 128 rows of
// one worker over 256 columns (a lane owns 8 adjacent columns, loaded as one 16-byte vector; the
// block's 8 warps take interleaved rows and are combined in a fixed order) into partial[chunk].
// Stage 2: per worker, the chunk partials are added in chunk order.  Deterministic.
constexpr int kBgRows = 128;
constexpr int kBgCols = 256;

__global__ void __launch_bounds__(256) bias_grad_partial_kernel(const __nv_bfloat16* __restrict__ delta, int ld,
                                                                int width, const int4* __restrict__ chunks,
                                                                float* __restrict__ partial) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[8][kBgCols + 8];
  const int4 ck = chunks[blockIdx.y];       // (worker, row begin, row end, unused)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c0 = blockIdx.x * kBgCols + lane * 8;
  float acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) acc[j] = 0.f;
  if (c0 < width) {
    const __nv_bfloat16* base = delta + c0;
    int r = ck.y + warp;
    for (; r + 24 < ck.z; r += 32) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = __ldcs(reinterpret_cast<const uint4*>(base + (int64_t)(r + 8 * u) * ld));
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v[u]);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[2 * j] += __low2float(h[j]);
          acc[2 * j + 1] += __high2float(h[j]);
        }
      }
    }
    for (; r < ck.z; r += 8) {
      const uint4 v = __ldcs(reinterpret_cast<const uint4*>(base + (int64_t)r * ld));
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        acc[2 * j] += __low2float(h[j]);
        acc[2 * j + 1] += __high2float(h[j]);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) red[warp][lane * 8 + j] = acc[j];
  __syncthreads();
  const int col = blockIdx.x * kBgCols + threadIdx.x;
  if (col < width) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += red[w][threadIdx.x];
    partial[(int64_t)blockIdx.y * width + col] = t;
  }
}

__global__ void bias_grad_combine_kernel(const float* __restrict__ partial, int width,
                                         const int32_t* __restrict__ chunk_begin, float* __restrict__ slabs,
                                         int64_t Ps, int64_t b_off) {
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.y;
  const int col = blockIdx.x * blockDim.x + threadIdx.x;
  if (col >= width) return;
  float t = 0.f;
  for (int c = chunk_begin[m]; c < chunk_begin[m + 1]; ++c) t += partial[(int64_t)c * width + col];
  slabs[(int64_t)m * Ps + b_off + col] = t;
}

int bias_grad_chunk_rows() { return kBgRows; }

void launch_bias_grad_bf16(const __nv_bfloat16* delta, int ld, int width, const int4* d_chunks, int n_chunks,
                           const int32_t* d_chunk_begin, int M, float* partial, float* slabs, int64_t Ps,
                           int64_t b_off, cudaStream_t s) {
  dim3 g1((width + kBgCols - 1) / kBgCols, n_chunks);
  launch_pdl(bias_grad_partial_kernel, g1, 256, 0, s, delta, ld, width, d_chunks, partial);
  dim3 g2((width + 255) / 256, M);
  launch_pdl(bias_grad_combine_kernel, g2, 256, 0, s, partial, width, d_chunk_begin, slabs, Ps, b_off);
}

void launch_bias_grad(const void* delta, bool delta_bf16, int ld, int width, const int32_t* d_offsets,
                      int M, float* slabs, int64_t Ps, int64_t b_off, cudaStream_t s) {
  dim3 grid((width + 127) / 128, M);
  if (delta_bf16)
    launch_pdl(bias_grad_kernel<true>, grid, 128, 0, s, delta, ld, width, d_offsets, slabs, Ps, b_off);
  else
    launch_pdl(bias_grad_kernel<false>, grid, 128, 0, s, delta, ld, width, d_offsets, slabs, Ps, b_off);
}

// ------------------------------------------------------------------ fused reduce + SGD update
// Section 1: g = sum_m w_m g^m (w_m = 1/M; Section 4.2: compute-power weights), then
// theta <- theta - lr * g.  One HBM pass: M slab reads + theta read, theta + bf16 shadow writes.
// kRecipe: the Section 5 training recipe on top of g: d = g + wd*theta, b = d (first step) or
// mu*b + d, theta <- theta - lr*b, with b kept in `mbuf` (one more read and write per parameter).
template <bool kRecipe>
__device__ __forceinline__ float apply_update(float t, float g, float lr, float* mb, float mu, float wd, int first) {
  if (!kRecipe) return fmaf(-lr, g, t);
  const float d = fmaf(wd, t, g);
  const float b = first ? d : fmaf(mu, *mb, d);
  *mb = b;
  return fmaf(-lr, b, t);
}

template <bool kRecipe>
__global__ void __launch_bounds__(512) reduce_update_kernel(
    float* __restrict__ theta, const float* __restrict__ slabs, int64_t Ps, int M,
    const float* __restrict__ w, float lr_arg, const float* __restrict__ lr_dev, int64_t P,
    __nv_bfloat16* __restrict__ shadow, float* __restrict__ gdebug, float* __restrict__ mbuf, float mu, float wd,
    int first) {
  pdl_wait();
  pdl_trigger();
  // the step's learning rate: the argument, or (a step replayed from a CUDA graph) device memory
  const float lr = lr_dev ? __ldg(lr_dev) : lr_arg;
  // The weights stay in global memory (read through the read-only cache): no shared memory, so
  // blocks of this kernel can share an SM with a resident tensor-core GEMM CTA.
  const float* __restrict__ sw = w;
  const int64_t nvec = P / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const float4* s4 = reinterpret_cast<const float4*>(slabs);
  const int64_t ps4 = Ps / 4;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    int m = 0;
    for (; m + 8 <= M; m += 8) {
      float4 g[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) g[u] = __ldcs(s4 + (int64_t)(m + u) * ps4 + v);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float wm = __ldg(sw + m + u);
        acc.x = fmaf(wm, g[u].x, acc.x);
        acc.y = fmaf(wm, g[u].y, acc.y);
        acc.z = fmaf(wm, g[u].z, acc.z);
        acc.w = fmaf(wm, g[u].w, acc.w);
      }
    }
    for (; m < M; ++m) {
      const float4 g = __ldcs(s4 + (int64_t)m * ps4 + v);
      const float wm = __ldg(sw + m);
      acc.x = fmaf(wm, g.x, acc.x);
      acc.y = fmaf(wm, g.y, acc.y);
      acc.z = fmaf(wm, g.z, acc.z);
      acc.w = fmaf(wm, g.w, acc.w);
    }
    float4 t = reinterpret_cast<float4*>(theta)[v];
    if (kRecipe) {
      float4 b = first ? make_float4(0.f, 0.f, 0.f, 0.f) : reinterpret_cast<const float4*>(mbuf)[v];
      t.x = apply_update<true>(t.x, acc.x, lr, &b.x, mu, wd, first);
      t.y = apply_update<true>(t.y, acc.y, lr, &b.y, mu, wd, first);
      t.z = apply_update<true>(t.z, acc.z, lr, &b.z, mu, wd, first);
      t.w = apply_update<true>(t.w, acc.w, lr, &b.w, mu, wd, first);
      reinterpret_cast<float4*>(mbuf)[v] = b;
    } else {
      t.x = fmaf(-lr, acc.x, t.x);
      t.y = fmaf(-lr, acc.y, t.y);
      t.z = fmaf(-lr, acc.z, t.z);
      t.w = fmaf(-lr, acc.w, t.w);
    }
    reinterpret_cast<float4*>(theta)[v] = t;
    if (shadow) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(t.x, t.y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(t.z, t.w);
      uint2 packed;
      packed.x = *reinterpret_cast<uint32_t*>(&lo);
      packed.y = *reinterpret_cast<uint32_t*>(&hi);
      reinterpret_cast<uint2*>(shadow)[v] = packed;
    }
    if (gdebug) reinterpret_cast<float4*>(gdebug)[v] = acc;
  }
  for (int64_t j = nvec * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < P; j += stride) {
    float acc = 0.f;
    for (int m = 0; m < M; ++m) acc = fmaf(__ldg(sw + m), slabs[(int64_t)m * Ps + j], acc);
    const float t = apply_update<kRecipe>(theta[j], acc, lr, kRecipe ? mbuf + j : nullptr, mu, wd, first);
    theta[j] = t;
    if (shadow) shadow[j] = __float2bfloat16_rn(t);
    if (gdebug) gdebug[j] = acc;
  }
}

void launch_reduce_update(float* theta, const float* slabs, int64_t Ps, int M, const float* d_w,
                          float lr, int64_t P, __nv_bfloat16* shadow, float* gdebug, int num_sms,
                          cudaStream_t s, int blocks_per_sm, const UpdateRecipe* recipe, const float* lr_dev) {
  const int threads = 512;
  int64_t blocks = (P / 4 + threads - 1) / threads;
  const int64_t cap = (int64_t)num_sms * blocks_per_sm;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  if (recipe && recipe->buf)
    launch_pdl(reduce_update_kernel<true>, (int)blocks, threads, 0, s, theta, slabs, Ps, M, d_w, lr, lr_dev, P, shadow,
               gdebug, recipe->buf, recipe->momentum, recipe->weight_decay, recipe->first);
  else
    launch_pdl(reduce_update_kernel<false>, (int)blocks, threads, 0, s, theta, slabs, Ps, M, d_w, lr, lr_dev, P, shadow,
               gdebug, nullptr, 0.f, 0.f, 0);
}

// *dst = v: the learning rate of a step replayed from a CUDA graph, written ahead of the replay.
__global__ void set_scalar_kernel(float* dst, float v) { *dst = v; }

void launch_set_scalar(float* dst, float v, cudaStream_t s) { set_scalar_kernel<<<1, 1, 0, s>>>(dst, v); }

}  // namespace hs
