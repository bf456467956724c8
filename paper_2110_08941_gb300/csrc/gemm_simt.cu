// fp32 CUDA-core GEMM for the HS_FP32_CHECK precision: the same contractions as the
// tensor-core path (forward, input-gradient and per-worker weight-gradient products of
// Eq. 1's per-worker losses), in plain fp32 FMA so the step can be compared with the fp64
// oracle at a tight tolerance.  Not a performance path.
#include "common.cuh"

namespace hs {

namespace {

constexpr int BM = 64, BN = 64, BK = 16;

// Acc = double for the forward products: the ReLU' decisions taken from their results then match
// an exact evaluation on the same fp32 operands; float (two-level) for the backward products.
template <typename Acc>
__global__ void __launch_bounds__(256) gemm_f32_kernel(GemmF32Args a) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int g = blockIdx.z;
  int kbeg = 0, kend = a.Kdim;
  float* C = a.C;
  if (a.k_offsets) {
    kbeg = a.k_offsets[g];
    kend = a.k_offsets[g + 1];
    C += (int64_t)g * a.c_gstride;
  }
  const bool a_kmajor = (a.a_sk == 1);
  const bool b_kmajor = (a.b_sk == 1);
  // Two-level fp32 sum: `acc` collects 16 k-tiles (256 products), then folds into `tot`, so the
  // rounding error grows with sqrt(256) + sqrt(K / 256) instead of sqrt(K) for long K (the
  // per-worker weight gradients of the convolutions sum over n_m * Ho * Wo rows).
  Acc acc[4][4], tot[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = tot[i][j] = 0.f;

  int tiles_done = 0;
  for (int k0 = kbeg; k0 < kend; k0 += BK) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int idx = tid + r * 256;
      int mm, kk;
      if (a_kmajor) { mm = idx / BK; kk = idx % BK; } else { mm = idx % BM; kk = idx / BM; }
      const int gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < a.Mdim && gk < kend) ? a.A[(int64_t)gm * a.a_sm + (int64_t)gk * a.a_sk] : 0.f;
      int nn;
      if (b_kmajor) { nn = idx / BK; kk = idx % BK; } else { nn = idx % BN; kk = idx / BN; }
      const int gn = n0 + nn;
      const int gk2 = k0 + kk;
      Bs[kk][nn] = (gn < a.Ndim && gk2 < kend) ? a.B[(int64_t)gk2 * a.b_sk + (int64_t)gn * a.b_sn] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float ar[4] = {av.x, av.y, av.z, av.w};
      const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fma((Acc)ar[i], (Acc)br[j], acc[i][j]);
    }
    __syncthreads();
    if (++tiles_done == 16) {
      tiles_done = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          tot[i][j] += acc[i][j];
          acc[i][j] = 0.f;
        }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] += tot[i][j];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= a.Mdim) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx * 4 + j;
      if (gn >= a.Ndim) continue;
      Acc v = acc[i][j];
      switch (a.epi) {
        case kEpiBias: v += (Acc)a.bias[gn]; break;
        case kEpiBiasRelu: v = v + (Acc)a.bias[gn] > (Acc)0 ? v + (Acc)a.bias[gn] : (Acc)0; break;
        case kEpiMask: v = (a.Z[(int64_t)gm * a.ldz + gn] > 0.f) ? v : (Acc)0; break;
        default: break;
      }
      C[(int64_t)gm * a.ldc + gn] = (float)v;
    }
  }
}

}  // namespace

void launch_gemm_f32(const GemmF32Args& a, cudaStream_t s) {
  if (a.Mdim <= 0 || a.Ndim <= 0) return;
  dim3 grid((a.Ndim + BN - 1) / BN, (a.Mdim + BM - 1) / BM, a.k_offsets ? a.groups : 1);
  if (a.epi == kEpiBias || a.epi == kEpiBiasRelu)
    gemm_f32_kernel<double><<<grid, 256, 0, s>>>(a);
  else
    gemm_f32_kernel<float><<<grid, 256, 0, s>>>(a);
}

}  // namespace hs
