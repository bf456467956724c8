// Internal declarations shared by the translation units of libhs (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/hs.h"

namespace hs {

constexpr int kMaxWorkers = 1024;

// Device-side error codes written to the context's status word (first error wins).
enum DevErr : int32_t {
  kDevOk = 0,
  kDevWaitTimeout = 1,   // a bounded mbarrier wait in a tensor-core kernel expired
  kDevBadLabel = 2,      // a label outside [0, classes) reached the loss kernel
};

// Programmatic dependent launch for the elementwise and reduction kernels (the tensor-core kernels
// do the same after their prologue): a kernel launched by launch_pdl may start while the previous
// kernel of its stream is finishing, so it first waits for that kernel's completion (pdl_wait, its
// first statement, before any global-memory access), then releases the next one (pdl_trigger).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

struct DevStatus {
  float loss;         // sum_m w_m L_m of the last step
  int32_t err;        // DevErr
  int32_t err_info;   // kernel-specific detail (which wait / which row)
};

hs_status partition_sizes_impl(int32_t M, int32_t N, const double* cp, int32_t* sizes,
                               double* cp_norm, const char** why);
// Sets the calling thread's message returned by hs_last_init_error() (calls without a context).
void set_init_error(const char* msg);

// ---------------------------------------------------------------- elementwise / reduction kernels
void launch_cast_f32_bf16(const float* x, __nv_bfloat16* y, int64_t n, cudaStream_t s);
void launch_partition_scatter(const int32_t* d_offsets, int M, int N, int32_t* index_map,
                              float* scale, int32_t* index_map_out, cudaStream_t s);
// out[i] = w[index_map[i]] * scale[i]
void launch_scale_by_weight(const int32_t* index_map, const float* scale, const float* w, int N, float* out,
                            cudaStream_t s);
// logits [N, ldl] fp32 -> ce[N], delta [N, ldd] (bf16 if delta_bf16 else fp32, columns >= C zeroed)
void launch_softmax_xent(const float* logits, int ldl, const int32_t* y, const float* scale, int N,
                         int C, void* delta, int ldd, bool delta_bf16, float* ce, DevStatus* st,
                         cudaStream_t s);
void launch_loss_reduce(const float* ce, const int32_t* d_offsets, int M, const float* d_w,
                        float* lm, DevStatus* st, unsigned int* ticket, cudaStream_t s);
// The same, and in the same launch the last layer's per-worker bias gradients from its bf16 delta
// (width <= loss_bias_max_width()): slabs[m*Ps + b_off + j] = sum_{i in seg_m} delta[i*ld + j].
int loss_bias_max_width();
// softmax_xent + launch_loss_bias_reduce in one launch (bf16 delta; at most 16 classes, ldd % 8 == 0,
// ldd <= 16, ldl % 4 == 0): softmax_loss_bias_ok says whether the shapes allow it.
bool softmax_loss_bias_ok(int C, int ldl, int ldd);
void launch_softmax_loss_bias(const float* logits, int ldl, const int32_t* y, const float* scale, int C,
                              __nv_bfloat16* delta, int ldd, float* ce, const int32_t* d_offsets, int M,
                              const float* d_w, float* lm, DevStatus* st, unsigned int* ticket, float* slabs,
                              int64_t Ps, int64_t b_off, cudaStream_t s);
void launch_loss_bias_reduce(const float* ce, const int32_t* d_offsets, int M, const float* d_w, float* lm,
                             DevStatus* st, unsigned int* ticket, const __nv_bfloat16* delta, int ld, int width,
                             float* slabs, int64_t Ps, int64_t b_off, cudaStream_t s);
// slabs[m*Ps + b_off + j] = sum_{i in seg_m} delta[i*ld + j], j < width
void launch_bias_grad(const void* delta, bool delta_bf16, int ld, int width, const int32_t* d_offsets,
                      int M, float* slabs, int64_t Ps, int64_t b_off, cudaStream_t s);
// Same reduction for bf16 delta with 16-byte rows (ld % 8 == 0): row chunks (worker, begin, end) of at
// most bias_grad_chunk_rows() rows, chunk_begin[m] = first chunk of worker m (M + 1 entries), partial
// scratch of n_chunks x width floats.  Launches two kernels.
int bias_grad_chunk_rows();
void launch_bias_grad_bf16(const __nv_bfloat16* delta, int ld, int width, const int4* d_chunks, int n_chunks,
                           const int32_t* d_chunk_begin, int M, float* partial, float* slabs, int64_t Ps,
                           int64_t b_off, cudaStream_t s);
// theta[j] -= lr * sum_m w[m] * slabs[m*Ps + j]; shadow[j] = bf16(theta[j]); gdebug[j] = g (optional)
// Works on any contiguous parameter range (pointers offset to its start, 16-byte aligned; slab m
// of the range at slabs + m*Ps).  blocks_per_sm = 1 leaves room for a resident GEMM CTA.
// The Section 5 recipe (momentum buffer at `buf`, offset like theta); null = plain SGD.
struct UpdateRecipe {
  float* buf;
  float momentum, weight_decay;
  int first;   // 1: the buffer starts as d (first step after the recipe was set)
};
// lr_dev: when non-null the kernel reads the learning rate there (a step replayed from a CUDA
// graph) instead of taking `lr`.
void launch_reduce_update(float* theta, const float* slabs, int64_t Ps, int M, const float* d_w,
                          float lr, int64_t P, __nv_bfloat16* shadow, float* gdebug, int num_sms,
                          cudaStream_t s, int blocks_per_sm = 4, const UpdateRecipe* recipe = nullptr,
                          const float* lr_dev = nullptr);
void launch_set_scalar(float* dst, float v, cudaStream_t s);

// ---------------------------------------------------------------- fp32 CUDA-core GEMM (check path)
// C(m, n) = sum_k A(m, k) B(k, n) with A(m,k) = A[m*a_sm + k*a_sk], B(k,n) = B[k*b_sk + n*b_sn],
// C[m*ldc + n].  Grouped form: blockIdx.z = g runs k over [k_offsets[g], k_offsets[g+1]) and writes
// C + g*c_gstride.  Epilogues below.
enum Epi : int32_t {
  kEpiStore = 0,      // C = acc
  kEpiBias = 1,       // C = acc + bias[n]
  kEpiBiasRelu = 2,   // C = max(acc + bias[n], 0)
  kEpiMask = 3,       // C = acc * (Z(m, n) > 0)
};

struct GemmF32Args {
  const float* A; int64_t a_sm, a_sk;
  const float* B; int64_t b_sk, b_sn;
  float* C; int64_t ldc;
  int Mdim, Ndim, Kdim;
  int epi;
  const float* bias;
  const float* Z; int64_t ldz;
  const int32_t* k_offsets;   // grouped if non-null
  int groups;
  int64_t c_gstride;
};
void launch_gemm_f32(const GemmF32Args& a, cudaStream_t s);

}  // namespace hs
