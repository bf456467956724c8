// hs_partition_noalloc: the sample -> worker map of Algorithm 1 for callers that cannot allocate
// device memory.
//
// hs_partition needs a context, and hs_init allocates the whole training workspace (gradient
// slabs, activations: gigabytes).  Some callers only want the partition and the device-side
// index map and cannot call cudaMalloc at all: a data-loading process that shares the GPU under a
// fixed memory budget, code running inside an allocator that forbids new device allocations after
// start-up, or a host thread that must not take the allocator's locks.  This entry point needs no
// context and allocates nothing: the one piece of device scratch it uses - the table of segment
// offsets the kernel searches - lives in a file-scope static device array of fixed size, present
// on every GPU that loads the library until the process exits.
#include <mutex>
#include <string>

#include "common.cuh"

namespace hs {
namespace {

constexpr int kNoAllocMaxWorkers = 1024;   // offsets table: 1025 int32 (4.1 KB)
constexpr int kNoAllocMaxDevices = 64;

// Device scratch shared by every call on a device: offsets[0..M] of the last call.
static __device__ __align__(256) int32_t g_noalloc_offsets[kNoAllocMaxWorkers + 1];

// Host-side device addresses of g_noalloc_offsets, one per device, filled on first use.
std::mutex g_setup_mu;
int32_t* g_offsets_addr[kNoAllocMaxDevices] = {nullptr};

// index_map[i] = m for offsets[m] <= i < offsets[m+1]; `offsets` is the static table's device address.
__global__ void index_map_from_static_offsets(const int32_t* __restrict__ offsets, int M, int N,
                                              int32_t* __restrict__ index_map) {
  __shared__ int32_t s_off[kNoAllocMaxWorkers + 1];
  for (int k = threadIdx.x; k <= M; k += blockDim.x) s_off[k] = offsets[k];
  __syncthreads();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  int lo = 0, hi = M - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_off[mid] <= i) lo = mid; else hi = mid - 1;
  }
  index_map[i] = lo;
}

hs_status fail(hs_status s, const char* msg) {
  set_init_error(msg);   // reported by hs_last_init_error()
  return s;
}

}  // namespace
}  // namespace hs

extern "C" hs_status hs_partition_noalloc(int32_t M, int32_t N, const double* cp, int32_t* counts_out,
                                          int32_t* index_map_out, void* stream) {
  using namespace hs;
  set_init_error("");
  if (M < 1 || M > kNoAllocMaxWorkers)
    return fail(HS_ERR_INVALID_ARG, "hs_partition_noalloc: M must be in [1, 1024] (size of its static offsets table)");
  if (!cp || !index_map_out) return fail(HS_ERR_INVALID_ARG, "hs_partition_noalloc: cp and index_map_out are required");
  int32_t sizes[kNoAllocMaxWorkers];
  double cpn[kNoAllocMaxWorkers];
  const char* why = nullptr;
  hs_status st = partition_sizes_impl(M, N, cp, sizes, cpn, &why);
  if (st != HS_OK) return fail(st, why);
  int32_t offsets[kNoAllocMaxWorkers + 1];
  offsets[0] = 0;
  for (int m = 0; m < M; ++m) offsets[m + 1] = offsets[m] + sizes[m];

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices) {
    cudaGetLastError();
    return fail(HS_ERR_CUDA, "hs_partition_noalloc: no usable current CUDA device");
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (s) {
    // The table's address is per device: a stream of another device would get the wrong one.
    int sdev = -1;
    if (cudaStreamGetDevice(s, &sdev) != cudaSuccess) {
      cudaGetLastError();
      return fail(HS_ERR_INVALID_ARG, "hs_partition_noalloc: stream is not a valid CUDA stream");
    }
    if (sdev != dev)
      return fail(HS_ERR_INVALID_ARG, "hs_partition_noalloc: stream belongs to another device than the current one");
  }
  int32_t* d_off = nullptr;
  {
    // Set-up, once per device with that device current: the host-side name of the static array is
    // not a device address, so look the address up and keep it.
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_offsets_addr[dev]) {
      void* p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_offsets);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        return fail(HS_ERR_CUDA, "hs_partition_noalloc: cudaGetSymbolAddress failed for the static offsets table");
      }
      g_offsets_addr[dev] = static_cast<int32_t*>(p);
    }
    d_off = g_offsets_addr[dev];
  }
  // Pageable source: the copy is staged before the call returns, so the stack table may go away.
  cudaError_t e = cudaMemcpyAsync(d_off, offsets, sizeof(int32_t) * (M + 1), cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return fail(HS_ERR_CUDA, cudaGetErrorString(e));
  const int threads = 256;
  index_map_from_static_offsets<<<(N + threads - 1) / threads, threads, 0, s>>>(d_off, M, N, index_map_out);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(HS_ERR_CUDA, cudaGetErrorString(e));
  if (counts_out)
    for (int m = 0; m < M; ++m) counts_out[m] = sizes[m];
  return HS_OK;
}
