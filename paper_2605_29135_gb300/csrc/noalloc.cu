// Routing (router GEMV, top-k, gates) for callers that cannot allocate device memory.
//
// Some callers run where cudaMalloc is not an option: an allocator-free inference runtime that
// owns all device memory up front, code that runs while another component holds the allocator
// lock, or a plug-in whose host process forbids device allocations after start-up. This entry
// point needs no handle and allocates nothing: the router logits live in a fixed device array
// of this file, so the caller only passes its own inputs and outputs.
//
// The scratch array is shared by every call in the process (on each device that loads the
// library it occupies MOE_NOALLOC_MAX_ROWS * MOE_NOALLOC_MAX_EXPERTS floats until exit). Each
// call overwrites the logits it later reads, so nothing in it has to start at zero; two calls
// whose work overlaps on the GPU (different streams, or different host threads) race on it.
//
// The arithmetic is the same as the router phase of the device-driven decode step: lane-owned
// 16-byte chunks in ascending order, a fixed XOR-shuffle reduction, fp32 accumulation, top-k by
// an order-preserving key with ties to the lower expert id, gates as a softmax over the k
// selected logits (or the full-softmax probabilities when renorm is 0).
#include <cuda_runtime.h>

#include <mutex>

#include "dev.cuh"
#include "moe.h"
#include "topk.cuh"

namespace {

using namespace moe;
using namespace moe::dev;

static __device__ __align__(256) float g_route_scratch[MOE_NOALLOC_MAX_ROWS * MOE_NOALLOC_MAX_EXPERTS];

constexpr int kMaxDevices = 64;
std::mutex g_lock;
float* g_scratch_addr[kMaxDevices] = {};

// Logits z[b][e] = W_r[e] . h_b; one warp per (row, expert), h_b staged in shared memory.
template <int WD>
__global__ void __launch_bounds__(256) k_route_logits(const uint8_t* w, const uint8_t* hidden, int E, int d,
                                                      float* z) {
  extern __shared__ uint4 xs4[];
  const uint8_t* xs = reinterpret_cast<const uint8_t*>(xs4);
  const int xbytes = d * (WD == WD_FP32 ? 4 : 2);
  const int b = blockIdx.y;
  stage16(xs4, hidden + (int64_t)b * xbytes, xbytes, threadIdx.x, blockDim.x);
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int e = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (e >= E) return;
  const uint8_t* row = w + (int64_t)e * xbytes;
  const int nch = xbytes / 16;
  float acc = 0.f;
  for (int c = lane; c < nch; c += 32) acc = dot_chunk<WD>(ld_stream(row + (int64_t)c * 16), xs + (int64_t)c * 16, acc);
  acc = warp_sum(acc);
  if (lane == 0) z[b * MOE_NOALLOC_MAX_EXPERTS + e] = acc;
}

// Top-k and gates of row blockIdx.x, one warp: the decode kernels' own selection code.
__global__ void __launch_bounds__(32) k_route_select(const float* z, int E, int k, int renorm, int32_t* idx,
                                                    float* gate) {
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  int my_i;
  float my_g;
  warp_topk(z + b * MOE_NOALLOC_MAX_EXPERTS, E, k, renorm, lane, my_i, my_g);
  if (lane < k) {
    idx[b * k + lane] = my_i;
    gate[b * k + lane] = my_g;
  }
}

// Device address of the scratch array on the current device, looked up once per device.
cudaError_t scratch_for_current_device(float** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> g(g_lock);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_route_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" moe_status moe_route_noalloc(const void* w_r, const void* hidden, int32_t rows, int32_t n_experts,
                                        int32_t d, int32_t top_k, int32_t renorm, int32_t wdtype, int32_t* idx,
                                        float* gate, void* stream) {
  if (!w_r || !hidden || !idx || !gate) return MOE_ERR_INVALID;
  if (rows > MOE_NOALLOC_MAX_ROWS || n_experts > MOE_NOALLOC_MAX_EXPERTS) return MOE_ERR_CAPACITY;
  if (rows < 1 || n_experts < 1 || top_k < 1 || top_k > 16 || top_k > n_experts || d < 1 ||
      (renorm != 0 && renorm != 1))
    return MOE_ERR_INVALID;
  if (wdtype != MOE_DTYPE_FP32 && wdtype != MOE_DTYPE_BF16) return MOE_ERR_INVALID;
  const int xbytes = d * (wdtype == MOE_DTYPE_FP32 ? 4 : 2);
  if (xbytes % 16 != 0 || xbytes > 48 * 1024) return MOE_ERR_INVALID;
  // w_r and hidden are read as 16-byte vectors, idx and gate written as 4-byte words: a
  // misaligned pointer is refused here rather than faulting the launch
  if ((((uintptr_t)w_r | (uintptr_t)hidden) & 15) != 0 || (((uintptr_t)idx | (uintptr_t)gate) & 3) != 0)
    return MOE_ERR_INVALID;
  float* z = nullptr;
  if (scratch_for_current_device(&z) != cudaSuccess) return MOE_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  const dim3 grid((n_experts + 7) / 8, rows);
  if (wdtype == MOE_DTYPE_FP32)
    k_route_logits<WD_FP32><<<grid, 256, xbytes, s>>>((const uint8_t*)w_r, (const uint8_t*)hidden, n_experts, d, z);
  else
    k_route_logits<WD_BF16><<<grid, 256, xbytes, s>>>((const uint8_t*)w_r, (const uint8_t*)hidden, n_experts, d, z);
  if (cudaGetLastError() != cudaSuccess) return MOE_ERR_CUDA;
  k_route_select<<<rows, 32, 0, s>>>(z, n_experts, top_k, renorm, idx, gate);
  if (cudaGetLastError() != cudaSuccess) return MOE_ERR_CUDA;
  return MOE_OK;
}
