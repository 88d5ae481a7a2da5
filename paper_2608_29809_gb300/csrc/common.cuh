// Shared device helpers of the region-sparse DiT library (sm_103a).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace rc {

// Device error-word bits (reported by rc_sync).
enum : unsigned {
  DEVERR_INDEX = 1u,    // a dirty index outside [0, N)
  DEVERR_COUNT = 2u,    // a device dirty count outside [0, bound]
  DEVERR_TIMEOUT = 4u,  // a bounded wait gave up
};

__device__ __forceinline__ float bf2f(__nv_bfloat16 v) { return __bfloat162float(v); }
__device__ __forceinline__ __nv_bfloat16 f2bf(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float2 unpack_bf16x2(uint32_t u) {
  __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
  return __bfloat1622float2(v);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// tanh on the special-function unit (relative error about 2^-11, below the
// bf16 rounding of every GELU output)
__device__ __forceinline__ float tanh_sfu(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float gelu_tanh(float z) {
  const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
  float inner = k0 * (z + 0.044715f * z * z * z);
  return 0.5f * z * (1.0f + tanh_sfu(inner));
}

__device__ __forceinline__ float silu(float z) { return z / (1.0f + expf(-z)); }

// Resolves the live dirty count: the device count when given (checked against
// the bound; a bad value raises DEVERR_COUNT and is treated as 0), else the
// host count.
__device__ __forceinline__ int live_count(const int* dcount, int bound, unsigned* err) {
  if (dcount == nullptr) return bound;
  int d = *dcount;
  if (d < 0 || d > bound) {
    if (err) atomicOr(err, DEVERR_COUNT);
    return 0;
  }
  return d;
}

// Programmatic dependent launch.  Every kernel of this library is launched
// with programmatic stream serialisation: it may start while its predecessor
// in the stream is still running, does its private set-up, then waits
// (griddepcontrol.wait) for the predecessor to complete before it touches
// any data another kernel writes, and lets its own successor start early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

}  // namespace rc

#ifndef __CUDACC_RTC__
namespace rc {
// Launches `kernel` on `st` with programmatic stream serialisation allowed.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
// launch_k with thread-block clusters of `cluster` CTAs along x.
template <class... KArgs, class... Args>
inline cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                    int cluster, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = unsigned(cluster);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
}  // namespace rc
#define RC_TRY(call)                         \
  do {                                       \
    cudaError_t e__ = (call);                \
    if (e__ != cudaSuccess) return e__;      \
  } while (0)
#endif
