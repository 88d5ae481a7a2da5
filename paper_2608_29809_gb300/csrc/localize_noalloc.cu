// rc_localize_mask_noalloc: the localisation mask with its scratch in a fixed
// device array of this library instead of a caller workspace, for callers
// that cannot allocate device memory (see include/regioncache.h).
#include <stdio.h>

#include <mutex>

#include "../../include/regioncache.h"
#include "kernels.h"

namespace {

// Scratch of every rc_localize_mask_noalloc call on a device: the workspace
// of the largest allowed problem (RC_NOALLOC_MAX_TOKENS tokens,
// RC_NOALLOC_MAX_DELTA delta tokens), checked against the workspace formula
// at every call.
static __device__ __align__(256) unsigned char g_noalloc_scratch[RC_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device, looked up once per
// device with that device current.  In host code the array's name is only a
// host-side stand-in, never a device address.
cudaError_t scratch_on_current_device(void** out, int* dev_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  *dev_out = dev;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" rc_status rc_localize_mask_noalloc(const float* xattn, int S, int N, int M, int grid_h,
                                              int grid_w, const int32_t* delta_ids_host,
                                              int n_delta, float threshold, int dilation,
                                              uint8_t* mask, int32_t* dirty_idx,
                                              int32_t* dirty_count, rc_stream stream) {
  char msg[256];
  if (N > RC_NOALLOC_MAX_TOKENS || n_delta > RC_NOALLOC_MAX_DELTA) {
    snprintf(msg, sizeof(msg),
             "rc_localize_mask_noalloc: N = %d, n_delta = %d exceed the fixed scratch "
             "(N <= %d, n_delta <= %d); use rc_localize_mask with a workspace",
             N, n_delta, RC_NOALLOC_MAX_TOKENS, RC_NOALLOC_MAX_DELTA);
    rc::set_last_error(msg);
    return RC_ERR_SHAPE;
  }
  if (N >= 1 && n_delta >= 1 &&
      rc::localize_workspace_bytes(N, n_delta) > size_t(RC_NOALLOC_SCRATCH_BYTES)) {
    snprintf(msg, sizeof(msg), "rc_localize_mask_noalloc: needs %zu scratch bytes > %d",
             rc::localize_workspace_bytes(N, n_delta), RC_NOALLOC_SCRATCH_BYTES);
    rc::set_last_error(msg);
    return RC_ERR_SHAPE;
  }
  void* scratch = nullptr;
  int dev = -1;
  cudaError_t e = scratch_on_current_device(&scratch, &dev);
  if (e != cudaSuccess) {
    snprintf(msg, sizeof(msg), "rc_localize_mask_noalloc: scratch address on device %d: %s",
             dev, cudaGetErrorString(e));
    rc::set_last_error(msg);
    return RC_ERR_CUDA;
  }
  // Same validation and kernels as rc_localize_mask, with the fixed scratch.
  return rc_localize_mask(xattn, S, N, M, grid_h, grid_w, delta_ids_host, n_delta, threshold,
                          dilation, mask, dirty_idx, dirty_count, scratch,
                          size_t(RC_NOALLOC_SCRATCH_BYTES), stream);
}
