// kvr_noalloc.cu -- kvr_decode_attend_score_noalloc: the attend+score step
// with its logit scratch in a static device array owned by the library.
//
// Who needs it: callers that cannot allocate device memory for a call.  A
// plug-in loaded into a host program that owns every device allocation (and
// hands the plug-in nothing but a call's tensors), or a service that fixes
// its device footprint at start-up and may not allocate afterwards, cannot
// provide working memory beyond the tensors it already has.  This entry
// point keeps the logits of every unit of the call in g_noalloc_logits
// instead of in the cache buffer's scratch area, and calls no allocator.
//
// Rules of use (also stated in include/kvr.h):
//  - The array is KVR_NOALLOC_SCRATCH_BYTES; a call whose logits would not
//    fit is rejected with KVR_EINVAL before anything is enqueued.
//  - Every GPU that loads the library holds the array until the process
//    exits.
//  - The first call on a device looks up the array's device address with
//    cudaGetSymbolAddress (a host-side stand-in is all the host sees of a
//    __device__ array); make that first call before any stream capture.
//  - All calls share the one array and it keeps the last call's contents:
//    each call writes every logit before reading it, so nothing needs
//    clearing, but calls that overlap on the GPU (other streams or threads)
//    race on it and must be serialised by the caller.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "../../include/kvr.h"
#include "kvr_internal.h"

namespace {

constexpr size_t kScratchFloats = KVR_NOALLOC_SCRATCH_BYTES / sizeof(float);

__device__ __align__(256) float g_noalloc_logits[kScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float *g_dev_ptr[kMaxDevices];  // device address of the array, per device

// Set-up, once per device, with that device current.
cudaError_t scratch_address(float **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_dev_ptr[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_logits);
    if (e != cudaSuccess) return e;
    g_dev_ptr[dev] = static_cast<float *>(p);
  }
  *out = g_dev_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" kvr_status kvr_decode_attend_score_noalloc(
    kvr_cache *cache, int layer_begin, int layer_end, const void *q,
    const void *k_new, const void *v_new, void *out, void *stream) {
  float *scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess)
    return static_cast<kvr_status>(kvr::report_cuda_error(
        "kvr_decode_attend_score_noalloc: cudaGetSymbolAddress", e));
  return static_cast<kvr_status>(kvr::decode_attend_score_ext(
      cache, layer_begin, layer_end, q, k_new, v_new, out, scratch,
      kScratchFloats, stream));
}
