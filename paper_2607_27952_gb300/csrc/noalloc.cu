// last_scores_noalloc: the scoring path (Eq. 6-8) with its scratch memory in a
// fixed, library-owned device array instead of a caller workspace.
//
// Some callers cannot allocate device memory at run time: for example an edge
// service that reserves all of its device memory at start-up and treats any
// later allocation as a failure, or a C program that links this library
// without a device allocator of its own.  They still pass their own q, k and
// w_out buffers; only the scratch (plan, per-chunk softmax statistics, visual
// logits) comes from the array below.
//
// The array is a file-scope static __device__ object of kNoAllocScratchBytes:
// every GPU that loads the library holds it until the process exits.  In host
// code its name is only a host-side stand-in, so the device address is looked up
// with cudaGetSymbolAddress, once per device, with that device current, the first
// time the entry point runs on it.  All calls share the array and it keeps the
// last call's contents; the only part that must start at zero (the device error
// word) is rewritten by every call's plan copy.  Calls whose executions overlap
// on the GPU (different streams, or different host threads on one device) race
// on the array.
#include "last_internal.h"

#include <mutex>
#include <string>

namespace last {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scores_scratch[kNoAllocScratchBytes];

namespace {

std::mutex g_scratch_mu;
void *g_scratch_ptr[kNoAllocMaxDevices] = {};

// Device address of g_scores_scratch on the current device (looked up once per device).
last_status scratch_for_current_device(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_error(std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    return LAST_ERR_CUDA;
  }
  if (dev < 0 || dev >= kNoAllocMaxDevices) {
    set_error("last_scores_noalloc supports device ordinals below 64");
    return LAST_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scores_scratch);
    if (e != cudaSuccess || p == nullptr) {
      set_error(std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
      return LAST_ERR_CUDA;
    }
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return LAST_OK;
}

}  // namespace
}  // namespace last

using namespace last;

extern "C" last_status last_scores_noalloc(const last_problem *p, const void *q, const void *k,
                                           float *w_out, void *stream) {
  Plan pl;
  last_status st = make_plan(p, true, false, &pl);
  if (st != LAST_OK) return st;
  if (pl.score_bytes > kNoAllocScratchBytes) {
    set_error("last_scores_noalloc: this problem needs " + std::to_string(pl.score_bytes) +
              " bytes of scratch, more than the library's fixed " +
              std::to_string(kNoAllocScratchBytes) + " bytes; use last_scores with a workspace");
    return LAST_ERR_UNSUPPORTED;
  }
  if (pl.total_vis > 0 && (q == nullptr || k == nullptr || w_out == nullptr)) {
    set_error("q, k and w_out are required");
    return LAST_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(q) & 15u) || (reinterpret_cast<uintptr_t>(k) & 15u)) {
    set_error("q and k must be 16-byte aligned");
    return LAST_ERR_INVALID_ARG;
  }
  void *scratch = nullptr;
  if ((st = scratch_for_current_device(&scratch)) != LAST_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the plan copy also clears the error word at the start of the scratch
  cudaError_t e = cudaMemcpyAsync(scratch, pl.host_blob.data(), pl.blob_bytes,
                                  cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) {
    set_error(std::string("plan copy: ") + cudaGetErrorString(e));
    return LAST_ERR_CUDA;
  }
  e = launch_scores(pl, q, k, w_out, static_cast<char *>(scratch), s);
  if (e != cudaSuccess) {
    set_error(std::string("scoring launch: ") + cudaGetErrorString(e));
    return LAST_ERR_CUDA;
  }
  return LAST_OK;
}
