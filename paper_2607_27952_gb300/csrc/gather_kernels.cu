// Eq. 12 (Sec. 3.4): X_S = [x_i], i in sort(S), for caller-given indices.
// One warp per output row, 16-byte vectors; the request of an output row is
// found by binary search over the per-request output offsets.
#include "last_device.cuh"
#include "last_internal.h"

namespace last {

__global__ void __launch_bounds__(kGatherThreads)
gather_kernel(const char *__restrict__ x, const int32_t *__restrict__ idx,
              char *__restrict__ x_out, const int32_t *__restrict__ meta, int B,
              long long total_keep, int row_bytes, unsigned *err) {
  const int lane = threadIdx.x & 31;
  const long long nwarps = (long long)gridDim.x * (kGatherThreads / 32);
  const int nvec = row_bytes / 16;
  for (long long r = (long long)blockIdx.x * (kGatherThreads / 32) + (threadIdx.x >> 5);
       r < total_keep; r += nwarps) {
    // last request whose output range starts at or before r (empty requests
    // share their offset with the next one, which is the one holding r)
    int lo = 0, hi = B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (meta[mid * kMetaFields + kKeepOff] <= r) lo = mid; else hi = mid - 1;
    }
    const int32_t *m = meta + lo * kMetaFields;
    const int i = idx[r];
    if (i < 0 || i >= m[kNumVis]) {
      if (lane == 0) atomicOr(err, kErrGatherIndex);
      continue;
    }
    const char *src = x + (long long)(m[kVisOff] + i) * row_bytes;
    char *dst = x_out + r * row_bytes;
    for (int v = lane; v < nvec; v += 32)
      reinterpret_cast<U4 *>(dst)[v] = ldg_stream(src + 16LL * v);
  }
}

cudaError_t launch_gather(const Plan &pl, const void *x, const int32_t *idx, void *x_out,
                          char *ws, cudaStream_t s) {
  if (pl.total_keep == 0) return cudaSuccess;
  const long long warps_needed = pl.total_keep;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  long long blocks = (warps_needed + kGatherThreads / 32 - 1) / (kGatherThreads / 32);
  const long long cap = (long long)sms * 8;
  if (blocks > cap) blocks = cap;
  gather_kernel<<<(unsigned)blocks, kGatherThreads, 0, s>>>(
      static_cast<const char *>(x), idx, static_cast<char *>(x_out),
      reinterpret_cast<const int32_t *>(ws + pl.off_meta), pl.B, pl.total_keep,
      pl.dv * pl.elem, reinterpret_cast<unsigned *>(ws + pl.off_err));
  return cudaGetLastError();
}

}  // namespace last

// Diagnostic of the bounded-wait path: one thread waits on an mbarrier that nothing
// completes, with a short iteration limit, and reports the expiry through the
// workspace error word -- the same path every device wait of the library takes.
namespace last {

__global__ void bounded_wait_check_kernel(unsigned *err, uint32_t limit) {
  __shared__ unsigned long long bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);   // expects one arrival that never comes
  fence_mbar_init();
  for (uint32_t i = 0; i < limit; ++i)
    if (mbar_try_wait(&bar, 0)) return;
  atomicOr(err, kErrTimeout);
}

}  // namespace last

extern "C" last_status last_check_bounded_wait(void *ws, void *stream) {
  using namespace last;
  if (ws == nullptr) {
    set_error("workspace is NULL");
    return LAST_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(unsigned), s);
  if (e == cudaSuccess) {
    bounded_wait_check_kernel<<<1, 32, 0, s>>>(static_cast<unsigned *>(ws), 1u << 12);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) {
    set_error(std::string("bounded-wait check: ") + cudaGetErrorString(e));
    return LAST_ERR_CUDA;
  }
  return LAST_OK;
}
