// Table 5 ("LAST (Top-k)"): the selection variant that keeps the k_b tokens of
// highest importance score w~ per request, ties to the lower index, returned in
// ascending index order (Eq. 12's sort(S)).
//
// topk_kernel: one CTA per request; a request of up to kTopkCacheTokens scores
// keeps them in shared memory for every pass.  Every token gets the 64-bit key
// (order-preserving bits of w~ << 32) | (0xffffffff - i), the same key the
// greedy's argmax uses: keys are unique, larger key = kept first.  An MSB-first
// radix select over 8-bit digits finds the k-th largest key T (stopping early
// once a digit bucket holds exactly the keys still needed), with integer shared
// memory histograms (warp-aggregated adds), so the result is exact and
// deterministic.  A block-wide ordered compaction then writes the indices of
// keys >= T in ascending order.
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>

namespace last {

constexpr int kTopkThreads = 1024;
constexpr int kTopkCacheTokens = 48 * 1024;   // 192 KB of scores

__global__ void __launch_bounds__(kTopkThreads)
topk_kernel(const float *__restrict__ w, const int32_t *__restrict__ meta,
            int32_t *__restrict__ idx_out, int cache_tokens) {
  extern __shared__ float wcache[];
  constexpr int kWarps = kTopkThreads / 32;
  __shared__ unsigned hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ unsigned s_need;
  __shared__ int s_done;
  __shared__ unsigned warp_cnt[kWarps];
  const int32_t *m = meta + blockIdx.x * kMetaFields;
  const int N = m[kNumVis], k = m[kNumKeep];
  if (k <= 0) return;
  const float *wg = w + m[kVisOff];
  int32_t *out = idx_out + m[kKeepOff];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool cached = N <= cache_tokens;
  if (cached) {
    for (int i = tid; i < N; i += kTopkThreads) wcache[i] = wg[i];
    __syncthreads();
  }
  const float *wb = cached ? wcache : wg;

  unsigned long long prefix = 0, mask = 0;
  unsigned need = static_cast<unsigned>(k);
  if (k < N) {
    for (int pos = 56; pos >= 0; pos -= 8) {
      for (int i = tid; i < 256; i += kTopkThreads) hist[i] = 0;
      __syncthreads();
      // keys of one warp mostly share a digit: one shared atomic per distinct digit
      for (int i0 = 0; i0 < N; i0 += kTopkThreads) {
        const int i = i0 + tid;
        unsigned digit = 256u + lane;   // distinct non-digits for lanes that count nothing
        if (i < N) {
          const unsigned long long key = argmax_key(wb[i], i);
          if ((key & mask) == prefix) digit = static_cast<unsigned>(key >> pos) & 255u;
        }
        // common case: every counting lane of the warp has the same digit -> one add
        const unsigned counting = __ballot_sync(0xffffffffu, digit < 256u);
        const unsigned dmin = __reduce_min_sync(0xffffffffu, digit);
        const unsigned dmax = __reduce_max_sync(0xffffffffu, digit < 256u ? digit : 0u);
        if (counting == 0u) {
          // nothing to count in this group of keys
        } else if (dmin == dmax) {
          if (lane == __ffs(counting) - 1) atomicAdd(&hist[dmin], __popc(counting));
        } else {
          const unsigned peers = __match_any_sync(0xffffffffu, digit);
          if (digit < 256u && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
        }
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns digits 255 - 8l down to 248 - 8l; scan from the top digit
        unsigned c[8], tot = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          c[j] = hist[255 - 8 * lane - j];
          tot += c[j];
        }
        unsigned incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned v = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += v;
        }
        const unsigned excl = incl - tot;   // keys with a higher digit than this lane's
        if (excl < need && need <= incl) {  // exactly one lane holds the need-th key
          unsigned above = excl;
          int j = 0;
          while (above + c[j] < need) above += c[j++];
          const unsigned digit = 255u - 8u * lane - j;
          s_prefix = prefix | (static_cast<unsigned long long>(digit) << pos);
          s_need = need - above;
          s_done = c[j] == need - above;   // every key of this bucket is kept
        }
      }
      __syncthreads();
      prefix = s_prefix;
      need = s_need;
      mask |= 0xffull << pos;
      const bool done = s_done;
      __syncthreads();   // the shared words are rewritten by the next pass
      if (done) break;
    }
  }
  // With the digits below the last pass zero in `prefix`, the keys >= prefix are
  // exactly the k largest (k == N keeps every key).
  const unsigned long long thr = k < N ? prefix : 0ull;

  unsigned base = 0;
  for (int i0 = 0; i0 < N; i0 += kTopkThreads) {
    const int i = i0 + tid;
    const bool sel = i < N && argmax_key(wb[i], i) >= thr;
    const unsigned bal = __ballot_sync(0xffffffffu, sel);
    if (lane == 0) warp_cnt[warp] = __popc(bal);
    __syncthreads();
    unsigned off = 0, tot = 0;
#pragma unroll
    for (int q = 0; q < kWarps; ++q) {
      const unsigned c = warp_cnt[q];
      off += q < warp ? c : 0u;
      tot += c;
    }
    if (sel) out[base + off + __popc(bal & ((1u << lane) - 1u))] = i;
    base += tot;
    __syncthreads();
  }
}

cudaError_t launch_topk(const Plan &pl, const float *w, int32_t *idx_out, char *ws,
                        cudaStream_t s) {
  if (pl.total_keep == 0 || pl.B == 0) return cudaSuccess;
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  // cache every request's scores when they fit (the shared memory of the
  // kernel's own arrays stays within the 48 KB static default)
  const int cache = std::min<int>(std::min(kTopkCacheTokens, pl.max_vis),
                                  std::max(0, (optin - 8 * 1024) / 4));
  const size_t smem = sizeof(float) * (size_t)cache;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  topk_kernel<<<pl.B, kTopkThreads, smem, s>>>(
      w, reinterpret_cast<const int32_t *>(ws + pl.off_meta), idx_out, cache);
  return cudaGetLastError();
}

}  // namespace last
