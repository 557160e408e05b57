// Eq. 9-12 (Sec. 3.4): importance-weighted greedy k-center selection and the
// order-restoring gather, fused in one kernel.
//
// One thread-block cluster of C CTAs per request.  CTA r owns the contiguous
// token range [r*T, min(N, (r+1)*T)), T = ceil(N / C), and keeps as many of its
// rows as fit resident in shared memory for all k iterations (the rest are
// re-read from global memory / L2 each iteration).  Per iteration t:
//   1. the row x_{j_{t-1}} is staged into every CTA's shared memory, from the
//      owner CTA's shared memory over DSMEM (or from global memory),
//   2. each warp takes its tokens two at a time and forms dot(x_i, x_j) in the
//      canonical order (lane l owns 8-coordinate groups l, l+32, ...; fp32 fma;
//      xor butterfly), then delta_i = min(delta_i, 1 - (dot r_i) r_j) and
//      p_i = w_i delta_i (Eq. 10, 11),
//   3. a (value, index) argmax key per warp -> per CTA -> pushed to every CTA
//      of the cluster over DSMEM; one cluster barrier; every CTA reduces the C
//      keys itself, so all of them agree on j_t and its r_{j_t}.
// Epilogue (Eq. 12): the CTAs exchange their selected counts, and each writes
// its selected indices (ascending) and copies their rows to x_out.
//
// The arithmetic is fp32 with explicit __fmaf_rn / __fmul_rn / __fsub_rn so
// nothing is re-associated or contracted: given the same w, the selection is
// bit-identical to the canonical definition in the public header.
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>
#include <cmath>

namespace last {

constexpr int kSelThreads = kSelectWarps * 32;
constexpr int kMaxCluster = 16;

struct SelectArgs {
  const void *x;
  const float *w;
  int32_t *idx_out;
  void *x_out;           // nullable
  const int32_t *meta;
  const int32_t *order;  // cluster -> request (longest first)
  int dv, row_bytes, tpc_max, cache_rows, csize;
};

// Shared-memory carve-up, identical on host (sizing) and device.
struct SelectSmem {
  size_t xcache, xj, w, r, dl, list, sel, red_key, red_r, slot_key, slot_r, cnt, total;
};
__host__ __device__ inline size_t align16(size_t v) { return (v + 15) & ~size_t(15); }
__host__ __device__ inline SelectSmem select_smem(int cache_rows, int row_bytes, int tpc_max) {
  SelectSmem s;
  size_t o = 0;
  s.xcache = o; o += (size_t)cache_rows * row_bytes;
  s.xj = o; o += align16(row_bytes);
  s.w = o; o += align16(sizeof(float) * tpc_max);
  s.r = o; o += align16(sizeof(float) * tpc_max);
  s.dl = o; o += align16(sizeof(float) * tpc_max);
  s.list = o; o += align16(sizeof(int) * tpc_max);
  s.sel = o; o += align16(tpc_max);
  s.red_key = o; o += sizeof(unsigned long long) * kSelectWarps;
  s.red_r = o; o += align16(sizeof(float) * kSelectWarps);
  s.slot_key = o; o += sizeof(unsigned long long) * 2 * kMaxCluster;
  s.slot_r = o; o += sizeof(float) * 2 * kMaxCluster;
  s.cnt = o; o += sizeof(int) * kMaxCluster;
  s.total = align16(o);
  return s;
}

// 8 consecutive elements starting at element `col` of a row, widened to fp32.
template <typename T, bool kShared>
__device__ __forceinline__ void load8(const char *row, int col, float *e) {
  if constexpr (sizeof(T) == 2) {
    const U4 v = kShared ? lds(row + col * 2) : ldg(row + col * 2);
    Elem<T>::widen(v, e);
  } else {
    const U4 v0 = kShared ? lds(row + col * 4) : ldg(row + col * 4);
    const U4 v1 = kShared ? lds(row + col * 4 + 16) : ldg(row + col * 4 + 16);
    Elem<T>::widen(v0, e);
    Elem<T>::widen(v1, e + 4);
  }
}

template <typename T, int NCH>
__device__ __forceinline__ void load8_any(const char *row, bool sh, int col, float *e) {
  if (sh) load8<T, true>(row, col, e);
  else load8<T, false>(row, col, e);
}

__device__ __forceinline__ float butterfly_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// max over the warp of (key, r) pairs; every lane ends with the winner
__device__ __forceinline__ void warp_argmax(unsigned long long &key, float &r) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long ok = shfl_xor_u64(key, o);
    const float orr = __shfl_xor_sync(0xffffffffu, r, o);
    if (ok > key) { key = ok; r = orr; }
  }
}

template <typename T, int NCH, bool kFull>
__global__ void __launch_bounds__(kSelThreads, 1)
select_kernel(const SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int C = a.csize;
  const uint32_t rank = cluster_ctarank();
  const int b = a.order[cluster_id_x()];
  const int32_t *m = a.meta + b * kMetaFields;
  const int voff = m[kVisOff], N = m[kNumVis], koff = m[kKeepOff], K = m[kNumKeep];
  if (K == 0) return;  // the whole cluster leaves together; no DSMEM traffic yet

  const SelectSmem L = select_smem(a.cache_rows, a.row_bytes, a.tpc_max);
  char *xcache = reinterpret_cast<char *>(smem + L.xcache);
  char *xj_s = reinterpret_cast<char *>(smem + L.xj);
  float *w_s = reinterpret_cast<float *>(smem + L.w);
  float *r_s = reinterpret_cast<float *>(smem + L.r);
  float *dl_s = reinterpret_cast<float *>(smem + L.dl);
  int *list_s = reinterpret_cast<int *>(smem + L.list);
  unsigned char *sel_s = smem + L.sel;
  unsigned long long *red_key = reinterpret_cast<unsigned long long *>(smem + L.red_key);
  float *red_r = reinterpret_cast<float *>(smem + L.red_r);
  unsigned long long *slot_key = reinterpret_cast<unsigned long long *>(smem + L.slot_key);
  float *slot_r = reinterpret_cast<float *>(smem + L.slot_r);
  int *cnt_s = reinterpret_cast<int *>(smem + L.cnt);

  const int tpr = (N + C - 1) / C;  // tokens per CTA for this request
  const int lo = min(N, (int)rank * tpr), hi = min(N, lo + tpr);
  const int nloc = hi - lo;
  const int ncache = min(nloc, a.cache_rows);
  const int rb = a.row_bytes;
  const char *xg = static_cast<const char *>(a.x) + (long long)(voff + lo) * rb;

  // ---- prologue: resident rows, weights, delta = +inf ----
  {
    const int nvec = ncache * (rb / 16);
    for (int v = threadIdx.x; v < nvec; v += kSelThreads)
      reinterpret_cast<U4 *>(xcache)[v] = ldg_stream(xg + (long long)v * 16);
    for (int t = threadIdx.x; t < nloc; t += kSelThreads) {
      w_s[t] = a.w[voff + lo + t];
      dl_s[t] = INFINITY;
      sel_s[t] = (K == N) ? 1 : 0;
    }
  }
  __syncthreads();

  if (K < N) {
    // ---- r_i = 1/sqrt(dot(x_i, x_i)) in the canonical order ----
    for (int t = warp; t < nloc; t += kSelectWarps) {
      const bool sh = t < ncache;
      const char *row = sh ? xcache + (long long)t * rb : xg + (long long)t * rb;
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const int col = 256 * c + 8 * lane;
        if (kFull || col < a.dv) {
          float e[8];
          load8_any<T, NCH>(row, sh, col, e);
#pragma unroll
          for (int q = 0; q < 8; ++q) acc = __fmaf_rn(e[q], e[q], acc);
        }
      }
      acc = butterfly_sum(acc);
      if (lane == 0) r_s[t] = acc > 0.f ? __fdiv_rn(1.0f, __fsqrt_rn(acc)) : 0.f;
    }
    __syncthreads();

    // cluster-wide argmax of (key, r); result identical in every CTA
    auto exchange = [&](int t, unsigned long long key, float r, int &j, float &rj) {
      if (lane == 0) { red_key[warp] = key; red_r[warp] = r; }
      __syncthreads();
      if (warp == 0) {
        unsigned long long k2 = lane < kSelectWarps ? red_key[lane] : 0ull;
        float r2 = lane < kSelectWarps ? red_r[lane] : 0.f;
        warp_argmax(k2, r2);
        if (lane < C) {
          const int s = (t & 1) * kMaxCluster + (int)rank;
          st_cluster_u64(map_shared(&slot_key[s], lane), k2);
          st_cluster_f32(map_shared(&slot_r[s], lane), r2);
        }
      }
      cluster_sync();
      unsigned long long best = 0ull;
      float br = 0.f;
      for (int q = 0; q < C; ++q) {
        const unsigned long long kq = slot_key[(t & 1) * kMaxCluster + q];
        if (kq > best) { best = kq; br = slot_r[(t & 1) * kMaxCluster + q]; }
      }
      j = key_index(best);
      rj = br;
      if (threadIdx.x == 0 && j >= lo && j < hi) sel_s[j - lo] = 1;
    };

    // ---- Eq. 9: j_1 = argmax w ----
    int j;
    float rj;
    {
      unsigned long long key = 0ull;
      float r = 0.f;
      for (int t = threadIdx.x; t < nloc; t += kSelThreads) {
        const unsigned long long kt = argmax_key(w_s[t], lo + t);
        if (kt > key) { key = kt; r = r_s[t]; }
      }
      warp_argmax(key, r);
      exchange(0, key, r, j, rj);
    }

    // ---- Eq. 10-11, t = 2..K ----
    for (int t = 1; t < K; ++t) {
      // stage x_j: from the owner's shared memory when resident there
      {
        const int owner = j / tpr, lj = j - owner * tpr;
        const int nvec = rb / 16;
        if (lj < a.cache_rows) {
          const uint32_t src = map_shared(xcache + (long long)lj * rb, owner);
          for (int v = threadIdx.x; v < nvec; v += kSelThreads)
            reinterpret_cast<U4 *>(xj_s)[v] = ld_cluster_v4(src + 16 * v);
        } else {
          const char *src = static_cast<const char *>(a.x) + (long long)(voff + j) * rb;
          for (int v = threadIdx.x; v < nvec; v += kSelThreads)
            reinterpret_cast<U4 *>(xj_s)[v] = ldg(src + 16 * v);
        }
      }
      __syncthreads();
      float xr[NCH][8];
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const int col = 256 * c + 8 * lane;
        if (kFull || col < a.dv) {
          load8<T, true>(xj_s, col, xr[c]);
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q) xr[c][q] = 0.f;
        }
      }

      unsigned long long wkey = 0ull;
      float wr = 0.f;
      for (int t0 = warp; t0 < nloc; t0 += 2 * kSelectWarps) {
        const int ta = t0, tb = t0 + kSelectWarps;
        const bool va = !sel_s[ta];
        const bool vb = tb < nloc && !sel_s[tb];
        if (!va && !vb) continue;
        const int tbb = vb ? tb : ta;
        const bool sha = ta < ncache, shb = tbb < ncache;
        const char *ra = sha ? xcache + (long long)ta * rb : xg + (long long)ta * rb;
        const char *rbp = shb ? xcache + (long long)tbb * rb : xg + (long long)tbb * rb;
        float acc_a = 0.f, acc_b = 0.f;
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          const int col = 256 * c + 8 * lane;
          if (kFull || col < a.dv) {
            float ea[8], eb[8];
            load8_any<T, NCH>(ra, sha, col, ea);
            load8_any<T, NCH>(rbp, shb, col, eb);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              acc_a = __fmaf_rn(ea[q], xr[c][q], acc_a);
              acc_b = __fmaf_rn(eb[q], xr[c][q], acc_b);
            }
          }
        }
        acc_a = butterfly_sum(acc_a);
        acc_b = butterfly_sum(acc_b);
        if (va) {
          const float cs = __fmul_rn(__fmul_rn(acc_a, r_s[ta]), rj);
          const float dl = fminf(dl_s[ta], __fsub_rn(1.0f, cs));
          if (lane == 0) dl_s[ta] = dl;
          const unsigned long long kt = argmax_key(__fmul_rn(w_s[ta], dl), lo + ta);
          if (kt > wkey) { wkey = kt; wr = r_s[ta]; }
        }
        if (vb) {
          const float cs = __fmul_rn(__fmul_rn(acc_b, r_s[tb]), rj);
          const float dl = fminf(dl_s[tb], __fsub_rn(1.0f, cs));
          if (lane == 0) dl_s[tb] = dl;
          const unsigned long long kt = argmax_key(__fmul_rn(w_s[tb], dl), lo + tb);
          if (kt > wkey) { wkey = kt; wr = r_s[tb]; }
        }
      }
      exchange(t, wkey, wr, j, rj);
    }
  }
  __syncthreads();

  // ---- Eq. 12: counts -> prefix over the cluster -> ascending indices + rows ----
  int cnt = 0;
  for (int t = threadIdx.x; t < nloc; t += kSelThreads) cnt += sel_s[t];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if (lane == 0) reinterpret_cast<int *>(red_key)[warp] = cnt;
  __syncthreads();
  if (warp == 0) {
    int v = lane < kSelectWarps ? reinterpret_cast<int *>(red_key)[lane] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane < C) st_cluster_s32(map_shared(&cnt_s[rank], lane), v);
  }
  cluster_sync();
  int prefix = 0, mine = 0;
  for (int q = 0; q < C; ++q) {
    if (q < (int)rank) prefix += cnt_s[q];
    if (q == (int)rank) mine = cnt_s[q];
  }
  if (warp == 0) {
    int run = 0;
    for (int base = 0; base < nloc; base += 32) {
      const int t = base + lane;
      const bool f = t < nloc && sel_s[t];
      const unsigned mask = __ballot_sync(0xffffffffu, f);
      const int pos = run + __popc(mask & ((1u << lane) - 1u));
      if (f) {
        list_s[pos] = t;
        a.idx_out[koff + prefix + pos] = lo + t;
      }
      run += __popc(mask);
    }
  }
  if (a.x_out != nullptr) {
    __syncthreads();
    const int nvec = rb / 16;
    char *out = static_cast<char *>(a.x_out) + (long long)(koff + prefix) * rb;
    for (int r = warp; r < mine; r += kSelectWarps) {
      const int t = list_s[r];
      const char *src = t < ncache ? xcache + (long long)t * rb : xg + (long long)t * rb;
      const bool sh = t < ncache;
      for (int v = lane; v < nvec; v += 32) {
        const U4 val = sh ? lds(src + 16 * v) : ldg(src + 16 * v);
        reinterpret_cast<U4 *>(out + (long long)r * rb)[v] = val;
      }
    }
  }
}

namespace {

template <typename T, int NCH>
void *pick2(bool full) {
  return full ? (void *)select_kernel<T, NCH, true> : (void *)select_kernel<T, NCH, false>;
}

template <typename T>
void *pick_select(int nch, bool full) {
  switch (nch) {
    case 1: return pick2<T, 1>(full);
    case 2: return pick2<T, 2>(full);
    case 3: return pick2<T, 3>(full);
    case 4: return pick2<T, 4>(full);
    case 5: return pick2<T, 5>(full);
    case 6: return pick2<T, 6>(full);
    case 7: return pick2<T, 7>(full);
    case 8: return pick2<T, 8>(full);
  }
  return nullptr;
}

int device_smem_optin() {
  int dev = 0, v = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  return v;
}

}  // namespace

bool select_supported(const Plan &pl, std::string *why) {
  if (pl.dv < 8 || pl.dv % 8 != 0 || pl.dv > kMaxFeatDim) {
    if (why) *why = "feat_dim must be a positive multiple of 8, at most 2048";
    return false;
  }
  return true;
}

cudaError_t launch_select(const Plan &pl, const float *w, const void *x, int32_t *idx_out,
                          void *x_out, char *ws, cudaStream_t s) {
  if (pl.B == 0 || pl.total_keep == 0) return cudaSuccess;
  const int rb = pl.dv * pl.elem;
  const int nch = (pl.dv + 255) / 256;
  const bool full = pl.dv == 256 * nch;
  void *fn = pl.dtype == LAST_DTYPE_BF16 ? pick_select<__nv_bfloat16>(nch, full)
                                         : pick_select<float>(nch, full);
  const int optin = device_smem_optin();
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  // Largest cluster (most shared memory per request) that the device can place.
  int C = 0, tpc = 0, cache_rows = 0;
  size_t smem = 0;
  for (int c = kMaxCluster; c >= 1; c /= 2) {
    tpc = (pl.max_vis + c - 1) / c;
    const size_t fixed = select_smem(0, rb, tpc).total;
    if (fixed > (size_t)optin) continue;
    cache_rows = (int)std::min<size_t>(tpc, (optin - fixed) / rb);
    smem = select_smem(cache_rows, rb, tpc).total;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t q = {};
    q.gridDim = dim3(c * pl.B);
    q.blockDim = dim3(kSelThreads);
    q.dynamicSmemBytes = smem;
    cudaLaunchAttribute qa[1];
    qa[0].id = cudaLaunchAttributeClusterDimension;
    qa[0].val.clusterDim.x = c;
    qa[0].val.clusterDim.y = 1;
    qa[0].val.clusterDim.z = 1;
    q.attrs = qa;
    q.numAttrs = 1;
    int active = 0;
    if (cudaOccupancyMaxActiveClusters(&active, fn, &q) == cudaSuccess && active > 0) {
      C = c;
      break;
    }
    cudaGetLastError();
  }
  if (C == 0) return cudaErrorInvalidConfiguration;

  SelectArgs a;
  a.x = x; a.w = w; a.idx_out = idx_out; a.x_out = x_out;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.order = reinterpret_cast<const int32_t *>(ws + pl.off_order);
  a.dv = pl.dv; a.row_bytes = rb; a.tpc_max = tpc; a.cache_rows = cache_rows; a.csize = C;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C * pl.B);
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void *args[] = {&a};
  return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace last
