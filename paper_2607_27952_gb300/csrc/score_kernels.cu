// Eq. 6-8 (Sec. 3.3): last-query-token attention scores.
//
// score_logits_kernel: one CTA per (request, chunk of keys, layer), 8 warps.  A
//   warp task is (kv-head g, 16 consecutive keys of the chunk); the two lanes of
//   a pair share one row K[key][g][0..D): lane h of the pair reads the 16-byte
//   segments h, h + 2, h + 4, ... so every warp-wide load fills whole 32-byte
//   sectors, and forms partial logits of the G = Hq/Hkv q-heads of g in
//   registers from q held in shared memory (broadcast reads): bf16 q as stored,
//   one mixed-precision fma.rn.f32.bf16 per element and the scale applied to the
//   dot; fp32 q pre-scaled.
//   One xor shuffle joins the pair.  The chunk's logits go to shared memory;
//   per (layer, head) the CTA then writes the chunk's max and its sums of
//   2^(z - max) over all keys and over the visual keys, and the visual logits.
//   Logits are in the log2 domain (q pre-scaled by scale * log2 e).
// score_tokens_kernel: one CTA per (request, 256 visual tokens).  It merges the
//   request's chunk statistics per (layer, head) in chunk order into the max M,
//   the total mass Z and the visual mass V, sums each visual token's
//   probabilities over layers then heads (Eq. 7) and divides by the request's
//   visual mass sum_lh V_lh / Z_lh (Eq. 8), which every CTA of the request
//   computes identically.  Fixed reduction trees: run-to-run deterministic.
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

namespace last {

struct ScoreArgs {
  const void *q;
  const void *k;
  const int32_t *meta;
  const int2 *items;     // (request, chunk)
  float4 *stats;         // [L][Hq][total_chunks]: max, sum all, sum visual, unused
  float *zlog;           // [L][Hq][total_vis]
  float *w;              // output scores
  long long total_keys;
  long long total_vis;
  int L, Hq, Hkv, D, total_chunks, chunk;
  float qscale;          // softmax scale * log2(e)
};

constexpr int kSegBatch = 8;        // 16-byte loads in flight per lane
constexpr int kRowsPerTask = 16;    // keys of one warp task (two lanes per key)

template <typename T, int G>
__global__ void __launch_bounds__(kScoreThreads, 3)
score_logits_kernel(const ScoreArgs a) {
  constexpr int V = Elem<T>::kPerVec;   // elements per 16-byte segment
  constexpr bool kBf16 = sizeof(T) == 2;
  extern __shared__ __align__(16) float smem_f[];
  const int Hq = a.Hq, D = a.D;
  // q of the item: bf16 as stored (one mixed-precision fma per element, the scale
  // applied to the dot), fp32 pre-scaled
  float *qs = smem_f;                   // [Hq][D] fp32, or bf16 in the first half
  const unsigned char *qs_b = reinterpret_cast<const unsigned char *>(smem_f);
  float *zbuf = smem_f + (kBf16 ? (Hq * D + 1) / 2 : Hq * D);   // [chunk][Hq + 1] logits
  const int ldz = Hq + 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nseg = D / V;                 // segments per row
  const int nhalf = (nseg + 1) >> 1;      // segments per lane of a pair
  const int half = lane & 1, r = lane >> 1;
  const int total_items = a.total_chunks * a.L;

  // persistent: items (layer-major, then request chunks) strided over the grid
  for (int it = blockIdx.x; it < total_items; it += gridDim.x) {
    const int l = it / a.total_chunks;
    const int2 item = a.items[it - l * a.total_chunks];
    const int b = item.x, chunk = item.y;
    const int32_t *m = a.meta + b * kMetaFields;
    const int seq0 = m[kSeqStart], P = m[kSeqLen], v0 = m[kVisStart];
    const int nvis = m[kNumVis], voff = m[kVisOff], cbase = m[kChunkBase];
    const int p_begin = chunk * a.chunk;
    const int nk = min(a.chunk, P - p_begin);
    const int ngrp = (nk + kRowsPerTask - 1) / kRowsPerTask;
    const int ntask = ngrp * a.Hkv;
    const T *kl = static_cast<const T *>(a.k) + ((long long)l * a.total_keys + seq0) * a.Hkv * D;

    auto row_of = [&](int task, bool *ok, int *kk, int *g) {
      const int grp = task / a.Hkv;
      *g = task - grp * a.Hkv;
      *kk = grp * kRowsPerTask + r;
      *ok = *kk < nk;
      return kl + ((long long)(p_begin + (*ok ? *kk : 0)) * a.Hkv + *g) * D;
    };
    auto issue = [&](const T *row, bool ok, int s0, U4 *buf) {
#pragma unroll
      for (int j = 0; j < kSegBatch; ++j) {
        const int seg = 2 * (s0 + j) + half;
        buf[j] = (ok && seg < nseg) ? ldg_nc(row + seg * V) : U4{0, 0, 0, 0};
      }
    };

    // the first key batch is in flight while q is staged
    U4 buf[kSegBatch];
    {
      bool ok = false;
      int kk, g;
      const T *row = warp < ntask ? row_of(warp, &ok, &kk, &g) : kl;
      issue(row, ok && warp < ntask, 0, buf);
    }
    __syncthreads();   // the previous item is done with qs and zbuf
    {
      const T *qb = static_cast<const T *>(a.q) + ((long long)b * a.L + l) * Hq * D;
      for (int v = tid; v < Hq * D / V; v += kScoreThreads) {
        if constexpr (kBf16) {
          reinterpret_cast<U4 *>(smem_f)[v] = ldg(qb + v * V);
        } else {
          float e[V];
          Elem<T>::widen(ldg(qb + v * V), e);
#pragma unroll
          for (int x = 0; x < V; ++x) qs[v * V + x] = e[x] * a.qscale;
        }
      }
    }
    __syncthreads();

    for (int task = warp; task < ntask; task += kScoreThreads / 32) {
      bool ok;
      int kk, g;
      const T *row = row_of(task, &ok, &kk, &g);
      const float *qg = qs + g * G * D;
      const unsigned char *qgb = qs_b + (size_t)g * G * D * 2;
      float acc[G];
#pragma unroll
      for (int gg = 0; gg < G; ++gg) acc[gg] = 0.f;
      for (int s0 = 0; s0 < nhalf; s0 += kSegBatch) {
        if (task != warp || s0 != 0) issue(row, ok, s0, buf);
#pragma unroll
        for (int j = 0; j < kSegBatch; ++j) {
          const int seg = 2 * (s0 + j) + half;
          if (seg < nseg) {
            if constexpr (kBf16) {
              const uint32_t kw[4] = {buf[j].x, buf[j].y, buf[j].z, buf[j].w};
#pragma unroll
              for (int gg = 0; gg < G; ++gg) {
                const U4 qv = lds(qgb + ((size_t)gg * D + seg * V) * 2);
                const uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
                for (int hw = 0; hw < 4; ++hw) {
                  acc[gg] = fma_bf16_lo(qw[hw], kw[hw], acc[gg]);
                  acc[gg] = fma_bf16_hi(qw[hw], kw[hw], acc[gg]);
                }
              }
            } else {
              float e[V];
              Elem<T>::widen(buf[j], e);
              const float *qc = qg + seg * V;
#pragma unroll
              for (int gg = 0; gg < G; ++gg) {
#pragma unroll
                for (int x = 0; x < V; x += 4) {
                  const float4 qv = *reinterpret_cast<const float4 *>(qc + gg * D + x);
                  acc[gg] = fmaf(qv.x, e[x], acc[gg]);
                  acc[gg] = fmaf(qv.y, e[x + 1], acc[gg]);
                  acc[gg] = fmaf(qv.z, e[x + 2], acc[gg]);
                  acc[gg] = fmaf(qv.w, e[x + 3], acc[gg]);
                }
              }
            }
          }
        }
      }
#pragma unroll
      for (int gg = 0; gg < G; ++gg) acc[gg] += __shfl_xor_sync(0xffffffffu, acc[gg], 1);
      if (ok && half == 0) {
        const float sc = kBf16 ? a.qscale : 1.0f;   // bf16: the scale goes on the dot
#pragma unroll
        for (int gg = 0; gg < G; ++gg) zbuf[kk * ldz + g * G + gg] = acc[gg] * sc;
      }
    }
    __syncthreads();

    // per-head chunk statistics: max, sums of 2^(z - max) over all and over visual keys
    const int vlo = max(p_begin, v0), vhi = min(p_begin + nk, v0 + nvis);
    for (int h = warp; h < Hq; h += kScoreThreads / 32) {
      float mx = -INFINITY;
      for (int kk = lane; kk < nk; kk += 32) mx = fmaxf(mx, zbuf[kk * ldz + h]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float sum = 0.f, vis = 0.f;
      for (int kk = lane; kk < nk; kk += 32) {
        const float e = exp2f(zbuf[kk * ldz + h] - mx);
        sum += e;
        const int p = p_begin + kk;
        if (p >= vlo && p < vhi) vis += e;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        sum += __shfl_xor_sync(0xffffffffu, sum, o);
        vis += __shfl_xor_sync(0xffffffffu, vis, o);
      }
      if (lane == 0)
        a.stats[((long long)l * Hq + h) * a.total_chunks + cbase + chunk] =
            make_float4(mx, sum, vis, 0.f);
    }

    // visual logits of this chunk
    const int nv = vhi - vlo;
    if (nv > 0) {
      for (int idx = tid; idx < nv * Hq; idx += kScoreThreads) {
        const int h = idx / nv, i = idx - h * nv;
        const int p = vlo + i;
        a.zlog[((long long)l * Hq + h) * a.total_vis + voff + (p - v0)] =
            zbuf[(p - p_begin) * ldz + h];
      }
    }
  }
  // the token kernel (launched as a programmatic dependent) may start its
  // prologue; it waits for this whole grid before reading any result
  asm volatile("griddepcontrol.launch_dependents;");
}

// Eq. 7-8: one CTA per (request b, tile of kTokenTile visual tokens).
__global__ void __launch_bounds__(kScoreThreads)
score_tokens_kernel(const ScoreArgs a) {
  extern __shared__ float coef[];   // [L*Hq] max, [L*Hq] 1/Z, [L*Hq] V/Z
  __shared__ float inv_total_s;
  const int b = blockIdx.y, tile = blockIdx.x;
  const int32_t *m = a.meta + b * kMetaFields;
  const int nvis = m[kNumVis], voff = m[kVisOff], cbase = m[kChunkBase];
  if (tile * kTokenTile >= nvis) return;
  // launched as a programmatic dependent of score_logits_kernel: wait until that
  // grid has completed and its writes are visible (a no-op for a plain launch)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int nch = (m[kSeqLen] + a.chunk - 1) / a.chunk;
  const int LH = a.L * a.Hq;
  float *cmax = coef, *cinv = coef + LH, *cvis = coef + 2 * LH;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // one warp per (layer, head): lanes stride over the request's chunks, then
  // fixed xor trees for the max and the rescaled sums
  for (int lh = warp; lh < LH; lh += kScoreThreads / 32) {
    const float4 *st = a.stats + (long long)lh * a.total_chunks + cbase;
    float mx = -INFINITY;
    for (int c = lane; c < nch; c += 32) mx = fmaxf(mx, st[c].x);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f, vz = 0.f;
    for (int c = lane; c < nch; c += 32) {
      const float4 v = st[c];
      const float f = exp2f(v.x - mx);
      z += v.y * f;
      vz += v.z * f;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      z += __shfl_xor_sync(0xffffffffu, z, o);
      vz += __shfl_xor_sync(0xffffffffu, vz, o);
    }
    if (lane == 0) {
      cmax[lh] = mx;
      cinv[lh] = 1.0f / z;
      cvis[lh] = vz / z;   // visual probability mass of (layer, head)
    }
  }
  __syncthreads();
  if (warp == 0) {   // sum_lh V_lh / Z_lh, strided over lanes then a fixed xor tree
    float t = 0.f;
    for (int lh = lane; lh < LH; lh += 32) t += cvis[lh];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) inv_total_s = 1.0f / t;
  }
  __syncthreads();
  const int i = tile * kTokenTile + threadIdx.x;
  if (i < nvis) {
    const float *z = a.zlog + voff + i;
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    int lh = 0;
    for (; lh + 4 <= LH; lh += 4) {   // four independent loads in flight
      const float z0 = z[(long long)(lh + 0) * a.total_vis];
      const float z1 = z[(long long)(lh + 1) * a.total_vis];
      const float z2 = z[(long long)(lh + 2) * a.total_vis];
      const float z3 = z[(long long)(lh + 3) * a.total_vis];
      s0 += exp2f(z0 - cmax[lh + 0]) * cinv[lh + 0];
      s1 += exp2f(z1 - cmax[lh + 1]) * cinv[lh + 1];
      s2 += exp2f(z2 - cmax[lh + 2]) * cinv[lh + 2];
      s3 += exp2f(z3 - cmax[lh + 3]) * cinv[lh + 3];
    }
    for (; lh < LH; ++lh) s0 += exp2f(z[(long long)lh * a.total_vis] - cmax[lh]) * cinv[lh];
    a.w[voff + i] = ((s0 + s1) + (s2 + s3)) * inv_total_s;
  }
}

namespace {

template <typename T>
void *pick_logits(int G) {
  switch (G) {
    case 1: return (void *)score_logits_kernel<T, 1>;
    case 2: return (void *)score_logits_kernel<T, 2>;
    case 3: return (void *)score_logits_kernel<T, 3>;
    case 4: return (void *)score_logits_kernel<T, 4>;
    case 5: return (void *)score_logits_kernel<T, 5>;
    case 6: return (void *)score_logits_kernel<T, 6>;
    case 7: return (void *)score_logits_kernel<T, 7>;
    case 8: return (void *)score_logits_kernel<T, 8>;
  }
  return nullptr;
}

size_t logits_smem(const Plan &pl) {
  return sizeof(float) * ((size_t)pl.Hq * pl.D + (size_t)pl.chunk * (pl.Hq + 1));
}

constexpr size_t kMaxScoreSmem = 100 * 1024;

// CTAs of `fn` resident on the whole current device (occupancy x SMs), cached
// per (device, kernel, shared memory).
cudaError_t resident_slots(const void *fn, size_t smem, int *slots) {
  static std::mutex mu;
  static std::map<std::tuple<int, const void *, size_t>, int> cache;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const auto key = std::make_tuple(dev, fn, smem);
  std::lock_guard<std::mutex> lock(mu);
  auto hit = cache.find(key);
  if (hit != cache.end()) {
    *slots = hit->second;
    return cudaSuccess;
  }
  int per_sm = 0, sms = 0;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kScoreThreads, smem)) != cudaSuccess)
    return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  *slots = std::max(per_sm, 1) * sms;
  cache.emplace(key, *slots);
  return cudaSuccess;
}

}  // namespace

int score_chunk_keys(int num_kv_heads) {
  // about 32 (kv-head, 16-key) warp tasks per CTA, 16..256 keys
  int c = 512 / std::max(num_kv_heads, 1) / kRowsPerTask * kRowsPerTask;
  return std::min(256, std::max(kRowsPerTask, c));
}

bool scores_supported(const Plan &pl, std::string *why) {
  if (pl.G < 1 || pl.G > kMaxGroup) {
    if (why) *why = "num_q_heads / num_kv_heads must be in [1, 8]";
    return false;
  }
  if ((pl.D * pl.elem) % 16) {
    if (why) *why = "head_dim * elem_bytes must be a multiple of 16";
    return false;
  }
  if (logits_smem(pl) > kMaxScoreSmem) {
    if (why) *why = "num_q_heads * head_dim too large for the scoring kernel's shared memory";
    return false;
  }
  return true;
}

cudaError_t launch_scores(const Plan &pl, const void *q, const void *k, float *w_out, char *ws,
                          cudaStream_t s) {
  if (pl.total_vis == 0 || pl.B == 0) return cudaSuccess;
  ScoreArgs a;
  a.q = q;
  a.k = k;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.items = reinterpret_cast<const int2 *>(ws + pl.off_items);
  a.stats = reinterpret_cast<float4 *>(ws + pl.off_stats);
  a.zlog = reinterpret_cast<float *>(ws + pl.off_zlog);
  a.w = w_out;
  a.total_keys = pl.total_keys;
  a.total_vis = pl.total_vis;
  a.L = pl.L; a.Hq = pl.Hq; a.Hkv = pl.Hkv; a.D = pl.D;
  a.total_chunks = pl.total_chunks;
  a.chunk = pl.chunk;
  a.qscale = pl.scale * 1.4426950408889634f;
  void *fn = pl.dtype == LAST_DTYPE_BF16 ? pick_logits<__nv_bfloat16>(pl.G)
                                         : pick_logits<float>(pl.G);
  const size_t smem = logits_smem(pl);
  cudaError_t e;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  int slots = 0;
  if ((e = resident_slots(fn, smem, &slots)) != cudaSuccess) return e;
  const long long items = (long long)pl.total_chunks * pl.L;
  const int grid = (int)std::min<long long>(items, slots);
  void *args[] = {&a};
  e = cudaLaunchKernel(fn, dim3(grid), dim3(kScoreThreads), args, smem, s);
  if (e != cudaSuccess) return e;
  const int max_tiles = (pl.max_vis + kTokenTile - 1) / kTokenTile;
  const size_t tsmem = sizeof(float) * 3 * pl.L * pl.Hq;
  if (tsmem > 48 * 1024) {
    e = cudaFuncSetAttribute(score_tokens_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)tsmem);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(max_tiles, pl.B);
  cfg.blockDim = dim3(kScoreThreads);
  cfg.dynamicSmemBytes = tsmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, score_tokens_kernel, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace last
