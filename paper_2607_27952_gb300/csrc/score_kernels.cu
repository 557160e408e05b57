// Eq. 6-8 (Sec. 3.3): last-query-token attention scores.
//
// score_logits_kernel: one CTA per (request, chunk of 128 keys, layer).  It
//   streams the chunk's keys once with 16-byte read-only loads (all kv-heads
//   of a key are contiguous, so consecutive threads read consecutive bytes),
//   forms the logits of the G = Hq/Hkv q-heads that share each kv-head from
//   that single read, and writes (a) per-(layer, head, chunk) softmax
//   statistics (max, sum of exp) and (b) the logits of the visual keys.
//   Logits are kept in the log2 domain (q is pre-scaled by scale*log2 e).
// score_reduce_kernel: one CTA per request.  Merges the chunk statistics of
//   every (layer, head) in chunk order, turns each visual logit into its
//   softmax probability, sums over layers then heads (Eq. 7), and normalises
//   over the visual span (Eq. 8).  Fixed reduction trees: run-to-run
//   deterministic.
#include "last_device.cuh"
#include "last_internal.h"

#include <cmath>

namespace last {

struct ScoreArgs {
  const void *q;
  const void *k;
  const int32_t *meta;
  const int2 *items;     // (request, chunk)
  float2 *stats;         // [L][Hq][total_chunks]
  float *zlog;           // [L][Hq][total_vis]
  long long total_keys;
  long long total_vis;
  int L, Hq, Hkv, D, total_chunks;
  float qscale;          // softmax scale * log2(e)
  int R, log2R;          // lanes per (key, kv-head) row, power of two
  int kpp;               // keys per pass = 256 / (Hkv * R)
};

template <typename T, int G, int SPL>
__global__ void __launch_bounds__(kScoreThreads)
score_logits_kernel(const ScoreArgs a) {
  constexpr int V = Elem<T>::kPerVec;   // elements per 16-byte vector
  constexpr int NE = V * SPL;           // elements of one row a lane owns
  constexpr int U = 4;                  // passes in flight per thread
  extern __shared__ float zbuf[];       // [kScoreChunk][Hq + 1]

  const int2 item = a.items[blockIdx.x];
  const int b = item.x, chunk = item.y, l = blockIdx.y;
  const int32_t *m = a.meta + b * kMetaFields;
  const int seq0 = m[kSeqStart], P = m[kSeqLen], v0 = m[kVisStart];
  const int nvis = m[kNumVis], voff = m[kVisOff], cbase = m[kChunkBase];
  const int p_begin = chunk * kScoreChunk;
  const int nk = min(kScoreChunk, P - p_begin);
  const int ldz = a.Hq + 1;

  const int tid = threadIdx.x;
  const int tpk = a.Hkv * a.R;
  const int slot = tid / tpk;
  const int within = tid - slot * tpk;
  const int g = within >> a.log2R;
  const int part = within & (a.R - 1);
  const bool active = slot < a.kpp;

  // this lane's q slice for the G heads of kv-head g, widened and pre-scaled
  float qv[G][NE];
  {
    const T *qb = static_cast<const T *>(a.q) + ((long long)b * a.L + l) * a.Hq * a.D;
#pragma unroll
    for (int gg = 0; gg < G; ++gg) {
      const T *qh = qb + (long long)(g * G + gg) * a.D;
#pragma unroll
      for (int j = 0; j < SPL; ++j) {
        float e[V];
        Elem<T>::widen(ldg(qh + (part + a.R * j) * V), e);
#pragma unroll
        for (int x = 0; x < V; ++x) qv[gg][j * V + x] = e[x] * a.qscale;
      }
    }
  }

  const T *kl = static_cast<const T *>(a.k) + ((long long)l * a.total_keys + seq0) * a.Hkv * a.D;
  const int passes = (nk + a.kpp - 1) / a.kpp;
  for (int pass0 = 0; pass0 < passes; pass0 += U) {
    U4 buf[U][SPL];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int kk = (pass0 + u) * a.kpp + slot;
      const bool ok = active && kk < nk;
      const T *row = kl + ((long long)(p_begin + kk) * a.Hkv + g) * a.D;
#pragma unroll
      for (int j = 0; j < SPL; ++j)
        buf[u][j] = ok ? ldg_stream(row + (part + a.R * j) * V) : U4{0, 0, 0, 0};
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float acc[G];
#pragma unroll
      for (int gg = 0; gg < G; ++gg) acc[gg] = 0.f;
#pragma unroll
      for (int j = 0; j < SPL; ++j) {
        float e[V];
        Elem<T>::widen(buf[u][j], e);
#pragma unroll
        for (int x = 0; x < V; ++x)
#pragma unroll
          for (int gg = 0; gg < G; ++gg) acc[gg] = fmaf(qv[gg][j * V + x], e[x], acc[gg]);
      }
      for (int o = a.R >> 1; o > 0; o >>= 1)
#pragma unroll
        for (int gg = 0; gg < G; ++gg) acc[gg] += __shfl_xor_sync(0xffffffffu, acc[gg], o);
      const int kk = (pass0 + u) * a.kpp + slot;
      if (active && part == 0 && kk < nk) {
#pragma unroll
        for (int gg = 0; gg < G; ++gg) zbuf[kk * ldz + g * G + gg] = acc[gg];
      }
    }
  }
  __syncthreads();

  // per-head chunk statistics: max and sum of 2^(z - max)
  const int warp = tid >> 5, lane = tid & 31;
  for (int h = warp; h < a.Hq; h += kScoreThreads / 32) {
    float mx = -INFINITY;
    for (int kk = lane; kk < nk; kk += 32) mx = fmaxf(mx, zbuf[kk * ldz + h]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
    for (int kk = lane; kk < nk; kk += 32) sum += exp2f(zbuf[kk * ldz + h] - mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0)
      a.stats[((long long)l * a.Hq + h) * a.total_chunks + cbase + chunk] = make_float2(mx, sum);
  }

  // visual logits of this chunk
  const int vlo = max(p_begin, v0), vhi = min(p_begin + nk, v0 + nvis);
  const int nv = vhi - vlo;
  if (nv > 0) {
    for (int idx = tid; idx < nv * a.Hq; idx += kScoreThreads) {
      const int h = idx / nv, i = idx - h * nv;
      const int p = vlo + i;
      a.zlog[((long long)l * a.Hq + h) * a.total_vis + voff + (p - v0)] =
          zbuf[(p - p_begin) * ldz + h];
    }
  }
}

__global__ void __launch_bounds__(kReduceThreads)
score_reduce_kernel(const int32_t *__restrict__ meta, const float2 *__restrict__ stats,
                    const float *__restrict__ zlog, float *__restrict__ w, int LH,
                    int total_chunks, long long total_vis) {
  extern __shared__ float coef[];      // [LH] max, [LH] 1/Z
  __shared__ float warp_sum[kReduceThreads / 32];
  const int b = blockIdx.x;
  const int32_t *m = meta + b * kMetaFields;
  const int nvis = m[kNumVis], voff = m[kVisOff], cbase = m[kChunkBase];
  const int nch = (m[kSeqLen] + kScoreChunk - 1) / kScoreChunk;
  if (nvis == 0) return;
  float *cmax = coef, *cinv = coef + LH;
  for (int lh = threadIdx.x; lh < LH; lh += blockDim.x) {
    const float2 *s = stats + (long long)lh * total_chunks + cbase;
    float mx = -INFINITY;
    for (int c = 0; c < nch; ++c) mx = fmaxf(mx, s[c].x);
    float z = 0.f;
    for (int c = 0; c < nch; ++c) z += s[c].y * exp2f(s[c].x - mx);
    cmax[lh] = mx;
    cinv[lh] = 1.0f / z;
  }
  __syncthreads();
  float local = 0.f;
  for (int i = threadIdx.x; i < nvis; i += blockDim.x) {
    float s = 0.f;
    for (int lh = 0; lh < LH; ++lh)
      s += exp2f(zlog[(long long)lh * total_vis + voff + i] - cmax[lh]) * cinv[lh];
    w[voff + i] = s;
    local += s;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) local += __shfl_xor_sync(0xffffffffu, local, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) warp_sum[warp] = local;
  __syncthreads();
  if (warp == 0) {
    float v = lane < (int)(blockDim.x >> 5) ? warp_sum[lane] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) warp_sum[0] = v;
  }
  __syncthreads();
  const float inv_total = 1.0f / warp_sum[0];
  for (int i = threadIdx.x; i < nvis; i += blockDim.x) w[voff + i] = w[voff + i] * inv_total;
}

namespace {

struct ScoreShape {
  int spl, R, log2R, kpp;
};

bool score_shape(const Plan &pl, ScoreShape *sh, std::string *why) {
  const int V = 16 / pl.elem;
  if (pl.D % V) { if (why) *why = "head_dim * elem_bytes must be a multiple of 16"; return false; }
  const int segs = pl.D / V;            // 16-byte vectors per (key, kv-head) row
  if (segs & (segs - 1)) {
    if (why) *why = "head_dim * elem_bytes must be 16 bytes times a power of two";
    return false;
  }
  int spl = pl.G <= 2 ? 2 : 1;
  if (spl > segs) spl = segs;
  const int R = segs / spl;
  if (R > 32) { if (why) *why = "head_dim * elem_bytes must be <= 512 (G>2) or 1024 bytes"; return false; }
  if (pl.Hkv * R > kScoreThreads) {
    if (why) *why = "num_kv_heads * head_dim * elem_bytes too large for one scoring CTA";
    return false;
  }
  int log2R = 0;
  while ((1 << log2R) < R) ++log2R;
  *sh = ScoreShape{spl, R, log2R, kScoreThreads / (pl.Hkv * R)};
  return true;
}

template <typename T, int G>
void *pick_logits(int spl) {
  return spl == 2 ? (void *)score_logits_kernel<T, G, 2> : (void *)score_logits_kernel<T, G, 1>;
}

template <typename T>
void *pick_logits_g(int G, int spl) {
  switch (G) {
    case 1: return pick_logits<T, 1>(spl);
    case 2: return pick_logits<T, 2>(spl);
    case 3: return (void *)score_logits_kernel<T, 3, 1>;
    case 4: return (void *)score_logits_kernel<T, 4, 1>;
    case 5: return (void *)score_logits_kernel<T, 5, 1>;
    case 6: return (void *)score_logits_kernel<T, 6, 1>;
    case 7: return (void *)score_logits_kernel<T, 7, 1>;
    case 8: return (void *)score_logits_kernel<T, 8, 1>;
  }
  return nullptr;
}

}  // namespace

bool scores_supported(const Plan &pl, std::string *why) {
  if (pl.G < 1 || pl.G > kMaxGroup) {
    if (why) *why = "num_q_heads / num_kv_heads must be in [1, 8]";
    return false;
  }
  ScoreShape sh;
  return score_shape(pl, &sh, why);
}

cudaError_t launch_scores(const Plan &pl, const void *q, const void *k, float *w_out, char *ws,
                          cudaStream_t s) {
  if (pl.total_vis == 0 || pl.B == 0) return cudaSuccess;
  ScoreShape sh;
  score_shape(pl, &sh, nullptr);
  ScoreArgs a;
  a.q = q;
  a.k = k;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.items = reinterpret_cast<const int2 *>(ws + pl.off_items);
  a.stats = reinterpret_cast<float2 *>(ws + pl.off_stats);
  a.zlog = reinterpret_cast<float *>(ws + pl.off_zlog);
  a.total_keys = pl.total_keys;
  a.total_vis = pl.total_vis;
  a.L = pl.L; a.Hq = pl.Hq; a.Hkv = pl.Hkv; a.D = pl.D;
  a.total_chunks = pl.total_chunks;
  a.qscale = pl.scale * 1.4426950408889634f;
  a.R = sh.R; a.log2R = sh.log2R; a.kpp = sh.kpp;
  void *fn = pl.dtype == LAST_DTYPE_BF16 ? pick_logits_g<__nv_bfloat16>(pl.G, sh.spl)
                                         : pick_logits_g<float>(pl.G, sh.spl);
  const size_t smem = sizeof(float) * kScoreChunk * (pl.Hq + 1);
  cudaError_t e;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  void *args[] = {&a};
  e = cudaLaunchKernel(fn, dim3(pl.total_chunks, pl.L), dim3(kScoreThreads), args, smem, s);
  if (e != cudaSuccess) return e;
  const int LH = pl.L * pl.Hq;
  score_reduce_kernel<<<pl.B, kReduceThreads, sizeof(float) * 2 * LH, s>>>(
      a.meta, a.stats, a.zlog, w_out, LH, pl.total_chunks, pl.total_vis);
  return cudaGetLastError();
}

}  // namespace last
