// Table 4 (attention sources): the importance of Eq. 7 from the attention rows of
// several query positions per request (First, Middle, All Mean), bf16 q and K.
//
// Request b has M_b query rows at positions row_pos (after its visual span); row m
// sees the keys 0 .. row_pos[m] (causal softmax, Eq. 6).  Scores are summed over
// rows, layers and q-heads at the visual positions and normalised (Eq. 8).  A
// "column" is one (row, q-head of kv-head g) pair: G = Hq / Hkv columns per row.
//
// Four launches, all deterministic (fixed reduction orders, no float atomics):
// rows_stats_kernel (request, 128-key chunk, layer, kv-head, 128-column tile):
//   tcgen05.mma with the query columns as M and the chunk's keys as N (bf16, fp32
//   accumulator in TMEM); thread t owns column t and takes, over its TMEM lane, the
//   masked max of its logits (log2 domain) and the sums of 2^(z - max) over all and
//   over the visual keys -- the chunk statistics of Eq. 6's softmax.
// rows_merge_kernel (request): merges each column's chunk statistics in chunk
//   order into (max, 1/Z) and the request's visual probability mass.
// rows_probs_kernel (request, visual 128-key chunk, layer, kv-head): the same
//   contraction with the keys as M; thread t owns key t and sums the probabilities
//   2^(z - max) / Z over the columns (every column sees every visual key).
// rows_final_kernel (request, 256 visual tokens): adds the (layer, kv-head)
//   partial sums and divides by the visual mass (Eq. 7-8).
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

namespace last {

namespace {

// Per-request metadata (int32 slots; the 64-bit statistics offset takes two slots
// and sits 8-byte aligned since a row is 12 slots).
enum RowsField : int {
  kRSeqStart = 0, kRSeqLen, kRVisStart, kRVisOff, kRNumVis, kRRowOff, kRNumRows,
  kRNumChunks, kRStatBase = 8, kRCoefBase = 10, kRowsFields = 12
};

constexpr int kRowsChunk = 128;     // keys per CTA
constexpr int kRowsThreads = 128;   // one thread per TMEM lane
constexpr int kRowsMaxN = 256;      // columns (rows x G) per request
constexpr int kRowsMaxRH = 6144;    // (row, layer, q-head) triples per request

struct RowsArgs {
  const __nv_bfloat16 *q, *k;
  const int32_t *meta;
  const int2 *items1, *items2;
  const int32_t *row_pos;
  float4 *stats;         // per column-layer-head triple x chunk: max, sum, visual sum
  float2 *coef;          // per triple: max, 1 / Z
  float *inv_total;      // per request: 1 / visual mass
  float *partial;        // [L][Hkv][total_vis] probability sums
  float *w;
  long long total_keys, total_vis;
  int L, Hq, Hkv, D, G, npad;
  uint32_t tmem_stats, tmem_probs;
  float qscale;          // softmax scale * log2(e)
  unsigned *err;
};

__device__ __forceinline__ long long stat_base(const int32_t *m) {
  return *reinterpret_cast<const long long *>(m + kRStatBase);
}

// 16-byte chunk j of row `row` of a K-major operand with 128-byte rows and the
// 128-byte swizzle; K blocks of `rows` rows each.
__device__ __forceinline__ unsigned char *sw128_chunk(unsigned char *base, int rows, int row, int j) {
  return base + (j >> 3) * (rows * 128) + row * 128 + (((j & 7) ^ (row & 7)) << 4);
}

// Keys c*128 .. c*128+127 of kv-head g (zero past P) into a 128-row operand.
__device__ __forceinline__ void stage_keys(unsigned char *dst, const RowsArgs &a, int seq0, int P,
                                           int c, int l, int g) {
  const int t = threadIdx.x, p = c * kRowsChunk + t;
  const __nv_bfloat16 *src = a.k + (((long long)l * a.total_keys + seq0 + p) * a.Hkv + g) * a.D;
  for (int j = 0; j < a.D / 8; ++j)
    *reinterpret_cast<U4 *>(sw128_chunk(dst, kRowsChunk, t, j)) =
        p < P ? ldg(src + 8 * j) : U4{0, 0, 0, 0};
}

// Query columns n0 .. n0+rows-1 (row n / G, q-head g*G + n % G; zero past ncol).
__device__ __forceinline__ void stage_queries(unsigned char *dst, const RowsArgs &a, int rows,
                                              int n0, int ncol, int row0, int l, int g) {
  for (int idx = threadIdx.x; idx < rows * (a.D / 8); idx += kRowsThreads) {
    const int i = idx / (a.D / 8), j = idx - i * (a.D / 8), n = n0 + i;
    U4 v = U4{0, 0, 0, 0};
    if (n < ncol) {
      const int r = n / a.G, gg = n - r * a.G;
      v = ldg(a.q + (((long long)(row0 + r) * a.L + l) * a.Hq + g * a.G + gg) * a.D + 8 * j);
    }
    *reinterpret_cast<U4 *>(sw128_chunk(dst, rows, i, j)) = v;
  }
}

// D[tmem] = A[128 x D] * B[n x D]^T over D / 64 K blocks, one thread; completion on bar.
__device__ __forceinline__ void rows_mma(uint32_t tmem, unsigned char *A, unsigned char *B, int n,
                                         int nkb, unsigned long long *bar) {
  const uint32_t idesc = umma_idesc_bf16(kRowsChunk, n);
  for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
    for (int k = 0; k < 4; ++k)
      umma_bf16(tmem, umma_desc_sw128(smem_addr(A + kb * (kRowsChunk * 128)) + k * 32),
                umma_desc_sw128(smem_addr(B + kb * (n * 128)) + k * 32), idesc, (kb | k) != 0 ? 1u : 0u);
  umma_commit(bar);
}

}  // namespace

__global__ void __launch_bounds__(kRowsThreads)
rows_stats_kernel(const RowsArgs a) {
  const int2 item = a.items1[blockIdx.x];
  const int b = item.x, c = item.y, l = blockIdx.y;
  const int g = blockIdx.z % a.Hkv, mt = blockIdx.z / a.Hkv;
  const int32_t *m = a.meta + b * kRowsFields;
  const int ncol = m[kRNumRows] * a.G;
  if (mt * kRowsThreads >= ncol) return;   // the whole CTA leaves before any allocation
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int nkb = a.D / 64;
  unsigned char *sQ = smem, *sK = smem + nkb * (kRowsChunk * 128);
  unsigned long long *bar = reinterpret_cast<unsigned long long *>(sK + nkb * (kRowsChunk * 128));
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);
  const int seq0 = m[kRSeqStart], P = m[kRSeqLen], v0 = m[kRVisStart], nvis = m[kRNumVis];
  const int row0 = m[kRRowOff], nch = m[kRNumChunks];
  const int t = threadIdx.x, warp = t >> 5;

  if (t == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, a.tmem_stats);
  stage_queries(sQ, a, kRowsThreads, mt * kRowsThreads, ncol, row0, l, g);
  stage_keys(sK, a, seq0, P, c, l, g);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  if (t == 0) rows_mma(tmem, sQ, sK, kRowsChunk, nkb, bar);
  __syncwarp();
  mbar_wait_bounded(bar, 0, a.err, kErrTimeout);
  tc_fence_after();

  // column n: its row's position bounds the keys it sees
  const int n = mt * kRowsThreads + t;
  const bool col_ok = n < ncol;
  const int r = col_ok ? n / a.G : 0;
  const int pos = col_ok ? a.row_pos[row0 + r] : -1;
  const uint32_t lane_addr = tmem + ((uint32_t)(32 * warp) << 16);
  const int p0 = c * kRowsChunk;
  float mx = -INFINITY;
  for (int j0 = 0; j0 < kRowsChunk; j0 += 16) {
    uint32_t raw[16];
    tmem_ld16(lane_addr + (uint32_t)j0, raw);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int p = p0 + j0 + j;
      if (p < P && p <= pos) mx = fmaxf(mx, __uint_as_float(raw[j]) * a.qscale);
    }
  }
  // (a column with no visible key in this chunk keeps max = -inf and adds nothing;
  // the TMEM loads stay warp-uniform)
  float sum = 0.f, vis = 0.f;
  for (int j0 = 0; j0 < kRowsChunk; j0 += 16) {
    uint32_t raw[16];
    tmem_ld16(lane_addr + (uint32_t)j0, raw);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int p = p0 + j0 + j;
      if (p < P && p <= pos) {
        const float e = exp2f(__uint_as_float(raw[j]) * a.qscale - mx);
        sum += e;
        if (p >= v0 && p < v0 + nvis) vis += e;
      }
    }
  }
  if (col_ok) {
    const int h = g * a.G + (n - r * a.G);
    const long long rh = ((long long)r * a.L + l) * a.Hq + h;
    a.stats[stat_base(m) + rh * nch + c] = make_float4(mx, sum, vis, 0.f);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, a.tmem_stats);
}

__global__ void __launch_bounds__(1024)
rows_merge_kernel(const RowsArgs a) {
  __shared__ float red[32];
  const int b = blockIdx.x;
  const int32_t *m = a.meta + b * kRowsFields;
  const int RH = m[kRNumRows] * a.L * a.Hq, nch = m[kRNumChunks], cb = m[kRCoefBase];
  const float4 *stats = a.stats + stat_base(m);
  float vis_mass = 0.f;
  for (int rh = threadIdx.x; rh < RH; rh += blockDim.x) {
    const float4 *st = stats + (long long)rh * nch;
    float mx = -INFINITY;
    for (int c = 0; c < nch; ++c) mx = fmaxf(mx, st[c].x);
    float z = 0.f, vz = 0.f;
    for (int c = 0; c < nch; ++c) {
      const float4 v = st[c];
      const float f = v.x == -INFINITY ? 0.f : exp2f(v.x - mx);   // chunks past the row
      z += v.y * f;
      vz += v.z * f;
    }
    a.coef[cb + rh] = make_float2(mx, 1.0f / z);
    vis_mass += vz / z;
  }
  // fixed-tree block sum of the visual masses
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) vis_mass += __shfl_xor_sync(0xffffffffu, vis_mass, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = vis_mass;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (int)(blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) a.inv_total[b] = 1.0f / v;
  }
}

__global__ void __launch_bounds__(kRowsThreads)
rows_probs_kernel(const RowsArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int nkb = a.D / 64, npad = a.npad;
  unsigned char *sK = smem, *sQ = smem + nkb * (kRowsChunk * 128);
  float2 *cf = reinterpret_cast<float2 *>(sQ + nkb * (npad * 128));
  unsigned long long *bar = reinterpret_cast<unsigned long long *>(cf + kRowsMaxN);
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);
  const int2 item = a.items2[blockIdx.x];
  const int b = item.x, c = item.y, l = blockIdx.y, g = blockIdx.z;
  const int32_t *m = a.meta + b * kRowsFields;
  const int seq0 = m[kRSeqStart], P = m[kRSeqLen], v0 = m[kRVisStart], nvis = m[kRNumVis];
  const int voff = m[kRVisOff], row0 = m[kRRowOff], ncol = m[kRNumRows] * a.G;
  const int cb = m[kRCoefBase];
  const int t = threadIdx.x, warp = t >> 5;

  if (t == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, a.tmem_probs);
  stage_keys(sK, a, seq0, P, c, l, g);
  stage_queries(sQ, a, npad, 0, ncol, row0, l, g);
  for (int n = t; n < ncol; n += kRowsThreads) {
    const int r = n / a.G, h = g * a.G + (n - r * a.G);
    cf[n] = a.coef[cb + ((long long)r * a.L + l) * a.Hq + h];
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  if (t == 0) rows_mma(tmem, sK, sQ, npad, nkb, bar);
  __syncwarp();
  mbar_wait_bounded(bar, 0, a.err, kErrTimeout);
  tc_fence_after();

  const int p = c * kRowsChunk + t;
  float s0 = 0.f, s1 = 0.f;
  for (int n0 = 0; n0 < ncol; n0 += 16) {
    uint32_t raw[16];
    tmem_ld16(tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)n0, raw);
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      if (n0 + j < ncol)
        s0 += exp2f(__uint_as_float(raw[j]) * a.qscale - cf[n0 + j].x) * cf[n0 + j].y;
      if (n0 + j + 1 < ncol)
        s1 += exp2f(__uint_as_float(raw[j + 1]) * a.qscale - cf[n0 + j + 1].x) * cf[n0 + j + 1].y;
    }
  }
  // every column's row sits after the visual span, so each visual key is unmasked
  if (p >= v0 && p < v0 + nvis && p < P)
    a.partial[((long long)l * a.Hkv + g) * a.total_vis + voff + (p - v0)] = s0 + s1;
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, a.tmem_probs);
}

__global__ void __launch_bounds__(kScoreThreads)
rows_final_kernel(const RowsArgs a) {
  const int b = blockIdx.y;
  const int32_t *m = a.meta + b * kRowsFields;
  const int i = blockIdx.x * kScoreThreads + threadIdx.x;
  if (i >= m[kRNumVis]) return;
  const long long tok = m[kRVisOff] + i;
  float s = 0.f;
  for (int lg = 0; lg < a.L * a.Hkv; ++lg) s += a.partial[(long long)lg * a.total_vis + tok];
  a.w[tok] = s * a.inv_total[b];
}

namespace {

struct RowsPlan {
  int B = 0, L = 0, Hq = 0, Hkv = 0, D = 0, G = 0, npad = 0, mtiles = 0, max_vis = 0;
  long long total_keys = 0, total_vis = 0, total_rows = 0, n_items1 = 0, n_items2 = 0;
  size_t off_meta = 0, off_items1 = 0, off_items2 = 0, off_pos = 0, blob_bytes = 0;
  size_t off_stats = 0, off_coef = 0, off_inv = 0, off_partial = 0, total_bytes = 0;
  std::vector<int32_t> blob;
  float scale = 0.f;
};

constexpr size_t kAlignR = 256;
size_t alignr(size_t v) { return (v + kAlignR - 1) / kAlignR * kAlignR; }

last_status rows_fail(last_status st, const std::string &msg) {
  set_error(msg);
  return st;
}

last_status make_rows_plan(const last_problem *p, const int32_t *cu_rows, const int32_t *row_pos,
                           RowsPlan *pl) {
  if (p == nullptr) return rows_fail(LAST_ERR_INVALID_ARG, "problem is NULL");
  if (cu_rows == nullptr || row_pos == nullptr)
    return rows_fail(LAST_ERR_INVALID_ARG, "cu_rows and row_pos are required");
  if (p->dtype != LAST_DTYPE_BF16)
    return rows_fail(LAST_ERR_UNSUPPORTED, "multi-row scoring takes bf16 q and K");
  if (p->batch < 0 || p->cu_seqlens == nullptr || p->vis_start == nullptr || p->cu_vis == nullptr)
    return rows_fail(LAST_ERR_INVALID_ARG, "batch, cu_seqlens, vis_start and cu_vis are required");
  if (p->num_layers < 1 || p->num_q_heads < 1 || p->num_kv_heads < 1 ||
      p->num_q_heads % p->num_kv_heads != 0)
    return rows_fail(LAST_ERR_INVALID_ARG, "layers and heads must be >= 1, Hq a multiple of Hkv");
  if (p->head_dim < 64 || p->head_dim % 64 != 0 || p->head_dim > 256)
    return rows_fail(LAST_ERR_UNSUPPORTED, "multi-row scoring takes head_dim 64, 128, 192 or 256");
  if (!std::isfinite(p->softmax_scale))
    return rows_fail(LAST_ERR_INVALID_ARG, "softmax_scale must be finite");
  if (p->cu_seqlens[0] != 0 || p->cu_vis[0] != 0 || cu_rows[0] != 0)
    return rows_fail(LAST_ERR_INVALID_ARG, "cu_seqlens[0], cu_vis[0] and cu_rows[0] must be 0");
  const int B = p->batch;
  pl->B = B; pl->L = p->num_layers; pl->Hq = p->num_q_heads; pl->Hkv = p->num_kv_heads;
  pl->D = p->head_dim; pl->G = pl->Hq / pl->Hkv;
  pl->scale = p->softmax_scale > 0.f ? p->softmax_scale : (float)(1.0 / std::sqrt((double)p->head_dim));
  int max_cols = 0;
  long long stats = 0, rh_total = 0;
  for (int b = 0; b < B; ++b) {
    const int P = p->cu_seqlens[b + 1] - p->cu_seqlens[b];
    const int N = p->cu_vis[b + 1] - p->cu_vis[b];
    const int M = cu_rows[b + 1] - cu_rows[b];
    if (P < 1 || N < 0 || p->vis_start[b] < 0 || (long long)p->vis_start[b] + N > (long long)P - 1)
      return rows_fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) +
                                                 ": visual span must end before the last position");
    if (M < 1) return rows_fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) + ": no query row");
    for (int r = cu_rows[b]; r < cu_rows[b + 1]; ++r)
      if (row_pos[r] < p->vis_start[b] + N || row_pos[r] > P - 1)
        return rows_fail(LAST_ERR_INVALID_ARG,
                         "request " + std::to_string(b) + ": a query row must sit after the visual "
                         "span and before P_b");
    max_cols = std::max(max_cols, M * pl->G);
    const long long rh = (long long)M * pl->L * pl->Hq;
    if (rh > kRowsMaxRH)
      return rows_fail(LAST_ERR_UNSUPPORTED, "rows x layers x q-heads must be <= 6144 per request");
    const int nch = (P + kRowsChunk - 1) / kRowsChunk;
    stats += rh * nch;
    rh_total += rh;
    pl->n_items1 += nch;
    if (N > 0)
      pl->n_items2 += (p->vis_start[b] + N - 1) / kRowsChunk - p->vis_start[b] / kRowsChunk + 1;
    pl->max_vis = std::max(pl->max_vis, N);
  }
  if (max_cols > kRowsMaxN)
    return rows_fail(LAST_ERR_UNSUPPORTED, "query rows x (num_q_heads / num_kv_heads) must be <= 256");
  if (rh_total > 0x7fffffffLL) return rows_fail(LAST_ERR_UNSUPPORTED, "too many query rows in all");
  pl->npad = std::max(16, (max_cols + 15) / 16 * 16);
  pl->mtiles = (max_cols + kRowsThreads - 1) / kRowsThreads;
  pl->total_keys = p->cu_seqlens[B];
  pl->total_vis = p->cu_vis[B];
  pl->total_rows = cu_rows[B];
  size_t o = alignr(64);                     // error word first
  pl->off_meta = o;
  o = alignr(o + sizeof(int32_t) * kRowsFields * std::max(B, 1));
  pl->off_items1 = o;
  o = alignr(o + sizeof(int32_t) * 2 * std::max<long long>(pl->n_items1, 1));
  pl->off_items2 = o;
  o = alignr(o + sizeof(int32_t) * 2 * std::max<long long>(pl->n_items2, 1));
  pl->off_pos = o;
  o = alignr(o + sizeof(int32_t) * std::max<long long>(pl->total_rows, 1));
  pl->blob_bytes = o;
  pl->off_stats = o;
  o = alignr(o + sizeof(float) * 4 * (size_t)std::max<long long>(stats, 1));
  pl->off_coef = o;
  o = alignr(o + sizeof(float) * 2 * (size_t)std::max<long long>(rh_total, 1));
  pl->off_inv = o;
  o = alignr(o + sizeof(float) * std::max(B, 1));
  pl->off_partial = o;
  o = alignr(o + sizeof(float) * (size_t)pl->L * pl->Hkv * (size_t)std::max<long long>(pl->total_vis, 1));
  pl->total_bytes = o;
  // staging blob: [error word][meta][items of every chunk][items of visual chunks][positions]
  pl->blob.assign(pl->blob_bytes / sizeof(int32_t), 0);
  int32_t *meta = pl->blob.data() + pl->off_meta / 4;
  int32_t *it1 = pl->blob.data() + pl->off_items1 / 4;
  int32_t *it2 = pl->blob.data() + pl->off_items2 / 4;
  int32_t *pos = pl->blob.data() + pl->off_pos / 4;
  long long sb = 0, i1 = 0, i2 = 0;
  int cb = 0;
  for (int b = 0; b < B; ++b) {
    int32_t *mm = meta + b * kRowsFields;
    const int P = p->cu_seqlens[b + 1] - p->cu_seqlens[b];
    const int N = p->cu_vis[b + 1] - p->cu_vis[b];
    const int M = cu_rows[b + 1] - cu_rows[b];
    const int nch = (P + kRowsChunk - 1) / kRowsChunk;
    mm[kRSeqStart] = p->cu_seqlens[b];
    mm[kRSeqLen] = P;
    mm[kRVisStart] = p->vis_start[b];
    mm[kRVisOff] = p->cu_vis[b];
    mm[kRNumVis] = N;
    mm[kRRowOff] = cu_rows[b];
    mm[kRNumRows] = M;
    mm[kRNumChunks] = nch;
    std::memcpy(mm + kRStatBase, &sb, sizeof sb);   // 64-bit offset in two int32 slots
    mm[kRCoefBase] = cb;
    const int rh = M * pl->L * pl->Hq;
    sb += (long long)rh * nch;
    cb += rh;
    for (int c = 0; c < nch; ++c, ++i1) {
      it1[2 * i1] = b;
      it1[2 * i1 + 1] = c;
    }
    if (N > 0)
      for (int c = p->vis_start[b] / kRowsChunk; c <= (p->vis_start[b] + N - 1) / kRowsChunk; ++c, ++i2) {
        it2[2 * i2] = b;
        it2[2 * i2 + 1] = c;
      }
  }
  for (long long r = 0; r < pl->total_rows; ++r) pos[r] = row_pos[r];
  return LAST_OK;
}

// Dynamic shared memory of a 128-thread kernel holding `cols` TMEM columns: the
// operands, and at least enough that at most 512 / cols CTAs share an SM, so every
// CTA's TMEM allocation is granted at once.
size_t tmem_safe_smem(size_t operands, uint32_t cols) {
  const size_t per_sm = 228 * 1024;
  return std::max(operands, per_sm / (512 / cols + 1) + 1);
}

// One query row per request: the row at position pos attends keys 0 .. pos, which
// is the last-row computation of Eq. 6-8 on the request cut after pos, so the
// last-row scoring kernels take it (the last_scores plan with P'_b = pos + 1).
// Returns LAST_OK only when that plan applies.
last_status single_row_plan(const last_problem *p, const int32_t *cu_rows, const int32_t *row_pos,
                            Plan *lp) {
  if (p->batch < 1 || cu_rows[p->batch] != p->batch) return LAST_ERR_UNSUPPORTED;
  std::vector<int32_t> len(p->batch);
  for (int b = 0; b < p->batch; ++b) len[b] = row_pos[b] + 1;
  last_problem pc = *p;
  if (pc.cu_keep == nullptr) pc.cu_keep = pc.cu_vis;   // scoring needs no budgets
  // a probe: when the plan does not apply, the multi-row kernels run instead and the
  // call's error message must not report the probe's rejection
  const std::string saved = get_error();
  const last_status st = make_plan(&pc, true, false, lp, len.data());
  if (st != LAST_OK) set_error(saved);
  return st;
}

}  // namespace
}  // namespace last

using namespace last;

extern "C" last_status last_scores_rows_workspace_size(const last_problem *p, const int32_t *cu_rows,
                                                       const int32_t *row_pos, size_t *bytes) {
  if (bytes == nullptr) return rows_fail(LAST_ERR_INVALID_ARG, "bytes is NULL");
  RowsPlan pl;
  last_status st = make_rows_plan(p, cu_rows, row_pos, &pl);
  if (st != LAST_OK) return st;
  Plan lp;
  *bytes = pl.total_bytes;
  if (single_row_plan(p, cu_rows, row_pos, &lp) == LAST_OK) *bytes = std::max(*bytes, lp.score_bytes);
  return LAST_OK;
}

extern "C" last_status last_scores_rows(const last_problem *p, const int32_t *cu_rows,
                                        const int32_t *row_pos, const void *q_rows, const void *k,
                                        float *w_out, void *ws, size_t ws_bytes, void *stream) {
  RowsPlan pl;
  last_status st = make_rows_plan(p, cu_rows, row_pos, &pl);
  if (st != LAST_OK) return st;
  Plan lp;
  const bool single = single_row_plan(p, cu_rows, row_pos, &lp) == LAST_OK;
  const size_t need = single ? std::max(pl.total_bytes, lp.score_bytes) : pl.total_bytes;
  if (ws == nullptr) return rows_fail(LAST_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlignR - 1)) != 0)
    return rows_fail(LAST_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return rows_fail(LAST_ERR_WORKSPACE_TOO_SMALL, "workspace needs " + std::to_string(need) + " bytes");
  if (pl.total_vis > 0 && (q_rows == nullptr || k == nullptr || w_out == nullptr))
    return rows_fail(LAST_ERR_INVALID_ARG, "q_rows, k and w_out are required");
  if ((reinterpret_cast<uintptr_t>(q_rows) & 15u) || (reinterpret_cast<uintptr_t>(k) & 15u))
    return rows_fail(LAST_ERR_INVALID_ARG, "q_rows and k must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char *wsc = static_cast<char *>(ws);
  if (single) {
    cudaError_t e = cudaMemcpyAsync(wsc, lp.host_blob.data(), lp.blob_bytes, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = launch_scores(lp, q_rows, k, w_out, wsc, s);
    if (e != cudaSuccess) return rows_fail(LAST_ERR_CUDA, std::string("single-row scoring: ") +
                                                            cudaGetErrorString(e));
    return LAST_OK;
  }
  cudaError_t e = cudaMemcpyAsync(wsc, pl.blob.data(), pl.blob_bytes, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return rows_fail(LAST_ERR_CUDA, std::string("plan copy: ") + cudaGetErrorString(e));
  if (pl.total_vis == 0 || pl.B == 0) return LAST_OK;

  RowsArgs a;
  a.q = static_cast<const __nv_bfloat16 *>(q_rows);
  a.k = static_cast<const __nv_bfloat16 *>(k);
  a.meta = reinterpret_cast<const int32_t *>(wsc + pl.off_meta);
  a.items1 = reinterpret_cast<const int2 *>(wsc + pl.off_items1);
  a.items2 = reinterpret_cast<const int2 *>(wsc + pl.off_items2);
  a.row_pos = reinterpret_cast<const int32_t *>(wsc + pl.off_pos);
  a.stats = reinterpret_cast<float4 *>(wsc + pl.off_stats);
  a.coef = reinterpret_cast<float2 *>(wsc + pl.off_coef);
  a.inv_total = reinterpret_cast<float *>(wsc + pl.off_inv);
  a.partial = reinterpret_cast<float *>(wsc + pl.off_partial);
  a.w = w_out;
  a.total_keys = pl.total_keys;
  a.total_vis = pl.total_vis;
  a.L = pl.L; a.Hq = pl.Hq; a.Hkv = pl.Hkv; a.D = pl.D; a.G = pl.G; a.npad = pl.npad;
  a.tmem_stats = 128;
  uint32_t tp = 32;
  while ((int)tp < pl.npad) tp *= 2;
  a.tmem_probs = tp;
  a.qscale = pl.scale * 1.4426950408889634f;
  a.err = reinterpret_cast<unsigned *>(wsc);
  auto fail_launch = [](cudaError_t err, const char *what) {
    return rows_fail(LAST_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(err));
  };

  const int nkb = pl.D / 64;
  const size_t op = 1024 + (size_t)2 * nkb * kRowsChunk * 128 + 64;
  const size_t smem1 = tmem_safe_smem(op, a.tmem_stats);
  if ((e = cudaFuncSetAttribute(rows_stats_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem1)) != cudaSuccess)
    return fail_launch(e, "rows stats");
  rows_stats_kernel<<<dim3((unsigned)pl.n_items1, pl.L, pl.Hkv * pl.mtiles), kRowsThreads, smem1, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return fail_launch(e, "rows stats launch");
  rows_merge_kernel<<<pl.B, 1024, 0, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return fail_launch(e, "rows merge launch");
  if (pl.n_items2 > 0) {
    const size_t op2 = 1024 + (size_t)nkb * kRowsChunk * 128 + (size_t)nkb * pl.npad * 128 +
                       sizeof(float2) * kRowsMaxN + 64;
    const size_t smem2 = tmem_safe_smem(op2, a.tmem_probs);
    if ((e = cudaFuncSetAttribute(rows_probs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)smem2)) != cudaSuccess)
      return fail_launch(e, "rows probs");
    rows_probs_kernel<<<dim3((unsigned)pl.n_items2, pl.L, pl.Hkv), kRowsThreads, smem2, s>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return fail_launch(e, "rows probs launch");
  }
  const int tiles = (pl.max_vis + kScoreThreads - 1) / kScoreThreads;
  rows_final_kernel<<<dim3(tiles, pl.B), kScoreThreads, 0, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return fail_launch(e, "rows final launch");
  return LAST_OK;
}
