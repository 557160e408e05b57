// Table 4 (attention sources): the importance of Eq. 7 from the attention rows of
// several query positions per request (First, Middle, All Mean), bf16 q and K.
//
// Request b has M_b query rows at positions row_pos (after its visual span); row m
// sees the keys 0 .. row_pos[m] (causal softmax, Eq. 6).  Scores are summed over
// rows, layers and q-heads at the visual positions and normalised (Eq. 8).
//
// rows_logits_kernel: one CTA of 128 threads per (request, 128-key chunk, layer,
//   kv-head g).  The chunk's keys of g (A, M = 128) and the request's query rows of
//   the G q-heads of g (B, N = M_b * G padded to a multiple of 16) are staged in
//   shared memory in the K-major 128-byte-swizzled layout; one thread issues
//   tcgen05.mma (bf16, fp32 accumulator in TMEM) over D / 64 K blocks.  Thread t
//   owns key t (TMEM lane t): per column (row, head) it masks keys past the row's
//   position, and the CTA reduces the column's max and its sums of 2^(z - max) over
//   all and over the visual keys (log2 domain), and writes the visual logits.
// rows_tokens_kernel: one CTA per (request, 256 visual tokens): merges each
//   (row, layer, head)'s chunk statistics in chunk order and sums the visual
//   tokens' probabilities over them, divided by the total visual mass.
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

namespace last {

namespace {

// Per-request metadata (int32 slots; the two 64-bit offsets take two slots each
// and sit 8-byte aligned since a row is 12 slots).
enum RowsField : int {
  kRSeqStart = 0, kRSeqLen, kRVisStart, kRVisOff, kRNumVis, kRRowOff, kRNumRows,
  kRNumChunks, kRStatBase = 8, kRZlogBase = 10, kRowsFields = 12
};

constexpr int kRowsChunk = 128;     // keys per CTA (MMA M)
constexpr int kRowsThreads = 128;
constexpr int kRowsMaxN = 256;      // query rows x heads per kv-head (MMA N)
constexpr int kRowsMaxRH = 6144;    // (row, layer, head) triples per request

struct RowsArgs {
  const __nv_bfloat16 *q, *k;
  const int32_t *meta;
  const int2 *items;
  const int32_t *row_pos;
  float4 *stats;
  float *zlog;
  float *w;
  long long total_keys;
  int L, Hq, Hkv, D, G, npad;
  uint32_t tmem_cols;
  float qscale;          // softmax scale * log2(e)
  unsigned *err;
};

}  // namespace

__global__ void __launch_bounds__(kRowsThreads)
rows_logits_kernel(const RowsArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int nkb = a.D / 64;
  const int npad = a.npad;
  unsigned char *sA = smem;                                   // nkb x [128 keys][128 B]
  unsigned char *sB = smem + nkb * kRowsChunk * 128;          // nkb x [npad rows][128 B]
  float *red = reinterpret_cast<float *>(sB + (size_t)nkb * npad * 128);   // [4][16] x 2
  float *colv = red + 2 * 4 * 16;                              // [16] column max
  unsigned long long *bar = reinterpret_cast<unsigned long long *>(colv + 16);
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int2 item = a.items[blockIdx.x];
  const int b = item.x, c = item.y, l = blockIdx.y, g = blockIdx.z;
  const int32_t *m = a.meta + b * kRowsFields;
  const int seq0 = m[kRSeqStart], P = m[kRSeqLen], v0 = m[kRVisStart];
  const int nvis = m[kRNumVis], row0 = m[kRRowOff], nrows = m[kRNumRows];
  const int nch = m[kRNumChunks];
  const long long sbase = ((const long long *)(m + kRStatBase))[0];
  const long long zbase = ((const long long *)(m + kRZlogBase))[0];
  const int G = a.G, ncol = nrows * G;

  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, a.tmem_cols);

  // A: key t of the chunk, 16-byte chunk j -> K block j / 8, row t, swizzled column
  {
    const int p = c * kRowsChunk + tid;
    const __nv_bfloat16 *src = a.k + (((long long)l * a.total_keys + seq0 + p) * a.Hkv + g) * a.D;
    for (int j = 0; j < a.D / 8; ++j) {
      const U4 v = p < P ? ldg(src + 8 * j) : U4{0, 0, 0, 0};
      *reinterpret_cast<U4 *>(sA + (j >> 3) * (kRowsChunk * 128) + tid * 128 +
                              (((j & 7) ^ (tid & 7)) << 4)) = v;
    }
  }
  // B: column n = (row n / G, head g * G + n % G)
  for (int idx = tid; idx < npad * (a.D / 8); idx += kRowsThreads) {
    const int n = idx / (a.D / 8), j = idx - n * (a.D / 8);
    U4 v = U4{0, 0, 0, 0};
    if (n < ncol) {
      const int r = n / G, gg = n - r * G;
      v = ldg(a.q + (((long long)(row0 + r) * a.L + l) * a.Hq + g * G + gg) * a.D + 8 * j);
    }
    *reinterpret_cast<U4 *>(sB + (j >> 3) * (npad * 128) + n * 128 + (((j & 7) ^ (n & 7)) << 4)) = v;
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (tid == 0) {
    const uint32_t idesc = umma_idesc_bf16(kRowsChunk, npad);
    for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
      for (int k = 0; k < 4; ++k)
        umma_bf16(tmem, umma_desc_sw128(smem_addr(sA + kb * (kRowsChunk * 128)) + k * 32),
                  umma_desc_sw128(smem_addr(sB + kb * (npad * 128)) + k * 32), idesc,
                  (kb | k) != 0 ? 1u : 0u);
    umma_commit(bar);
  }
  __syncwarp();
  mbar_wait_bounded(bar, 0, a.err, kErrTimeout);
  tc_fence_after();

  const int p = c * kRowsChunk + tid;                  // this thread's key
  const bool key_ok = p < P;
  const bool vis = p >= v0 && p < v0 + nvis;
  for (int n0 = 0; n0 < ncol; n0 += 16) {
    uint32_t raw[16];
    tmem_ld16(tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)n0, raw);
    float z[16];
    bool use[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int n = n0 + j;
      const int pos = n < ncol ? a.row_pos[row0 + n / G] : -1;
      use[j] = key_ok && n < ncol && p <= pos;
      z[j] = use[j] ? __uint_as_float(raw[j]) * a.qscale : -INFINITY;
    }
    // column max over the 128 keys
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float v = z[j];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
      if (lane == 0) red[warp * 16 + j] = v;
    }
    __syncthreads();
    if (tid < 16)
      colv[tid] = fmaxf(fmaxf(red[tid], red[16 + tid]), fmaxf(red[32 + tid], red[48 + tid]));
    __syncthreads();
    // sums of 2^(z - max) over all keys and over the visual keys
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float e = use[j] ? exp2f(z[j] - colv[j]) : 0.f;
      float ev = vis ? e : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        e += __shfl_xor_sync(0xffffffffu, e, o);
        ev += __shfl_xor_sync(0xffffffffu, ev, o);
      }
      if (lane == 0) {
        red[warp * 16 + j] = e;
        red[64 + warp * 16 + j] = ev;
      }
    }
    __syncthreads();
    if (tid < 16 && n0 + tid < ncol) {
      const int n = n0 + tid, r = n / G, h = g * G + (n - r * G);
      const float s = (red[tid] + red[16 + tid]) + (red[32 + tid] + red[48 + tid]);
      const float sv = (red[64 + tid] + red[80 + tid]) + (red[96 + tid] + red[112 + tid]);
      const long long rh = ((long long)r * a.L + l) * a.Hq + h;
      a.stats[sbase + rh * nch + c] = make_float4(colv[tid], s, sv, 0.f);
    }
    // visual logits
    if (vis && key_ok) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int n = n0 + j;
        if (n < ncol) {
          const int r = n / G, h = g * G + (n - r * G);
          const long long rh = ((long long)r * a.L + l) * a.Hq + h;
          a.zlog[zbase + rh * nvis + (p - v0)] = z[j];
        }
      }
    }
    __syncthreads();   // red / colv are reused by the next column group
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, a.tmem_cols);
}

__global__ void __launch_bounds__(kScoreThreads)
rows_tokens_kernel(const RowsArgs a) {
  extern __shared__ float coef[];     // [RH] max, [RH] 1/Z, [RH] V/Z
  __shared__ float inv_total_s;
  const int b = blockIdx.y, tile = blockIdx.x;
  const int32_t *m = a.meta + b * kRowsFields;
  const int nvis = m[kRNumVis], voff = m[kRVisOff], nrows = m[kRNumRows], nch = m[kRNumChunks];
  if (tile * kTokenTile >= nvis) return;
  const long long sbase = ((const long long *)(m + kRStatBase))[0];
  const long long zbase = ((const long long *)(m + kRZlogBase))[0];
  const int RH = nrows * a.L * a.Hq;
  float *cmax = coef, *cinv = coef + RH, *cvis = coef + 2 * RH;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int rh = warp; rh < RH; rh += kScoreThreads / 32) {
    const float4 *st = a.stats + sbase + (long long)rh * nch;
    float mx = -INFINITY;
    for (int cc = lane; cc < nch; cc += 32) mx = fmaxf(mx, st[cc].x);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f, vz = 0.f;
    for (int cc = lane; cc < nch; cc += 32) {
      const float4 v = st[cc];
      const float f = v.x == -INFINITY ? 0.f : exp2f(v.x - mx);   // chunks past the row
      z += v.y * f;
      vz += v.z * f;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      z += __shfl_xor_sync(0xffffffffu, z, o);
      vz += __shfl_xor_sync(0xffffffffu, vz, o);
    }
    if (lane == 0) {
      cmax[rh] = mx;
      cinv[rh] = 1.0f / z;
      cvis[rh] = vz / z;
    }
  }
  __syncthreads();
  if (warp == 0) {
    float t = 0.f;
    for (int rh = lane; rh < RH; rh += 32) t += cvis[rh];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) inv_total_s = 1.0f / t;
  }
  __syncthreads();
  const int i = tile * kTokenTile + threadIdx.x;
  if (i < nvis) {
    const float *zl = a.zlog + zbase + i;
    float s0 = 0.f, s1 = 0.f;
    int rh = 0;
    for (; rh + 2 <= RH; rh += 2) {
      s0 += exp2f(zl[(long long)rh * nvis] - cmax[rh]) * cinv[rh];
      s1 += exp2f(zl[(long long)(rh + 1) * nvis] - cmax[rh + 1]) * cinv[rh + 1];
    }
    if (rh < RH) s0 += exp2f(zl[(long long)rh * nvis] - cmax[rh]) * cinv[rh];
    a.w[voff + i] = (s0 + s1) * inv_total_s;
  }
}

namespace {

struct RowsPlan {
  int B = 0, L = 0, Hq = 0, Hkv = 0, D = 0, G = 0, npad = 0, max_vis = 0, max_rh = 0;
  long long total_keys = 0, total_vis = 0, total_rows = 0, total_items = 0;
  size_t off_meta = 0, off_items = 0, off_pos = 0, off_stats = 0, off_zlog = 0, total_bytes = 0;
  size_t blob_bytes = 0;
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
  long long stats = 0, zlog = 0;
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
    pl->max_rh = std::max<int>(pl->max_rh, (int)rh);
    const int nch = (P + kRowsChunk - 1) / kRowsChunk;
    stats += rh * nch;
    zlog += rh * N;
    pl->total_items += nch;
    pl->max_vis = std::max(pl->max_vis, N);
  }
  if (max_cols > kRowsMaxN)
    return rows_fail(LAST_ERR_UNSUPPORTED, "query rows x (num_q_heads / num_kv_heads) must be <= 256");
  pl->npad = std::max(16, (max_cols + 15) / 16 * 16);
  pl->total_keys = p->cu_seqlens[B];
  pl->total_vis = p->cu_vis[B];
  pl->total_rows = cu_rows[B];
  size_t o = 0;
  o = alignr(o + 64);                       // error word
  pl->off_meta = o;
  o = alignr(o + sizeof(int32_t) * kRowsFields * std::max(B, 1));
  pl->off_items = o;
  o = alignr(o + sizeof(int32_t) * 2 * std::max<long long>(pl->total_items, 1));
  pl->off_pos = o;
  o = alignr(o + sizeof(int32_t) * std::max<long long>(pl->total_rows, 1));
  pl->blob_bytes = o;
  pl->off_stats = o;
  o = alignr(o + sizeof(float) * 4 * (size_t)std::max<long long>(stats, 1));
  pl->off_zlog = o;
  o = alignr(o + sizeof(float) * (size_t)std::max<long long>(zlog, 1));
  pl->total_bytes = o;
  // staging blob: [error word][meta][items][row positions]
  pl->blob.assign(pl->blob_bytes / sizeof(int32_t), 0);
  int32_t *meta = pl->blob.data() + pl->off_meta / 4;
  int32_t *items = pl->blob.data() + pl->off_items / 4;
  int32_t *pos = pl->blob.data() + pl->off_pos / 4;
  long long sb = 0, zb = 0, it = 0;
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
    std::memcpy(mm + kRStatBase, &sb, sizeof sb);   // 64-bit offsets in two int32 slots
    std::memcpy(mm + kRZlogBase, &zb, sizeof zb);
    const long long rh = (long long)M * pl->L * pl->Hq;
    sb += rh * nch;
    zb += rh * N;
    for (int c = 0; c < nch; ++c, ++it) {
      items[2 * it] = b;
      items[2 * it + 1] = c;
    }
  }
  for (long long r = 0; r < pl->total_rows; ++r) pos[r] = row_pos[r];
  return LAST_OK;
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
  *bytes = pl.total_bytes;
  return LAST_OK;
}

extern "C" last_status last_scores_rows(const last_problem *p, const int32_t *cu_rows,
                                        const int32_t *row_pos, const void *q_rows, const void *k,
                                        float *w_out, void *ws, size_t ws_bytes, void *stream) {
  RowsPlan pl;
  last_status st = make_rows_plan(p, cu_rows, row_pos, &pl);
  if (st != LAST_OK) return st;
  if (ws == nullptr) return rows_fail(LAST_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlignR - 1)) != 0)
    return rows_fail(LAST_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (ws_bytes < pl.total_bytes)
    return rows_fail(LAST_ERR_WORKSPACE_TOO_SMALL,
                     "workspace needs " + std::to_string(pl.total_bytes) + " bytes");
  if (pl.total_vis > 0 && (q_rows == nullptr || k == nullptr || w_out == nullptr))
    return rows_fail(LAST_ERR_INVALID_ARG, "q_rows, k and w_out are required");
  if ((reinterpret_cast<uintptr_t>(q_rows) & 15u) || (reinterpret_cast<uintptr_t>(k) & 15u))
    return rows_fail(LAST_ERR_INVALID_ARG, "q_rows and k must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char *wsc = static_cast<char *>(ws);
  cudaError_t e = cudaMemcpyAsync(wsc, pl.blob.data(), pl.blob_bytes, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return rows_fail(LAST_ERR_CUDA, std::string("plan copy: ") + cudaGetErrorString(e));
  if (pl.total_vis == 0 || pl.B == 0) return LAST_OK;

  RowsArgs a;
  a.q = static_cast<const __nv_bfloat16 *>(q_rows);
  a.k = static_cast<const __nv_bfloat16 *>(k);
  a.meta = reinterpret_cast<const int32_t *>(wsc + pl.off_meta);
  a.items = reinterpret_cast<const int2 *>(wsc + pl.off_items);
  a.row_pos = reinterpret_cast<const int32_t *>(wsc + pl.off_pos);
  a.stats = reinterpret_cast<float4 *>(wsc + pl.off_stats);
  a.zlog = reinterpret_cast<float *>(wsc + pl.off_zlog);
  a.w = w_out;
  a.total_keys = pl.total_keys;
  a.L = pl.L; a.Hq = pl.Hq; a.Hkv = pl.Hkv; a.D = pl.D; a.G = pl.G; a.npad = pl.npad;
  uint32_t tcols = 32;
  while ((int)tcols < pl.npad) tcols *= 2;
  a.tmem_cols = tcols;
  a.qscale = pl.scale * 1.4426950408889634f;
  a.err = reinterpret_cast<unsigned *>(wsc);

  // Shared memory: the operands, plus enough that at most 512 / tmem_cols CTAs share
  // an SM, so every CTA's TMEM allocation is granted at once.
  const int nkb = pl.D / 64;
  size_t smem = 1024 + (size_t)nkb * kRowsChunk * 128 + (size_t)nkb * pl.npad * 128 + 1024;
  const size_t per_sm = 228 * 1024;
  const size_t floor_smem = per_sm / (512 / tcols + 1) + 1;
  smem = std::max(smem, floor_smem);
  e = cudaFuncSetAttribute(rows_logits_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return rows_fail(LAST_ERR_CUDA, std::string("rows logits: ") + cudaGetErrorString(e));
  rows_logits_kernel<<<dim3((unsigned)pl.total_items, pl.L, pl.Hkv), kRowsThreads, smem, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess)
    return rows_fail(LAST_ERR_CUDA, std::string("rows logits launch: ") + cudaGetErrorString(e));
  const size_t tsmem = sizeof(float) * 3 * pl.max_rh;
  if (tsmem > 48 * 1024) {
    e = cudaFuncSetAttribute(rows_tokens_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tsmem);
    if (e != cudaSuccess) return rows_fail(LAST_ERR_CUDA, std::string("rows tokens: ") + cudaGetErrorString(e));
  }
  const int tiles = (pl.max_vis + kTokenTile - 1) / kTokenTile;
  rows_tokens_kernel<<<dim3(tiles, pl.B), kScoreThreads, tsmem, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess)
    return rows_fail(LAST_ERR_CUDA, std::string("rows tokens launch: ") + cudaGetErrorString(e));
  return LAST_OK;
}
