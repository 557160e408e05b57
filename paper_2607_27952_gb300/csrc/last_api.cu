// C-ABI entry points of liblast: argument validation, workspace layout, the
// small host->device plan copy, and the kernel launch sequence.
#include "last_internal.h"

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <numeric>

namespace last {

namespace {
thread_local std::string g_error;

constexpr size_t kAlign = 256;
size_t align_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

last_status fail(last_status st, const std::string &msg) {
  g_error = msg;
  return st;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

void set_error(const std::string &msg) { g_error = msg; }
std::string get_error() { return g_error; }

last_status make_plan(const last_problem *p, bool need_scores, bool need_select, Plan *pl,
                      const int32_t *seq_len) {
  if (p == nullptr) return fail(LAST_ERR_INVALID_ARG, "problem is NULL");
  if (p->batch < 0) return fail(LAST_ERR_INVALID_ARG, "batch < 0");
  if (p->dtype != LAST_DTYPE_F32 && p->dtype != LAST_DTYPE_BF16)
    return fail(LAST_ERR_INVALID_ARG, "dtype must be LAST_DTYPE_F32 or LAST_DTYPE_BF16");
  const int B = p->batch;
  pl->B = B;
  pl->L = p->num_layers;
  pl->Hq = p->num_q_heads;
  pl->Hkv = p->num_kv_heads;
  pl->D = p->head_dim;
  pl->dv = p->feat_dim;
  pl->dtype = p->dtype;
  pl->elem = p->dtype == LAST_DTYPE_F32 ? 4 : 2;

  if (p->cu_vis == nullptr || p->cu_keep == nullptr)
    return fail(LAST_ERR_INVALID_ARG, "cu_vis and cu_keep are required");
  if (p->cu_vis[0] != 0 || p->cu_keep[0] != 0)
    return fail(LAST_ERR_INVALID_ARG, "cu_vis[0] and cu_keep[0] must be 0");
  for (int b = 0; b < B; ++b) {
    const int n = p->cu_vis[b + 1] - p->cu_vis[b];
    const int kb = p->cu_keep[b + 1] - p->cu_keep[b];
    if (n < 0) return fail(LAST_ERR_INVALID_ARG, "cu_vis must be non-decreasing");
    if (kb < 0 || kb > n)
      return fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) + ": need 0 <= k_b <= N_b");
    pl->max_vis = std::max(pl->max_vis, n);
    pl->max_keep = std::max(pl->max_keep, kb);
  }
  pl->total_vis = p->cu_vis[B];
  pl->total_keep = p->cu_keep[B];

  if (need_select) {
    if (p->feat_dim < 8 || p->feat_dim % 8 != 0)
      return fail(LAST_ERR_INVALID_ARG, "feat_dim must be a positive multiple of 8");
    std::string why;
    if (!select_supported(*pl, &why)) return fail(LAST_ERR_UNSUPPORTED, why);
  }

  pl->total_chunks = 0;
  const bool have_seq = p->cu_seqlens != nullptr && p->vis_start != nullptr;
  if (need_scores && !have_seq)
    return fail(LAST_ERR_INVALID_ARG, "cu_seqlens and vis_start are required for scoring");
  if (have_seq && p->num_layers > 0) {
    if (p->num_layers < 1 || p->num_q_heads < 1 || p->num_kv_heads < 1 || p->head_dim < 1)
      return fail(LAST_ERR_INVALID_ARG, "layers, heads and head_dim must be >= 1");
    if (p->num_q_heads % p->num_kv_heads != 0)
      return fail(LAST_ERR_INVALID_ARG, "num_q_heads must be a multiple of num_kv_heads");
    if (!std::isfinite(p->softmax_scale))
      return fail(LAST_ERR_INVALID_ARG, "softmax_scale must be finite");
    if ((long long)p->num_layers * p->num_q_heads > 6144)
      return fail(LAST_ERR_UNSUPPORTED, "num_layers * num_q_heads must be <= 6144");
    if (p->cu_seqlens[0] != 0) return fail(LAST_ERR_INVALID_ARG, "cu_seqlens[0] must be 0");
    pl->G = p->num_q_heads / p->num_kv_heads;
    pl->chunk = score_chunk_keys(p->num_kv_heads);
    pl->scale = p->softmax_scale > 0.f ? p->softmax_scale
                                       : (float)(1.0 / std::sqrt((double)p->head_dim));
    for (int b = 0; b < B; ++b) {
      const int P_full = p->cu_seqlens[b + 1] - p->cu_seqlens[b];
      const int P = seq_len != nullptr ? seq_len[b] : P_full;
      const int n = p->cu_vis[b + 1] - p->cu_vis[b];
      if (P > P_full)
        return fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) + ": cut beyond P_b");
      if (P < 1)
        return fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) +
                                              ": P_b must be >= 1 (the query position)");
      if (p->vis_start[b] < 0 || (long long)p->vis_start[b] + n > (long long)P - 1)
        return fail(LAST_ERR_INVALID_ARG, "request " + std::to_string(b) +
                                              ": visual span must end before the query position");
      pl->max_seq = std::max(pl->max_seq, P);
      pl->total_chunks += (P + pl->chunk - 1) / pl->chunk;
    }
    pl->total_keys = p->cu_seqlens[B];
    if (need_scores) {
      std::string why;
      if (!scores_supported(*pl, &why)) return fail(LAST_ERR_UNSUPPORTED, why);
    }
  } else if (need_scores) {
    return fail(LAST_ERR_INVALID_ARG, "num_layers must be >= 1 for scoring");
  }

  // ---- workspace layout ----
  size_t o = 0;
  pl->off_err = o;
  o = align_up(o + 64);
  pl->off_meta = o;
  o = align_up(o + sizeof(int32_t) * kMetaFields * std::max(B, 1));
  pl->off_items = o;
  o = align_up(o + sizeof(int32_t) * 2 * std::max(pl->total_chunks, 1));
  pl->off_order = o;
  o = align_up(o + sizeof(int32_t) * std::max(B, 1));
  pl->off_gbar = o;   // abort word and one barrier counter per request slot
  o = align_up(o + sizeof(uint32_t) * (1 + kGridMaxReq));
  const size_t blob_end = o;
  pl->off_stats = o;
  o = align_up(o + sizeof(float) * 4 * (size_t)std::max(pl->L, 0) * std::max(pl->Hq, 0) *
                       pl->total_chunks);
  pl->off_zlog = o;
  o = align_up(o + sizeof(float) * (size_t)std::max(pl->L, 0) * std::max(pl->Hq, 0) *
                       (size_t)pl->total_vis);
  pl->off_w = o;
  o = align_up(o + sizeof(float) * (size_t)pl->total_vis);
  pl->score_bytes = o;
  // The bf16 greedy's row skipping keeps up to kRootsPerRequest feature rows per
  // request (min(k_b, kRootsPerRequest) rounded up to whole groups of 16, each row
  // padded to whole 64-element blocks) and a table of bounds per root.
  pl->root_rows = 0;
  const bool sel_scratch = p->dtype == LAST_DTYPE_BF16 && p->feat_dim >= 8 &&
                           p->feat_dim % 8 == 0 && p->feat_dim <= kMaxFeatDim;
  auto root_cap = [&](int b) {
    return (std::min(p->cu_keep[b + 1] - p->cu_keep[b], kRootsPerRequest) + 15) / 16 * 16;
  };
  if (sel_scratch)
    for (int b = 0; b < B; ++b) pl->root_rows += root_cap(b);
  pl->off_roots = o;
  o = align_up(o + (size_t)pl->root_rows * (size_t)((std::max(p->feat_dim, 0) + 63) / 64) * 128);
  pl->off_rtab = o;
  o = align_up(o + (size_t)pl->root_rows * kRootTableCols * sizeof(float));
  // the whole-GPU selection's published keys, for launches that may take it
  pl->off_gpub = o;
  if (B <= kGridMaxReq && pl->max_vis >= kGridMinTokens) o = align_up(o + grid_pub_bytes());
  pl->total_bytes = o;

  // ---- host staging: [err words][meta][items][order], one copy ----
  pl->blob_bytes = blob_end;
  pl->host_blob.assign(blob_end / sizeof(int32_t), 0);
  int32_t *meta = pl->host_blob.data() + pl->off_meta / 4;
  int32_t *items = pl->host_blob.data() + pl->off_items / 4;
  int32_t *order = pl->host_blob.data() + pl->off_order / 4;
  int chunk = 0;
  long long root_off = 0;
  for (int b = 0; b < B; ++b) {
    int32_t *m = meta + b * kMetaFields;
    m[kRootOff] = (int32_t)root_off;
    if (sel_scratch) root_off += root_cap(b);
    m[kVisOff] = p->cu_vis[b];
    m[kNumVis] = p->cu_vis[b + 1] - p->cu_vis[b];
    m[kKeepOff] = p->cu_keep[b];
    m[kNumKeep] = p->cu_keep[b + 1] - p->cu_keep[b];
    if (have_seq && p->num_layers > 0) {
      m[kSeqStart] = p->cu_seqlens[b];
      m[kSeqLen] = seq_len != nullptr ? seq_len[b] : p->cu_seqlens[b + 1] - p->cu_seqlens[b];
      m[kVisStart] = p->vis_start[b];
      m[kChunkBase] = chunk;
      const int nch = (m[kSeqLen] + pl->chunk - 1) / pl->chunk;
      for (int c = 0; c < nch; ++c) {
        items[2 * (chunk + c)] = b;
        items[2 * (chunk + c) + 1] = c;
      }
      chunk += nch;
    }
  }
  // selection clusters take the most expensive requests (k_b * N_b) first
  std::vector<int> ord(B);
  std::iota(ord.begin(), ord.end(), 0);
  std::stable_sort(ord.begin(), ord.end(), [&](int a, int c) {
    const long long wa = (long long)meta[a * kMetaFields + kNumKeep] * meta[a * kMetaFields + kNumVis];
    const long long wc = (long long)meta[c * kMetaFields + kNumKeep] * meta[c * kMetaFields + kNumVis];
    return wa > wc;
  });
  for (int b = 0; b < B; ++b) order[b] = ord[b];
  return LAST_OK;
}

namespace {

last_status check_ws(const Plan &pl, const void *ws, size_t ws_bytes, bool scores_only = false) {
  if (ws == nullptr) return fail(LAST_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0)
    return fail(LAST_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const size_t need = scores_only ? pl.score_bytes : pl.total_bytes;
  if (ws_bytes < need)
    return fail(LAST_ERR_WORKSPACE_TOO_SMALL, "workspace needs " + std::to_string(need) + " bytes");
  return LAST_OK;
}

last_status cuda_fail(cudaError_t e, const char *what) {
  return fail(LAST_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// Device copies of last_prune_host's tensors after the plan workspace, each
// 256-byte aligned.
struct HostLayout {
  size_t q, k, x, w, idx, xo, total;
  size_t q_bytes, k_bytes, x_bytes, w_bytes, idx_bytes, xo_bytes;
};
HostLayout host_layout(const Plan &pl) {
  auto al = [](size_t v) { return (v + kAlign - 1) & ~(size_t)(kAlign - 1); };
  HostLayout h;
  h.q_bytes = (size_t)pl.B * pl.L * pl.Hq * pl.D * pl.elem;
  h.k_bytes = (size_t)pl.L * pl.total_keys * pl.Hkv * pl.D * pl.elem;
  h.x_bytes = (size_t)pl.total_vis * pl.dv * pl.elem;
  h.w_bytes = (size_t)pl.total_vis * sizeof(float);
  h.idx_bytes = (size_t)pl.total_keep * sizeof(int32_t);
  h.xo_bytes = (size_t)pl.total_keep * pl.dv * pl.elem;
  size_t o = al(pl.total_bytes);
  h.q = o; o += al(h.q_bytes);
  h.k = o; o += al(h.k_bytes);
  h.x = o; o += al(h.x_bytes);
  h.w = o; o += al(h.w_bytes);
  h.idx = o; o += al(h.idx_bytes);
  h.xo = o; o += al(h.xo_bytes);
  h.total = o;
  return h;
}

last_status stage(const Plan &pl, void *ws, cudaStream_t s) {
  cudaError_t e = cudaMemcpyAsync(ws, pl.host_blob.data(), pl.blob_bytes, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e, "plan copy");
  return LAST_OK;
}

}  // namespace
}  // namespace last

using namespace last;

extern "C" {

last_status last_workspace_size(const last_problem *p, size_t *bytes) {
  if (bytes == nullptr) return fail(LAST_ERR_INVALID_ARG, "bytes is NULL");
  Plan pl;
  const bool have_seq = p != nullptr && p->cu_seqlens != nullptr && p->vis_start != nullptr &&
                        p->num_layers > 0;
  last_status st = make_plan(p, have_seq, false, &pl);
  if (st != LAST_OK) return st;
  *bytes = pl.total_bytes;
  return LAST_OK;
}

last_status last_scores(const last_problem *p, const void *q, const void *k, float *w_out,
                        void *ws, size_t ws_bytes, void *stream) {
  Plan pl;
  last_status st = make_plan(p, true, false, &pl);
  if (st != LAST_OK) return st;
  if ((st = check_ws(pl, ws, ws_bytes, true)) != LAST_OK) return st;
  if (pl.total_vis > 0 && (q == nullptr || k == nullptr || w_out == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "q, k and w_out are required");
  if (!aligned16(q) || !aligned16(k)) return fail(LAST_ERR_INVALID_ARG, "q and k must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  cudaError_t e = launch_scores(pl, q, k, w_out, static_cast<char *>(ws), s);
  if (e != cudaSuccess) return cuda_fail(e, "scoring launch");
  return LAST_OK;
}

namespace {
last_status check_select_fits(const last::Plan &pl) {
  std::string why;
  return last::select_fits(pl, &why) ? LAST_OK : fail(LAST_ERR_UNSUPPORTED, why);
}
}  // namespace

last_status last_select(const last_problem *p, const float *w, const void *x, int32_t *idx_out,
                        void *x_out, void *ws, size_t ws_bytes, void *stream) {
  Plan pl;
  last_status st = make_plan(p, false, true, &pl);
  if (st != LAST_OK) return st;
  if ((st = check_select_fits(pl)) != LAST_OK) return st;
  if ((st = check_ws(pl, ws, ws_bytes)) != LAST_OK) return st;
  if (pl.total_keep > 0 && (w == nullptr || x == nullptr || idx_out == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "w, x and idx_out are required");
  if (!aligned16(x) || !aligned16(x_out))
    return fail(LAST_ERR_INVALID_ARG, "x and x_out must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  cudaError_t e = launch_select(pl, w, x, idx_out, x_out, static_cast<char *>(ws), s);
  if (e != cudaSuccess) return cuda_fail(e, "selection launch");
  return LAST_OK;
}

last_status last_select_topk(const last_problem *p, const float *w, const void *x,
                             int32_t *idx_out, void *x_out, void *ws, size_t ws_bytes,
                             void *stream) {
  Plan pl;
  last_status st = make_plan(p, false, false, &pl);
  if (st != LAST_OK) return st;
  if ((st = check_ws(pl, ws, ws_bytes)) != LAST_OK) return st;
  if (pl.total_keep > 0 && (w == nullptr || idx_out == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "w and idx_out are required");
  if (x_out != nullptr) {
    if (p->feat_dim < 8 || p->feat_dim % 8 != 0)
      return fail(LAST_ERR_INVALID_ARG, "feat_dim must be a positive multiple of 8");
    if (pl.total_keep > 0 && x == nullptr)
      return fail(LAST_ERR_INVALID_ARG, "x is required when x_out is given");
    if (!aligned16(x) || !aligned16(x_out))
      return fail(LAST_ERR_INVALID_ARG, "x and x_out must be 16-byte aligned");
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  char *wsc = static_cast<char *>(ws);
  cudaError_t e = launch_topk(pl, w, idx_out, wsc, s);
  if (e != cudaSuccess) return cuda_fail(e, "top-k launch");
  if (x_out != nullptr) {
    e = launch_gather(pl, x, idx_out, x_out, wsc, s);
    if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  }
  return LAST_OK;
}

last_status last_gather(const last_problem *p, const void *x, const int32_t *idx, void *x_out,
                        void *ws, size_t ws_bytes, void *stream) {
  Plan pl;
  // Eq. 12 is a row copy: only the row width must suit the kernel's 16-byte copies
  // (the selection's own feature-width limit does not apply)
  last_status st = make_plan(p, false, false, &pl);
  if (st != LAST_OK) return st;
  if (p->feat_dim < 8 || p->feat_dim % 8 != 0)
    return fail(LAST_ERR_INVALID_ARG, "feat_dim must be a positive multiple of 8");
  if ((st = check_ws(pl, ws, ws_bytes)) != LAST_OK) return st;
  if (pl.total_keep > 0 && (x == nullptr || idx == nullptr || x_out == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "x, idx and x_out are required");
  if (!aligned16(x) || !aligned16(x_out))
    return fail(LAST_ERR_INVALID_ARG, "x and x_out must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  cudaError_t e = launch_gather(pl, x, idx, x_out, static_cast<char *>(ws), s);
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  return LAST_OK;
}

last_status last_prune(const last_problem *p, const void *q, const void *k, const void *x,
                       float *w_out, int32_t *idx_out, void *x_out, void *ws, size_t ws_bytes,
                       void *stream) {
  Plan pl;
  last_status st = make_plan(p, true, true, &pl);
  if (st != LAST_OK) return st;
  if ((st = check_select_fits(pl)) != LAST_OK) return st;
  if ((st = check_ws(pl, ws, ws_bytes)) != LAST_OK) return st;
  if (pl.total_vis > 0 && (q == nullptr || k == nullptr || x == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "q, k and x are required");
  if (pl.total_keep > 0 && idx_out == nullptr)
    return fail(LAST_ERR_INVALID_ARG, "idx_out is required");
  if (!aligned16(q) || !aligned16(k) || !aligned16(x) || !aligned16(x_out))
    return fail(LAST_ERR_INVALID_ARG, "q, k, x and x_out must be 16-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char *wsc = static_cast<char *>(ws);
  float *w = w_out != nullptr ? w_out : reinterpret_cast<float *>(wsc + pl.off_w);
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  cudaError_t e = launch_scores(pl, q, k, w, wsc, s);
  if (e != cudaSuccess) return cuda_fail(e, "scoring launch");
  e = launch_select(pl, w, x, idx_out, x_out, wsc, s);
  if (e != cudaSuccess) return cuda_fail(e, "selection launch");
  return LAST_OK;
}

last_status last_host_workspace_size(const last_problem *p, size_t *bytes) {
  if (bytes == nullptr) return fail(LAST_ERR_INVALID_ARG, "bytes is NULL");
  Plan pl;
  last_status st = make_plan(p, true, true, &pl);
  if (st != LAST_OK) return st;
  *bytes = host_layout(pl).total;
  return LAST_OK;
}

last_status last_prune_host(const last_problem *p, const void *q, const void *k, const void *x,
                            float *w_out, int32_t *idx_out, void *x_out, void *ws, size_t ws_bytes,
                            void *stream) {
  Plan pl;
  last_status st = make_plan(p, true, true, &pl);
  if (st != LAST_OK) return st;
  if ((st = check_select_fits(pl)) != LAST_OK) return st;
  const HostLayout h = host_layout(pl);
  if (ws == nullptr) return fail(LAST_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0)
    return fail(LAST_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (ws_bytes < h.total)
    return fail(LAST_ERR_WORKSPACE_TOO_SMALL,
                "last_prune_host's workspace needs " + std::to_string(h.total) + " bytes");
  if (pl.total_vis > 0 && (q == nullptr || k == nullptr || x == nullptr))
    return fail(LAST_ERR_INVALID_ARG, "q, k and x are required");
  if (pl.total_keep > 0 && idx_out == nullptr)
    return fail(LAST_ERR_INVALID_ARG, "idx_out is required");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char *wsc = static_cast<char *>(ws);
  void *qd = wsc + h.q, *kd = wsc + h.k, *xd = wsc + h.x, *xod = wsc + h.xo;
  float *wd = reinterpret_cast<float *>(wsc + h.w);
  int32_t *idd = reinterpret_cast<int32_t *>(wsc + h.idx);
  cudaError_t e = cudaSuccess;
  // one copy per tensor
  if (h.q_bytes && e == cudaSuccess) e = cudaMemcpyAsync(qd, q, h.q_bytes, cudaMemcpyHostToDevice, s);
  if (h.k_bytes && e == cudaSuccess) e = cudaMemcpyAsync(kd, k, h.k_bytes, cudaMemcpyHostToDevice, s);
  if (h.x_bytes && e == cudaSuccess) e = cudaMemcpyAsync(xd, x, h.x_bytes, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e, "host-to-device copy");
  if ((st = stage(pl, ws, s)) != LAST_OK) return st;
  e = launch_scores(pl, qd, kd, wd, wsc, s);
  if (e != cudaSuccess) return cuda_fail(e, "scoring launch");
  e = launch_select(pl, wd, xd, idd, x_out != nullptr ? xod : nullptr, wsc, s);
  if (e != cudaSuccess) return cuda_fail(e, "selection launch");
  if (h.idx_bytes && e == cudaSuccess)
    e = cudaMemcpyAsync(idx_out, idd, h.idx_bytes, cudaMemcpyDeviceToHost, s);
  if (x_out != nullptr && h.xo_bytes && e == cudaSuccess)
    e = cudaMemcpyAsync(x_out, xod, h.xo_bytes, cudaMemcpyDeviceToHost, s);
  if (w_out != nullptr && h.w_bytes && e == cudaSuccess)
    e = cudaMemcpyAsync(w_out, wd, h.w_bytes, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return cuda_fail(e, "device-to-host copy");
  return LAST_OK;
}

last_status last_poll(const void *ws, void *stream) {
  if (ws == nullptr) return fail(LAST_ERR_INVALID_ARG, "workspace is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned flag = 0;
  cudaError_t e = cudaMemcpyAsync(&flag, ws, sizeof flag, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "poll");
  if (flag & kErrConfig)
    return fail(LAST_ERR_CUDA, "internal error: a kernel's shared-memory plan exceeded its launch; "
                               "outputs of that call are invalid");
  if (flag & kErrTimeout)
    return fail(LAST_ERR_TIMEOUT, "a bounded device wait expired; outputs of that call are invalid");
  if (flag & kErrGatherIndex)
    return fail(LAST_ERR_DEVICE_INDEX, "a gather index was outside [0, N_b)");
  return LAST_OK;
}

int32_t last_budget(int32_t n_vis, int32_t num, int32_t den) {
  if (n_vis < 0 || num < 0 || den <= 0) return -1;
  const long long prod = (long long)num * n_vis;
  long long kq = prod / den;
  if (kq * den < prod) ++kq;
  return kq > 0x7fffffffLL ? -1 : (int32_t)kq;
}

const char *last_status_string(last_status s) {
  switch (s) {
    case LAST_OK: return "LAST_OK";
    case LAST_ERR_INVALID_ARG: return "LAST_ERR_INVALID_ARG";
    case LAST_ERR_UNSUPPORTED: return "LAST_ERR_UNSUPPORTED";
    case LAST_ERR_WORKSPACE_TOO_SMALL: return "LAST_ERR_WORKSPACE_TOO_SMALL";
    case LAST_ERR_CUDA: return "LAST_ERR_CUDA";
    case LAST_ERR_DEVICE_INDEX: return "LAST_ERR_DEVICE_INDEX";
    case LAST_ERR_TIMEOUT: return "LAST_ERR_TIMEOUT";
  }
  return "LAST_ERR_UNKNOWN";
}

const char *last_error_message(void) { return g_error.c_str(); }

}  // extern "C"
