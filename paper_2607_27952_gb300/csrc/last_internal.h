// Host-side plan shared by the entry points and the kernel launchers.
#pragma once

#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "last.h"

namespace last {

// Per-request metadata row staged into the workspace (int32 each).
enum MetaField : int {
  kSeqStart = 0,   // cu_seqlens[b]
  kSeqLen,         // P_b
  kVisStart,       // v_b (position of the first visual token)
  kVisOff,         // cu_vis[b]
  kNumVis,         // N_b
  kKeepOff,        // cu_keep[b]
  kNumKeep,        // k_b
  kChunkBase,      // first score chunk of request b
  kRootOff,        // first row of request b in the selection's root rows
  kMetaFields
};

constexpr int kScoreThreads = 256;
constexpr int kTokenTile = kScoreThreads;   // visual tokens per score_tokens_kernel CTA
constexpr int kMaxGroup = 8;         // q-heads per kv-head supported by the scoring kernel
constexpr int kMaxFeatDim = 2048;    // selection keeps x_j in 64 fp32 registers per lane
constexpr int kRootsPerRequest = 1024;   // root rows per request (the selection's kMaxRoots)
constexpr int kRootTableCols = 32;       // bound-table columns per root (the selection's kMaxAccept)
constexpr int kSelectWarps = 8;
constexpr int kGridMaxReq = 4;      // requests of one whole-GPU selection launch
constexpr int kGridMaxCtas = 256;   // CTAs of one whole-GPU selection launch at most
constexpr int kGatherThreads = 256;

// Device error flags (first word of the workspace).
constexpr unsigned kErrGatherIndex = 1u;
constexpr unsigned kErrTimeout = 2u;      // a bounded wait on a bulk copy expired
constexpr unsigned kErrConfig = 4u;       // a kernel's shared-memory plan exceeded its launch

struct Plan {
  // problem
  int B = 0, L = 0, Hq = 0, Hkv = 0, D = 0, dv = 0, dtype = 0;
  int G = 0, elem = 0;
  float scale = 0.f;
  long long total_keys = 0, total_vis = 0, total_keep = 0;
  int max_seq = 0, max_vis = 0, max_keep = 0;
  int chunk = 0;          // keys per scoring CTA (score_chunk_keys)
  int total_chunks = 0;
  // workspace byte offsets
  size_t off_err = 0, off_meta = 0, off_items = 0, off_order = 0;
  size_t off_stats = 0, off_zlog = 0, off_w = 0, total_bytes = 0;
  // bf16 selection scratch: root rows [root_rows][dv] and the bound table
  // [root_rows][kRootTableCols] (after the scoring scratch; score_bytes excludes them)
  size_t off_roots = 0, off_rtab = 0, score_bytes = 0;
  // whole-GPU selection: barrier counters (zeroed with the staged plan) and the
  // published keys
  size_t off_gbar = 0, off_gpub = 0;
  long long root_rows = 0;
  // host staging (error word, meta rows, score items, selection order) in ws order
  std::vector<int32_t> host_blob;
  size_t blob_bytes = 0;  // bytes from off_meta to the end of the order array
};

// Validation + layout.  `need_scores` / `need_select` widen the checks to the
// parts a call uses.  Returns LAST_OK or an error with a message set.
// seq_len (nullable): per-request key counts P'_b <= P_b to score instead of P_b
// (keys 0 .. P'_b - 1 of each request, whose last one is then the query row).
last_status make_plan(const last_problem *p, bool need_scores, bool need_select, Plan *plan,
                      const int32_t *seq_len = nullptr);

void set_error(const std::string &msg);
std::string get_error();   // the message last_error_message() returns on this thread

// Kernel launchers (return cudaSuccess or the launch error).
cudaError_t launch_scores(const Plan &pl, const void *q, const void *k, float *w_out,
                          char *ws, cudaStream_t s);
cudaError_t launch_select(const Plan &pl, const float *w, const void *x, int32_t *idx_out,
                          void *x_out, char *ws, cudaStream_t s);
cudaError_t launch_gather(const Plan &pl, const void *x, const int32_t *idx, void *x_out,
                          char *ws, cudaStream_t s);
// The whole-GPU selection of a few long requests (select_grid.cu).
cudaError_t launch_select_grid(const Plan &pl, const float *w, const void *x, int32_t *idx_out,
                               void *x_out, char *ws, cudaStream_t s);
size_t grid_select_smem(int row_bytes, int tpc);
size_t grid_pub_bytes();
// Whether the whole-GPU selection can run the plan's requests on the current device
// (it takes requests too long for any thread-block cluster, at most kGridMaxReq).
bool grid_select_fits(const Plan &pl);
// Requests shorter than this always fit a cluster: their workspace needs no
// room for the whole-GPU selection.
constexpr int kGridMinTokens = 4096;

cudaError_t launch_topk(const Plan &pl, const float *w, int32_t *idx_out, char *ws,
                        cudaStream_t s);

// Keys per scoring CTA for a given number of kv-heads (a multiple of 16).
int score_chunk_keys(int num_kv_heads);

// Checks the compiled limits of the scoring / selection kernels.
bool scores_supported(const Plan &pl, std::string *why);
bool select_supported(const Plan &pl, std::string *why);
// Whether the greedy selection's shared-memory plan holds the longest request.
bool select_fits(const Plan &pl, std::string *why);

}  // namespace last
