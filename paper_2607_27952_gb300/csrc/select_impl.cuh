// Eq. 9-12 (Sec. 3.4): importance-weighted greedy k-center selection and the
// order-restoring gather, fused in one kernel.
//
// One thread-block cluster of C CTAs per request.  CTA r owns the contiguous
// token range [r*T, min(N, (r+1)*T)), T = ceil(N / C), keeps as many of those
// rows resident in shared memory as fit, and holds w~, r = 1/||x||, delta and
// the selected flag of its tokens.
//
// The greedy runs in rounds, each of which accepts a batch of consecutive
// greedy picks at once and yields exactly the sequential Eq. 10-11 sequence:
//   1. every CTA publishes its 4 best unselected keys (w~_i delta_i, index)
//      and the 5th-best key to every CTA of the cluster (DSMEM; barrier);
//   2. the published entries above U = max over CTAs of the 5th-best key form
//      the candidate list L (best first, at most 16; U grows to the first
//      key cut off).  Every token outside L has a key <= U, and keys never
//      increase (delta only shrinks), so U bounds them for the whole round;
//   3. the rows of L are copied into every CTA's shared memory, the CTAs split
//      the pairwise dot products of L between them and broadcast them (barrier);
//   4. every CTA replays the greedy on L alone: take the member with the
//      largest current key; if it is above U it is the true next pick
//      (nothing outside L can beat it), so accept it and fold its distance into
//      the remaining members' delta; stop at U, at the budget, or when L runs out;
//   5. one pass over the CTA's tokens folds all accepted centres into delta
//      (4 tokens x up to 16 centres register-blocked dot products), then
//      recomputes the keys and the CTA's best candidates for the next round.
// The seed (Eq. 9, argmax w~) is a round that accepts exactly one token.
//
// Arithmetic is the canonical fp32 of the public header: lane l of a warp owns
// 8-coordinate groups l, l+32, ...; explicit __fmaf_rn / __fmul_rn / __fsub_rn,
// xor butterfly, argmax ties to the lowest index.  Every dot product of the same
// pair is evaluated identically wherever it is needed, so the result is
// bit-identical to the sequential definition.
//
// Epilogue (Eq. 12): the CTAs exchange their selected counts, then each writes
// its selected indices in ascending order and copies their rows to x_out.
#pragma once

#include "last_device.cuh"
#include "last_internal.h"

#include <cuda.h>   // CUtensorMap (types only; the encoder comes from the runtime's driver entry point)

#include <type_traits>

namespace last {

constexpr int kSelThreads = kSelectWarps * 32;
constexpr int kMaxCluster = 16;
constexpr int kLcap = 32;                          // candidate list capacity (runtime a.lcap <= kLcap)
constexpr int kMaxAccept = 32;                     // picks folded into delta per round (runtime a.max_accept)
constexpr int kTopMax = 17;                        // ranked keys per warp / CTA: <= 16 published + bound
// ranked keys the kernel keeps: 8 + bound on the CUDA-core update (register
// budget), 16 + bound with the tensor-core update
template <bool TC> __host__ __device__ constexpr int top_width() { return TC ? 17 : 9; }
constexpr int kMaxPairs = kLcap * (kLcap - 1) / 2;
constexpr int kRing = 4;                           // async-copy ring depth (groups in flight)

// Tensor-core update (bf16): 128-row tiles of X against up to 16 new centres.
constexpr int kTcBM = 128, kTcBK = 64;             // MMA M; K elements per 128-byte row
                                                   // (MMA N = the candidate list length)
constexpr int kTcMaxStages = 12;                   // TMA ring depth (runtime a.tc_stages)
constexpr int kTcBoxBytes = kTcBM * kTcBK * 2;     // one A box (128 rows x 64 elements): 16 KB
constexpr int kTmemCols = 512;                     // TMEM columns per SM
constexpr int kGramChains = 4;                     // accumulators of the list's Gram

// Row skipping by the triangle inequality (tensor-core variant).  Every accepted
// centre is either a "root" (no earlier root within chordal distance kTriTau) or is
// attached to its nearest root R with an upper bound e >= rho(centre, R), where
// rho(a, b) = |a/|a| - b/|b|| = sqrt(2 (1 - cos(a, b))) is the chordal metric on the
// unit sphere.  Token i with nearest centre o (delta_i = d(i, o)) and o's root R
// satisfies, for a new centre c,
//   rho(i, c) >= rho(R, c) - rho(R, o) - rho(o, i) >= rho_lb(R, c) - e_o - rho_up(i),
// so rho_lb(R, c) >= 2 rho_up(i) + e_o proves d(i, c) >= delta_i and c cannot lower
// delta_i.  The bounds carry the rounding of every computed distance (kTriEpsC for
// the canonical fp32 order against exact arithmetic, plus the tensor-core bound for
// the root table) and are evaluated with directed rounding, so a skipped pair is
// one whose canonical fminf would have left delta_i unchanged: the selection stays
// bit-identical.  Rows outside a safe norm range (no underflow or overflow in the
// canonical dot) are never skipped.
constexpr int kMaxRoots = kRootsPerRequest;        // roots per request (workspace rows)
// Candidate list of the tensor-core variant: each CTA keeps up to kDeep of its
// highest keys w~_i delta_i (sorted) and a bound theta that every other token's key
// stays below (keys never increase).  After a round the entries still above theta
// are exactly the CTA's top keys, so the CTA re-ranks all of its tokens only when
// fewer than the published count remain.
constexpr int kDeep = 64;
static_assert(kMaxAccept == kRootTableCols, "the bound table has one column per accepted centre");
constexpr int kRootGroup = 16;                     // roots per group: the table MMA's N
// Root rows are stored in groups of 16 in the MMA's shared-memory image: K block kb
// of the group at kb * 2048, row i at i * 128, 16-byte chunk c at (c ^ (i % 8)) * 16
// (K-major, 128-byte swizzle).  One bulk copy then moves any run of K blocks.
constexpr int kRootGroupKbBytes = kRootGroup * 128;
// The root table streams through the update's ring (idle while it runs) in slots
// of one K block of 128 root rows, at most kTabSt of them, with barriers of their
// own, so that its copies are in flight while the candidate list is processed.
constexpr int kTabSt = 8;
constexpr float kTriTau = 0.5f;                    // chordal radius that makes a centre a root
// |canonical fp32 distance - exact distance| for rows of norm in [2^-50, 2^50] and
// d_v <= 2048: the dot's at most 64 fmas per lane and 5 butterfly additions give
// 69 u relative to |x_i||x_j|, each reciprocal norm 36.5 u, the two scalings and the
// subtraction 3 u more: 8.9e-6 in all (u = 2^-24); taken with a 3x margin.
constexpr float kTriEpsC = 3e-5f;

struct SelectArgs {
  CUtensorMap tmap;      // X as [total_vis][dv] bf16, box 64 x 128, 128-byte swizzle (tc only)
  const void *x;
  const float *w;
  int32_t *idx_out;
  void *x_out;           // nullable
  const int32_t *meta;
  const int32_t *order;  // cluster -> request (most work first)
  int dv, row_bytes, tpc_max, cache_rows, csize;
  int mc;                // candidates each CTA publishes per round (< top_width)
  int max_accept;        // picks accepted per round (<= kMaxAccept; 16 on the CUDA-core update)
  int ring;              // 1: rows beyond the resident cache stream through an async-copy ring
  int lcap;              // candidate list length (16 or 32)
  unsigned *err;         // workspace error word
  uint32_t tmem_cols;    // tc: TMEM columns allocated (power of two >= 32)
  int tc_stages;         // tc: TMA ring depth (2..kTcMaxStages)
  int tc_kps;            // tc: K blocks (boxes) per ring stage
  float tc_eps;          // tc: bound on |tensor-core distance - canonical distance|
  // triangle-inequality skipping (tc only)
  char *roots;           // root row groups: request b's from row meta kRootOff (a multiple of 16)
  float *rtab;           // per round: rho lower bounds [root row][kMaxAccept]
  int tri;               // 1: skip rows by the triangle inequality
  int gram;              // tc: 1 when the list's Gram may be taken (its buffers exist)
  int root_cap;          // roots per request (<= kMaxRoots, <= s_cap * csize)
  float tri_eps_x;       // bound on |root-table distance - exact distance| (tc_eps + kTriEpsC)
};

// Shared-memory carve-up, identical on host (sizing) and device.
struct SelectSmem {
  size_t aring, xcache, cbuf, ring, blk, w, r, dl, list, sel, wtop, pub_key, pub_f, lp_key,
      lp_f, lp_idx, lp_row, pair, acc, misc, bar, cnt, tbar, tslot, fidx, fmask, fcnt, gram, plist,
      oroot, oe, mr, rootr, part, croot, ce, rowj, nrl, hard, deep, total;
};
// K blocks of kTcBK elements covering a feature row.
__host__ __device__ inline int tc_kblocks(int dv) { return (dv + kTcBK - 1) / kTcBK; }
__host__ __device__ inline size_t align16(size_t v) { return (v + 15) & ~size_t(15); }
// Bytes of the per-warp async-copy rings: kRing groups x tb rows x (8 coordinates x
// elem bytes) per lane.
__host__ __device__ inline size_t ring_bytes(int ring, int tb, int elem) {
  return ring ? (size_t)kSelectWarps * kRing * tb * 8 * elem * 32 : 0;
}
__host__ __device__ inline int blocks_per_warp(int tpc_max, int tb) {
  return (tpc_max + kSelectWarps * tb - 1) / (kSelectWarps * tb);
}
__host__ __device__ inline SelectSmem select_smem(int cache_rows, int row_bytes, int tpc_max,
                                                  int ring, int tb, int elem, int lcap,
                                                  int tc = 0, int stages = 0, int kps = 1,
                                                  int roots = 0, int csize = kMaxCluster,
                                                  int gram = 1) {
  SelectSmem s;
  size_t o = 0;
  if (tc) {
    // the candidate rows double as the MMA's B operand (K-major, 128-byte swizzle):
    // K block kb of list row j at kb * lcap * 128 + j * 128; both regions are
    // multiples of 1024 bytes from a 1024-aligned base
    s.cbuf = o; o += (size_t)tc_kblocks(row_bytes / elem) * lcap * 128;
    s.aring = o; o += (size_t)stages * kps * kTcBoxBytes;
    s.xcache = o;
    s.ring = o;
    s.blk = o;
  } else {
    s.aring = o;
    s.xcache = o; o += (size_t)cache_rows * row_bytes;
    s.cbuf = o; o += (size_t)lcap * row_bytes;
    s.ring = o; o += ring_bytes(ring, tb, elem);
    s.blk = o; o += align16(sizeof(int) * kSelectWarps * blocks_per_warp(tpc_max, tb));
  }
  s.w = o; o += align16(sizeof(float) * tpc_max);
  s.r = o; o += align16(sizeof(float) * tpc_max);
  s.dl = o; o += align16(sizeof(float) * tpc_max);
  s.list = o; o += tc ? 0 : align16(sizeof(int) * tpc_max);   // tensor-core variant: aliases fidx
  s.sel = o; o += align16(tpc_max);
  s.wtop = o; o += sizeof(unsigned long long) * kSelectWarps * kTopMax;
  s.pub_key = o; o += sizeof(unsigned long long) * 2 * csize * kTopMax;   // [parity][CTA][entry]
  s.pub_f = o; o += sizeof(float4) * 2 * csize * kTopMax;
  s.lp_key = o; o += sizeof(unsigned long long) * kLcap;
  s.lp_f = o; o += sizeof(float) * kLcap * 3;
  s.lp_idx = o; o += sizeof(int) * kLcap;
  s.lp_row = o; o += sizeof(int) * kLcap;
  s.pair = o; o += sizeof(float) * 2 * kMaxPairs;
  s.acc = o; o += sizeof(int) * kMaxAccept;
  s.misc = o; o += sizeof(unsigned long long) * (4 + kTopMax);
  s.bar = o; o += sizeof(unsigned long long);
  s.cnt = o; o += sizeof(int) * kMaxCluster;
  o = align16(o);
  s.tbar = o; o += tc ? sizeof(unsigned long long) * (2 * kTcMaxStages + 3 + 2 * kTabSt) : 0;
  o = align16(o);   // later regions take 16-byte vector accesses (mr: v4 loads and cluster stores)
  s.tslot = o; o += tc ? 16 : 0;
  s.fidx = o; o += tc ? align16(sizeof(int) * tpc_max) : 0;
  if (tc) s.list = s.fidx;   // the epilogue's list of kept tokens, after the last update
  s.fmask = o; o += tc ? align16(sizeof(uint32_t) * tpc_max) : 0;
  s.fcnt = o; o += tc ? 16 : 0;
  // list Gram (tensor cores) and the pairs it leaves, when the launch may take it
  s.gram = o; o += tc && gram ? sizeof(float) * kLcap * kLcap : 0;
  s.plist = o; o += tc && gram ? align16(sizeof(int) * (kMaxPairs + 1)) : 0;
  // triangle-inequality state: per token the root of its nearest centre and the bound
  // e of that centre; per root the round's smallest rho lower bound and its 1/|x|;
  // per accepted centre its root and e; the cluster's partial nearest-root searches
  // (sized 0 when the launch does not skip rows: roots == 0)
  const bool tri = tc && roots > 0;
  s.oroot = o; o += tri ? align16(sizeof(int16_t) * tpc_max) : 0;   // roots < 2^15
  s.oe = o; o += tri ? align16(sizeof(float) * tpc_max) : 0;
  s.mr = o; o += tri ? align16(sizeof(float) * roots) : 0;
  s.rootr = o; o += tri ? align16(sizeof(float) * roots) : 0;
  s.part = o; o += tri ? sizeof(float2) * kMaxCluster * kMaxAccept : 0;
  s.croot = o; o += tri ? sizeof(int) * kMaxAccept : 0;
  s.ce = o; o += tri ? sizeof(float) * kMaxAccept : 0;
  s.rowj = o; o += tri ? sizeof(int) * kLcap : 0;
  s.nrl = o; o += tri ? sizeof(int2) * (kMaxAccept + 1) : 0;
  s.hard = o; o += tri ? sizeof(int2) * kMaxCluster : 0;   // every CTA's (hard, live) counts
  s.deep = o; o += tc ? sizeof(unsigned long long) * kDeep + 16 : 0;   // candidate list + flag
  s.total = align16(o) + 1024;   // slack for aligning the base to 1024 bytes
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
template <typename T>
__device__ __forceinline__ void load8_any(const char *row, bool sh, int col, float *e) {
  if (sh) load8<T, true>(row, col, e);
  else load8<T, false>(row, col, e);
}

__device__ __forceinline__ float butterfly_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// canonical dot of two rows (warp-cooperative; every lane returns the result)
template <typename T, int NCH>
__device__ __forceinline__ float dot_rows(const char *ra, bool sha, const char *rb, bool shb,
                                          int dv, int lane) {
  float acc = 0.f;
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int col = 256 * c + 8 * lane;
    if (col < dv) {
      float ea[8], eb[8];
      load8_any<T>(ra, sha, col, ea);
      load8_any<T>(rb, shb, col, eb);
#pragma unroll
      for (int q = 0; q < 8; ++q) acc = __fmaf_rn(ea[q], eb[q], acc);
    }
  }
  return butterfly_sum(acc);
}

// max over the warp of (key, payload); every lane ends with the winner
__device__ __forceinline__ void warp_argmax(unsigned long long &key, int &payload) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long ok = shfl_xor_u64(key, o);
    const int op = __shfl_xor_sync(0xffffffffu, payload, o);
    if (ok > key) { key = ok; payload = op; }
  }
}

// maximum over the warp of a 64-bit key (every lane returns it)
__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
  const uint32_t hi = __reduce_max_sync(0xffffffffu, (uint32_t)(v >> 32));
  const uint32_t lo = __reduce_max_sync(0xffffffffu, (uint32_t)(v >> 32) == hi ? (uint32_t)v : 0u);
  return ((unsigned long long)hi << 32) | lo;
}

// descending top-W list held in (warp-uniform) registers
template <int W>
struct TopList {
  unsigned long long k[W];
  __device__ __forceinline__ void clear() {
#pragma unroll
    for (int i = 0; i < W; ++i) k[i] = 0ull;
  }
  __device__ __forceinline__ void insert(unsigned long long v) {
    if (v <= k[W - 1]) return;
#pragma unroll
    for (int i = W - 1; i > 0; --i) {
      if (v > k[i - 1]) k[i] = k[i - 1];
      else if (v > k[i]) { k[i] = v; v = 0ull; }
    }
    if (v > k[0]) k[0] = v;
  }
};

// ---- triangle-inequality bounds (directed rounding: each is a true bound) ----
// 1/|x| of a row whose canonical dot products obey the kTriEpsC bound
__device__ __forceinline__ bool tri_in_range(float r) { return r >= 0x1p-50f && r <= 0x1p50f; }
// upper bound on rho(i, o) from delta_i = d(i, o) (canonical), +inf when unbounded
__device__ __forceinline__ float tri_rho_up(float delta) {
  if (!(delta <= 4.0f)) return INFINITY;
  return __fsqrt_ru(__fmul_ru(2.0f, fmaxf(__fadd_ru(delta, kTriEpsC), 0.0f)));
}
// lower bound on rho(a, b) from a computed distance d with |d - exact| <= eps
__device__ __forceinline__ float tri_rho_lb(float d, float eps) {
  const float v = __fsub_rd(d, eps);
  return v > 0.0f ? __fsqrt_rd(__fmul_rd(2.0f, v)) : 0.0f;   // NaN -> 0 (never skips)
}
// upper bound on rho(a, b) from a computed distance d with |d - exact| <= eps
__device__ __forceinline__ float tri_rho_ub(float d, float eps) {
  const float v = __fadd_ru(d, eps);
  if (!(v <= 4.0f)) return INFINITY;
  return __fsqrt_ru(__fmul_ru(2.0f, fmaxf(v, 0.0f)));
}
// rho_lb(R, c) >= 2 rho_up(i) + e_o: c cannot lower delta_i
__device__ __forceinline__ float tri_need(float delta, float e) {
  return __fadd_ru(__fmul_ru(2.0f, tri_rho_up(delta)), e);
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

template <typename T, int NCH, int TB, bool TC>
__global__ void __launch_bounds__(kSelThreads, 1)
select_kernel(const __grid_constant__ SelectArgs a) {
  constexpr int kTop = top_width<TC>();
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int C = a.csize;
  const uint32_t rank = cluster_ctarank();
  const int b = a.order[cluster_id_x()];
  const int32_t *m = a.meta + b * kMetaFields;
  const int voff = m[kVisOff], N = m[kNumVis], koff = m[kKeepOff], K = m[kNumKeep];
  if (K == 0) return;  // the whole cluster leaves together; no DSMEM traffic yet
  const int rootoff = m[kRootOff];

  const SelectSmem S = select_smem(a.cache_rows, a.row_bytes, a.tpc_max, a.ring, TB, (int)sizeof(T),
                                   a.lcap, TC ? 1 : 0, TC ? a.tc_stages : 0, TC ? a.tc_kps : 1,
                                   TC && a.tri ? a.root_cap : 0, a.csize, TC ? a.gram : 1);
  {
    // The host sizes the launch with the same plan; should they ever disagree, every
    // CTA of every cluster leaves here together (before any cluster barrier)
    // instead of touching shared memory past the allocation.
    uint32_t dyn;
    asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn));
    if (S.total > dyn) {
      if (threadIdx.x == 0) atomicOr(a.err, kErrConfig);
      return;
    }
  }
  const int lcap = a.lcap;
  char *xcache = reinterpret_cast<char *>(smem + S.xcache);
  char *cbuf = reinterpret_cast<char *>(smem + S.cbuf);
  const uint32_t ring_base = smem_addr(smem + S.ring);
  int *blk_s = reinterpret_cast<int *>(smem + S.blk);
  float *w_s = reinterpret_cast<float *>(smem + S.w);
  float *r_s = reinterpret_cast<float *>(smem + S.r);
  float *dl_s = reinterpret_cast<float *>(smem + S.dl);
  int *list_s = reinterpret_cast<int *>(smem + S.list);
  unsigned char *sel_s = smem + S.sel;
  unsigned long long *wtop = reinterpret_cast<unsigned long long *>(smem + S.wtop);
  unsigned long long *pub_key = reinterpret_cast<unsigned long long *>(smem + S.pub_key);
  float4 *pub_f = reinterpret_cast<float4 *>(smem + S.pub_f);
  unsigned long long *lp_key = reinterpret_cast<unsigned long long *>(smem + S.lp_key);
  float *lp_f = reinterpret_cast<float *>(smem + S.lp_f);       // [kLcap][3]: delta, w, r
  int *lp_idx = reinterpret_cast<int *>(smem + S.lp_idx);
  int *lp_row = reinterpret_cast<int *>(smem + S.lp_row);   // cbuf row of each member
  unsigned long long *bar = reinterpret_cast<unsigned long long *>(smem + S.bar);
  float *pairbuf = reinterpret_cast<float *>(smem + S.pair);
  int *acc_s = reinterpret_cast<int *>(smem + S.acc);
  unsigned long long *misc = reinterpret_cast<unsigned long long *>(smem + S.misc);
  int *cnt_s = reinterpret_cast<int *>(smem + S.cnt);
  // triangle-inequality state (tensor-core variant)
  const bool tri = TC && a.tri != 0;
  int16_t *oroot_s = reinterpret_cast<int16_t *>(smem + S.oroot);
  float *oe_s = reinterpret_cast<float *>(smem + S.oe);
  float *mr_s = reinterpret_cast<float *>(smem + S.mr);
  float *rootr_s = reinterpret_cast<float *>(smem + S.rootr);
  float2 *part_s = reinterpret_cast<float2 *>(smem + S.part);   // [kMaxCluster][kMaxAccept]
  int *croot_s = reinterpret_cast<int *>(smem + S.croot);
  float *ce_s = reinterpret_cast<float *>(smem + S.ce);
  int *rowj_s = reinterpret_cast<int *>(smem + S.rowj);
  int2 *nrl_s = reinterpret_cast<int2 *>(smem + S.nrl);         // new roots: (root id, token)
  const int rcap = tri ? min(a.root_cap, K) : 0;
  int nroot = 0;   // roots of this request (the same in every CTA of the cluster)

  const int tpr = (N + C - 1) / C;  // tokens per CTA for this request
  const int lo = min(N, (int)rank * tpr), hi = min(N, lo + tpr);
  const int nloc = hi - lo;
  const int ncache = min(nloc, a.cache_rows);
  const int rb = a.row_bytes;
  const int dv = a.dv;
  const char *xreq = static_cast<const char *>(a.x) + (long long)voff * rb;
  const char *xg = xreq + (long long)lo * rb;

  // ---- prologue: resident rows (one bulk copy), weights, delta = +inf ----
  // `bar` tracks the bulk copies into this CTA's shared memory; `phase` is the
  // parity of the next phase to wait for.
  uint32_t phase = 0;
  unsigned long long *tfull = reinterpret_cast<unsigned long long *>(smem + S.tbar);
  const int nstage = TC ? a.tc_stages : 1;
  unsigned long long *tempty = tfull + kTcMaxStages;
  unsigned long long *tdone = tempty + kTcMaxStages;
  unsigned long long *tpair = tdone + 1;
  unsigned long long *ttab = tpair + 1;   // the round's root table is in TMEM
  unsigned long long *tbf = ttab + 1;     // root-table stages: landed
  unsigned long long *tbe = tbf + kTabSt; // root-table stages: consumed by the MMAs
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    if constexpr (TC) {
      for (int i = 0; i < nstage; ++i) {
        mbar_init(&tfull[i], 1);
        mbar_init(&tempty[i], 1);
      }
      mbar_init(tdone, 1);
      mbar_init(tpair, 1);
      mbar_init(ttab, 1);
      for (int i = 0; i < kTabSt; ++i) {
        mbar_init(&tbf[i], 1);
        mbar_init(&tbe[i], 1);
      }
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && ncache > 0) {
    mbar_expect_tx(bar, (uint32_t)(ncache * rb));
    bulk_g2s(xcache, xg, (uint32_t)(ncache * rb), bar);
  }
  for (int t = threadIdx.x; t < nloc; t += kSelThreads) {
    w_s[t] = a.w[voff + lo + t];
    dl_s[t] = INFINITY;
    sel_s[t] = (K == N) ? 1 : 0;
    if (tri) {
      oroot_s[t] = -1;      // no nearest centre yet: never skipped
      oe_s[t] = INFINITY;
    }
  }
  if (ncache > 0) {
    mbar_wait_bounded(bar, phase, a.err, kErrTimeout);
    phase ^= 1u;
  }
  __syncthreads();

  if (K < N) {
    // tensor-core accumulators: lcap fp32 columns per 128-row tile of this CTA's tokens
    uint32_t tmem = 0;
    if constexpr (TC) {
      uint32_t *tslot = reinterpret_cast<uint32_t *>(smem + S.tslot);
      if (threadIdx.x == 0) tslot[1] = 0;   // abort word: a tensor-core wait expired
      if (warp == 0) tmem_alloc(tslot, a.tmem_cols);
      // the candidate rows start at zero: K chunks past d_v stay zero for the MMA and
      // rows never staged hold finite values
      for (size_t v = threadIdx.x; v < (S.aring - S.cbuf) / 16; v += kSelThreads)
        reinterpret_cast<U4 *>(smem + S.cbuf)[v] = U4{0, 0, 0, 0};
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      tmem = *tslot;
    }
    // r_i = 1/sqrt(dot(x_i, x_i)); each warp also ranks its tokens by w~ for the seed
    TopList<kTop> top;
    top.clear();
    for (int t = warp; t < nloc; t += kSelectWarps) {
      const bool sh = t < ncache;
      const char *row = sh ? xcache + (long long)t * rb : xg + (long long)t * rb;
      const float ss = dot_rows<T, NCH>(row, sh, row, sh, dv, lane);
      if (lane == 0) r_s[t] = ss > 0.f ? __fdiv_rn(1.0f, __fsqrt_rn(ss)) : 0.f;
      top.insert(argmax_key(w_s[t], lo + t));
    }
    if (lane == 0) {
#pragma unroll
      for (int i = 0; i < kTop; ++i) wtop[warp * kTop + i] = top.k[i];
    }
    __syncthreads();

    // Merge the warps' lists into the CTA's kTop best and publish them (key and
    // {delta, w, r}) to every CTA of the cluster, into buffer `par`.
    unsigned long long *top5 = misc + 4;  // misc[4..4+kTop)
    unsigned long long *dkey = reinterpret_cast<unsigned long long *>(smem + S.deep);
    int *drescan = reinterpret_cast<int *>(smem + S.deep + sizeof(unsigned long long) * kDeep);
    unsigned long long d_theta = 0ull;   // warp 0: bound on every key outside dkey
    int d_n = 0;                         // warp 0: entries of dkey
    // warp 0: the list holds keys w~ delta (not the seed round's w~ alone: a key w~
    // delta can exceed w~ when delta > 1, so that first list bounds nothing later)
    bool d_bounds = false;
    // warp 0: the union of the warps' ranked lists -> the candidate list.  Every
    // token a warp left out has a key below that warp's last entry, so the union's
    // entries above the largest such entry are the CTA's top keys, in order.
    auto deep_rebuild = [&](bool bounds) {
      if (warp != 0) return;
      d_bounds = bounds;
      constexpr int nk = kSelectWarps * kTop;
      constexpr int kPerLane = (nk + 31) / 32;
      unsigned long long kl[kPerLane];
      int rl[kPerLane];
#pragma unroll
      for (int j = 0; j < kPerLane; ++j) {
        kl[j] = lane + 32 * j < nk ? wtop[lane + 32 * j] : 0ull;
        rl[j] = 0;
      }
      unsigned long long th = lane < kSelectWarps ? wtop[lane * kTop + kTop - 1] : 0ull;
      {
        const uint32_t hi = __reduce_max_sync(0xffffffffu, (uint32_t)(th >> 32));
        const uint32_t lo_ = __reduce_max_sync(0xffffffffu, (uint32_t)(th >> 32) == hi ? (uint32_t)th : 0u);
        th = ((unsigned long long)hi << 32) | lo_;
      }
#pragma unroll
      for (int f = 0; f < nk; ++f) {
        const unsigned long long kf = wtop[f];
#pragma unroll
        for (int j = 0; j < kPerLane; ++j) rl[j] += kf > kl[j] ? 1 : 0;
      }
      int above = 0;
      unsigned long long cut = 0ull;
#pragma unroll
      for (int j = 0; j < kPerLane; ++j) {
        const bool up = kl[j] > th;
        above += __popc(__ballot_sync(0xffffffffu, up));
        if (up && rl[j] < kDeep) dkey[rl[j]] = kl[j];
        if (up && rl[j] == kDeep) cut = kl[j];
      }
      {
        const uint32_t hi = __reduce_max_sync(0xffffffffu, (uint32_t)(cut >> 32));
        const uint32_t lo_ = __reduce_max_sync(0xffffffffu, (uint32_t)(cut >> 32) == hi ? (uint32_t)cut : 0u);
        cut = ((unsigned long long)hi << 32) | lo_;
      }
      d_n = min(above, kDeep);
      d_theta = above > kDeep ? cut : th;
      __syncwarp();
    };
    // warp 0, after an update: the list's keys from the new deltas; entries that fell
    // to theta or below (or were selected) leave it.  Sets *drescan when fewer than
    // the published count remain while other tokens exist.
    auto deep_refresh = [&]() {
      if (warp != 0) return;
      if (!d_bounds) {
        if (lane == 0) *drescan = 1;
        __syncwarp();
        return;
      }
      unsigned long long k[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int e = lane + 32 * h;
        k[h] = 0ull;
        if (e < d_n) {
          const int gi = key_index(dkey[e]);
          const int t = gi - lo;
          const unsigned long long nk = sel_s[t] ? 0ull : argmax_key(__fmul_rn(w_s[t], dl_s[t]), gi);
          k[h] = nk > d_theta ? nk : 0ull;
        }
      }
      int r0 = 0, r1 = 0;
#pragma unroll 8
      for (int src = 0; src < 32; ++src) {
        const unsigned long long a0 = shfl_u64(k[0], src), a1 = shfl_u64(k[1], src);
        r0 += (a0 > k[0] ? 1 : 0) + (a1 > k[0] ? 1 : 0);
        r1 += (a0 > k[1] ? 1 : 0) + (a1 > k[1] ? 1 : 0);
      }
      const int kept = __popc(__ballot_sync(0xffffffffu, k[0] != 0ull)) +
                       __popc(__ballot_sync(0xffffffffu, k[1] != 0ull));
      __syncwarp();
      if (k[0] != 0ull) dkey[r0] = k[0];
      if (k[1] != 0ull) dkey[r1] = k[1];
      d_n = kept;
      if (lane == 0) *drescan = (d_n >= a.mc + 1 || d_theta == 0ull) ? 0 : 1;
      __syncwarp();
    };
    auto publish = [&](int par) {
      if (warp == 0) {
        if constexpr (TC) {
          // the candidate list holds the CTA's top keys, and every live token outside
          // it has a key at or below theta.  A rebuild can leave only mc of them (when
          // one warp owns the CTA's best mc + 1 keys, its last one is theta itself), so
          // the bound slot mc takes theta whenever the list is that short.
          if (lane < kTop) top5[lane] = lane < d_n ? dkey[lane] : (lane == a.mc ? d_theta : 0ull);
        } else {
        constexpr int nk = kSelectWarps * kTop;   // the warps' ranked keys
        constexpr int kPerLane = (nk + 31) / 32;
        static_assert(kPerLane <= 5, "publish ranks at most 160 keys");
        unsigned long long kl[kPerLane];
        int rl[kPerLane];
#pragma unroll
        for (int j = 0; j < kPerLane; ++j) {
          kl[j] = lane + 32 * j < nk ? wtop[lane + 32 * j] : 0ull;
          rl[j] = 0;
        }
        if (lane < kTop) top5[lane] = 0ull;
#pragma unroll
        for (int f = 0; f < nk; ++f) {
          const unsigned long long kf = wtop[f];
#pragma unroll
          for (int j = 0; j < kPerLane; ++j) rl[j] += kf > kl[j] ? 1 : 0;
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < kPerLane; ++j)
          if (kl[j] != 0ull && rl[j] < kTop) top5[rl[j]] = kl[j];
        }
        __syncwarp();
        if (lane < C) {
          for (int i = 0; i <= a.mc; ++i) {
            const unsigned long long key = top5[i];
            const int slot = (par * C + (int)rank) * kTopMax + i;
            float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
            if (key != 0ull) {
              const int lt = key_index(key) - lo;
              f = make_float4(dl_s[lt], w_s[lt], r_s[lt], 0.f);
            }
            st_cluster_u64(map_shared(&pub_key[slot], lane), key);
            st_cluster_v4f(map_shared(&pub_f[slot], lane), f);
          }
        }
      }
    };

    // Shared address of the 8 elements at column `col` (a multiple of 8) of cbuf row
    // j: plain rows, or for the tensor-core update the K-major 128-byte swizzled
    // layout (K block col / 64, 16-byte chunk (col / 8) % 8 stored at chunk ^ (j % 8)).
    const uint32_t cbuf_sa = smem_addr(cbuf);
    auto cb_chunk = [&](int j, int col) -> uint32_t {
      if constexpr (TC) {
        const int kb = col >> 6, c = (col >> 3) & 7;
        return cbuf_sa + (uint32_t)(kb * lcap * 128 + j * 128 + ((c ^ (j & 7)) << 4));
      } else {
        return cbuf_sa + (uint32_t)(j * rb + col * (int)sizeof(T));
      }
    };
    // Row `gi` of the request into cbuf row j, 16 bytes per copy, by the threads
    // [t0, t0 + nt) (tensor-core layout; completion with cp.async wait).
    auto copy_row_tc = [&](int j, int gi, int t0, int nt) {
      const char *src = xreq + (long long)gi * rb;
      for (int cc = (int)threadIdx.x - t0; cc < dv / 8; cc += nt)
        cp_async16(cb_chunk(j, cc * 8), src + cc * 16);
    };
    // Copy the rows of list members 0..nL-1 into cbuf rows 0..nL-1: one bulk copy
    // per row (completion on `bar`), or, for the tensor-core layout, 16-byte async
    // copies by every thread.  Every thread then waits for them (wait_rows).
    auto stage_list = [&](int nL) {
      if constexpr (TC) {
        for (int u = 0; u < nL; ++u) copy_row_tc(u, lp_idx[u], 0, kSelThreads);
        cp_async_commit();
        if (threadIdx.x < nL) lp_row[threadIdx.x] = threadIdx.x;
      } else if (threadIdx.x == 0) {
        mbar_expect_tx(bar, (uint32_t)(nL * rb));
        for (int u = 0; u < nL; ++u) {
          lp_row[u] = u;
          bulk_g2s(cbuf + (long long)u * rb, xreq + (long long)lp_idx[u] * rb, (uint32_t)rb, bar);
        }
      }
    };
    auto wait_rows = [&]() {
      if constexpr (TC) {
        cp_async_wait<0>();
      } else {
        mbar_wait_bounded(bar, phase, a.err, kErrTimeout);
        phase ^= 1u;
      }
    };
    // With few CTAs every published candidate fits in cbuf: copy them all right after
    // the exchange (published entry e of CTA q -> cbuf row q * mc + e), overlapping the
    // copies with the list construction.
    const bool early = C * a.mc <= lcap;

    // delta_i <- min(delta_i, 1 - (dot(x_i, x_c) r_i) r_c) over the nA accepted
    // centres (cbuf rows acc_s[0..nA)), for every unselected local token; then the
    // warps' best keys for the next round.  A warp takes TB tokens at a time and all
    // centres at once; accumulators pair two tokens per __ffma2_rn (two independent
    // correctly rounded fp32 fmas, so the canonical order is unchanged).  The body is
    // compiled for NB = 4, 8, 12, 16 centres without branches (slots past nA repeat
    // centre 0 and are ignored) so that the independent chains interleave.
    auto update_nb = [&](auto nb_tag, int nA) {
      constexpr int NB = decltype(nb_tag)::value;
      constexpr int NP = NB / 2;   // centre pairs: one __ffma2_rn serves two centres (fp32)
      (void)NP;
      constexpr int V = Elem<T>::kPerVec;
      constexpr int VPG = 8 / V;   // 16-byte vectors per 8-coordinate group
      int coff[NB];
#pragma unroll
      for (int c = 0; c < NB; ++c) coff[c] = lp_row[acc_s[c < nA ? c : 0]] * rb;
      // this warp's token blocks that still hold an unselected token
      int *blist = blk_s + warp * blocks_per_warp(a.tpc_max, TB);
      int nact = 0;
      for (int k0 = 0; (warp + k0 * kSelectWarps) * TB < nloc; k0 += 32) {
        const int t0 = (warp + (k0 + lane) * kSelectWarps) * TB;
        bool act = false;
        if (t0 < nloc) {
#pragma unroll
          for (int q = 0; q < TB; ++q) act |= t0 + q < nloc && !sel_s[t0 + q];
        }
        const unsigned m = __ballot_sync(0xffffffffu, act);
        if (act) blist[nact + __popc(m & ((1u << lane) - 1u))] = t0;
        nact += __popc(m);
      }
      __syncwarp();
      // Items (block j, group g) flow through a per-lane ring: each lane copies its own
      // 16-byte pieces of the streamed rows kRing-1 items ahead and reads back only what
      // it copied, so the ring needs no cross-lane synchronisation.  Fully resident
      // blocks issue nothing.
      const uint32_t wring = ring_base + (uint32_t)(warp * kRing * TB * VPG * 512) + lane * 16;
      const uint32_t xc_base = smem_addr(xcache) + lane * 8 * (int)sizeof(T);
      const uint32_t cb_base = smem_addr(cbuf) + lane * (int)sizeof(T) * 8;
      const bool streams = a.ring && ncache < nloc;
      int ij = 0, ig = 0;       // issue cursor: block, group
      uint32_t islot = 0;       // ring slot of the next issue
      auto issue = [&]() {
        if (streams && ij < nact) {
          const int t0 = blist[ij];
          const int col = 256 * ig + 8 * lane;
          if (col < dv) {
            const char *src = xg + (long long)t0 * rb + col * (int)sizeof(T);
#pragma unroll
            for (int q = 0; q < TB; ++q)
              if (t0 + q < nloc && t0 + q >= ncache)
#pragma unroll
                for (int h = 0; h < VPG; ++h)
                  cp_async16(wring + (islot * TB * VPG + q * VPG + h) * 512, src + (long long)q * rb + 16 * h);
          }
          if (++ig == NCH) { ig = 0; ++ij; }
        }
        islot = (islot + 1) & (kRing - 1);
        cp_async_commit();
      };
      if (streams)
        for (int i = 0; i < kRing - 1; ++i) issue();
      TopList<kTop> tl;
      tl.clear();
      uint32_t cslot = 0;       // ring slot of the item being computed
      for (int j = 0; j < nact; ++j) {
        const int t0 = blist[j];
        uint32_t tok[TB];       // per-token shared address of group 0 (resident) or ring base
        bool res[TB];
#pragma unroll
        for (int q = 0; q < TB; ++q) {
          const int tq = t0 + q < nloc ? t0 + q : t0;   // padding slots reuse a real row
          res[q] = tq < ncache;
          tok[q] = res[q] ? xc_base + (uint32_t)(tq * rb) : wring + (uint32_t)((tq - t0) * VPG * 512);
        }
        float acc[TB][NB];
#pragma unroll
        for (int q = 0; q < TB; ++q)
#pragma unroll
          for (int c = 0; c < NB; ++c) acc[q][c] = 0.f;
#pragma unroll 1
        for (int g = 0; g < NCH; ++g) {
          if (streams) {
            issue();
            cp_async_wait<kRing - 1>();
          }
          if (256 * g + 8 * lane < dv) {
            U4 cur[TB][VPG];
#pragma unroll
            for (int q = 0; q < TB; ++q)
#pragma unroll
              for (int h = 0; h < VPG; ++h)
                cur[q][h] = lds32(res[q] ? tok[q] + (uint32_t)(g * 8 * sizeof(T) * 32 + 16 * h)
                                         : tok[q] + (uint32_t)((cslot * TB * VPG + h) * 512));
            const uint32_t cg = cb_base + (uint32_t)(g * 8 * sizeof(T) * 32);
            // bf16: one mixed-precision fma per coordinate straight from the packed words;
            // fp32: paired fmas over two centres.  Both follow the canonical order.
            if constexpr (sizeof(T) == 2) {
#pragma unroll
              for (int c = 0; c < NB; ++c) {
                const U4 cv = lds32(cg + (uint32_t)coff[c]);
                const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
                for (int hw = 0; hw < 4; ++hw) {
#pragma unroll
                  for (int q = 0; q < TB; ++q) {
                    const uint32_t tw = hw == 0 ? cur[q][0].x : hw == 1 ? cur[q][0].y
                                      : hw == 2 ? cur[q][0].z : cur[q][0].w;
                    acc[q][c] = fma_bf16_lo(tw, cw[hw], acc[q][c]);
                    acc[q][c] = fma_bf16_hi(tw, cw[hw], acc[q][c]);
                  }
                }
              }
            } else {
              float tk[TB][8];
#pragma unroll
              for (int q = 0; q < TB; ++q)
#pragma unroll
                for (int h = 0; h < VPG; ++h) Elem<T>::widen(cur[q][h], tk[q] + h * V);
#pragma unroll
              for (int p = 0; p < NP; ++p) {
                float c0[8], c1[8];
                Elem<T>::widen(lds32(cg + (uint32_t)coff[2 * p]), c0);
                Elem<T>::widen(lds32(cg + (uint32_t)coff[2 * p] + 16), c0 + 4);
                Elem<T>::widen(lds32(cg + (uint32_t)coff[2 * p + 1]), c1);
                Elem<T>::widen(lds32(cg + (uint32_t)coff[2 * p + 1] + 16), c1 + 4);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                  const float2 cc = make_float2(c0[e], c1[e]);
#pragma unroll
                  for (int q = 0; q < TB; ++q) {
                    const float2 r2 = __ffma2_rn(make_float2(tk[q][e], tk[q][e]), cc,
                                                 make_float2(acc[q][2 * p], acc[q][2 * p + 1]));
                    acc[q][2 * p] = r2.x;
                    acc[q][2 * p + 1] = r2.y;
                  }
                }
              }
            }
          }
          cslot = (cslot + 1) & (kRing - 1);
        }
#pragma unroll
        for (int q = 0; q < TB; ++q) {
          const bool valid = t0 + q < nloc && !sel_s[t0 + q];
          float dl = valid ? dl_s[t0 + q] : 0.f;
          const float ri = valid ? r_s[t0 + q] : 0.f;
#pragma unroll
          for (int c = 0; c < NB; ++c) {
            if (c < nA) {
              const float dot = butterfly_sum(acc[q][c]);
              const float rc = lp_f[acc_s[c] * 3 + 2];
              dl = fminf(dl, __fsub_rn(1.0f, __fmul_rn(__fmul_rn(dot, ri), rc)));
            }
          }
          if (valid) {
            const int tq = t0 + q;
            if (lane == 0) dl_s[tq] = dl;
            tl.insert(argmax_key(__fmul_rn(w_s[tq], dl), lo + tq));
          }
        }
      }
      cp_async_wait<0>();
      if (lane == 0) {
#pragma unroll
        for (int i = 0; i < kTop; ++i) wtop[warp * kTop + i] = tl.k[i];
      }
    };
    // Tensor-core form of the same update (bf16).  X's rows of this CTA stream
    // through TMA in 128 x 64 boxes; one thread issues tcgen05.mma against every
    // list row (cbuf, K-major with the 128-byte swizzle) into one TMEM accumulator
    // of lcap columns per 128-row tile; the accepted centres are the columns
    // lp_row[acc_s[j]].  Each token's tensor-core
    // distances d~ are within tc_eps of the canonical ones, so a centre with
    // d~ - tc_eps >= delta_i cannot lower delta_i; every other (token, centre)
    // pair is recomputed in the canonical order.  delta thus stays bit-identical
    // to the CUDA-core update.
    uint32_t tc_pit = 0, tc_mit = 0, tc_dph = 0;   // producer / MMA / done phase counters
    uint32_t tc_pph = 0;                            // list-Gram phase
    // After one expired wait every later tensor-core wait returns at once, so a
    // broken call ends quickly (reporting LAST_ERR_TIMEOUT) instead of waiting out
    // each limit in turn.
    auto twait = [&](unsigned long long *b, uint32_t par) -> bool {
      volatile uint32_t *abort_w = reinterpret_cast<volatile uint32_t *>(smem + S.tslot) + 1;
      if (*abort_w) return false;
      if (mbar_wait_bounded(b, par, a.err, kErrTimeout)) return true;
      *abort_w = 1u;
      return false;
    };
    auto update_tc = [&](int nA, bool tri_round) {
      const int nkb = tc_kblocks(dv);
      char *aring = reinterpret_cast<char *>(smem + S.aring);
      int *fidx = reinterpret_cast<int *>(smem + S.fidx);
      uint32_t *fmask = reinterpret_cast<uint32_t *>(smem + S.fmask);
      int *fcnt = reinterpret_cast<int *>(smem + S.fcnt);
      // 1. the B operand is cbuf as staged (every list row; the accepted centres are
      //    the accumulator columns lp_row[acc_s[j]])
      if (threadIdx.x == 0) *fcnt = 0;
      fence_proxy_async_smem();
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      // 1b. triangle test: a token survives unless the round's root table proves that
      //     no accepted centre can lower its delta.  A survivor is "hard" when no
      //     bound can exclude any centre for it (2 rho_up + e above 2, the largest
      //     chordal distance: its delta is still near 1); its pairs all need a
      //     distance.  With few survivors their pairs are evaluated exactly (step 4)
      //     without streaming X; otherwise the dense tensor-core pass decides every
      //     pair.  The choice compares the bytes the dense pass streams with the
      //     survivors' rows plus their exact pairs (about 5/16 of a row each).
      bool dense = true;
      if (tri_round) {
        if (threadIdx.x == 0) fcnt[1] = 0;
        __syncthreads();
        for (int t0 = warp * 32; t0 < nloc; t0 += kSelThreads) {
          const int t = t0 + lane;
          bool act = false, hard = false;
          if (t < nloc && !sel_s[t]) {
            act = hard = true;
            const int R = oroot_s[t];
            if (R >= 0 && tri_in_range(r_s[t])) {
              const float nd = tri_need(dl_s[t], oe_s[t]);
              act = !(mr_s[R] >= nd);
              hard = !(nd <= 2.0f);
            }
          }
          const unsigned bal = __ballot_sync(0xffffffffu, act);
          const unsigned hb = __ballot_sync(0xffffffffu, act && hard);
          int base = 0;
          if (lane == 0 && bal != 0u) {
            base = atomicAdd(fcnt, __popc(bal));
            if (hb != 0u) atomicAdd(fcnt + 1, __popc(hb));
          }
          base = __shfl_sync(0xffffffffu, base, 0);
          if (act) fidx[base + __popc(bal & ((1u << lane) - 1u))] = t;
        }
        __syncthreads();
        const int nact = fcnt[0], nhard = fcnt[1];
        const long long pair_bytes = (long long)dv * 5 / 16;
        const long long sparse_cost = (long long)nact * rb * 5 / 4 +
                                      ((long long)nhard * nA + 2LL * (nact - nhard)) * pair_bytes;
        dense = sparse_cost > (long long)nloc * rb;
        __syncthreads();   // every thread has read the counts
        if (dense) {
          if (threadIdx.x == 0) *fcnt = 0;
        } else {
          // the centres the survivor's root bound does not exclude (table rows written
          // by the slice owners before the last cluster barrier; read past L1); four
          // survivors per warp at a time keep their table loads in flight together
          for (int f0 = warp; f0 < nact; f0 += 4 * kSelectWarps) {
            float tv[4], nd[4];
            bool chk[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int f = f0 + u * kSelectWarps;
              chk[u] = false;
              tv[u] = 0.f;
              nd[u] = 0.f;
              if (f < nact && lane < nA) {
                const int t = fidx[f];
                const int R = oroot_s[t];
                if (R >= 0 && tri_in_range(r_s[t])) {
                  nd[u] = tri_need(dl_s[t], oe_s[t]);
                  if (nd[u] <= 2.0f) {
                    chk[u] = true;
                    tv[u] = __ldcg(a.rtab + (size_t)(rootoff + R) * kMaxAccept + lane);
                  }
                }
              }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int f = f0 + u * kSelectWarps;
              if (f < nact) {
                const unsigned msk = __ballot_sync(0xffffffffu, lane < nA && !(chk[u] && tv[u] >= nd[u]));
                if (lane == 0) fmask[f] = msk;
              }
            }
          }
        }
        __syncthreads();
      }
      if (dense) {
      // 2. TMA producer (thread 0) and MMA issuer (thread 32)
      const int ntile = (nloc + kTcBM - 1) / kTcBM;
      // a ring stage holds kps consecutive K blocks of one tile (one barrier, one
      // commit): the per-stage hand-off costs the same whatever the stage size
      const int kps = a.tc_kps;
      const int stage_bytes = kps * kTcBoxBytes;
      const int ngrp = (nkb + kps - 1) / kps;
      if (threadIdx.x == 0) {
        for (int tile = 0; tile < ntile; ++tile)
          for (int gq = 0; gq < ngrp; ++gq, ++tc_pit) {
            const int st = tc_pit % nstage;
            if (tc_pit >= (uint32_t)nstage && !twait(&tempty[st], ((tc_pit / nstage) - 1) & 1))
              continue;   // expired: the stage is skipped and the call reports the timeout
            const int nb = min(kps, nkb - gq * kps);
            mbar_expect_tx(&tfull[st], (uint32_t)(nb * kTcBoxBytes));
            for (int q = 0; q < nb; ++q)
              tma_load_2d(aring + st * stage_bytes + q * kTcBoxBytes, &a.tmap, (gq * kps + q) * kTcBK,
                          voff + lo + tile * kTcBM, &tfull[st]);
          }
      } else if (threadIdx.x == 32) {
        const uint32_t idesc = umma_idesc_bf16(kTcBM, lcap);
        for (int tile = 0; tile < ntile; ++tile)
          for (int gq = 0; gq < ngrp; ++gq, ++tc_mit) {
            const int st = tc_mit % nstage;
            const bool ok = twait(&tfull[st], (tc_mit / nstage) & 1);
            tc_fence_after();
            if (ok) {
              const int nb = min(kps, nkb - gq * kps);
              for (int q = 0; q < nb; ++q) {
                const int kb = gq * kps + q;
#pragma unroll
                for (int k = 0; k < kTcBK / 16; ++k)
                  umma_bf16(tmem + tile * lcap,
                            umma_desc_sw128(smem_addr(aring + st * stage_bytes + q * kTcBoxBytes) + k * 32),
                            umma_desc_sw128(cbuf_sa + kb * lcap * 128 + k * 32), idesc,
                            (kb | k) != 0 ? 1u : 0u);
              }
            }
            umma_commit(&tempty[st]);   // frees the stage once these MMAs have read it
          }
        umma_commit(tdone);
      }
      __syncwarp();
      twait(tdone, tc_dph);
      tc_dph ^= 1u;
      tc_fence_after();
      // 3. certify: flag (token, centre) pairs the tensor-core distance cannot decide
      const float eps = a.tc_eps;
      for (int tt = warp >> 2; tt < ntile; tt += 2) {
        const uint32_t tbase = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)(tt * lcap);
        const int t = tt * kTcBM + 32 * (warp & 3) + lane;
        const bool live = t < nloc && !sel_s[t];
        const float ri = live ? r_s[t] : 0.f, dl = live ? dl_s[t] : 0.f;
        uint32_t msk = 0;
        // the accepted centres 16 at a time: one TMEM column each
        for (int j0 = 0; j0 < nA; j0 += 16) {
          uint32_t dv_[16];
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (j0 + j < nA) tmem_ld1(tbase + (uint32_t)lp_row[acc_s[j0 + j]], &dv_[j]);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            if (j0 + j < nA) {
              const float rcj = lp_f[acc_s[j0 + j] * 3 + 2];
              const float d = __fsub_rn(1.0f, __fmul_rn(__fmul_rn(__uint_as_float(dv_[j]), ri), rcj));
              if (!(__fsub_rn(d, eps) >= dl)) msk |= 1u << (j0 + j);   // NaN also goes to the exact path
            }
          }
        }
        if (live && msk) {
          const int pos = atomicAdd(fcnt, 1);
          fidx[pos] = t;
          fmask[pos] = msk;
        }
      }
      tc_fence_before();
      __syncthreads();
      }   // dense
      // 4. exact canonical distances for the flagged pairs.  A warp per flagged token
      //    reads the token's row straight from global memory (the next token's row is
      //    in flight while the current one is evaluated) and evaluates its pairs in the
      //    canonical order against the centre rows in shared memory.
      const int nf = *fcnt;
      auto exact_token = [&](int t, unsigned msk, const U4 *xv) {
        const float ri = r_s[t];
        float dl = dl_s[t];
        int own = -1;   // the accepted centre that last lowered delta (nearest centre)
        while (msk) {
          const int j = __ffs(msk) - 1;
          msk &= msk - 1;
          const int crow = lp_row[acc_s[j]];
          float acc = 0.f;
#pragma unroll
          for (int g = 0; g < NCH; ++g) {
            const int col = 256 * g + 8 * lane;
            if (col < dv) {
              const U4 cv = lds32(cb_chunk(crow, col));
              const uint32_t xw[4] = {xv[g].x, xv[g].y, xv[g].z, xv[g].w};
              const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
              for (int hw = 0; hw < 4; ++hw) {
                acc = fma_bf16_lo(xw[hw], cw[hw], acc);
                acc = fma_bf16_hi(xw[hw], cw[hw], acc);
              }
            }
          }
          const float dot = butterfly_sum(acc);
          const float d = __fsub_rn(1.0f, __fmul_rn(__fmul_rn(dot, ri), lp_f[acc_s[j] * 3 + 2]));
          if (d < dl) own = j;
          dl = fminf(dl, d);
        }
        if (lane == 0) {
          dl_s[t] = dl;
          if (tri && own >= 0) {
            oroot_s[t] = (int16_t)croot_s[own];
            oe_s[t] = ce_s[own];
          }
        }
      };
      auto load_row = [&](int t, U4 *xv) {
        const char *row = xg + (long long)t * rb;
#pragma unroll
        for (int g = 0; g < NCH; ++g) {
          const int col = 256 * g + 8 * lane;
          xv[g] = col < dv ? ldg_stream(row + col * 2) : U4{0, 0, 0, 0};
        }
      };
      {
        U4 xa[NCH], xb[NCH];
        int f = warp;
        if (f < nf) load_row(fidx[f], xa);
        while (f < nf) {
          if (f + kSelectWarps < nf) load_row(fidx[f + kSelectWarps], xb);
          exact_token(fidx[f], fmask[f], xa);
          f += kSelectWarps;
          if (f >= nf) break;
          if (f + kSelectWarps < nf) load_row(fidx[f + kSelectWarps], xa);
          exact_token(fidx[f], fmask[f], xb);
          f += kSelectWarps;
        }
      }
      __syncthreads();
      // 5. the candidate list from the new deltas; all tokens are re-ranked only when
      //    too few of its entries are still known to lead
      deep_refresh();
      __syncthreads();
      if (*drescan == 0) return;
      TopList<kTop> tl;
      tl.clear();
      for (int t0 = warp * 32; t0 < nloc; t0 += kSelectWarps * 32) {
        const int t = t0 + lane;
        const unsigned long long key =
            (t < nloc && !sel_s[t]) ? argmax_key(__fmul_rn(w_s[t], dl_s[t]), lo + t) : 0ull;
        // the warp's 32 keys enter the list in descending order
        unsigned long long kk = key;
        for (int i = 0; i < kTop; ++i) {
          const uint32_t hi = __reduce_max_sync(0xffffffffu, (uint32_t)(kk >> 32));
          const uint32_t lo_ = __reduce_max_sync(0xffffffffu, (uint32_t)(kk >> 32) == hi ? (uint32_t)kk : 0u);
          const unsigned long long best = ((unsigned long long)hi << 32) | lo_;
          if (best == 0ull || best <= tl.k[kTop - 1]) break;
          tl.insert(best);
          if (kk == best) kk = 0ull;
        }
      }
      if (lane == 0) {
#pragma unroll
        for (int i = 0; i < kTop; ++i) wtop[warp * kTop + i] = tl.k[i];
      }
      __syncthreads();
      deep_rebuild(true);
    };
    auto update = [&](int nA, bool tri_round) {
      if constexpr (TC) {
        update_tc(nA, tri_round);
      } else {
        (void)tri_round;
        if (nA <= 4) update_nb(std::integral_constant<int, 4>{}, nA);
        else if (nA <= 8) update_nb(std::integral_constant<int, 8>{}, nA);
        else if (nA <= 12) update_nb(std::integral_constant<int, 12>{}, nA);
        else update_nb(std::integral_constant<int, 16>{}, nA);
      }
    };

    // ---- triangle-inequality bookkeeping (tensor-core variant) ----
    // Each round the cluster's CTAs split the request's roots: CTA `rank` takes roots
    // [tr_s0, tr_s0 + tr_cnt) (at most 128) and forms their dot products with every
    // list row on the tensor cores: A = the slice's root rows (M = 128, one TMEM lane
    // per root), B = the list rows in cbuf (N = lcap), fp32 accumulators in TMEM
    // columns [0, lcap), which the update's first tile reuses later.  The root rows
    // stream through the ring one K block per stage: the slice's groups of 16 rows
    // land side by side, so a stage is the K-major 128-byte-swizzled image of up to
    // 128 rows (rows past the slice hold stale data and only reach unused lanes).
    int tr_s0 = 0, tr_cnt = 0, tr_w = 0, tr_ngrp = 0, tr_nts = 0, tr_pre = 0;
    int tab_slots = 2, tab_stride = 0;   // stage slots and their spacing
    int tr_issued = 0, tr_mma = 0;   // thread 64: stages issued; thread 32: stages consumed
    // Per-slot barrier phases (the slot count changes from round to round): thread 64
    // keeps the parity of each slot's fills so far and which slots were ever filled,
    // thread 32 the parity of each slot's consumptions so far.
    uint32_t tb_fpar = 0, tb_fused = 0, tb_cpar = 0;
    uint32_t tc_tph = 0;   // root-table phase
    constexpr int kTabSlot = kTcBM * 128;   // one K block of 128 root rows
    const int tab_ring = nstage * a.tc_kps * kTcBoxBytes;
    auto tri_slice = [&]() {
      const int per = ((nroot + C - 1) / C + kRootGroup - 1) / kRootGroup * kRootGroup;
      tr_s0 = min(nroot, (int)rank * per);
      tr_cnt = min(nroot, tr_s0 + per) - tr_s0;
      tr_w = per;
      tr_ngrp = (tr_cnt + kRootGroup - 1) / kRootGroup;
      tr_nts = tr_cnt > 0 ? tc_kblocks(dv) : 0;
      tab_stride = kTabSlot;
      tab_slots = min(kTabSt, tab_ring / kTabSlot);
      tr_pre = min(tr_nts, tab_slots);
      tr_issued = 0;
      tr_mma = 0;
    };
    // thread 64: bulk copies of table stages [tr_issued, upto) into the ring; stage s
    // is K block s of every group of the slice.  A stage slot is reused once the MMAs
    // of its previous stage are done; `block` false issues only what is free now.
    auto table_load = [&](int upto, bool block) {
      char *aring = reinterpret_cast<char *>(smem + S.aring);
      const int nkb = tc_kblocks(dv);
      for (; tr_issued < upto; ++tr_issued) {
        const int st = tr_issued % tab_slots;
        if ((tb_fused >> st) & 1u) {   // the slot's previous fill must have been consumed
          const uint32_t par = ((tb_fpar >> st) & 1u) ^ 1u;
          if (!block && !mbar_try_wait(&tbe[st], par)) break;
          if (block && !twait(&tbe[st], par)) {
            tb_fpar ^= 1u << st;   // the stage is skipped: the call reports the timeout
            continue;
          }
        }
        tb_fpar ^= 1u << st;
        tb_fused |= 1u << st;
        const char *src = a.roots + (long long)(rootoff + tr_s0) * (nkb * 128) +
                          (long long)tr_issued * kRootGroupKbBytes;
        mbar_expect_tx(&tbf[st], (uint32_t)(tr_ngrp * kRootGroupKbBytes));
        for (int g = 0; g < tr_ngrp; ++g)
          bulk_g2s(aring + st * tab_stride + g * kRootGroupKbBytes,
                   src + (long long)g * nkb * kRootGroupKbBytes, (uint32_t)kRootGroupKbBytes, &tbf[st]);
      }
    };
    // thread 32: the table's MMAs (M = 128 root lanes, N = lcap list rows, one K
    // block per stage) for stages that have landed; `block` waits for all of them and
    // then commits to ttab
    auto table_mma = [&](bool block) {
      const uint32_t aring_sa = smem_addr(smem + S.aring);
      const uint32_t idesc = umma_idesc_bf16(kTcBM, lcap);
      for (; tr_mma < tr_nts; ++tr_mma) {
        const int st = tr_mma % tab_slots;
        const uint32_t par = (tb_cpar >> st) & 1u;
        if (!block && !mbar_try_wait(&tbf[st], par)) return;
        const bool ok = !block || twait(&tbf[st], par);
        tb_cpar ^= 1u << st;
        tc_fence_after();
        if (ok) {
          const int kb = tr_mma;
#pragma unroll
          for (int k = 0; k < kTcBK / 16; ++k)
            umma_bf16(tmem, umma_desc_sw128(aring_sa + st * tab_stride + k * 32),
                      umma_desc_sw128(cbuf_sa + kb * lcap * 128 + k * 32), idesc,
                      (kb | k) != 0 ? 1u : 0u);
        }
        umma_commit(&tbe[st]);
      }
      if (block) umma_commit(ttab);
    };
    // the table's service threads at a point where they are otherwise idle
    auto table_poll = [&]() {
      if (!tri || tr_nts == 0) return;
      if (threadIdx.x == 32) table_mma(false);
      else if (threadIdx.x == 64) table_load(tr_nts, false);
    };
    // warps 0-3 (TMEM lane = root of the slice): for the thread's root, the lower
    // bound rho_lb(R, c_j) per accepted centre into the global table and their minimum
    // into every CTA's mr_s[R]; per accepted centre, the nearest root of the slice
    // (the lowest root on ties) into every CTA's part_s[rank][j]
    auto table_epilogue = [&]() {
      if (warp >= 4) return;
      unsigned long long *near = wtop;   // [4 warps][kMaxAccept] (idle until the update)
      const int si = 32 * warp + lane;
      const bool valid = si < tr_cnt;
      const int R = tr_s0 + si;
      const float rr = valid ? rootr_s[R] : 0.f;
      float *trow = a.rtab + (size_t)(rootoff + (valid ? R : tr_s0)) * kMaxAccept;
      float mn = INFINITY;
      for (int c0 = 0; c0 < lcap; c0 += 16) {
        uint32_t raw[16];
        tmem_ld16(tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)c0, raw);
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int jl = rowj_s[c0 + q];   // the same for every thread
          if (jl >= 0) {
            const float rc = lp_f[acc_s[jl] * 3 + 2];
            const bool cin = tri_in_range(rc);
            const float d = __fsub_rn(1.0f, __fmul_rn(__fmul_rn(__uint_as_float(raw[q]), rc), rr));
            const float lb = cin ? tri_rho_lb(d, a.tri_eps_x) : 0.f;
            if (valid) {
              trow[jl] = lb;
              mn = fminf(mn, lb);
            }
            // (d, R) as one ordered key; NaN and invalid lanes never win
            const uint32_t dk = (valid && cin && d == d) ? (__float_as_uint(d) ^
                                ((__float_as_uint(d) & 0x80000000u) ? 0xffffffffu : 0x80000000u))
                                                          : 0xffffffffu;
            const uint32_t hk = __reduce_min_sync(0xffffffffu, dk);
            const uint32_t rk = __reduce_min_sync(0xffffffffu, dk == hk ? (uint32_t)R : 0xffffffffu);
            if (lane == 0) near[warp * kMaxAccept + jl] = ((unsigned long long)hk << 32) | rk;
          }
        }
      }
      if (valid) mr_s[R] = mn;
      asm volatile("bar.sync 1, 128;" ::: "memory");   // warps 0-3
      if (warp == 0) {
        const int jl = lane < lcap ? rowj_s[lane] : -1;
        if (jl >= 0) {
          unsigned long long best = near[jl];
#pragma unroll
          for (int w = 1; w < 4; ++w) best = min(best, near[w * kMaxAccept + jl]);
          const uint32_t hk = (uint32_t)(best >> 32);
          const bool any = hk != 0xffffffffu;
          const float bd = any ? __uint_as_float(hk ^ ((hk & 0x80000000u) ? 0x80000000u : 0xffffffffu))
                               : INFINITY;
          const int bR = any ? (int)(uint32_t)best : -1;
          for (int q = 0; q < C; ++q)
            st_cluster_v2f(map_shared(&part_s[(int)rank * kMaxAccept + jl], q), make_float2(bd, __int_as_float(bR)));
        }
        // the slice's minima to every other CTA, four at a time (tr_s0 is a multiple of 16)
        if (lane < C && lane != (int)rank)
          for (int s4 = 0; s4 < tr_cnt; s4 += 4) {
            const U4 v = lds(&mr_s[tr_s0 + s4]);
            asm volatile("st.shared::cluster.v4.u32 [%0], {%1,%2,%3,%4};"
                         :: "r"(map_shared(&mr_s[tr_s0 + s4], lane)), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                         : "memory");
          }
      }
    };
    // every CTA alike: each accepted centre's nearest root over the slices that
    // existed this round (the lowest root on ties); a centre farther than kTriTau
    // from every root becomes a root (while the request has room), else it is
    // attached to that root with e = rho_ub; then the new roots' rows are copied to
    // the request's root rows (for the next rounds' tables)
    auto tri_merge = [&](int nA, int nroot_start) {
      if (warp == 0) {
        float bd = INFINITY;
        int bR = -1;
        if (lane < nA)
          for (int q = 0; q < C; ++q)
            if (q * tr_w < nroot_start) {
              const float2 pv = part_s[q * kMaxAccept + lane];
              const int R = __float_as_int(pv.y);
              if (R >= 0 && pv.x < bd) {
                bd = pv.x;
                bR = R;
              }
            }
        const float rc = lane < nA ? lp_f[acc_s[lane] * 3 + 2] : 0.f;
        const bool cin = lane < nA && tri_in_range(rc);
        float e = INFINITY;
        int root = -1;
        bool want = false;
        if (cin) {
          if (bR < 0) {
            want = true;
          } else {
            root = bR;
            e = tri_rho_ub(bd, a.tri_eps_x);
            want = !(e <= kTriTau);
          }
        }
        const unsigned bal = __ballot_sync(0xffffffffu, want);
        const int id = nroot + __popc(bal & ((1u << lane) - 1u));
        const bool made = want && id < rcap;
        if (made) {
          root = id;
          e = 0.f;
          rootr_s[id] = rc;
        }
        if (lane < nA) {
          croot_s[lane] = root;
          ce_s[lane] = e;
        }
        const unsigned mb = __ballot_sync(0xffffffffu, made);
        if (made) nrl_s[__popc(mb & ((1u << lane) - 1u))] = make_int2(id, lp_idx[acc_s[lane]]);
        if (lane == 0) nrl_s[kMaxAccept] = make_int2(__popc(mb), 0);
      }
      __syncthreads();
      const int nnew = nrl_s[kMaxAccept].x;
      for (int u = (int)rank + C * warp; u < nnew; u += C * kSelectWarps) {
        const int2 nr = nrl_s[u];
        const char *src = xreq + (long long)nr.y * rb;
        const int i = nr.x % kRootGroup;
        const int nkb = tc_kblocks(dv);   // rows are padded to whole K blocks (zeros)
        char *grp = a.roots + (long long)(rootoff + nr.x - i) * (nkb * 128) + i * 128;
        for (int v = lane; v < nkb * 8; v += 32)   // chunk v: K block v / 8, chunk v % 8
          *reinterpret_cast<U4 *>(grp + (v >> 3) * kRootGroupKbBytes + (((v & 7) ^ (i & 7)) << 4)) =
              v < rb / 16 ? ldg(src + 16 * v) : U4{0, 0, 0, 0};
      }
      fence_proxy_async_global();   // the next rounds read these rows through TMA
      nroot += nnew;
    };

    // After an update: this CTA's live tokens and how many of them are "hard" (no
    // centre near enough for a root bound to exclude any new centre: no root, a row
    // outside the safe norm range, or 2 rho_up + e above 2), sent to every CTA.  A
    // round whose live tokens are mostly hard skips the root table: its update
    // streams every row anyway, and its accepted centres simply become roots.
    int2 *hard_s = reinterpret_cast<int2 *>(smem + S.hard);
    auto tri_count = [&]() {
      int nh = 0, nl = 0;
      for (int t = threadIdx.x; t < nloc; t += kSelThreads) {
        if (!sel_s[t]) {
          ++nl;
          const int R = oroot_s[t];
          const bool easy = R >= 0 && tri_in_range(r_s[t]) && tri_need(dl_s[t], oe_s[t]) <= 2.0f;
          nh += easy ? 0 : 1;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        nh += __shfl_xor_sync(0xffffffffu, nh, o);
        nl += __shfl_xor_sync(0xffffffffu, nl, o);
      }
      int *red = reinterpret_cast<int *>(wtop);   // idle between updates
      if (lane == 0) {
        red[2 * warp] = nh;
        red[2 * warp + 1] = nl;
      }
      __syncthreads();
      if (warp == 0) {
        int h = 0, l = 0;
#pragma unroll
        for (int w8 = 0; w8 < kSelectWarps; ++w8) {
          h += red[2 * w8];
          l += red[2 * w8 + 1];
        }
        if (lane < C) st_cluster_v2f(map_shared(&hard_s[rank], lane), make_float2(__int_as_float(h), __int_as_float(l)));
      }
    };

    // ---- seed (Eq. 9): one round that accepts argmax w~ ----
    if constexpr (TC) deep_rebuild(false);
    publish(0);
    cluster_sync();
    if (threadIdx.x == 0) {
      unsigned long long best = 0ull;
      int bq = 0;
      for (int q = 0; q < C; ++q) {
        const unsigned long long kq = pub_key[q * kTopMax];
        if (kq > best) { best = kq; bq = q; }
      }
      const int slot = bq * kTopMax;
      lp_key[0] = best;
      lp_idx[0] = key_index(best);
      const float4 f = pub_f[slot];
      lp_f[0] = f.x;
      lp_f[1] = f.y;
      lp_f[2] = f.z;
      acc_s[0] = 0;
      const int gi = lp_idx[0];
      if (gi >= lo && gi < hi) sel_s[gi - lo] = 1;
    }
    __syncthreads();
    int taken = 1;
    if (taken < K) {
      stage_list(1);
      wait_rows();
      __syncthreads();
      if (tri) tri_merge(1, 0);   // the seed is the first root
      update(1, false);
      __syncthreads();
      if (tri) tri_count();
    }

    // ---- rounds (Eq. 10-11) ----
    for (int round = 1; taken < K; ++round) {
      const int par = round & 1;
      publish(par);
      cluster_sync();
      // the root table this round only if most live tokens of the request are not hard
      // (the counts were sent before the barrier above; every CTA decides alike)
      bool table_on = false;
      if (tri) {
        int hs = 0, ls = 0;
        for (int q = 0; q < C; ++q) {
          hs += hard_s[q].x;
          ls += hard_s[q].y;
        }
        table_on = 2 * hs <= ls;
      }
      tr_s0 = tr_cnt = tr_nts = tr_pre = 0;
      if (table_on) {
        // this round's slice of the roots: its rows start streaming now, while the
        // candidate list is built (every ring stage is free at a round's start).  The
        // barrier above orders the last merge's root-row copies (any CTA) before these
        // tensor loads.
        tri_slice();
        if (threadIdx.x == 64 && tr_pre > 0) {
          fence_proxy_async_global();
          fence_proxy_async_smem();
          table_load(tr_pre, true);   // every slot is free at a round's start
        }
      }
      if (TC && early && warp > 0) {   // warps 1.. copy while warp 0 builds the list
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e) {
            const unsigned long long kq = pub_key[(par * C + q) * kTopMax + e];
            if (kq != 0ull) copy_row_tc(q * a.mc + e, key_index(kq), 32, kSelThreads - 32);
          }
        cp_async_commit();
      } else if (!TC && early && threadIdx.x == 32) {   // one lane of warp 1 issues the copies
        uint32_t bytes = 0;
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e)
            bytes += pub_key[(par * C + q) * kTopMax + e] != 0ull ? (uint32_t)rb : 0u;
        mbar_expect_tx(bar, bytes);
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e) {
            const unsigned long long kq = pub_key[(par * C + q) * kTopMax + e];
            if (kq != 0ull)
              bulk_g2s(cbuf + (long long)(q * a.mc + e) * rb, xreq + (long long)key_index(kq) * rb,
                       (uint32_t)rb, bar);
          }
      }
      // candidate list: published entries above U, best first, at most lcap.  Each
      // CTA's published entries are sorted, so the list is a C-way merge: lane q
      // holds the head of CTA q's entries and the warp takes the largest head.
      if (warp == 0) {
        const int kPer = a.mc;
        const int base = (par * C + lane) * kTopMax;
        const unsigned long long u5 = lane < C ? pub_key[base + kPer] : 0ull;
        const unsigned long long U = warp_max_u64(u5);
        int ptr = 0, n = 0;
        unsigned long long head = (lane < C && kPer > 0) ? pub_key[base] : 0ull;
        unsigned long long cut = 0ull;
        while (true) {
          const unsigned long long best = warp_max_u64(head);
          if (best <= U) break;            // also the end of every list (key 0)
          if (n == lcap) {
            cut = best;                    // the first candidate the list cannot hold
            break;
          }
          if (head == best) {              // keys are unique: one lane
            const float4 f = pub_f[base + ptr];
            lp_key[n] = best;
            lp_idx[n] = key_index(best);
            lp_row[n] = ptr + lane * kPer;  // the early copy's row of this entry
            lp_f[n * 3 + 0] = f.x;
            lp_f[n * 3 + 1] = f.y;
            lp_f[n * 3 + 2] = f.z;
            ++ptr;
            head = ptr < kPer ? pub_key[base + ptr] : 0ull;
          }
          ++n;
        }
        if (lane == 0) {
          misc[0] = cut > U ? cut : U;               // U' bounds everything outside L
          misc[1] = (unsigned long long)n;
        }
      }
      __syncthreads();
      const int nL = (int)misc[1];
      if (!early) stage_list(nL);
      wait_rows();
      if constexpr (TC) fence_proxy_async_smem();   // the list rows are MMA operands next
      __syncthreads();
      // pairwise dots of L, split over the cluster (4 interleaved pairs per warp),
      // broadcast to every CTA.  With the tensor-core update and more pairs than the
      // cluster's warps take in one pass, the list's Gram is first taken on the
      // tensor cores: a pair whose tensor-core distance is at least tc_eps above both
      // members' delta can lower neither member's delta during the replay (delta only
      // shrinks), so its dot is stored as -inf (distance +inf) and only the other
      // pairs are evaluated in the canonical order.  When one pass covers every pair
      // the Gram would only add its latency.
      {
        const int npairs = nL * (nL - 1) / 2;
        int nwork = npairs;              // pairs evaluated exactly
        int *plist = reinterpret_cast<int *>(smem + S.plist);
        const bool use_gram = TC && a.gram != 0 && npairs > C * kSelectWarps * 4;
        if constexpr (TC) if (use_gram) {
          float *gram = reinterpret_cast<float *>(smem + S.gram);
          fence_proxy_async_smem();
          tc_fence_before();
          __syncthreads();
          tc_fence_after();
          const uint32_t gcol = (uint32_t)(((a.tpc_max + kTcBM - 1) / kTcBM) * lcap);
          // K blocks alternate over kGramChains accumulators (independent MMA chains),
          // added in the epilogue
          if (threadIdx.x == 32) {
            const uint32_t idesc = umma_idesc_bf16(kTcBM, lcap);
            const int nkb = tc_kblocks(dv);
            for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
              for (int k = 0; k < kTcBK / 16; ++k)
                umma_bf16(tmem + gcol + (uint32_t)((kb % kGramChains) * lcap),
                          umma_desc_sw128(cbuf_sa + kb * lcap * 128 + k * 32),
                          umma_desc_sw128(cbuf_sa + kb * lcap * 128 + k * 32), idesc,
                          (kb >= kGramChains || k != 0) ? 1u : 0u);
            umma_commit(tpair);
          }
          table_poll();   // root-table stages that have landed
          __syncwarp();
          twait(tpair, tc_pph);
          tc_pph ^= 1u;
          tc_fence_after();
          if (warp == 0) {   // TMEM lanes 0..31 and the columns: cbuf rows
            const int nch = min(kGramChains, tc_kblocks(dv));
            for (int v0 = 0; v0 < lcap; v0 += 16) {
              float sum[16];
#pragma unroll
              for (int j = 0; j < 16; ++j) sum[j] = 0.f;
              for (int ch = 0; ch < nch; ++ch) {
                uint32_t raw[16];
                tmem_ld16(tmem + gcol + (uint32_t)(ch * lcap + v0), raw);
#pragma unroll
                for (int j = 0; j < 16; ++j) sum[j] += __uint_as_float(raw[j]);
              }
#pragma unroll
              for (int j = 0; j < 16; ++j)
                if (lane < lcap) gram[lane * kLcap + v0 + j] = sum[j];
            }
          }
          tc_fence_before();
          __syncthreads();
          // pairs that still need the canonical dot, compacted in pair order
          int base = 0;
          for (int q0 = 0; q0 < npairs; q0 += kSelThreads) {
            const int p = q0 + (int)threadIdx.x;
            bool need = false;
            if (p < npairs) {
              int u = 0, rem = p;
              while (rem >= nL - 1 - u) { rem -= nL - 1 - u; ++u; }
              const int v = u + 1 + rem;
              const float ru = lp_f[u * 3 + 2], rv = lp_f[v * 3 + 2];
              const float du = lp_f[u * 3 + 0], dv_ = lp_f[v * 3 + 0];
              const float g = gram[lp_row[u] * kLcap + lp_row[v]];
              const float d = __fsub_rn(1.0f, __fmul_rn(__fmul_rn(g, ru), rv));
              need = ru == 0.f || rv == 0.f || !(__fsub_rn(d, a.tc_eps) >= fmaxf(du, dv_));
              if (!need) pairbuf[par * kMaxPairs + p] = -INFINITY;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, need);
            if (lane == 0) cnt_s[warp] = __popc(bal);   // scratch: cnt_s is idle until the epilogue
            __syncthreads();
            int off = base, tot = 0;
#pragma unroll
            for (int w8 = 0; w8 < kSelectWarps; ++w8) {
              off += w8 < warp ? cnt_s[w8] : 0;
              tot += cnt_s[w8];
            }
            if (need) plist[off + __popc(bal & ((1u << lane) - 1u))] = p;
            base += tot;
            __syncthreads();
          }
          nwork = base;
        }
        // From here on threads 32 and 64 feed the root table until it is complete (its
        // copies and MMAs overlap the pair dots and the replay); warps 1 and 2 then
        // take no pairs, and the two service threads arrive at the cluster barrier
        // before their work (they write no pair dots) and wait on it after.
        // The split of the pairs over the warps must be the same in every CTA, so it
        // depends on the request's root count (the same everywhere), not on whether
        // this CTA's slice of the roots is empty.
        const bool tsvc = table_on && nroot > 0;
        const bool svc = tsvc && tr_nts > 0 && (threadIdx.x == 32 || threadIdx.x == 64);
        const int nwk = tsvc ? kSelectWarps - 2 : kSelectWarps;   // pair workers per CTA
        const int wk = (tsvc && warp > 0) ? warp - 2 : warp;       // this warp's worker index
        if (svc) {
          cluster_arrive_release();
          if (threadIdx.x == 32) table_mma(true);
          else table_load(tr_nts, true);
        }
        if (!(tsvc && (warp == 1 || warp == 2)))
        for (int p0 = ((int)rank + C * wk) * 4; p0 < nwork; p0 += C * nwk * 4) {
          int ja[4], jv[4];   // cbuf rows of the two members of each pair
          int pj[4];          // pair index of each work item
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int wi = min(p0 + j, nwork - 1);
            const int p = use_gram ? plist[wi] : wi;
            pj[j] = p;
            int u = 0, rem = p;
            while (rem >= nL - 1 - u) { rem -= nL - 1 - u; ++u; }
            ja[j] = lp_row[u];
            jv[j] = lp_row[u + 1 + rem];
          }
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int g = 0; g < NCH; ++g) {
            const int col = 256 * g + 8 * lane;
            if (col < dv) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                if constexpr (TC) {
                  // bf16 rows: one mixed-precision fma per coordinate, in the same order
                  const U4 va = lds32(cb_chunk(ja[j], col)), vb = lds32(cb_chunk(jv[j], col));
                  const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
                  for (int hw = 0; hw < 4; ++hw) {
                    acc[j] = fma_bf16_lo(wa[hw], wb[hw], acc[j]);
                    acc[j] = fma_bf16_hi(wa[hw], wb[hw], acc[j]);
                  }
                } else {
                  float ea[8], eb[8];
                  load8<T, true>(cbuf + (long long)ja[j] * rb, col, ea);
                  load8<T, true>(cbuf + (long long)jv[j] * rb, col, eb);
#pragma unroll
                  for (int q = 0; q < 8; ++q) acc[j] = __fmaf_rn(ea[q], eb[q], acc[j]);
                }
              }
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float d = butterfly_sum(acc[j]);
            if (p0 + j < nwork && lane < C)
              st_cluster_f32(map_shared(&pairbuf[par * kMaxPairs + pj[j]], lane), d);
          }
        }
        // the pair dots are visible cluster-wide after this barrier (non-aligned: the
        // service threads arrived early)
        if (!svc) cluster_arrive_release();
        cluster_wait_acquire();
      }
      // replay the greedy on L (warp 0; lane u holds member u); meanwhile the root
      // table's service threads finish its copies and MMAs
      if (warp == 0) {
        const unsigned long long Up = misc[0];
        bool pending = lane < nL;
        unsigned long long key = pending ? lp_key[lane] : 0ull;
        float cd = pending ? lp_f[lane * 3 + 0] : 0.f;
        const float wv = pending ? lp_f[lane * 3 + 1] : 0.f;
        const float rv = pending ? lp_f[lane * 3 + 2] : 0.f;
        const int gi = pending ? lp_idx[lane] : 0;
        int nA = 0;
        while (taken + nA < K && nA < a.max_accept) {
          // argmax of the pending keys: high word (ordered value) then low word (index)
          const uint32_t khi = pending ? (uint32_t)(key >> 32) : 0u;
          const uint32_t mhi = __reduce_max_sync(0xffffffffu, khi);
          const uint32_t klo = (pending && khi == mhi) ? (uint32_t)key : 0u;
          const uint32_t mlo = __reduce_max_sync(0xffffffffu, klo);
          const unsigned long long bk = ((unsigned long long)mhi << 32) | mlo;
          if (bk <= Up) break;
          const int bl = __ffs(__ballot_sync(0xffffffffu, pending && khi == mhi && (uint32_t)key == mlo)) - 1;
          if (lane == 0) acc_s[nA] = bl;
          ++nA;
          if (lane == bl) pending = false;
          if (taken + nA == K) break;
          const float rb_ = __shfl_sync(0xffffffffu, rv, bl);
          if (pending) {
            const int u = min(lane, bl), v = max(lane, bl);
            const int p = u * (2 * nL - u - 1) / 2 + (v - u - 1);
            const float dot = pairbuf[par * kMaxPairs + p];
            cd = fminf(cd, __fsub_rn(1.0f, __fmul_rn(__fmul_rn(dot, rv), rb_)));
            key = argmax_key(__fmul_rn(wv, cd), gi);
          }
        }
        if (lane == 0) misc[2] = (unsigned long long)nA;
      }
      __syncthreads();
      const int nA = (int)misc[2];
      if (threadIdx.x < nA) {
        const int gi = lp_idx[acc_s[threadIdx.x]];
        if (gi >= lo && gi < hi) sel_s[gi - lo] = 1;
      }
      taken += nA;
      __syncthreads();
      if (taken < K) {
        const int nroot_start = nroot;
        if (table_on) {
          if (warp == 0) {   // cbuf row -> accepted slot
            if (lane < kLcap) rowj_s[lane] = -1;
            __syncwarp();
            if (lane < nA) rowj_s[lp_row[acc_s[lane]]] = lane;
          }
          if (tr_nts > 0) {
            __syncthreads();   // the service threads finished their part during the replay
            twait(ttab, tc_tph);
            tc_tph ^= 1u;
            tc_fence_after();
          }
          __syncthreads();
          if (tr_cnt > 0) table_epilogue();
          tc_fence_before();
          cluster_sync();
          tc_fence_after();
        }
        // without a table this round no root is known near the new centres: each
        // becomes a root (while the request has room)
        if (tri) tri_merge(nA, table_on ? nroot_start : 0);
        update(nA, table_on && nroot_start > 0);
        __syncthreads();
        if (tri) tri_count();
      } else if (tri && tr_nts > 0) {
        // the selection ended this round: the table's copies and MMAs still complete
        // (nothing may be in flight when the CTA exits)
        __syncthreads();
        twait(ttab, tc_tph);
        tc_tph ^= 1u;
        tc_fence_after();
      }
    }
    if constexpr (TC) {
      tc_fence_before();
      __syncthreads();
      if (warp == 0) tmem_dealloc(tmem, a.tmem_cols);
    }
  }
  __syncthreads();

  // ---- Eq. 12: counts -> prefix over the cluster -> ascending indices + rows ----
  int cnt = 0;
  for (int t = threadIdx.x; t < nloc; t += kSelThreads) cnt += sel_s[t];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  int *red = reinterpret_cast<int *>(wtop);
  if (lane == 0) red[warp] = cnt;
  __syncthreads();
  if (warp == 0) {
    int v = lane < kSelectWarps ? red[lane] : 0;
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
      const bool sh = t < ncache;
      const char *src = sh ? xcache + (long long)t * rb : xg + (long long)t * rb;
      for (int v = lane; v < nvec; v += 32) {
        const U4 val = sh ? lds(src + 16 * v) : ldg(src + 16 * v);
        reinterpret_cast<U4 *>(out + (long long)r * rb)[v] = val;
      }
    }
  }
}

}  // namespace last
