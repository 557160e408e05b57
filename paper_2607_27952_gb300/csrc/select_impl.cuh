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
};

// Shared-memory carve-up, identical on host (sizing) and device.
struct SelectSmem {
  size_t aring, xcache, cbuf, ring, blk, w, r, dl, list, sel, wtop, pub_key, pub_f, lp_key,
      lp_f, lp_idx, lp_row, pair, acc, misc, bar, cnt, tbar, tslot, fidx, fmask, fcnt, gram, plist,
      total;
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
                                                  int tc = 0, int stages = 0, int kps = 1) {
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
  s.list = o; o += align16(sizeof(int) * tpc_max);
  s.sel = o; o += align16(tpc_max);
  s.wtop = o; o += sizeof(unsigned long long) * kSelectWarps * kTopMax;
  s.pub_key = o; o += sizeof(unsigned long long) * 2 * kMaxCluster * kTopMax;
  s.pub_f = o; o += sizeof(float4) * 2 * kMaxCluster * kTopMax;
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
  s.tbar = o; o += tc ? sizeof(unsigned long long) * (2 * kTcMaxStages + 2) : 0;
  s.tslot = o; o += tc ? 16 : 0;
  s.fidx = o; o += tc ? align16(sizeof(int) * tpc_max) : 0;
  s.fmask = o; o += tc ? align16(sizeof(uint32_t) * tpc_max) : 0;
  s.fcnt = o; o += tc ? 16 : 0;
  s.gram = o; o += tc ? sizeof(float) * kLcap * kLcap : 0;       // list Gram (tensor cores)
  s.plist = o; o += tc ? align16(sizeof(int) * (kMaxPairs + 1)) : 0;   // pairs to evaluate
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

  const SelectSmem S = select_smem(a.cache_rows, a.row_bytes, a.tpc_max, a.ring, TB, (int)sizeof(T),
                                   a.lcap, TC ? 1 : 0, TC ? a.tc_stages : 0, TC ? a.tc_kps : 1);
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
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    if constexpr (TC) {
      for (int i = 0; i < nstage; ++i) {
        mbar_init(&tfull[i], 1);
        mbar_init(&tempty[i], 1);
      }
      mbar_init(tdone, 1);
      mbar_init(tpair, 1);
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
    auto publish = [&](int par) {
      if (warp == 0) {
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
        __syncwarp();
        if (lane < C) {
          for (int i = 0; i <= a.mc; ++i) {
            const unsigned long long key = top5[i];
            const int slot = (par * kMaxCluster + (int)rank) * kTopMax + i;
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
    auto update_tc = [&](int nA) {
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
      // 4. exact canonical distances for the flagged pairs (a warp per token, two
      //    tokens' rows in flight)
      const int nf = *fcnt;
      auto exact_token = [&](int t, unsigned msk, const U4 *xv) {
        const float ri = r_s[t];
        float dl = dl_s[t];
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
          dl = fminf(dl, __fsub_rn(1.0f, __fmul_rn(__fmul_rn(dot, ri), lp_f[acc_s[j] * 3 + 2])));
        }
        if (lane == 0) dl_s[t] = dl;
      };
      for (int f = warp; f < nf; f += 2 * kSelectWarps) {
        const int f2 = f + kSelectWarps;
        const int t0 = fidx[f], t1 = f2 < nf ? fidx[f2] : t0;
        U4 xa[NCH], xb[NCH];
#pragma unroll
        for (int g = 0; g < NCH; ++g) {
          const int col = 256 * g + 8 * lane;
          xa[g] = col < dv ? ldg(xg + (long long)t0 * rb + col * 2) : U4{0, 0, 0, 0};
          xb[g] = col < dv ? ldg(xg + (long long)t1 * rb + col * 2) : U4{0, 0, 0, 0};
        }
        exact_token(t0, fmask[f], xa);
        if (f2 < nf) exact_token(t1, fmask[f2], xb);
      }
      __syncthreads();
      // 5. keys of the unselected tokens -> the warp's ranked list for the next round
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
    };
    auto update = [&](int nA) {
      if constexpr (TC) {
        update_tc(nA);
      } else {
        if (nA <= 4) update_nb(std::integral_constant<int, 4>{}, nA);
        else if (nA <= 8) update_nb(std::integral_constant<int, 8>{}, nA);
        else if (nA <= 12) update_nb(std::integral_constant<int, 12>{}, nA);
        else update_nb(std::integral_constant<int, 16>{}, nA);
      }
    };

    // ---- seed (Eq. 9): one round that accepts argmax w~ ----
    publish(0);
    cluster_sync();
    if (threadIdx.x == 0) {
      unsigned long long best = 0ull;
      int bq = 0;
      for (int q = 0; q < C; ++q) {
        const unsigned long long kq = pub_key[(0 * kMaxCluster + q) * kTopMax];
        if (kq > best) { best = kq; bq = q; }
      }
      const int slot = (0 * kMaxCluster + bq) * kTopMax;
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
      update(1);
      __syncthreads();
    }

    // ---- rounds (Eq. 10-11) ----
    for (int round = 1; taken < K; ++round) {
      const int par = round & 1;
      publish(par);
      cluster_sync();
      if (TC && early && warp > 0) {   // warps 1.. copy while warp 0 builds the list
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e) {
            const unsigned long long kq = pub_key[(par * kMaxCluster + q) * kTopMax + e];
            if (kq != 0ull) copy_row_tc(q * a.mc + e, key_index(kq), 32, kSelThreads - 32);
          }
        cp_async_commit();
      } else if (!TC && early && threadIdx.x == 32) {   // one lane of warp 1 issues the copies
        uint32_t bytes = 0;
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e)
            bytes += pub_key[(par * kMaxCluster + q) * kTopMax + e] != 0ull ? (uint32_t)rb : 0u;
        mbar_expect_tx(bar, bytes);
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e) {
            const unsigned long long kq = pub_key[(par * kMaxCluster + q) * kTopMax + e];
            if (kq != 0ull)
              bulk_g2s(cbuf + (long long)(q * a.mc + e) * rb, xreq + (long long)key_index(kq) * rb,
                       (uint32_t)rb, bar);
          }
      }
      // candidate list: published top-mc entries above U, best first, at most lcap
      if (warp == 0) {
        const int kPer = a.mc;
        const int ne = C * kPer;
        const unsigned long long u5 = lane < C ? pub_key[(par * kMaxCluster + lane) * kTopMax + kPer] : 0ull;
        const uint32_t uhi = __reduce_max_sync(0xffffffffu, (uint32_t)(u5 >> 32));
        const uint32_t ulo = __reduce_max_sync(0xffffffffu, (uint32_t)(u5 >> 32) == uhi ? (uint32_t)u5 : 0u);
        const unsigned long long U = ((unsigned long long)uhi << 32) | ulo;
        int slot0 = 0, slot1 = 0;
        unsigned long long ke0 = 0ull, ke1 = 0ull;
        if (lane < ne) {
          slot0 = (par * kMaxCluster + lane / kPer) * kTopMax + lane % kPer;
          ke0 = pub_key[slot0];
        }
        if (lane + 32 < ne) {
          slot1 = (par * kMaxCluster + (lane + 32) / kPer) * kTopMax + (lane + 32) % kPer;
          ke1 = pub_key[slot1];
        }
        const bool c0 = ke0 > U, c1 = ke1 > U;
        // rank among the candidates: non-candidates are masked to 0 (below every candidate)
        const unsigned long long m0 = c0 ? ke0 : 0ull, m1 = c1 ? ke1 : 0ull;
        int pos0 = 0, pos1 = 0;
#pragma unroll
        for (int src = 0; src < 32; ++src) {
          const unsigned long long a0 = shfl_u64(m0, src), a1 = shfl_u64(m1, src);
          pos0 += (a0 > ke0 ? 1 : 0) + (a1 > ke0 ? 1 : 0);
          pos1 += (a0 > ke1 ? 1 : 0) + (a1 > ke1 ? 1 : 0);
        }
        unsigned long long cut = 0ull;
        auto place = [&](bool cand, int pos, unsigned long long ke, int slot) {
          if (!cand) return;
          if (pos < lcap) {
            const float4 f = pub_f[slot];
            lp_key[pos] = ke;
            lp_idx[pos] = key_index(ke);
            lp_row[pos] = (slot % kTopMax) + (slot / kTopMax - par * kMaxCluster) * a.mc;
            lp_f[pos * 3 + 0] = f.x;
            lp_f[pos * 3 + 1] = f.y;
            lp_f[pos * 3 + 2] = f.z;
          } else if (pos == lcap) {
            cut = ke;
          }
        };
        place(c0, pos0, ke0, slot0);
        place(c1, pos1, ke1, slot1);
        const int ncand = __popc(__ballot_sync(0xffffffffu, c0)) + __popc(__ballot_sync(0xffffffffu, c1));
        {
          const uint32_t chi = __reduce_max_sync(0xffffffffu, (uint32_t)(cut >> 32));
          const uint32_t clo = __reduce_max_sync(0xffffffffu, (uint32_t)(cut >> 32) == chi ? (uint32_t)cut : 0u);
          cut = ((unsigned long long)chi << 32) | clo;
        }
        if (lane == 0) {
          misc[0] = cut > U ? cut : U;               // U' bounds everything outside L
          misc[1] = (unsigned long long)min(ncand, lcap);
        }
      }
      __syncthreads();
      const int nL = (int)misc[1];
      if (!early) stage_list(nL);
      wait_rows();
      __syncthreads();
      // pairwise dots of L, split over the cluster (4 interleaved pairs per warp),
      // broadcast to every CTA.  With the tensor-core update the list's Gram is first
      // taken on the tensor cores: a pair whose tensor-core distance is at least
      // tc_eps above both members' delta can lower neither member's delta during the
      // replay (delta only shrinks), so its dot is stored as -inf (distance +inf) and
      // only the other pairs are evaluated in the canonical order.
      {
        const int npairs = nL * (nL - 1) / 2;
        int nwork = npairs;              // pairs evaluated exactly
        int *plist = reinterpret_cast<int *>(smem + S.plist);
        if constexpr (TC) {
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
        for (int p0 = ((int)rank + C * warp) * 4; p0 < nwork; p0 += C * kSelectWarps * 4) {
          int ja[4], jv[4];   // cbuf rows of the two members of each pair
          int pj[4];          // pair index of each work item
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int wi = min(p0 + j, nwork - 1);
            const int p = TC ? plist[wi] : wi;
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
      }
      cluster_sync();
      // replay the greedy on L (warp 0; lane u holds member u)
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
        update(nA);
        __syncthreads();
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
