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
#include "last_device.cuh"
#include "last_internal.h"

#include <algorithm>
#include <cmath>
#include <type_traits>

namespace last {

constexpr int kSelThreads = kSelectWarps * 32;
constexpr int kMaxCluster = 16;
constexpr int kLcap = 32;                          // candidate list capacity (runtime a.lcap <= kLcap)
constexpr int kMaxAccept = 16;                     // picks folded into delta per round
constexpr int kTopM = 9;                           // per-warp / per-CTA ranked keys (<= 8 + bound)
constexpr int kMaxPairs = kLcap * (kLcap - 1) / 2;
constexpr int kRing = 4;                           // async-copy ring depth (groups in flight)

struct SelectArgs {
  const void *x;
  const float *w;
  int32_t *idx_out;
  void *x_out;           // nullable
  const int32_t *meta;
  const int32_t *order;  // cluster -> request (most work first)
  int dv, row_bytes, tpc_max, cache_rows, csize;
  int mc;                // candidates each CTA publishes per round (<= kTopM - 1)
  int ring;              // 1: rows beyond the resident cache stream through an async-copy ring
  int lcap;              // candidate list length (16 or 32)
  unsigned *err;         // workspace error word
};

// Shared-memory carve-up, identical on host (sizing) and device.
struct SelectSmem {
  size_t xcache, cbuf, ring, blk, w, r, dl, list, sel, wtop, pub_key, pub_f, lp_key, lp_f, lp_idx,
      lp_row, pair, acc, misc, bar, cnt, total;
};
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
                                                  int ring, int tb, int elem, int lcap) {
  SelectSmem s;
  size_t o = 0;
  s.xcache = o; o += (size_t)cache_rows * row_bytes;
  s.cbuf = o; o += (size_t)lcap * row_bytes;
  s.ring = o; o += ring_bytes(ring, tb, elem);
  s.blk = o; o += align16(sizeof(int) * kSelectWarps * blocks_per_warp(tpc_max, tb));
  s.w = o; o += align16(sizeof(float) * tpc_max);
  s.r = o; o += align16(sizeof(float) * tpc_max);
  s.dl = o; o += align16(sizeof(float) * tpc_max);
  s.list = o; o += align16(sizeof(int) * tpc_max);
  s.sel = o; o += align16(tpc_max);
  s.wtop = o; o += sizeof(unsigned long long) * kSelectWarps * kTopM;
  s.pub_key = o; o += sizeof(unsigned long long) * 2 * kMaxCluster * kTopM;
  s.pub_f = o; o += sizeof(float4) * 2 * kMaxCluster * kTopM;
  s.lp_key = o; o += sizeof(unsigned long long) * kLcap;
  s.lp_f = o; o += sizeof(float) * kLcap * 3;
  s.lp_idx = o; o += sizeof(int) * kLcap;
  s.lp_row = o; o += sizeof(int) * kLcap;
  s.pair = o; o += sizeof(float) * 2 * kMaxPairs;
  s.acc = o; o += sizeof(int) * kMaxAccept;
  s.misc = o; o += sizeof(unsigned long long) * (4 + kTopM);
  s.bar = o; o += sizeof(unsigned long long);
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

// descending top-kTopM list held in (warp-uniform) registers
struct TopList {
  unsigned long long k[kTopM];
  __device__ __forceinline__ void clear() {
#pragma unroll
    for (int i = 0; i < kTopM; ++i) k[i] = 0ull;
  }
  __device__ __forceinline__ void insert(unsigned long long v) {
    if (v <= k[kTopM - 1]) return;
#pragma unroll
    for (int i = kTopM - 1; i > 0; --i) {
      if (v > k[i - 1]) k[i] = k[i - 1];
      else if (v > k[i]) { k[i] = v; v = 0ull; }
    }
    if (v > k[0]) k[0] = v;
  }
};

template <typename T, int NCH, int TB>
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

  const SelectSmem S = select_smem(a.cache_rows, a.row_bytes, a.tpc_max, a.ring, TB, (int)sizeof(T),
                                   a.lcap);
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
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
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
    // r_i = 1/sqrt(dot(x_i, x_i)); each warp also ranks its tokens by w~ for the seed
    TopList top;
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
      for (int i = 0; i < kTopM; ++i) wtop[warp * kTopM + i] = top.k[i];
    }
    __syncthreads();

    // Merge the warps' lists into the CTA's kTopM best and publish them (key and
    // {delta, w, r}) to every CTA of the cluster, into buffer `par`.
    unsigned long long *top5 = misc + 4;  // misc[4..4+kTopM)
    auto publish = [&](int par) {
      if (warp == 0) {
        constexpr int nk = kSelectWarps * kTopM;   // the warps' ranked keys
        constexpr int kPerLane = (nk + 31) / 32;
        static_assert(kPerLane <= 3, "publish ranks at most 96 keys");
        unsigned long long kl[kPerLane];
        int rl[kPerLane];
#pragma unroll
        for (int j = 0; j < kPerLane; ++j) {
          kl[j] = lane + 32 * j < nk ? wtop[lane + 32 * j] : 0ull;
          rl[j] = 0;
        }
        if (lane < kTopM) top5[lane] = 0ull;
#pragma unroll
        for (int f = 0; f < nk; ++f) {
          const unsigned long long kf = wtop[f];
#pragma unroll
          for (int j = 0; j < kPerLane; ++j) rl[j] += kf > kl[j] ? 1 : 0;
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < kPerLane; ++j)
          if (kl[j] != 0ull && rl[j] < kTopM) top5[rl[j]] = kl[j];
        __syncwarp();
        if (lane < C) {
          for (int i = 0; i <= a.mc; ++i) {
            const unsigned long long key = top5[i];
            const int slot = (par * kMaxCluster + (int)rank) * kTopM + i;
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

    // Bulk-copy the rows of list members 0..nL-1 into cbuf rows 0..nL-1 (TMA,
    // completion on `bar`); every thread then waits for them.
    auto stage_list = [&](int nL) {
      if (threadIdx.x == 0) {
        mbar_expect_tx(bar, (uint32_t)(nL * rb));
        for (int u = 0; u < nL; ++u) {
          lp_row[u] = u;
          bulk_g2s(cbuf + (long long)u * rb, xreq + (long long)lp_idx[u] * rb, (uint32_t)rb, bar);
        }
      }
    };
    auto wait_rows = [&]() {
      mbar_wait_bounded(bar, phase, a.err, kErrTimeout);
      phase ^= 1u;
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
      TopList tl;
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
        for (int i = 0; i < kTopM; ++i) wtop[warp * kTopM + i] = tl.k[i];
      }
    };
    auto update = [&](int nA) {
      if (nA <= 4) update_nb(std::integral_constant<int, 4>{}, nA);
      else if (nA <= 8) update_nb(std::integral_constant<int, 8>{}, nA);
      else if (nA <= 12) update_nb(std::integral_constant<int, 12>{}, nA);
      else update_nb(std::integral_constant<int, 16>{}, nA);
    };

    // ---- seed (Eq. 9): one round that accepts argmax w~ ----
    publish(0);
    cluster_sync();
    if (threadIdx.x == 0) {
      unsigned long long best = 0ull;
      int bq = 0;
      for (int q = 0; q < C; ++q) {
        const unsigned long long kq = pub_key[(0 * kMaxCluster + q) * kTopM];
        if (kq > best) { best = kq; bq = q; }
      }
      const int slot = (0 * kMaxCluster + bq) * kTopM;
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
      if (early && threadIdx.x == 32) {   // one lane of warp 1 issues the copies
        uint32_t bytes = 0;
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e)
            bytes += pub_key[(par * kMaxCluster + q) * kTopM + e] != 0ull ? (uint32_t)rb : 0u;
        mbar_expect_tx(bar, bytes);
        for (int q = 0; q < C; ++q)
          for (int e = 0; e < a.mc; ++e) {
            const unsigned long long kq = pub_key[(par * kMaxCluster + q) * kTopM + e];
            if (kq != 0ull)
              bulk_g2s(cbuf + (long long)(q * a.mc + e) * rb, xreq + (long long)key_index(kq) * rb,
                       (uint32_t)rb, bar);
          }
      }
      // candidate list: published top-mc entries above U, best first, at most lcap
      if (warp == 0) {
        const int kPer = a.mc;
        const int ne = C * kPer;
        const unsigned long long u5 = lane < C ? pub_key[(par * kMaxCluster + lane) * kTopM + kPer] : 0ull;
        const uint32_t uhi = __reduce_max_sync(0xffffffffu, (uint32_t)(u5 >> 32));
        const uint32_t ulo = __reduce_max_sync(0xffffffffu, (uint32_t)(u5 >> 32) == uhi ? (uint32_t)u5 : 0u);
        const unsigned long long U = ((unsigned long long)uhi << 32) | ulo;
        int slot0 = 0, slot1 = 0;
        unsigned long long ke0 = 0ull, ke1 = 0ull;
        if (lane < ne) {
          slot0 = (par * kMaxCluster + lane / kPer) * kTopM + lane % kPer;
          ke0 = pub_key[slot0];
        }
        if (lane + 32 < ne) {
          slot1 = (par * kMaxCluster + (lane + 32) / kPer) * kTopM + (lane + 32) % kPer;
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
            lp_row[pos] = (slot % kTopM) + (slot / kTopM - par * kMaxCluster) * a.mc;
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
      // broadcast to every CTA
      {
        const int npairs = nL * (nL - 1) / 2;
        for (int p0 = ((int)rank + C * warp) * 4; p0 < npairs; p0 += C * kSelectWarps * 4) {
          const char *ra[4], *rv[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int p = min(p0 + j, npairs - 1);
            int u = 0, rem = p;
            while (rem >= nL - 1 - u) { rem -= nL - 1 - u; ++u; }
            ra[j] = cbuf + (long long)lp_row[u] * rb;
            rv[j] = cbuf + (long long)lp_row[u + 1 + rem] * rb;
          }
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int g = 0; g < NCH; ++g) {
            const int col = 256 * g + 8 * lane;
            if (col < dv) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                float ea[8], eb[8];
                load8<T, true>(ra[j], col, ea);
                load8<T, true>(rv[j], col, eb);
#pragma unroll
                for (int q = 0; q < 8; ++q) acc[j] = __fmaf_rn(ea[q], eb[q], acc[j]);
              }
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float d = butterfly_sum(acc[j]);
            if (p0 + j < npairs && lane < C)
              st_cluster_f32(map_shared(&pairbuf[par * kMaxPairs + p0 + j], lane), d);
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
        while (taken + nA < K && nA < kMaxAccept) {
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

namespace {

template <typename T, int TB>
void *pick_select_tb(int nch) {
  switch (nch) {
    case 1: return (void *)select_kernel<T, 1, TB>;
    case 2: return (void *)select_kernel<T, 2, TB>;
    case 3: return (void *)select_kernel<T, 3, TB>;
    case 4: return (void *)select_kernel<T, 4, TB>;
    case 5: return (void *)select_kernel<T, 5, TB>;
    case 6: return (void *)select_kernel<T, 6, TB>;
    case 7: return (void *)select_kernel<T, 7, TB>;
    case 8: return (void *)select_kernel<T, 8, TB>;
  }
  return nullptr;
}

template <typename T>
void *pick_select(int nch, int tb) {
  // fp32 rows take twice the registers per prefetched group: 2-token blocks only
  if constexpr (sizeof(T) == 4) return pick_select_tb<T, 2>(nch);
  else return tb == 4 ? pick_select_tb<T, 4>(nch) : pick_select_tb<T, 2>(nch);
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
  // 4-token register blocks amortise the centre loads best; 2-token blocks balance
  // the warps better when a CTA owns few tokens
  auto pick = [&](int tb) {
    return pl.dtype == LAST_DTYPE_BF16 ? pick_select<__nv_bfloat16>(nch, tb)
                                       : pick_select<float>(nch, tb);
  };
  void *fn = pick(4);   // sizes the cluster; both block widths have the same footprint
  const int optin = device_smem_optin();
  double l2 = 0.0;
  {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev);
    l2 = v;
  }
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  // Cluster size: every cluster size the device can place is costed as
  //   waves x (tokens per CTA x d_v x centres per round / FMA rate + round overhead)
  // (the round count of a request does not depend on C to first order); small
  // clusters raise the number of requests in flight, large ones shorten each round.
  int C = 0, tpc = 0, cache_rows = 0;
  size_t smem = 0;
  double best = 0.0;
  int ring = 0, lcap = kLcap / 2;
  for (int c = 1; c <= kMaxCluster; c *= 2) {
    const int tpc_c = (pl.max_vis + c - 1) / c;
    const int tb_c = (pl.elem == 4 || tpc_c < 64) ? 2 : 4;
    const int lcap_c = c <= 4 ? kLcap : kLcap / 2;
    // rows that fit without a ring; otherwise reserve the ring and cache what is left
    const size_t fixed0 = select_smem(0, rb, tpc_c, 0, tb_c, pl.elem, lcap_c).total;
    if (fixed0 > (size_t)optin) continue;
    int ring_c = 0;
    int cache_c = (int)std::min<size_t>(tpc_c, (optin - fixed0) / rb);
    if (cache_c < tpc_c) {
      ring_c = 1;
      const size_t fixed1 = select_smem(0, rb, tpc_c, 1, tb_c, pl.elem, lcap_c).total;
      if (fixed1 > (size_t)optin) continue;
      cache_c = (int)std::min<size_t>(tpc_c, (optin - fixed1) / rb);
    }
    const size_t smem_c = select_smem(cache_c, rb, tpc_c, ring_c, tb_c, pl.elem, lcap_c).total;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_c);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t q = {};
    q.gridDim = dim3(c * pl.B);
    q.blockDim = dim3(kSelThreads);
    q.dynamicSmemBytes = smem_c;
    cudaLaunchAttribute qa[1];
    qa[0].id = cudaLaunchAttributeClusterDimension;
    qa[0].val.clusterDim.x = c;
    qa[0].val.clusterDim.y = 1;
    qa[0].val.clusterDim.z = 1;
    q.attrs = qa;
    q.numAttrs = 1;
    int active = 0;
    if (cudaOccupancyMaxActiveClusters(&active, fn, &q) != cudaSuccess || active <= 0) {
      cudaGetLastError();
      continue;
    }
    const double waves = std::ceil((double)pl.B / active);
    // features of the requests in flight beyond L2 stream from HBM (about 3x slower
    // per row than from L2 or shared memory)
    const double in_flight = std::min<double>(pl.B, active) * pl.max_vis * (double)rb;
    const double stream_penalty = in_flight > 0.7 * l2 ? 3.0 : 1.0;
    const double streamed = std::max(0, tpc_c - cache_c), cached = std::min(tpc_c, cache_c);
    const double round_cycles =
        (cached + stream_penalty * streamed) * pl.dv * 8.0 / 56.0 + 16000.0 + 400.0 * c;
    const double cost = waves * round_cycles;
    if (C == 0 || cost < best) {
      best = cost; C = c; tpc = tpc_c; cache_rows = cache_c; smem = smem_c; ring = ring_c;
      lcap = lcap_c;
    }
  }
  if (C == 0) return cudaErrorInvalidConfiguration;
  // 4-token register blocks amortise the centre loads best; 2-token blocks balance
  // the warps better when a CTA owns few tokens
  fn = pick(pl.elem == 4 || tpc < 64 ? 2 : 4);
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;

  SelectArgs a;
  a.x = x; a.w = w; a.idx_out = idx_out; a.x_out = x_out;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.order = reinterpret_cast<const int32_t *>(ws + pl.off_order);
  a.dv = pl.dv; a.row_bytes = rb; a.tpc_max = tpc; a.cache_rows = cache_rows; a.csize = C;
  // enough candidates per CTA that the list approximates the global top 16
  a.mc = C <= 4 ? kTopM - 1 : 4;
  a.ring = ring;
  a.lcap = lcap;
  a.err = reinterpret_cast<unsigned *>(ws + pl.off_err);

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
