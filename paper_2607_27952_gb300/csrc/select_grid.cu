// Eq. 9-12 (Sec. 3.4) for a few long requests on the whole GPU.
//
// The clustered selection (select_impl.cuh) gives a request one thread-block
// cluster of at most 16 CTAs, so a batch of one to four long requests leaves most
// SMs idle, and a request longer than 16 CTAs' shared memory holds cannot run.
// Here one cooperative launch spreads the requests over every SM: request b gets
// a share of the CTAs proportional to its work k_b * N_b, each CTA owns a
// contiguous range of its tokens (w~, 1/|x|, delta and the selected flag in shared
// memory), and the CTAs of a request meet at one grid barrier per round through
// global memory.
//
// A round accepts a batch of consecutive greedy picks, exactly the sequential
// Eq. 10-11 sequence:
//   1. every CTA ranks its live tokens by w~ delta and publishes its 16 best keys
//      (with delta, w~, 1/|x|) and its 17th key to global memory; grid barrier;
//   2. every CTA reads all published keys of the request: the entries above
//      U = the largest 17th key form the candidate list (best first, at most 16;
//      U grows to the first entry cut off).  No token outside the list has a key
//      above U, and keys never increase, so U bounds them for the whole round;
//   3. every CTA copies the list rows, forms their pairwise dot products in the
//      canonical order and replays the greedy on the list: the member with the
//      largest current key is the true next pick while it is above U;
//   4. every CTA folds the accepted centres into the delta of its own tokens
//      (canonical order, four centres at a time per warp).
// Every CTA of a request computes the same list and the same picks.  The seed
// (Eq. 9) is a round on keys w~ that accepts exactly one token.
//
// Arithmetic is the canonical fp32 of the public header, as in the clustered
// kernel, so the kept indices are bit-identical to it and to the oracle.
//
// Every grid-barrier wait is bounded: on expiry the CTA sets kErrTimeout and an
// abort word that ends every later wait of the launch at once, so a broken launch
// finishes (reporting LAST_ERR_TIMEOUT through last_poll) instead of hanging.
#include "select_impl.cuh"

#include <algorithm>
#include <cstring>

namespace last {

constexpr int kGridTop = 17;       // keys each CTA publishes: 16 candidates and the bound
constexpr int kGridLcap = 16;      // candidate list
constexpr int kGridPairs = kGridLcap * (kGridLcap - 1) / 2;
constexpr int kGridAccept = 16;    // picks accepted per round at most
constexpr uint32_t kGridWaitLimit = 1u << 21;   // polls of one barrier wait (a second or two)

struct GridArgs {
  const void *x;
  const float *w;
  int32_t *idx_out;
  void *x_out;             // nullable
  const int32_t *meta;
  unsigned *err;           // workspace error word
  unsigned *gbar;          // [0] abort word, [1 + s] barrier counter of request slot s
  unsigned long long *pub_key;   // [2][kGridMaxCtas][kGridTop]
  float4 *pub_f;                 // [2][kGridMaxCtas][kGridTop]: delta, w~, 1/|x|
  int *gcnt;                     // [kGridMaxCtas] kept tokens per CTA (the epilogue)
  int cta0[kGridMaxReq + 1];     // slot s owns CTAs [cta0[s], cta0[s + 1])
  int req[kGridMaxReq];          // request of slot s
  int nslot, dv, row_bytes, tpc_max;
};

// Shared memory (host sizing and device carve-up alike).
struct GridSmem {
  size_t cbuf, w, r, dl, sel, list, wtop, lp_key, lp_f, lp_idx, pair, acc, misc, total;
};
__host__ __device__ inline GridSmem grid_smem(int row_bytes, int tpc) {
  GridSmem s;
  size_t o = 0;
  s.cbuf = o; o += (size_t)kGridLcap * row_bytes;
  s.w = o; o += align16(sizeof(float) * tpc);
  s.r = o; o += align16(sizeof(float) * tpc);
  s.dl = o; o += align16(sizeof(float) * tpc);
  s.sel = o; o += align16(tpc);
  s.list = o; o += align16(sizeof(int) * tpc);   // the epilogue's kept tokens
  s.wtop = o; o += sizeof(unsigned long long) * kSelectWarps * kGridTop;
  s.lp_key = o; o += sizeof(unsigned long long) * (kGridLcap + 1);
  s.lp_f = o; o += sizeof(float) * 3 * kGridLcap;
  s.lp_idx = o; o += sizeof(int) * kGridLcap;
  s.pair = o; o += sizeof(float) * kGridPairs;
  s.acc = o; o += sizeof(int) * kGridAccept;
  s.misc = o; o += sizeof(unsigned long long) * (4 + kSelectWarps);
  s.total = align16(o);
  return s;
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

template <typename T, int NCH>
__global__ void __launch_bounds__(kSelThreads, 1) select_grid_kernel(const __grid_constant__ GridArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int slot = 0;
  while (slot + 1 < a.nslot && (int)blockIdx.x >= a.cta0[slot + 1]) ++slot;
  const int q = (int)blockIdx.x - a.cta0[slot], G = a.cta0[slot + 1] - a.cta0[slot];
  const int b = a.req[slot];
  const int32_t *m = a.meta + b * kMetaFields;
  const int voff = m[kVisOff], N = m[kNumVis], koff = m[kKeepOff], K = m[kNumKeep];
  if (K == 0) return;   // every CTA of the request leaves: no barrier is reached
  const int tpc = (N + G - 1) / G;
  const int lo = min(N, q * tpc), hi = min(N, lo + tpc), nloc = hi - lo;
  const int rb = a.row_bytes, dv = a.dv;
  const char *xreq = static_cast<const char *>(a.x) + (long long)voff * rb;
  const char *xg = xreq + (long long)lo * rb;
  unsigned *ctr = a.gbar + 1 + slot;
  unsigned *abort_w = a.gbar;

  const GridSmem S = grid_smem(rb, a.tpc_max);
  char *cbuf = reinterpret_cast<char *>(smem + S.cbuf);
  float *w_s = reinterpret_cast<float *>(smem + S.w);
  float *r_s = reinterpret_cast<float *>(smem + S.r);
  float *dl_s = reinterpret_cast<float *>(smem + S.dl);
  unsigned char *sel_s = smem + S.sel;
  unsigned long long *wtop = reinterpret_cast<unsigned long long *>(smem + S.wtop);
  unsigned long long *lp_key = reinterpret_cast<unsigned long long *>(smem + S.lp_key);
  float *lp_f = reinterpret_cast<float *>(smem + S.lp_f);
  int *lp_idx = reinterpret_cast<int *>(smem + S.lp_idx);
  float *pairbuf = reinterpret_cast<float *>(smem + S.pair);
  int *acc_s = reinterpret_cast<int *>(smem + S.acc);
  unsigned long long *misc = reinterpret_cast<unsigned long long *>(smem + S.misc);

  // grid barrier of the request's CTAs: generation `gen` completes when all G have
  // arrived for the gen-th time (the counter starts at zero every call)
  unsigned gen = 0;
  auto gsync = [&]() {
    __syncthreads();
    if (threadIdx.x == 0) {
      ++gen;
      __threadfence();   // this CTA's global writes before its arrival
      atomicAdd(ctr, 1u);
      const unsigned target = gen * (unsigned)G;
      bool ok = false;
      for (uint32_t i = 0; i < kGridWaitLimit; ++i) {
        if (ld_acquire_u32(ctr) >= target) { ok = true; break; }
        if (ld_acquire_u32(abort_w) != 0u) break;
      }
      if (!ok) {
        atomicOr(a.err, kErrTimeout);
        atomicExch(abort_w, 1u);
      }
      __threadfence();
    }
    __syncthreads();
  };

  // ---- prologue: w~, delta = +inf, 1/|x| of the own tokens ----
  for (int t = threadIdx.x; t < nloc; t += kSelThreads) {
    w_s[t] = a.w[voff + lo + t];
    dl_s[t] = INFINITY;
    sel_s[t] = (K == N) ? 1 : 0;
  }
  __syncthreads();
  int taken = K == N ? K : 0;   // K == N keeps every token (selected above)
  if (K < N) {
    for (int t = warp; t < nloc; t += kSelectWarps) {
      const char *row = xg + (long long)t * rb;
      const float ss = dot_rows<T, NCH>(row, false, row, false, dv, lane);
      if (lane == 0) r_s[t] = ss > 0.f ? __fdiv_rn(1.0f, __fsqrt_rn(ss)) : 0.f;
    }
    __syncthreads();
  }

  // the warps' best keys of the own live tokens (key w~ delta, or w~ for the seed)
  auto rank_own = [&](bool seed) {
    TopList<kGridTop> tl;
    tl.clear();
    for (int t0 = warp * 32; t0 < nloc; t0 += kSelectWarps * 32) {
      const int t = t0 + lane;
      const unsigned long long key =
          (t < nloc && !sel_s[t]) ? argmax_key(seed ? w_s[t] : __fmul_rn(w_s[t], dl_s[t]), lo + t) : 0ull;
      unsigned long long kk = key;
      for (int i = 0; i < kGridTop; ++i) {
        const unsigned long long best = warp_max_u64(kk);
        if (best == 0ull || best <= tl.k[kGridTop - 1]) break;
        tl.insert(best);
        if (kk == best) kk = 0ull;
      }
    }
    if (lane == 0)
      for (int i = 0; i < kGridTop; ++i) wtop[warp * kGridTop + i] = tl.k[i];
    __syncthreads();
  };
  // warp 0: the best `n` of the keys at src[0 .. cnt) into out (descending, zero-padded)
  auto merge_top = [&](const unsigned long long *src, int cnt, unsigned long long *out, int n) {
    TopList<kGridTop> tl;
    tl.clear();
    for (int f0 = 0; f0 < cnt; f0 += 32) {
      unsigned long long kk = f0 + lane < cnt ? src[f0 + lane] : 0ull;
      for (int i = 0; i < n; ++i) {
        const unsigned long long best = warp_max_u64(kk);
        if (best == 0ull || best <= tl.k[n - 1]) break;
        tl.insert(best);
        if (kk == best) kk = 0ull;
      }
    }
    if (lane < n) out[lane] = tl.k[lane];
    __syncwarp();
  };
  // this CTA's kGridTop best keys and their (delta, w~, 1/|x|) to global, parity par
  auto publish = [&](int par) {
    if (warp == 0) {
      merge_top(wtop, kSelectWarps * kGridTop, lp_key, kGridTop);   // lp_key holds kGridLcap + 1
      const size_t base = ((size_t)par * kGridMaxCtas + blockIdx.x) * kGridTop;
      if (lane < kGridTop) {
        const unsigned long long key = lp_key[lane];
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (key != 0ull) {
          const int lt = key_index(key) - lo;
          f = make_float4(dl_s[lt], w_s[lt], r_s[lt], 0.f);
        }
        a.pub_key[base + lane] = key;
        a.pub_f[base + lane] = f;
      }
    }
  };

  // ---- rounds (the seed is round 0: keys w~, one pick) ----
  for (int round = 0; taken < K; ++round) {
    const int par = round & 1;
    rank_own(round == 0);
    publish(par);
    gsync();
    // candidate list: published entries above U = the largest bound, best first
    {
      const size_t base = ((size_t)par * kGridMaxCtas + a.cta0[slot]) * kGridTop;
      // each warp: its share of the request's candidate entries -> its best kGridLcap + 1
      TopList<kGridTop> tl;
      tl.clear();
      unsigned long long ub = 0ull;
      for (int f0 = warp * 32; f0 < G * kGridTop; f0 += kSelectWarps * 32) {
        const int f = f0 + lane;
        unsigned long long kk = 0ull;
        if (f < G * kGridTop) {
          const unsigned long long v = __ldcg(a.pub_key + base + f);
          if (f % kGridTop == kGridTop - 1) ub = max(ub, v);
          else kk = v;
        }
        for (int i = 0; i < kGridTop; ++i) {
          const unsigned long long best = warp_max_u64(kk);
          if (best == 0ull || best <= tl.k[kGridTop - 1]) break;
          tl.insert(best);
          if (kk == best) kk = 0ull;
        }
      }
      ub = warp_max_u64(ub);
      if (lane == 0) {
        for (int i = 0; i < kGridTop; ++i) wtop[warp * kGridTop + i] = tl.k[i];
        misc[4 + warp] = ub;
      }
      __syncthreads();
      if (warp == 0) {
        unsigned long long U = lane < kSelectWarps ? misc[4 + lane] : 0ull;
        U = warp_max_u64(U);
        merge_top(wtop, kSelectWarps * kGridTop, lp_key, kGridLcap + 1);
        int n = 0;
        for (int i = 0; i < kGridLcap; ++i) n += lp_key[i] > U ? 1 : 0;
        const unsigned long long cut = lp_key[kGridLcap] > U ? lp_key[kGridLcap] : 0ull;
        if (round == 0) n = min(n, 1);   // the seed round takes exactly argmax w~
        if (lane == 0) {
          misc[0] = cut > U ? cut : U;   // U' bounds every token outside the list
          misc[1] = (unsigned long long)n;
        }
        if (lane < n) lp_idx[lane] = key_index(lp_key[lane]);
      }
      __syncthreads();
      // the members' (delta, w~, 1/|x|) from the published payload: every thread
      // matches its share of the request's published entries against the list
      {
        const int n = (int)misc[1];
        for (int f = threadIdx.x; f < G * kGridTop; f += kSelThreads) {
          if (f % kGridTop == kGridTop - 1) continue;
          const unsigned long long v = __ldcg(a.pub_key + base + f);
          for (int u = 0; u < n; ++u)
            if (v == lp_key[u]) {
              const float4 pf = __ldcg(a.pub_f + base + f);
              lp_f[u * 3 + 0] = pf.x;
              lp_f[u * 3 + 1] = pf.y;
              lp_f[u * 3 + 2] = pf.z;
            }
        }
      }
      __syncthreads();
    }
    const int nL = (int)misc[1];
    // the list rows into shared memory (16-byte loads of every thread)
    {
      const int nvec = rb / 16;
      for (int v = threadIdx.x; v < nL * nvec; v += kSelThreads) {
        const int u = v / nvec, c = v - u * nvec;
        reinterpret_cast<U4 *>(cbuf + (long long)u * rb)[c] = ldg(xreq + (long long)lp_idx[u] * rb + 16 * c);
      }
    }
    __syncthreads();
    // pairwise canonical dots of the list, four interleaved pairs per warp
    const int npairs = nL * (nL - 1) / 2;
    for (int p0 = warp * 4; p0 < npairs; p0 += kSelectWarps * 4) {
      int ja[4], jv[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int p = min(p0 + j, npairs - 1);
        int u = 0, rem = p;
        while (rem >= nL - 1 - u) { rem -= nL - 1 - u; ++u; }
        ja[j] = u;
        jv[j] = u + 1 + rem;
      }
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int g = 0; g < NCH; ++g) {
        const int col = 256 * g + 8 * lane;
        if (col < dv) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float ea[8], eb[8];
            load8<T, true>(cbuf + (long long)ja[j] * rb, col, ea);
            load8<T, true>(cbuf + (long long)jv[j] * rb, col, eb);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[j] = __fmaf_rn(ea[e], eb[e], acc[j]);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float d = butterfly_sum(acc[j]);
        if (p0 + j < npairs && lane == 0) pairbuf[p0 + j] = d;
      }
    }
    __syncthreads();
    // replay the greedy on the list (warp 0; lane u holds member u)
    if (warp == 0) {
      const unsigned long long Up = misc[0];
      bool pending = lane < nL;
      unsigned long long key = pending ? lp_key[lane] : 0ull;
      float cd = pending ? lp_f[lane * 3 + 0] : 0.f;
      const float wv = pending ? lp_f[lane * 3 + 1] : 0.f;
      const float rv = pending ? lp_f[lane * 3 + 2] : 0.f;
      const int gi = pending ? lp_idx[lane] : 0;
      int nA = 0;
      while (taken + nA < K && nA < kGridAccept && nA < nL) {
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
        if (taken + nA == K || round == 0) break;
        const float rb_ = __shfl_sync(0xffffffffu, rv, bl);
        if (pending) {
          const int u = min(lane, bl), v = max(lane, bl);
          const int p = u * (2 * nL - u - 1) / 2 + (v - u - 1);
          cd = fminf(cd, __fsub_rn(1.0f, __fmul_rn(__fmul_rn(pairbuf[p], rv), rb_)));
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
    if (taken >= K || nA == 0) {
      if (nA == 0 && threadIdx.x == 0) atomicOr(a.err, kErrConfig);   // cannot happen: U bounds
      if (nA == 0) break;
      continue;
    }
    // delta <- min(delta, d(i, c)) over the accepted centres in acceptance order,
    // four centres at a time (independent canonical fma chains) per warp and token;
    // the warp's next token row is in flight while the current one is evaluated
    {
      constexpr bool kBf16 = sizeof(T) == 2;
      constexpr int kVec = kBf16 ? 1 : 2;   // 16-byte vectors per 8-coordinate group
      auto load_tok = [&](int t, U4 (*xv)[kVec]) {
        const char *row = xg + (long long)t * rb;
#pragma unroll
        for (int g = 0; g < NCH; ++g) {
          const int col = 256 * g + 8 * lane;
#pragma unroll
          for (int h = 0; h < kVec; ++h)
            xv[g][h] = col < dv ? ldg_stream(row + col * (int)sizeof(T) + 16 * h) : U4{0, 0, 0, 0};
        }
      };
      auto eval_tok = [&](int t, U4 (*xv)[kVec]) {
        const float ri = r_s[t];
        float dl = dl_s[t];
        for (int j0 = 0; j0 < nA; j0 += 4) {
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
          const char *crow[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) crow[j] = cbuf + (long long)acc_s[min(j0 + j, nA - 1)] * rb;
#pragma unroll
          for (int g = 0; g < NCH; ++g) {
            const int col = 256 * g + 8 * lane;
            if (col < dv) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                if (kBf16) {
                  const U4 cv = lds(crow[j] + col * 2);
                  const uint32_t xw[4] = {xv[g][0].x, xv[g][0].y, xv[g][0].z, xv[g][0].w};
                  const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
                  for (int hw = 0; hw < 4; ++hw) {
                    acc[j] = fma_bf16_lo(xw[hw], cw[hw], acc[j]);
                    acc[j] = fma_bf16_hi(xw[hw], cw[hw], acc[j]);
                  }
                } else {
                  float ec[8], ex[8];
                  load8<T, true>(crow[j], col, ec);
                  Elem<T>::widen(xv[g][0], ex);
                  Elem<T>::widen(xv[g][kVec - 1], ex + 4);
#pragma unroll
                  for (int e = 0; e < 8; ++e) acc[j] = __fmaf_rn(ex[e], ec[e], acc[j]);
                }
              }
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (j0 + j < nA) {
              const float dot = butterfly_sum(acc[j]);
              const float rc = lp_f[acc_s[j0 + j] * 3 + 2];
              dl = fminf(dl, __fsub_rn(1.0f, __fmul_rn(__fmul_rn(dot, ri), rc)));
            }
          }
        }
        if (lane == 0) dl_s[t] = dl;
      };
      // the warp's live tokens t = warp, warp + 8, ... (selected ones skipped)
      auto next_live = [&](int t) {
        while (t < nloc && sel_s[t]) t += kSelectWarps;
        return t;
      };
      U4 xa[NCH][kVec], xb[NCH][kVec];
      int t = next_live(warp);
      if (t < nloc) load_tok(t, xa);
      while (t < nloc) {
        int tn = next_live(t + kSelectWarps);
        if (tn < nloc) load_tok(tn, xb);
        eval_tok(t, xa);
        t = tn;
        if (t >= nloc) break;
        tn = next_live(t + kSelectWarps);
        if (tn < nloc) load_tok(tn, xa);
        eval_tok(t, xb);
        t = tn;
      }
    }
    __syncthreads();
  }

  // ---- Eq. 12: counts of the request's CTAs -> prefix -> ascending indices + rows ----
  int cnt = 0;
  for (int t = threadIdx.x; t < nloc; t += kSelThreads) cnt += sel_s[t];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  int *red = reinterpret_cast<int *>(wtop);
  if (lane == 0) red[warp] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int v = 0;
    for (int w8 = 0; w8 < kSelectWarps; ++w8) v += red[w8];
    a.gcnt[blockIdx.x] = v;
  }
  gsync();
  int prefix = 0;
  for (int qq = 0; qq < q; ++qq) prefix += __ldcg(a.gcnt + a.cta0[slot] + qq);
  int *list_s = reinterpret_cast<int *>(smem + S.list);
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
    if (lane == 0) misc[3] = (unsigned long long)run;
  }
  __syncthreads();
  if (a.x_out != nullptr) {
    const int mine = (int)misc[3];
    const int nvec = rb / 16;
    char *out = static_cast<char *>(a.x_out) + (long long)(koff + prefix) * rb;
    for (int r = warp; r < mine; r += kSelectWarps) {
      const char *src = xg + (long long)list_s[r] * rb;
      for (int v = lane; v < nvec; v += 32)
        reinterpret_cast<U4 *>(out + (long long)r * rb)[v] = ldg(src + 16 * v);
    }
  }
}

namespace {

template <typename T>
void *pick_grid(int nch) {
  switch (nch) {
    case 1: return (void *)select_grid_kernel<T, 1>;
    case 2: return (void *)select_grid_kernel<T, 2>;
    case 3: return (void *)select_grid_kernel<T, 3>;
    case 4: return (void *)select_grid_kernel<T, 4>;
    case 5: return (void *)select_grid_kernel<T, 5>;
    case 6: return (void *)select_grid_kernel<T, 6>;
    case 7: return (void *)select_grid_kernel<T, 7>;
    case 8: return (void *)select_grid_kernel<T, 8>;
  }
  return nullptr;
}

}  // namespace

size_t grid_select_smem(int row_bytes, int tpc) { return grid_smem(row_bytes, tpc).total; }

namespace {

// CTAs per request: first as many as its tokens need to fit one CTA's shared
// memory (`optin` bytes), then the rest in proportion to k_b * N_b; `ctas` in
// all.  Returns the largest tokens-per-CTA, or 0 when the requests do not fit.
int grid_assign(const Plan &pl, int ctas, size_t optin, int *cta0) {
  const int32_t *meta = pl.host_blob.data() + pl.off_meta / 4;
  const int rb = pl.dv * pl.elem;
  int lo = 0, hi = 1 << 22;   // tokens per CTA that fit: the largest t with a plan <= optin
  while (lo < hi) {
    const int t = lo + (hi - lo + 1) / 2;
    if (grid_smem(rb, t).total <= optin) lo = t;
    else hi = t - 1;
  }
  if (lo < 1) return 0;
  int g[kGridMaxReq], need = 0;
  double total = 0.0;
  for (int b = 0; b < pl.B; ++b) {
    const int n = meta[b * kMetaFields + kNumVis];
    g[b] = std::max(1, (n + lo - 1) / lo);
    need += g[b];
    total += std::max(1.0, (double)meta[b * kMetaFields + kNumKeep] * n);
  }
  if (need > ctas) return 0;
  int left = ctas - need;
  for (int b = 0; b < pl.B && left > 0; ++b) {
    const double wk = std::max(1.0, (double)meta[b * kMetaFields + kNumKeep] * meta[b * kMetaFields + kNumVis]);
    const int extra = std::min(left, (int)std::floor((ctas - need) * wk / total));
    g[b] += extra;
    left -= extra;
  }
  for (int b = 0; left > 0; b = (b + 1) % pl.B, --left) ++g[b];   // the rounding remainder
  int used = 0, tpc = 1;
  for (int b = 0; b < pl.B; ++b) {
    cta0[b] = used;
    used += g[b];
    tpc = std::max(tpc, (meta[b * kMetaFields + kNumVis] + g[b] - 1) / g[b]);
  }
  cta0[pl.B] = used;
  return tpc;
}

// SMs of the current device and its opt-in shared memory per CTA (0, 0 on error).
void device_limits(int *sms, int *optin) {
  int dev = 0;
  *sms = *optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
    cudaGetLastError();
    *sms = *optin = 0;
  }
}

}  // namespace

bool grid_select_fits(const Plan &pl) {
  // (the workspace holds the published keys only for such launches)
  if (pl.B < 1 || pl.B > kGridMaxReq || pl.max_vis < kGridMinTokens) return false;
  int sms = 0, optin = 0;
  device_limits(&sms, &optin);
  const int ctas = std::min(sms, kGridMaxCtas);
  if (ctas < pl.B) return false;
  int cta0[kGridMaxReq + 1];
  const int tpc = grid_assign(pl, ctas, (size_t)optin, cta0);
  return tpc > 0 && grid_smem(pl.dv * pl.elem, tpc).total <= (size_t)optin;
}

cudaError_t launch_select_grid(const Plan &pl, const float *w, const void *x, int32_t *idx_out,
                               void *x_out, char *ws, cudaStream_t s) {
  const int rb = pl.dv * pl.elem;
  const int nch = (pl.dv + 255) / 256;
  void *fn = pl.dtype == LAST_DTYPE_BF16 ? pick_grid<__nv_bfloat16>(nch) : pick_grid<float>(nch);
  if (fn == nullptr || pl.B < 1 || pl.B > kGridMaxReq) return cudaErrorInvalidConfiguration;
  int sms = 0, optin = 0;
  device_limits(&sms, &optin);
  const int ctas = std::min(sms, kGridMaxCtas);
  if (ctas < pl.B) return cudaErrorInvalidConfiguration;
  GridArgs a;
  std::memset(&a, 0, sizeof a);
  a.nslot = pl.B;
  const int tpc = grid_assign(pl, ctas, (size_t)optin, a.cta0);
  for (int b = 0; b < pl.B; ++b) a.req[b] = b;
  const size_t smem = grid_smem(rb, tpc).total;
  if (tpc == 0 || smem > (size_t)optin) return cudaErrorInvalidConfiguration;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  a.x = x; a.w = w; a.idx_out = idx_out; a.x_out = x_out;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.err = reinterpret_cast<unsigned *>(ws + pl.off_err);
  a.gbar = reinterpret_cast<unsigned *>(ws + pl.off_gbar);
  a.pub_key = reinterpret_cast<unsigned long long *>(ws + pl.off_gpub);
  a.pub_f = reinterpret_cast<float4 *>(ws + pl.off_gpub + sizeof(unsigned long long) * 2 * kGridMaxCtas * kGridTop);
  a.gcnt = reinterpret_cast<int *>(ws + pl.off_gpub + (sizeof(unsigned long long) + sizeof(float4)) * 2 *
                                   kGridMaxCtas * kGridTop);
  a.dv = pl.dv; a.row_bytes = rb; a.tpc_max = tpc;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.cta0[pl.B]);
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;   // every CTA resident at once (they wait on one another)
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void *args[] = {&a};
  return cudaLaunchKernelExC(&cfg, fn, args);
}

size_t grid_pub_bytes() {
  return (sizeof(unsigned long long) + sizeof(float4)) * 2 * kGridMaxCtas * kGridTop + sizeof(int) * kGridMaxCtas;
}

}  // namespace last
