/*
 * Plain, slow, single-threaded CPU oracle for LAST's edge-side token-selection
 * path (last-query-token attention scoring, importance-weighted greedy k-center
 * selection, order-restoring gather).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may call this file.  It shares no code,
 * header, table or helper with the CUDA library, and the CUDA library never
 * calls it.
 *
 * Every function follows the paper's equations literally, in the order the
 * paper states them:
 *   oracle_last_row        Eq. 6  (one row p* of the causal softmax attention)
 *   oracle_scores          Eq. 6, 7, 8 (sum over layers and heads, normalise)
 *   oracle_scores_rows     Table 4's attention sources: Eq. 6-8 with the rows of
 *                          several query positions summed (First, Middle, All Mean)
 *   oracle_select_fp32     Eq. 9, 10, 11 in "canonical fp32" arithmetic
 *   oracle_select_fp64     Eq. 9, 10, 11 in plain fp64 arithmetic
 *   oracle_select_topk     Table 5's "Top-k" selection: the k highest scores
 *   oracle_restore_order   Eq. 12 (sort(S))
 *   oracle_gather          Eq. 12 (X_S = [x_i], i in sort(S))
 *   oracle_budget          Eq. 2  (K = ceil(rho N))
 *
 * Build: gcc -O2 -ffp-contract=off -std=c99 -fPIC -shared (no fast-math), so
 * every fused multiply-add is the explicit fmaf() written below and nothing
 * else is contracted.
 *
 * Readings where the paper is silent (also listed in the design notes):
 *  - scores sum over the layers and q-heads passed in; q-head h reads kv-head
 *    floor(h / (Hq/Hkv)) (consecutive grouping);
 *  - softmax scale defaults to 1/sqrt(D); the row p* = P_b - 1 is unmasked over
 *    all P_b keys (visual, text and itself);
 *  - argmax ties go to the lowest index; selected tokens are excluded by the
 *    selected set, never by their delta value; no clamp of delta;
 *  - x_bar^T x_bar_j is evaluated as (dot(x_i, x_j) * r_i) * r_j with
 *    r = 1/sqrt(dot(x, x)) (r = 0 for a zero vector).
 *
 * Parity status: scores are pinned by closed forms, a brute-force P x P
 * causal attention and invariants; selection is pinned by brute-force
 * enumeration of greedy sequences on tiny inputs and by special cases with
 * known answers (orthogonal features -> top-k, identical features, uniform
 * weights -> farthest-point order).  The paper prints no worked numerical
 * example, so no value is pinned to a number printed in the paper.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_DTYPE_F32 0
#define ORACLE_DTYPE_BF16 1

/* Exact widening of one stored element to double (bf16 is the upper half of
 * an IEEE single). */
static double load_elem(const void *base, int dtype, int64_t i) {
  if (dtype == ORACLE_DTYPE_F32) return (double)((const float *)base)[i];
  uint32_t u = (uint32_t)((const uint16_t *)base)[i] << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static float load_elem_f(const void *base, int dtype, int64_t i) {
  return (float)load_elem(base, dtype, i);
}

/* ------------------------------------------------------------------------ */
/* Eq. 6: the softmax-normalised causal attention row of the last position   */
/* p* = P_b - 1 for one (request b, layer l, q-head h).  Writes P_b values.  */
/* q: [B][L][Hq][D]; k: [L][sum P][Hkv][D].                                  */
/* ------------------------------------------------------------------------ */
int oracle_last_row(int B, int L, int Hq, int Hkv, int D, int dtype, double scale,
                    const int32_t *cu_seqlens, const void *q, const void *k,
                    int b, int l, int h, double *a_out) {
  if (b < 0 || b >= B || l < 0 || l >= L || h < 0 || h >= Hq) return 1;
  if (Hkv <= 0 || Hq % Hkv != 0) return 1;
  if (scale <= 0.0) scale = 1.0 / sqrt((double)D);
  const int group = Hq / Hkv;
  const int g = h / group;
  const int64_t total_keys = cu_seqlens[B];
  const int64_t p0 = cu_seqlens[b];
  const int P = cu_seqlens[b + 1] - cu_seqlens[b];
  if (P <= 0) return 1;
  const int64_t qoff = (((int64_t)b * L + l) * Hq + h) * D;
  /* logits z_p = scale * q . k_p over every key the last row can see */
  double zmax = -INFINITY;
  for (int p = 0; p < P; ++p) {
    const int64_t koff = (((int64_t)l * total_keys + p0 + p) * Hkv + g) * D;
    double acc = 0.0;
    for (int d = 0; d < D; ++d) acc += load_elem(q, dtype, qoff + d) * load_elem(k, dtype, koff + d);
    a_out[p] = scale * acc;
    if (a_out[p] > zmax) zmax = a_out[p];
  }
  double zsum = 0.0;
  for (int p = 0; p < P; ++p) {
    a_out[p] = exp(a_out[p] - zmax);
    zsum += a_out[p];
  }
  for (int p = 0; p < P; ++p) a_out[p] /= zsum;
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Eq. 7 and 8: s_i = sum_l sum_h A^(l,h)[p*, p_i], w_i = s_i / sum_j s_j.     */
/* Visual token i of request b sits at position vis_start[b] + i; its score  */
/* goes to w_out[cu_vis[b] + i].                                             */
/* ------------------------------------------------------------------------ */
int oracle_scores(int B, int L, int Hq, int Hkv, int D, int dtype, double scale,
                  const int32_t *cu_seqlens, const int32_t *vis_start, const int32_t *cu_vis,
                  const void *q, const void *k, double *w_out) {
  int max_p = 0;
  for (int b = 0; b < B; ++b) {
    int P = cu_seqlens[b + 1] - cu_seqlens[b];
    int N = cu_vis[b + 1] - cu_vis[b];
    if (P <= 0 || N < 0 || vis_start[b] < 0 || vis_start[b] + N > P - 1) return 1;
    if (P > max_p) max_p = P;
  }
  double *row = (double *)malloc(sizeof(double) * (size_t)(max_p > 0 ? max_p : 1));
  if (!row) return 2;
  for (int b = 0; b < B; ++b) {
    const int N = cu_vis[b + 1] - cu_vis[b];
    double *s = w_out + cu_vis[b];
    for (int i = 0; i < N; ++i) s[i] = 0.0;
    for (int l = 0; l < L; ++l) {
      for (int h = 0; h < Hq; ++h) {
        int rc = oracle_last_row(B, L, Hq, Hkv, D, dtype, scale, cu_seqlens, q, k, b, l, h, row);
        if (rc) { free(row); return rc; }
        for (int i = 0; i < N; ++i) s[i] += row[vis_start[b] + i];
      }
    }
    double total = 0.0;
    for (int i = 0; i < N; ++i) total += s[i];
    for (int i = 0; i < N; ++i) s[i] = s[i] / total;
  }
  free(row);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Canonical fp32 dot product.  The coordinate set is cut into groups of     */
/* `vec` consecutive coordinates; group g belongs to lane (g mod lanes).     */
/* Each lane accumulates its groups in increasing order, coordinates inside  */
/* a group in increasing order, one fmaf per coordinate into one fp32        */
/* accumulator that starts at +0.  The lane sums are then combined by a      */
/* butterfly: at offsets lanes/2, ..., 2, 1 every lane adds its partner's     */
/* value (acc[l] + acc[l ^ o]); addition commutes, so all lanes end equal.   */
/* `lanes` must be a power of two <= 64.                                     */
/* ------------------------------------------------------------------------ */
static float dot_canonical(const float *a, const float *b, int n, int lanes, int vec) {
  float acc[64], nxt[64];
  for (int l = 0; l < lanes; ++l) acc[l] = 0.0f;
  const int stride = lanes * vec;
  for (int base = 0; base < n; base += stride)
    for (int l = 0; l < lanes; ++l)
      for (int e = 0; e < vec; ++e) {
        int c = base + l * vec + e;
        if (c < n) acc[l] = fmaf(a[c], b[c], acc[l]);
      }
  for (int o = lanes / 2; o >= 1; o /= 2) {
    for (int l = 0; l < lanes; ++l) nxt[l] = acc[l] + acc[l ^ o];
    for (int l = 0; l < lanes; ++l) acc[l] = nxt[l];
  }
  return acc[0];
}

float oracle_dot_canonical(const float *a, const float *b, int n, int lanes, int vec) {
  return dot_canonical(a, b, n, lanes, vec);
}

static int valid_lanes(int lanes) {
  return lanes >= 1 && lanes <= 64 && (lanes & (lanes - 1)) == 0;
}

/* ------------------------------------------------------------------------ */
/* Eq. 9-11, canonical fp32 arithmetic (the precision the selection kernel   */
/* decides in).  x: N rows of d elements (dtype), w: N fp32 weights.         */
/* Writes the selection sequence j_1..j_k (0-based) to order_out.            */
/*   r_i   = dot(x_i,x_i) > 0 ? 1/sqrtf(dot(x_i,x_i)) : 0                     */
/*   c     = (dot(x_i, x_j) * r_i) * r_j      (two fp32 roundings)           */
/*   delta = min(delta, 1 - c)                                               */
/*   p_i   = w_i * delta_i                                                   */
/* j_1 = argmax w; j_t = argmax over unselected of p; ties -> lowest index.   */
/* ------------------------------------------------------------------------ */
int oracle_select_fp32(int N, int d, int dtype, const void *x, const float *w, int k,
                       int lanes, int vec, int32_t *order_out) {
  if (N < 0 || d <= 0 || k < 0 || k > N || !valid_lanes(lanes) || vec <= 0) return 1;
  if (k == 0) return 0;
  float *xf = (float *)malloc(sizeof(float) * (size_t)N * (size_t)d);
  float *r = (float *)malloc(sizeof(float) * (size_t)N);
  float *delta = (float *)malloc(sizeof(float) * (size_t)N);
  unsigned char *in_s = (unsigned char *)calloc((size_t)N, 1);
  if (!xf || !r || !delta || !in_s) { free(xf); free(r); free(delta); free(in_s); return 2; }
  for (int64_t i = 0; i < (int64_t)N * d; ++i) xf[i] = load_elem_f(x, dtype, i);
  for (int i = 0; i < N; ++i) {
    const float *xi = xf + (int64_t)i * d;
    float ss = dot_canonical(xi, xi, d, lanes, vec);
    r[i] = ss > 0.0f ? 1.0f / sqrtf(ss) : 0.0f;
    delta[i] = INFINITY;
  }
  /* Eq. 9: seed with the most query-relevant token */
  int j = 0;
  for (int i = 1; i < N; ++i)
    if (w[i] > w[j]) j = i;
  order_out[0] = j;
  in_s[j] = 1;
  for (int t = 1; t < k; ++t) {
    /* Eq. 10, incrementally: fold the newest centre j into every delta */
    const float *xj = xf + (int64_t)j * d;
    for (int i = 0; i < N; ++i) {
      if (in_s[i]) continue;
      float dot = dot_canonical(xf + (int64_t)i * d, xj, d, lanes, vec);
      float c = (dot * r[i]) * r[j];
      float dist = 1.0f - c;
      delta[i] = fminf(delta[i], dist);
    }
    /* Eq. 11: the unselected token with the largest w_i * delta_i */
    int best = -1;
    float best_p = 0.0f;
    for (int i = 0; i < N; ++i) {
      if (in_s[i]) continue;
      float p = w[i] * delta[i];
      if (best < 0 || p > best_p) { best = i; best_p = p; }
    }
    j = best;
    order_out[t] = j;
    in_s[j] = 1;
  }
  free(xf); free(r); free(delta); free(in_s);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Eq. 9-11 in plain fp64: sequential dot, exact sqrt/div of doubles.        */
/* Checks the semantics; decisions agree with the fp32 mode except at        */
/* near-ties.                                                                */
/* ------------------------------------------------------------------------ */
int oracle_select_fp64(int N, int d, int dtype, const void *x, const double *w, int k,
                       int32_t *order_out) {
  if (N < 0 || d <= 0 || k < 0 || k > N) return 1;
  if (k == 0) return 0;
  double *xd = (double *)malloc(sizeof(double) * (size_t)N * (size_t)d);
  double *r = (double *)malloc(sizeof(double) * (size_t)N);
  double *delta = (double *)malloc(sizeof(double) * (size_t)N);
  unsigned char *in_s = (unsigned char *)calloc((size_t)N, 1);
  if (!xd || !r || !delta || !in_s) { free(xd); free(r); free(delta); free(in_s); return 2; }
  for (int64_t i = 0; i < (int64_t)N * d; ++i) xd[i] = load_elem(x, dtype, i);
  for (int i = 0; i < N; ++i) {
    double ss = 0.0;
    for (int c = 0; c < d; ++c) ss += xd[(int64_t)i * d + c] * xd[(int64_t)i * d + c];
    r[i] = ss > 0.0 ? 1.0 / sqrt(ss) : 0.0;
    delta[i] = INFINITY;
  }
  int j = 0;
  for (int i = 1; i < N; ++i)
    if (w[i] > w[j]) j = i;
  order_out[0] = j;
  in_s[j] = 1;
  for (int t = 1; t < k; ++t) {
    for (int i = 0; i < N; ++i) {
      if (in_s[i]) continue;
      double dot = 0.0;
      for (int c = 0; c < d; ++c) dot += xd[(int64_t)i * d + c] * xd[(int64_t)j * d + c];
      double dist = 1.0 - dot * r[i] * r[j];
      if (dist < delta[i]) delta[i] = dist;
    }
    int best = -1;
    double best_p = 0.0;
    for (int i = 0; i < N; ++i) {
      if (in_s[i]) continue;
      double p = w[i] * delta[i];
      if (best < 0 || p > best_p) { best = i; best_p = p; }
    }
    j = best;
    order_out[t] = j;
    in_s[j] = 1;
  }
  free(xd); free(r); free(delta); free(in_s);
  return 0;
}

/* Table 5 ("LAST (Top-k)"): keep the k tokens with the highest importance
 * score w~, with no diversity term.  Written as k repeated argmaxes over the
 * tokens not yet taken (ties to the lowest index, IEEE '>' so -0 == +0), which
 * is the greedy of Eq. 9-11 with every delta fixed at 1.  order_out receives
 * the selection order (descending score). */
int oracle_select_topk(int N, const float *w, int k, int32_t *order_out) {
  if (N < 0 || k < 0 || k > N) return 1;
  unsigned char *taken = (unsigned char *)calloc((size_t)N + 1, 1);
  if (!taken) return 2;
  for (int t = 0; t < k; ++t) {
    int best = -1;
    for (int i = 0; i < N; ++i) {
      if (taken[i]) continue;
      if (best < 0 || w[i] > w[best]) best = i;
    }
    order_out[t] = best;
    taken[best] = 1;
  }
  free(taken);
  return 0;
}

/* Table 4 (attention sources): the importance of Eq. 7 taken from the attention
 * rows of several query positions instead of p* alone.  Request b has the query
 * rows cu_rows[b] .. cu_rows[b+1]-1; row r sits at request-local position
 * row_pos[r], after the visual span (vis_start[b] + N_b <= row_pos[r] <= P_b - 1),
 * and its causal softmax runs over the keys 0 .. row_pos[r].  q holds one query
 * vector per row, layer and q-head: [cu_rows[B]][L][Hq][D].  The rows' probabilities
 * at the visual positions are summed over rows, layers and heads (a mean over the
 * rows is the same after Eq. 8's normalisation), then normalised. */
int oracle_scores_rows(int B, int L, int Hq, int Hkv, int D, int dtype, double scale,
                       const int32_t *cu_seqlens, const int32_t *vis_start, const int32_t *cu_vis,
                       const int32_t *cu_rows, const int32_t *row_pos, const void *q,
                       const void *k, double *w_out) {
  if (Hkv <= 0 || Hq % Hkv != 0 || cu_rows[0] != 0) return 1;
  if (scale <= 0.0) scale = 1.0 / sqrt((double)D);
  const int group = Hq / Hkv;
  const int64_t total_keys = cu_seqlens[B];
  int max_p = 1;
  for (int b = 0; b < B; ++b) {
    const int P = cu_seqlens[b + 1] - cu_seqlens[b];
    const int N = cu_vis[b + 1] - cu_vis[b];
    if (P <= 0 || N < 0 || vis_start[b] < 0) return 1;
    if (cu_rows[b + 1] <= cu_rows[b]) return 1;          /* at least one row */
    for (int r = cu_rows[b]; r < cu_rows[b + 1]; ++r)
      if (row_pos[r] < vis_start[b] + N || row_pos[r] > P - 1) return 1;
    if (P > max_p) max_p = P;
  }
  double *a = (double *)malloc(sizeof(double) * (size_t)max_p);
  if (!a) return 2;
  for (int b = 0; b < B; ++b) {
    const int N = cu_vis[b + 1] - cu_vis[b];
    const int64_t p0 = cu_seqlens[b];
    double *s = w_out + cu_vis[b];
    for (int i = 0; i < N; ++i) s[i] = 0.0;
    for (int r = cu_rows[b]; r < cu_rows[b + 1]; ++r) {
      const int pos = row_pos[r];
      for (int l = 0; l < L; ++l) {
        for (int h = 0; h < Hq; ++h) {
          const int g = h / group;
          const int64_t qoff = (((int64_t)r * L + l) * Hq + h) * D;
          /* Eq. 6 for this row: causal softmax over keys 0..pos */
          double zmax = -INFINITY;
          for (int p = 0; p <= pos; ++p) {
            const int64_t koff = (((int64_t)l * total_keys + p0 + p) * Hkv + g) * D;
            double acc = 0.0;
            for (int d = 0; d < D; ++d)
              acc += load_elem(q, dtype, qoff + d) * load_elem(k, dtype, koff + d);
            a[p] = scale * acc;
            if (a[p] > zmax) zmax = a[p];
          }
          double zsum = 0.0;
          for (int p = 0; p <= pos; ++p) {
            a[p] = exp(a[p] - zmax);
            zsum += a[p];
          }
          /* Eq. 7: accumulate the visual positions */
          for (int i = 0; i < N; ++i) s[i] += a[vis_start[b] + i] / zsum;
        }
      }
    }
    /* Eq. 8 */
    double total = 0.0;
    for (int i = 0; i < N; ++i) total += s[i];
    for (int i = 0; i < N; ++i) s[i] = s[i] / total;
  }
  free(a);
  return 0;
}

/* Eq. 12: sort(S) -- the selected indices in their original (ascending) order. */
void oracle_restore_order(int k, const int32_t *order, int32_t *idx_out) {
  for (int t = 0; t < k; ++t) idx_out[t] = order[t];
  for (int a = 1; a < k; ++a) { /* insertion sort */
    int32_t v = idx_out[a];
    int b = a - 1;
    while (b >= 0 && idx_out[b] > v) { idx_out[b + 1] = idx_out[b]; --b; }
    idx_out[b + 1] = v;
  }
}

/* Eq. 12: X_S[r] = x_{idx[r]}, a bitwise copy of each selected row. */
int oracle_gather(int N, int d, int elem_bytes, const void *x, int k, const int32_t *idx,
                  void *x_out) {
  const size_t row = (size_t)d * (size_t)elem_bytes;
  for (int r = 0; r < k; ++r) {
    if (idx[r] < 0 || idx[r] >= N) return 1;
    memcpy((char *)x_out + (size_t)r * row, (const char *)x + (size_t)idx[r] * row, row);
  }
  return 0;
}

/* Eq. 2: K = ceil(rho N) for rho = num/den, in exact integer arithmetic. */
int32_t oracle_budget(int32_t n, int32_t num, int32_t den) {
  if (n < 0 || num < 0 || den <= 0) return -1;
  int64_t prod = (int64_t)num * (int64_t)n;
  int64_t q = prod / den;
  if (q * den < prod) q += 1;
  return (int32_t)q;
}
