/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the target model's tree
 * verification step in DREAM-S speculative decoding (arXiv 2606.00535).
 *
 * TEST INFRASTRUCTURE. Only the test suite, the package smoke check and the
 * benchmark's CPU-baseline leg may load or run this file. The CUDA library
 * never calls it, and this file includes nothing from the CUDA library: the
 * two implementations share no code, constants or helpers.
 *
 * Every routine is the plain definition written out as straight loops, in
 * double precision, single-threaded, without blocking, fusion or reordering:
 *
 *   - oracle_tree_attention : softmax(scale * q K^T) V over the prefix KV cache
 *                             plus the query node's own ancestors in the draft
 *                             tree (paper Sec. 2, "Speculative decoding": the
 *                             target evaluates all draft tokens in one pass;
 *                             Sec. 2, "Vision-Language Models": every cached
 *                             visual and text token takes part in attention at
 *                             every decoding step; Sec. 3.2 writes the
 *                             attention matrix as softmax(Q K^T / sqrt(z))).
 *   - oracle_argmax_*       : the target's own greedy prediction per node,
 *                             temperature 0 (Sec. 2 "Speculative decoding";
 *                             Table 2, Temperature = 0), a linear scan.
 *   - oracle_sample_*       : the target's own sample per node at temperature
 *                             tau > 0 (Sec. 2 "Speculative decoding": each
 *                             draft token is checked against the output of the
 *                             target's own sampling; Table 2, Temperature = 1),
 *                             by inverse transform of softmax(x / tau).
 *   - oracle_accept_path    : sequential acceptance -- drafts are accepted in
 *                             order while they equal the target's prediction,
 *                             and the target's own token replaces the first
 *                             mismatch (Sec. 2 "Speculative decoding"),
 *                             generalised from a chain to the longest matching
 *                             root path of a draft tree.
 *   - oracle_spec_path_*    : speculative sampling over the draft tree
 *                             (Leviathan et al., cited in Sec. 1): each draft
 *                             is accepted with probability min(1, p / q),
 *                             and a rejection moves the target to the
 *                             renormalised residual max(0, p - q) from which
 *                             the bonus token is drawn (Table 2, T = 1).
 *   - oracle_kv_compact     : the accepted nodes' K/V are moved into the
 *                             contiguous slots that follow the prefix, so the
 *                             cache stays a plain sequence for the next step
 *                             (Sec. 2 "Vision-Language Models": the cache
 *                             persists across decoding steps).
 *
 * Readings of points the paper leaves open (the paper describes chains only):
 *   - a draft tree is a parent array with parent[0] = -1 and
 *     0 <= parent[i] < i for i >= 1; node 0 is the root, i.e. the last
 *     committed token, whose K/V are computed in this pass and sit in slot L;
 *     tree node i sits in cache slot L + i;
 *   - the attention scale is passed in (1/sqrt(head_dim) in practice);
 *   - argmax ties go to the lowest index, +0 equals -0, NaN is greater than
 *     every number and the first NaN wins;
 *   - the accepted path is the longest root path whose drafts all match the
 *     target's prediction at their parents; among equally long matching
 *     paths the lexicographically smallest node sequence wins (with distinct
 *     sibling tokens the matching path is unique); the root's own token is
 *     never checked; the accepted length counts the bonus (target) token;
 *   - at most max_path - 1 drafts are accepted (path and out_tokens rows hold
 *     max_path entries); entries past the accepted length are set to -1;
 *   - at temperature tau > 0 the target's own output at a node is one draw
 *     from softmax(x / tau), taken by inverse transform with a uniform u that
 *     the caller passes in: the smallest v whose cumulative weight exceeds
 *     u times the total; acceptance then compares drafts with these draws
 *     exactly as with the argmax at temperature 0.
 *
 * bf16 values are handled as their raw 16-bit patterns; widening bf16 to
 * double is exact.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Per-sequence data-error bits (the same meanings as the library's status
 * word; defined here independently from the written specification). */
#define ORACLE_BAD_PARENT 0x1
#define ORACLE_BAD_TREE_LEN 0x2
#define ORACLE_BAD_KV_LEN 0x4
#define ORACLE_BAD_PAGE 0x8
#define ORACLE_BAD_PATH 0x10

static double bf16_bits_to_double(uint16_t h) {
  uint32_t u = ((uint32_t)h) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* Description of one layer's K or V cache.
 *   contiguous (page_table == NULL): element [b][s][g][d] at
 *       ((b * capacity + s) * Hkv + g) * D + d
 *   paged: logical slot s of sequence b lives in physical page
 *       p = page_table[b * pages_per_seq + s / page_size], row s % page_size,
 *       element at ((p * page_size + s % page_size) * Hkv + g) * D + d
 */
typedef struct {
  int64_t capacity;
  const int32_t *page_table;
  int64_t page_size;
  int64_t pages_per_seq;
  int64_t num_pages;
  int64_t Hkv;
  int64_t D;
} oracle_kv_layout;

/* Element offset of (b, s, g, 0); -1 if the page id is out of range. */
static int64_t kv_row_offset(const oracle_kv_layout *L, int64_t b, int64_t s, int64_t g) {
  if (L->page_table == NULL) {
    return ((b * L->capacity + s) * L->Hkv + g) * L->D;
  }
  int64_t p = L->page_table[b * L->pages_per_seq + s / L->page_size];
  if (p < 0 || p >= L->num_pages) return -1;
  return ((p * L->page_size + s % L->page_size) * L->Hkv + g) * L->D;
}

/* Checks the tree of one sequence: tree_len in [1, T_max], parent[0] == -1,
 * 0 <= parent[i] < i. Returns 0 or data-error bits. */
static int check_tree(const int32_t *parent_row, int32_t tree_len, int32_t T_max) {
  if (tree_len < 1 || tree_len > T_max) return ORACLE_BAD_TREE_LEN;
  if (parent_row[0] != -1) return ORACLE_BAD_PARENT;
  for (int32_t i = 1; i < tree_len; ++i) {
    if (parent_row[i] < 0 || parent_row[i] >= i) return ORACLE_BAD_PARENT;
  }
  return 0;
}

/*
 * oracle_ancestor_mask: mask[i * T + a] = 1 iff node a is node i or one of
 * its ancestors, found by following parent links from i to the root.
 * Returns 0, or data-error bits for a malformed tree.
 */
int oracle_ancestor_mask(const int32_t *parent, int32_t T, uint8_t *mask) {
  int bad = check_tree(parent, T, T);
  if (bad) return bad;
  memset(mask, 0, (size_t)T * (size_t)T);
  for (int32_t i = 0; i < T; ++i) {
    int32_t a = i;
    while (a >= 0) {
      mask[(int64_t)i * T + a] = 1;
      a = parent[a];
    }
  }
  return 0;
}

/*
 * oracle_tree_attention: for each selected (b, t, h) triple, with
 * G = Hq / Hkv and KV head g = h / G, the query row q = Q[b, t, h, :] attends
 * to the key set
 *     J = { prefix slots 0 .. L_b - 1 } U { slot L_b + a : a in anc*(t) },
 * where anc*(t) is t and all its ancestors, and
 *     s_j = scale * sum_d q[d] K[b, j, g, d]
 *     m   = max_j s_j,  w_j = exp(s_j - m),  den = sum_j w_j
 *     out = sum_j w_j V[b, j, g, :] / den,   lse = m + log(den).
 *
 * q: bf16 bits [B, T_max, Hq, D]; k, v: bf16 bits of one layer cache (layout
 * above); sel: n_sel triples (b, t, h); out: [n_sel, D]; lse: [n_sel].
 * Returns the OR of data-error bits met; a triple of a bad sequence or with
 * t >= tree_len[b] gets NaN outputs.
 */
int oracle_tree_attention(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                          int64_t capacity, const int32_t *page_table, int64_t page_size,
                          int64_t pages_per_seq, int64_t num_pages, const int32_t *parent,
                          const int32_t *tree_len, const int32_t *kv_len, int64_t B,
                          int64_t T_max, int64_t Hq, int64_t Hkv, int64_t D, double scale,
                          const int32_t *sel, int64_t n_sel, double *out, double *lse) {
  oracle_kv_layout lay = {capacity, page_table, page_size, pages_per_seq, num_pages, Hkv, D};
  int64_t G = Hq / Hkv;
  int status = 0;
  int64_t max_keys = capacity;
  double *s = (double *)malloc(sizeof(double) * (size_t)(max_keys > 0 ? max_keys : 1));
  int64_t *kv_off = (int64_t *)malloc(sizeof(int64_t) * (size_t)(max_keys > 0 ? max_keys : 1));
  int32_t *anc = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T_max > 0 ? T_max : 1));

  for (int64_t n = 0; n < n_sel; ++n) {
    int64_t b = sel[3 * n], t = sel[3 * n + 1], h = sel[3 * n + 2];
    double *o = out + n * D;
    for (int64_t d = 0; d < D; ++d) o[d] = NAN;
    lse[n] = NAN;

    const int32_t *par = parent + b * T_max;
    int64_t L = kv_len[b], T = tree_len[b];
    int bad = check_tree(par, tree_len[b], (int32_t)T_max);
    if (!bad && (L < 0 || L + T > capacity)) bad = ORACLE_BAD_KV_LEN;
    if (bad) {
      status |= bad;
      continue;
    }
    if (t >= T) continue;

    /* Key set J: the whole prefix, then the ancestors of t (root first). */
    int64_t n_anc = 0;
    for (int32_t a = (int32_t)t; a >= 0; a = par[a]) anc[n_anc++] = a;
    int64_t nk = 0;
    for (int64_t j = 0; j < L; ++j) kv_off[nk++] = kv_row_offset(&lay, b, j, h / G);
    for (int64_t x = n_anc - 1; x >= 0; --x) kv_off[nk++] = kv_row_offset(&lay, b, L + anc[x], h / G);
    int page_bad = 0;
    for (int64_t j = 0; j < nk; ++j)
      if (kv_off[j] < 0) page_bad = 1;
    if (page_bad) {
      status |= ORACLE_BAD_PAGE;
      continue;
    }

    const uint16_t *qrow = q + ((b * T_max + t) * Hq + h) * D;
    double m = -INFINITY;
    for (int64_t j = 0; j < nk; ++j) {
      double acc = 0.0;
      for (int64_t d = 0; d < D; ++d)
        acc += bf16_bits_to_double(qrow[d]) * bf16_bits_to_double(k[kv_off[j] + d]);
      s[j] = scale * acc;
      if (s[j] > m) m = s[j];
    }
    double den = 0.0;
    for (int64_t j = 0; j < nk; ++j) {
      s[j] = exp(s[j] - m); /* s now holds the unnormalised weight w_j */
      den += s[j];
    }
    for (int64_t d = 0; d < D; ++d) {
      double acc = 0.0;
      for (int64_t j = 0; j < nk; ++j) acc += s[j] * bf16_bits_to_double(v[kv_off[j] + d]);
      o[d] = acc / den;
    }
    lse[n] = m + log(den);
  }
  free(s);
  free(kv_off);
  free(anc);
  return status;
}

/* The total order of the argmax: is a (at a later index) strictly better than
 * the current best b? NaN beats every number; among equals (+0 == -0) and
 * among NaNs the earlier index stays. */
static int argmax_better(double a, double b) {
  if (isnan(b)) return 0;
  if (isnan(a)) return 1;
  return a > b;
}

/* oracle_argmax_f32: out[r] = index of the greatest logits[r * row_stride + v]
 * over v = 0 .. V-1, by a linear scan in increasing v. */
void oracle_argmax_f32(const float *logits, int64_t rows, int64_t V, int64_t row_stride,
                       int32_t *out) {
  for (int64_t r = 0; r < rows; ++r) {
    const float *x = logits + r * row_stride;
    int64_t best = 0;
    for (int64_t i = 1; i < V; ++i)
      if (argmax_better((double)x[i], (double)x[best])) best = i;
    out[r] = (int32_t)best;
  }
}

/* oracle_argmax_bf16: the same scan over bf16 bit patterns widened to double. */
void oracle_argmax_bf16(const uint16_t *logits, int64_t rows, int64_t V, int64_t row_stride,
                        int32_t *out) {
  for (int64_t r = 0; r < rows; ++r) {
    const uint16_t *x = logits + r * row_stride;
    int64_t best = 0;
    for (int64_t i = 1; i < V; ++i)
      if (argmax_better(bf16_bits_to_double(x[i]), bf16_bits_to_double(x[best]))) best = i;
    out[r] = (int32_t)best;
  }
}

/* One draw from softmax(x / tau) by inverse transform (x has V values):
 *   M = max_v x_v,  w_v = exp((x_v - M) / tau),  Z = sum_v w_v,
 *   draw = min { v : w_0 + ... + w_v > u * Z },
 * with u clamped to [0, 1] (NaN counts as 0); when no v qualifies (u = 1), the
 * last v with w_v > 0. A row holding a NaN, with maximum +inf, or with every
 * value -inf has no such distribution: its draw is its argmax (the first NaN,
 * else the first +inf, else index 0). */
static int64_t sample_row(const double *x, int64_t V, double tau, double u) {
  int64_t best = 0;
  for (int64_t i = 1; i < V; ++i)
    if (argmax_better(x[i], x[best])) best = i;
  const double M = x[best];
  if (isnan(M) || isinf(M)) return best;
  if (!(u > 0.0)) u = 0.0;
  if (u > 1.0) u = 1.0;
  double Z = 0.0;
  for (int64_t v = 0; v < V; ++v) Z += exp((x[v] - M) / tau);
  const double target = u * Z;
  double cum = 0.0;
  int64_t last_pos = best;
  for (int64_t v = 0; v < V; ++v) {
    const double w = exp((x[v] - M) / tau);
    cum += w;
    if (w > 0.0) last_pos = v;
    if (cum > target) return v;
  }
  return last_pos;
}

/* oracle_sample_f32: out[r] = one draw from softmax(logits[r, 0 .. V-1] / tau)
 * with the uniform u[r] (see sample_row). */
void oracle_sample_f32(const float *logits, int64_t rows, int64_t V, int64_t row_stride, double tau,
                       const float *u, int32_t *out) {
  double *x = (double *)malloc((size_t)V * sizeof(double));
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t v = 0; v < V; ++v) x[v] = (double)logits[r * row_stride + v];
    out[r] = (int32_t)sample_row(x, V, tau, (double)u[r]);
  }
  free(x);
}

/* oracle_sample_bf16: the same over bf16 bit patterns widened to double. */
void oracle_sample_bf16(const uint16_t *logits, int64_t rows, int64_t V, int64_t row_stride, double tau,
                        const float *u, int32_t *out) {
  double *x = (double *)malloc((size_t)V * sizeof(double));
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t v = 0; v < V; ++v) x[v] = bf16_bits_to_double(logits[r * row_stride + v]);
    out[r] = (int32_t)sample_row(x, V, tau, (double)u[r]);
  }
  free(x);
}

/* Depth of node c (edges from the root); the tree is already checked. */
static int32_t node_depth(const int32_t *par, int32_t c) {
  int32_t d = 0;
  for (; c > 0; c = par[c]) ++d;
  return d;
}

/* Does every draft node x on the root path of c carry the target's
 * prediction at its parent, tokens[x] == am[parent[x]]? */
static int path_matches(const int32_t *par, const int32_t *tok, const int32_t *pred, int32_t c) {
  for (; c > 0; c = par[c])
    if (tok[c] != pred[par[c]]) return 0;
  return 1;
}

/* Writes the root path of c (root first) into out; returns its length. */
static int32_t root_path(const int32_t *par, int32_t c, int32_t *out) {
  int32_t n = node_depth(par, c) + 1;
  for (int32_t k = n - 1; k >= 0; --k, c = par[c]) out[k] = c;
  return n;
}

/*
 * oracle_accept_path: greedy (temperature-0) acceptance over a draft tree,
 * per sequence b. A root path 0 -> c1 -> ... -> cn matches when every draft
 * on it equals the target's prediction at its parent, tokens[ck] ==
 * am[c(k-1)] -- on a chain this is "accept t_1 .. t_(i-1), stop at the first
 * mismatch". The accepted path is the longest matching root path, cut to at
 * most max_path - 1 drafts; among matching paths of that length the
 * lexicographically smallest node sequence wins. With n drafts accepted and
 * last node c_n:
 *     path       = (0, c1, ..., cn)
 *     out_tokens = (tokens[c1], ..., tokens[cn], am[cn])   (bonus token last)
 *     accept_len = n + 1,  new_kv_len = kv_len + n + 1
 * am: [B, T_max]; path, out_tokens: [B, max_path], entries past accept_len
 * are -1. A sequence with a malformed tree or kv_len < 0 gets accept_len 0,
 * new_kv_len = kv_len and rows of -1; its error bits are OR-ed into the
 * return value.
 */
int oracle_accept_path(const int32_t *am, const int32_t *parent, const int32_t *tokens,
                       const int32_t *tree_len, const int32_t *kv_len, int64_t B, int64_t T_max,
                       int64_t max_path, int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                       int32_t *new_kv_len) {
  int status = 0;
  int32_t *best = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T_max + 1));
  int32_t *cand = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T_max + 1));
  for (int64_t b = 0; b < B; ++b) {
    const int32_t *par = parent + b * T_max;
    const int32_t *tok = tokens + b * T_max;
    const int32_t *pred = am + b * T_max;
    int32_t *pb = path + b * max_path;
    int32_t *ob = out_tokens + b * max_path;
    for (int64_t k = 0; k < max_path; ++k) pb[k] = ob[k] = -1;
    int bad = check_tree(par, tree_len[b], (int32_t)T_max);
    if (!bad && kv_len[b] < 0) bad = ORACLE_BAD_KV_LEN;
    if (bad || max_path < 1) {
      status |= bad;
      accept_len[b] = 0;
      new_kv_len[b] = kv_len[b];
      continue;
    }
    int32_t T = tree_len[b];
    /* longest matching root path, capped at max_path - 1 drafts */
    int32_t n = 0;
    for (int32_t c = 1; c < T; ++c) {
      if (path_matches(par, tok, pred, c)) {
        int32_t d = node_depth(par, c);
        if (d > n) n = d;
      }
    }
    if (n > max_path - 1) n = (int32_t)(max_path - 1);
    /* lexicographically smallest matching root path with n drafts: among the
     * nodes c whose whole root path matches and has depth >= n, compare the
     * first n + 1 nodes of their root paths */
    int32_t have = 0;
    best[0] = 0;
    for (int32_t c = 1; c < T && n > 0; ++c) {
      if (!path_matches(par, tok, pred, c) || node_depth(par, c) < n) continue;
      root_path(par, c, cand);
      int less = !have;
      for (int32_t k = 0; k <= n && !less; ++k) {
        if (cand[k] != best[k]) {
          less = cand[k] < best[k];
          break;
        }
      }
      if (less) {
        memcpy(best, cand, sizeof(int32_t) * (size_t)(n + 1));
        have = 1;
      }
    }
    for (int32_t k = 0; k <= n; ++k) pb[k] = best[k];
    for (int32_t k = 1; k <= n; ++k) ob[k - 1] = tok[best[k]];
    ob[n] = pred[best[n]];
    accept_len[b] = n + 1;
    new_kv_len[b] = kv_len[b] + n + 1;
  }
  free(best);
  free(cand);
  return status;
}

/* Target or draft distribution of a row: w_v = exp((x_v - M) / tau) / Z. */
static void row_softmax(const double *x, int64_t V, double tau, double *w) {
  double M = -INFINITY;
  for (int64_t v = 0; v < V; ++v)
    if (x[v] > M) M = x[v];
  double Z = 0.0;
  for (int64_t v = 0; v < V; ++v) {
    w[v] = exp((x[v] - M) / tau);
    Z += w[v];
  }
  for (int64_t v = 0; v < V; ++v) w[v] /= Z;
}

/* Inverse-transform draw from a distribution w (sums to 1 up to rounding):
 * the smallest v with w_0 + ... + w_v > u, u clamped to [0, 1] (NaN counts as
 * 0); none (u = 1): the last v with w_v > 0. *margin gets min(its current
 * value, the distance of u from the nearest cumulative sum). */
static int64_t draw_dist(const double *w, int64_t V, double u, double *margin) {
  if (!(u > 0.0)) u = 0.0;
  if (u > 1.0) u = 1.0;
  double cum = 0.0;
  int64_t last = 0;
  for (int64_t v = 0; v < V; ++v) {
    const double before = cum;
    cum += w[v];
    if (w[v] > 0.0) last = v;
    if (cum > u) {
      const double d = fmin(u - before, cum - u);
      if (d < *margin) *margin = d;
      return v;
    }
  }
  return last;
}

/*
 * Speculative sampling over a draft tree (Leviathan et al., cited in Sec. 1;
 * the verification at temperature 1 of Table 2), walked from the root: at
 * node cur the target's distribution is p = softmax(target[cur] / tau) and
 * the draft's is q = softmax(draft[cur] / tau), the distribution the drafts
 * of cur's children were drawn from. The children are tried in index order,
 * with the residual r = p at first: child c with draft token x is accepted
 * when u_acc[c] < min(1, r(x) / q(x)) (q(x) = 0: accepted when r(x) > 0);
 * a rejection replaces r by max(0, r - q) / sum max(0, r - q) (kept as it is
 * when that sum is 0, i.e. r == q). An accepted child becomes cur. When no
 * child is accepted, at a leaf, or once max_path - 1 drafts are accepted,
 * the bonus token is drawn from r (p at a leaf or at the cut) by inverse
 * transform with u_res[cur], and the walk stops. Outputs as
 * oracle_accept_path: path, out_tokens (accepted drafts then the bonus),
 * accept_len = n + 1, new_kv_len = kv_len + n + 1; a malformed tree or
 * kv_len < 0 gets accept_len 0 and rows of -1. margin[b] (may be NULL): the
 * smallest distance of a uniform from the threshold it was compared with
 * (|u_acc - min(1, r/q)| per tested child, the distance to the nearest
 * cumulative sum for the draw), so a test can tell which decisions a
 * rounding difference could flip. target / draft: B * T_max rows of V values
 * (row b * T_max + i is node i of sequence b), row_stride apart; the draft
 * rows of leaves are not read.
 */
static int spec_path(const void *target, const void *draft, int bf16, int64_t V, int64_t row_stride,
                     const int32_t *parent, const int32_t *tokens, const int32_t *tree_len, const int32_t *kv_len,
                     int64_t B, int64_t T_max, int64_t max_path, double tau, const float *u_acc,
                     const float *u_res, int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                     int32_t *new_kv_len, double *margin) {
  int status = 0;
  double *x = (double *)malloc((size_t)V * sizeof(double));
  double *p = (double *)malloc((size_t)V * sizeof(double));
  double *q = (double *)malloc((size_t)V * sizeof(double));
  for (int64_t b = 0; b < B; ++b) {
    const int32_t *par = parent + b * T_max;
    const int32_t *tok = tokens + b * T_max;
    int32_t *pb = path + b * max_path;
    int32_t *ob = out_tokens + b * max_path;
    double mg = INFINITY;
    for (int64_t k = 0; k < max_path; ++k) pb[k] = ob[k] = -1;
    int bad = check_tree(par, tree_len[b], (int32_t)T_max);
    if (!bad && kv_len[b] < 0) bad = ORACLE_BAD_KV_LEN;
    if (bad || max_path < 1) {
      status |= bad;
      accept_len[b] = 0;
      new_kv_len[b] = kv_len[b];
      if (margin) margin[b] = mg;
      continue;
    }
    const int32_t T = tree_len[b];
    int32_t cur = 0, n = 0;
    pb[0] = 0;
    for (;;) {
      const int64_t row = b * T_max + cur;
      for (int64_t v = 0; v < V; ++v)
        x[v] = bf16 ? bf16_bits_to_double(((const uint16_t *)target)[row * row_stride + v])
                    : (double)((const float *)target)[row * row_stride + v];
      row_softmax(x, V, tau, p); /* p now holds the residual r, which starts as the target */
      int32_t next = -1;
      if (n < max_path - 1) {
        int have_q = 0;
        for (int32_t c = cur + 1; c < T && next < 0; ++c) {
          if (par[c] != cur) continue;
          if (!have_q) {
            for (int64_t v = 0; v < V; ++v)
              x[v] = bf16 ? bf16_bits_to_double(((const uint16_t *)draft)[row * row_stride + v])
                          : (double)((const float *)draft)[row * row_stride + v];
            row_softmax(x, V, tau, q);
            have_q = 1;
          }
          const int32_t t = tok[c];
          const double r_t = (t >= 0 && t < V) ? p[t] : 0.0;
          const double q_t = (t >= 0 && t < V) ? q[t] : 0.0;
          const double a = q_t > 0.0 ? fmin(1.0, r_t / q_t) : (r_t > 0.0 ? 1.0 : 0.0);
          const double u = (double)u_acc[b * T_max + c];
          if (fabs(u - a) < mg) mg = fabs(u - a);
          if (u < a) {
            next = c;
          } else {
            double Z = 0.0;
            for (int64_t v = 0; v < V; ++v) Z += fmax(0.0, p[v] - q[v]);
            if (Z > 0.0)
              for (int64_t v = 0; v < V; ++v) p[v] = fmax(0.0, p[v] - q[v]) / Z;
          }
        }
      }
      if (next < 0) {
        const int64_t bonus = draw_dist(p, V, (double)u_res[b * T_max + cur], &mg);
        ob[n] = (int32_t)bonus;
        break;
      }
      ++n;
      pb[n] = next;
      ob[n - 1] = tok[next];
      cur = next;
    }
    accept_len[b] = n + 1;
    new_kv_len[b] = kv_len[b] + n + 1;
    if (margin) margin[b] = mg;
  }
  free(x);
  free(p);
  free(q);
  return status;
}

int oracle_spec_path_f32(const float *target, const float *draft, int64_t V, int64_t row_stride,
                         const int32_t *parent, const int32_t *tokens, const int32_t *tree_len,
                         const int32_t *kv_len, int64_t B, int64_t T_max, int64_t max_path, double tau,
                         const float *u_acc, const float *u_res, int32_t *accept_len, int32_t *path,
                         int32_t *out_tokens, int32_t *new_kv_len, double *margin) {
  return spec_path(target, draft, 0, V, row_stride, parent, tokens, tree_len, kv_len, B, T_max, max_path, tau,
                   u_acc, u_res, accept_len, path, out_tokens, new_kv_len, margin);
}

int oracle_spec_path_bf16(const uint16_t *target, const uint16_t *draft, int64_t V, int64_t row_stride,
                          const int32_t *parent, const int32_t *tokens, const int32_t *tree_len,
                          const int32_t *kv_len, int64_t B, int64_t T_max, int64_t max_path, double tau,
                          const float *u_acc, const float *u_res, int32_t *accept_len, int32_t *path,
                          int32_t *out_tokens, int32_t *new_kv_len, double *margin) {
  return spec_path(target, draft, 1, V, row_stride, parent, tokens, tree_len, kv_len, B, T_max, max_path, tau,
                   u_acc, u_res, accept_len, path, out_tokens, new_kv_len, margin);
}

/*
 * oracle_kv_compact: for each sequence b with accept_len[b] = A > 0 and each
 * layer, KV head and of K and V:
 *     tmp[x] = cache[b, L_b + path[b][x]]   for x = 0 .. A-1   (all reads)
 *     cache[b, L_b + x] = tmp[x]            for x = 0 .. A-1   (then writes)
 * Every other slot keeps its bytes. k, v: bf16 bits, n_layers caches each
 * layer_stride elements apart. A path is what the acceptance walk returns:
 * path[0] = 0 and strictly increasing. Returns data-error bits (a path that
 * is not of that form, slots beyond the capacity, bad page ids); such a
 * sequence is left untouched.
 */
int oracle_kv_compact(uint16_t *k, uint16_t *v, int64_t n_layers, int64_t layer_stride,
                      int64_t capacity, const int32_t *page_table, int64_t page_size,
                      int64_t pages_per_seq, int64_t num_pages, int64_t Hkv, int64_t D, int64_t B,
                      const int32_t *kv_len, const int32_t *accept_len, const int32_t *path,
                      int64_t max_path) {
  oracle_kv_layout lay = {capacity, page_table, page_size, pages_per_seq, num_pages, Hkv, D};
  int status = 0;
  uint16_t *tmp = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)(max_path * D + 1));
  for (int64_t b = 0; b < B; ++b) {
    int64_t A = accept_len[b], L = kv_len[b];
    if (A <= 0) continue;
    int bad = 0;
    if (A > max_path || L < 0) bad = ORACLE_BAD_KV_LEN;
    if (!bad && path[b * max_path] != 0) bad = ORACLE_BAD_PATH;
    for (int64_t x = 1; !bad && x < A; ++x)
      if (path[b * max_path + x] <= path[b * max_path + x - 1]) bad = ORACLE_BAD_PATH;
    for (int64_t x = 0; !bad && x < A; ++x) {
      int64_t src = path[b * max_path + x];
      if (L + src >= capacity || L + x >= capacity) bad = ORACLE_BAD_KV_LEN;
      else if (kv_row_offset(&lay, b, L + src, 0) < 0 || kv_row_offset(&lay, b, L + x, 0) < 0)
        bad = ORACLE_BAD_PAGE;
    }
    if (bad) {
      status |= bad;
      continue;
    }
    for (int64_t layer = 0; layer < n_layers; ++layer) {
      for (int which = 0; which < 2; ++which) {
        uint16_t *cache = (which == 0 ? k : v) + layer * layer_stride;
        for (int64_t g = 0; g < Hkv; ++g) {
          for (int64_t x = 0; x < A; ++x) {
            int64_t off = kv_row_offset(&lay, b, L + path[b * max_path + x], g);
            memcpy(tmp + x * D, cache + off, sizeof(uint16_t) * (size_t)D);
          }
          for (int64_t x = 0; x < A; ++x) {
            int64_t off = kv_row_offset(&lay, b, L + x, g);
            memcpy(cache + off, tmp + x * D, sizeof(uint16_t) * (size_t)D);
          }
        }
      }
    }
  }
  free(tmp);
  return status;
}
