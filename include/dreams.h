/*
 * dreams.h -- C ABI of the GB300 (sm_103a) library for the target model's
 * tree verification step of DREAM-S speculative decoding for vision-language
 * models (arXiv 2606.00535).
 *
 * One verification step (paper Sec. 2, "Speculative decoding"): the target
 * model scores every draft token in one parallel pass, then accepts drafts in
 * order while they equal its own prediction, replacing the first mismatch by
 * its own token. Here the drafts form a tree (parent array), so the step is
 *
 *   1. dreams_tree_verify_attn  tree-masked attention of the T tree tokens
 *                               against the image-plus-text KV cache (Sec. 2,
 *                               "Vision-Language Models": every cached visual
 *                               and text token takes part in attention at each
 *                               decoding step), once per layer;
 *   2. dreams_vocab_argmax      the target's greedy prediction per tree node
 *                               (temperature 0, Table 2);
 *   3. dreams_accept_path       the longest root path whose drafts match, plus
 *                               the target's bonus token;
 *   4. dreams_kv_compact        the accepted nodes' K/V moved into contiguous
 *                               cache slots for the next step;
 *   5. dreams_verify_step       2 + 3 + 4 in one call (two launches).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All data pointers are DEVICE pointers owned by the caller; the library
 *    allocates no memory. Scratch comes from a caller-supplied workspace
 *    (16-byte aligned) whose size the matching *_workspace_size function
 *    returns. The attention workspace holds no state between calls. The
 *    argmax and verify-step workspaces hold counters that reset themselves:
 *    zero-fill such a workspace once when it is allocated, and every call
 *    leaves it zero-filled again, whatever its shape arguments. Calls that
 *    overlap in time must not share a workspace.
 *  - Every call is asynchronous on the given stream (NULL = the legacy
 *    default stream) and runs on the current CUDA device.
 *  - Host-side checks (null pointers, sizes, alignment, supported shapes)
 *    run before any launch. A failed check returns DREAMS_ERR_INVALID_ARG or
 *    DREAMS_ERR_UNSUPPORTED and launches nothing.
 *  - Malformed device data (a bad parent array, tree or cache length, page
 *    id or path) is never trapped: the kernels OR a DREAMS_DATA_* bit into
 *    *status_word (a device int32, may be NULL) and skip the affected
 *    sequence, whose outputs are then as documented per call.
 *  - A launch failure returns DREAMS_ERR_CUDA; dreams_last_cuda_error()
 *    gives the CUDA error code of the calling thread's last failure.
 *
 * Shapes (B sequences; T_max tree nodes per sequence including the root;
 * Hq query heads; Hkv KV heads with Hq % Hkv == 0; head dim D in {64, 128}):
 *  - tree node 0 is the root: the last committed token, whose K/V this pass
 *    has just written to cache slot kv_len[b]; node i sits in slot
 *    kv_len[b] + i. parent[b][0] = -1 and 0 <= parent[b][i] < i.
 */
#ifndef DREAMS_H_
#define DREAMS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DREAMS_VERSION 10000 /* 1.0.0 */

/* Same type as cudaStream_t. */
typedef struct CUstream_st *dreams_stream_t;

typedef enum dreams_status {
  DREAMS_OK = 0,
  DREAMS_ERR_INVALID_ARG = 1, /* null pointer, bad size, misaligned pointer */
  DREAMS_ERR_UNSUPPORTED = 2, /* valid but unsupported shape or dtype */
  DREAMS_ERR_WORKSPACE = 3,   /* workspace missing or too small */
  DREAMS_ERR_CUDA = 4,        /* a CUDA call failed; see dreams_last_cuda_error */
  DREAMS_ERR_SCRATCH_LIMIT = 5 /* larger than a no-allocation entry point's fixed scratch */
} dreams_status_t;

typedef enum dreams_dtype { DREAMS_F32 = 0, DREAMS_BF16 = 1 } dreams_dtype_t;

/* Bits OR-ed into *status_word by the kernels. */
#define DREAMS_DATA_BAD_PARENT 0x1   /* parent[0] != -1 or parent[i] outside [0, i) */
#define DREAMS_DATA_BAD_TREE_LEN 0x2 /* tree_len outside [1, T_max] */
#define DREAMS_DATA_BAD_KV_LEN 0x4   /* kv_len < 0 or kv_len + tree_len > capacity */
#define DREAMS_DATA_BAD_PAGE 0x8     /* page-table entry outside [0, num_pages) */
#define DREAMS_DATA_BAD_PATH 0x10    /* path[0] != 0 or not strictly increasing */
#define DREAMS_DATA_TIMEOUT 0x20     /* a kernel gave up waiting on its own pipeline (2 s) */

/*
 * One attention layer's K and V cache (bf16), or n_layers of them.
 *  - contiguous (page_table == NULL): element (b, s, g, d) at
 *        ((b * capacity + s) * Hkv + g) * D + d
 *  - paged: logical slot s of sequence b is row s % page_size of physical
 *    page p = page_table[b * pages_per_seq + s / page_size], and element
 *    (b, s, g, d) is at ((p * page_size + s % page_size) * Hkv + g) * D + d;
 *    capacity must equal pages_per_seq * page_size. Only page_size 64.
 *  - layer l's cache starts layer_stride elements after layer l-1's (k and v
 *    alike). k, v and layer_stride * 2 bytes must be 16-byte aligned.
 *  - The struct carries no batch size: a call that addresses sequences
 *    0 .. B-1 reads (and the compaction writes) their slots, so the caller's
 *    buffers must hold at least B sequences (contiguous: B * capacity slots
 *    per layer; paged: B rows of the page table). The Python binding checks
 *    this; the library cannot.
 */
typedef struct dreams_kv_cache {
  void *k;
  void *v;
  int32_t n_layers;
  int64_t layer_stride;
  int32_t Hkv;
  int32_t D;
  int32_t capacity;
  const int32_t *page_table;
  int32_t page_size;
  int32_t pages_per_seq;
  int32_t num_pages;
} dreams_kv_cache_t;

/* The draft trees of a batch (all device int32 arrays). */
typedef struct dreams_tree {
  const int32_t *parent;   /* [B, T_max] */
  const int32_t *tokens;   /* [B, T_max] draft token ids; tokens[b][0] is never checked */
  const int32_t *tree_len; /* [B] nodes in use, 1..T_max */
  const int32_t *kv_len;   /* [B] committed prefix length L_b */
  int32_t B;
  int32_t T_max; /* 1..64 */
} dreams_tree_t;

/*
 * Tree-masked verification attention for one layer (Sec. 2, "Speculative
 * decoding" and "Vision-Language Models"; attention = softmax(Q K^T * scale)
 * as in Sec. 3.2). For every sequence b, tree node t < tree_len[b] and query
 * head h, with KV head g = h / (Hq / Hkv):
 *     keys  J = { slots 0 .. L_b - 1 } U { slot L_b + a : a = t or an ancestor of t }
 *     out[b, t, h, :] = sum_{j in J} softmax_j(scale * <q, K[b, j, g]>) V[b, j, g, :]
 *     lse[b, t, h]    = log sum_{j in J} exp(scale * <q, K[b, j, g]>)
 * Hq must be a multiple of kv->Hkv with at most 128 query heads per KV head.
 * q: bf16, element (b, t, h, d) at q[b * q_stride_b + t * q_stride_t + h * D + d]:
 * each token's Hq head rows are dense, tokens and sequences are strided, so Q
 * may be a view into a fused QKV projection output (e.g. [B, T, 3, Hq, D]:
 * q_stride_t = 3 Hq D, q_stride_b = T_max q_stride_t). Both strides are in
 * elements, at least Hq * D, multiples of 8 (16 bytes) and below 2^38;
 * q_stride_b is ignored when B == 1. out: bf16 [B, T_max, Hq, D], dense.
 * q and out 16-byte aligned. lse: f32 [B, T_max, Hq] or NULL. Rows
 * t >= tree_len[b] of out and lse are left untouched, and so are all rows of a
 * sequence with bad data, and the rows a call that flags DREAMS_DATA_TIMEOUT
 * did not finish. layer selects the cache (0 <= layer < kv->n_layers). scale
 * must be finite and > 0. Accumulation is fp32 (the probabilities enter the
 * PV product as bf16); the output is rounded to bf16 once.
 */
size_t dreams_tree_verify_attn_workspace_size(const dreams_kv_cache_t *kv, const dreams_tree_t *tree,
                                              int32_t Hq);
/* Kernel launches one dreams_tree_verify_attn call with these shapes makes
 * (1 to 3: an ordering pass when more than 64 (sequence, KV split) pairs are
 * scheduled longest first (up to 64, every CTA ranks them itself), the
 * attention, a merge of the KV splits when the cache is split); 0 for shapes
 * the call rejects. */
int32_t dreams_tree_verify_attn_launches(const dreams_kv_cache_t *kv, const dreams_tree_t *tree, int32_t Hq);
dreams_status_t dreams_tree_verify_attn(const void *q, int64_t q_stride_b, int64_t q_stride_t,
                                        const dreams_kv_cache_t *kv, int32_t layer,
                                        const dreams_tree_t *tree, int32_t Hq, float scale, void *out,
                                        float *lse, void *workspace, size_t workspace_bytes,
                                        int32_t *status_word, dreams_stream_t stream);

/*
 * Attention without a tree: the draft's cross-attention to target features,
 * and the prefill self-attention of a target layer, optionally with each query
 * row's attention entropy.
 *   DREAMS_ATTN_FULL   query t of sequence b attends slots 0 .. kv_len[b] - 1:
 *                      the cross-attention through which the draft reads the
 *                      target's features S^l' (keys and values) with its own
 *                      intermediate features E^j as queries (Sec. 3.2,
 *                      "Adaptive Target Feature Injection");
 *   DREAMS_ATTN_CAUSAL query t attends slots 0 .. kv_len[b] + t: its own slot
 *                      is kv_len[b] + t (prefill of a layer, A = softmax(QK^T /
 *                      sqrt(z)) of Sec. 3.3).
 * q (strided as for dreams_tree_verify_attn), out: bf16 [B, T_max, Hq, D];
 * q_len[b] in [1, T_max] query rows are computed (T_max <= 2^20); kv as for
 * dreams_tree_verify_attn (FULL needs
 * kv_len >= 1, CAUSAL kv_len + q_len <= capacity). lse and entropy: f32
 * [B, T_max, Hq] or NULL. entropy[b][t][h] = -sum_j a_j ln a_j over the row's
 * attention weights a (nats); the average over rows and heads is AE(l) of
 * Sec. 3.3 (Adaptive Intermediate Feature Distillation). Accumulation as in
 * dreams_tree_verify_attn; the entropy adds one f32 sum per row.
 */
#define DREAMS_ATTN_FULL 1
#define DREAMS_ATTN_CAUSAL 2
size_t dreams_attention_workspace_size(const dreams_kv_cache_t *kv, int32_t B, int32_t T_max, int32_t Hq,
                                       int32_t mode, int32_t want_entropy);
dreams_status_t dreams_attention(const void *q, int64_t q_stride_b, int64_t q_stride_t, const dreams_kv_cache_t *kv,
                                 int32_t layer, const int32_t *q_len,
                                 const int32_t *kv_len, int32_t B, int32_t T_max, int32_t Hq, float scale,
                                 int32_t mode, void *out, float *lse, float *entropy, void *workspace,
                                 size_t workspace_bytes, int32_t *status_word, dreams_stream_t stream);

/*
 * Row-wise argmax (the target's greedy prediction, Sec. 2 "Speculative
 * decoding" at temperature 0): out_idx[r] = argmax_v logits[r * row_stride + v]
 * for v < V, under the total order "greater value wins, equal values (+0 ==
 * -0) go to the lower index, NaN is above every number and the first NaN
 * wins" -- the same result as torch.argmax. logits: f32 or bf16, rows x
 * row_stride elements; row_stride >= V. Rows that start 16-byte aligned are
 * read with 16-byte loads.
 */
size_t dreams_vocab_argmax_workspace_size(int64_t rows, int64_t V);
dreams_status_t dreams_vocab_argmax(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V,
                                    int64_t row_stride, int32_t *out_idx, void *workspace,
                                    size_t workspace_bytes, dreams_stream_t stream);

/*
 * Greedy acceptance over the draft tree (Sec. 2 "Speculative decoding",
 * generalised from a chain to a tree). argmax: [B, T_max] target predictions
 * (row b * T_max + i is node i of sequence b). A root path 0 -> c1 -> ... -> cn
 * matches when tokens[ck] == argmax[c(k-1)] for every k. The accepted path is
 * the longest matching root path, cut to at most max_path - 1 drafts, ties to
 * the lexicographically smallest node sequence. Outputs per sequence b:
 *     path[b]       = (0, c1, ..., cn, -1, ...)                  [B, max_path]
 *     out_tokens[b] = (tokens[c1], ..., tokens[cn], argmax[cn], -1, ...)
 *     accept_len[b] = n + 1 (drafts plus the bonus token)
 *     new_kv_len[b] = kv_len[b] + n + 1
 * A sequence with a bad tree or kv_len < 0 gets accept_len 0, new_kv_len =
 * kv_len and rows of -1. max_path >= 1.
 */
dreams_status_t dreams_accept_path(const int32_t *argmax, const dreams_tree_t *tree, int32_t max_path,
                                   int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                                   int32_t *new_kv_len, int32_t *status_word, dreams_stream_t stream);

/*
 * KV compaction (keeps the cache a plain sequence for the next step, Sec. 2
 * "Vision-Language Models"): for every sequence b with A = accept_len[b] > 0,
 * every layer, K and V and every KV head,
 *     slot L_b + x  <-  slot L_b + path[b][x]     for x = 0 .. A-1
 * as if all A source rows were read before any is written. All other bytes are
 * unchanged. path: [B, max_path], as returned by dreams_accept_path
 * (path[b][0] = 0, strictly increasing); a sequence whose path is not of that
 * form, or whose slots fall outside the capacity or on a bad page, is left
 * untouched and flagged. kv->Hkv, kv->D give the head shape.
 */
dreams_status_t dreams_kv_compact(const dreams_kv_cache_t *kv, int32_t B, const int32_t *kv_len,
                                  const int32_t *accept_len, const int32_t *path, int32_t max_path,
                                  int32_t *status_word, dreams_stream_t stream);

/*
 * The verification tail in one call: dreams_vocab_argmax over the rows of
 * tree nodes (row b * T_max + i for i < tree_len[b]; logits [B, T_max, V]
 * with row_stride), then dreams_accept_path, then dreams_kv_compact on all
 * kv->n_layers layers, with the semantics documented above. argmax_out
 * ([B, T_max], may be NULL) receives the predictions of the rows computed;
 * other rows are untouched. The call makes two kernel launches on the
 * stream: the argmax, then the walk and compaction (one CTA per sequence),
 * chained by programmatic dependent launch.
 */
size_t dreams_verify_step_workspace_size(const dreams_tree_t *tree, int64_t V);
dreams_status_t dreams_verify_step(const void *logits, dreams_dtype_t dtype, int64_t V,
                                   int64_t row_stride, const dreams_tree_t *tree,
                                   const dreams_kv_cache_t *kv, int32_t max_path, int32_t *argmax_out,
                                   int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                                   int32_t *new_kv_len, void *workspace, size_t workspace_bytes,
                                   int32_t *status_word, dreams_stream_t stream);

/*
 * Temperature sampling: one draw per row from softmax(x / temperature), the
 * target's own sample at temperature tau > 0 (Sec. 2 "Speculative decoding":
 * each draft token is checked against the output of the target's own
 * sampling; Table 2, Temperature = 1), by inverse transform with the row's
 * uniform u_r = uniforms[r]:
 *     M = max_v x_v,  w_v = exp((x_v - M) / tau),  Z = sum_v w_v
 *     out_idx[r] = min { v : w_0 + ... + w_v > u_r Z }
 * with u_r clamped to [0, 1] (NaN counts as 0); when no v qualifies (u_r = 1)
 * the last v with w_v > 0. Rows holding a NaN, with maximum +inf, or with
 * every value -inf take their argmax (the order of dreams_vocab_argmax).
 * logits: f32 or bf16, rows x row_stride elements, row_stride >= V.
 * uniforms: device f32 [rows] (the caller's random numbers). temperature:
 * finite, > 0, with log2(e) / temperature finite in f32. The weights are f32
 * (hardware exp2 of the scaled difference, subnormals flushed) summed in a
 * fixed order per row, so a draw can differ from the exact-arithmetic draw
 * only when u_r Z lies within rounding of a cumulative sum. Two launches,
 * chained by programmatic dependent launch: CTAs over (row, range of
 * 1024-value segments) store each segment's maximum and weight sum in the
 * workspace (8 bytes per 1024 values per row); then one warp per row finds
 * the segment and the value. The workspace holds no state between calls.
 */
size_t dreams_vocab_sample_workspace_size(int64_t rows, int64_t V);
dreams_status_t dreams_vocab_sample(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V,
                                    int64_t row_stride, float temperature, const float *uniforms,
                                    int32_t *out_idx, void *workspace, size_t workspace_bytes,
                                    dreams_stream_t stream);

/*
 * The verification tail at temperature tau > 0: the draw of
 * dreams_vocab_sample for the rows of tree nodes (row b * T_max + i for
 * i < tree_len[b], uniforms [B, T_max]) takes the place of the argmax, then
 * dreams_accept_path and dreams_kv_compact run as in dreams_verify_step: a
 * draft is accepted when it equals the target's draw at its parent, and the
 * draw at the last accepted node is the bonus token (Sec. 2 "Speculative
 * decoding"). sample_out ([B, T_max], may be NULL) receives the draws of the
 * rows computed. Three kernel launches, chained by programmatic dependent
 * launch: the two stages of the draws over the node rows, then the walk and
 * the compaction (one CTA per sequence). The workspace holds no state between
 * calls.
 */
size_t dreams_verify_step_sampled_workspace_size(const dreams_tree_t *tree, int64_t V);
dreams_status_t dreams_verify_step_sampled(const void *logits, dreams_dtype_t dtype, int64_t V,
                                           int64_t row_stride, const dreams_tree_t *tree,
                                           const dreams_kv_cache_t *kv, int32_t max_path, float temperature,
                                           const float *uniforms, int32_t *sample_out, int32_t *accept_len,
                                           int32_t *path, int32_t *out_tokens, int32_t *new_kv_len,
                                           void *workspace, size_t workspace_bytes, int32_t *status_word,
                                           dreams_stream_t stream);

/*
 * The verification tail at temperature tau > 0 by speculative sampling
 * (Leviathan et al., cited in Sec. 1; Table 2, Temperature = 1), over the
 * draft tree: the accepted tokens are distributed as the target's own samples
 * whatever the draft proposes. At node cur the target's distribution is
 * p = softmax(target[cur] / tau) and the draft's q = softmax(draft[cur] / tau),
 * the distribution the drafts of cur's children were drawn from. The walk
 * starts at the root with the residual r = p and tries cur's children in index
 * order: child c with draft token x is accepted when
 *     u_accept[b][c] < min(1, r(x) / q(x))        (q(x) = 0: accepted iff r(x) > 0)
 * and then becomes cur (r restarts as the target at c); a rejection replaces r
 * by max(0, r - q) / sum_v max(0, r - q) (kept when that sum is 0, r == q).
 * When no child is accepted, at a leaf, or once max_path - 1 drafts are
 * accepted, the bonus token is drawn from r by inverse transform with
 * u_resample[b][cur] (the smallest v whose cumulative weight exceeds u, u
 * clamped to [0, 1]; none: the last v of positive weight). accept_len, path,
 * out_tokens, new_kv_len and the KV compaction are as in dreams_verify_step.
 * target_logits, draft_logits: f32 or bf16, [B, T_max, V] with row_stride
 * (the same for both); only the rows of the nodes the walk visits are read
 * (the draft row only where children are tried). u_accept, u_resample:
 * device f32 [B, T_max] (the caller's random numbers). Logits must be finite
 * (with non-finite values the tokens drawn are unspecified but lie in
 * [0, V)). V <= 393216 (beyond 196608 the kernel needs clusters of 16 CTAs),
 * max_path <= 65. Arithmetic is f32 (hardware exp2 of the scaled
 * differences), so a decision can differ from the exact-arithmetic one only
 * when a uniform lies within rounding of its threshold. The kernel holds the
 * residual in closed form, r = max(0, p - s q) / P with P = sum_v max(0, p -
 * s q) (s = 0 at the node; a rejection sets s to s + P), which is the
 * recursion above. One launch, no workspace: a cluster of up to 16 CTAs per
 * sequence, each holding a slice of the visited node's rows in shared memory;
 * a rejection costs one sum over the slices, combined across the cluster in
 * distributed shared memory. The cluster then draws the bonus, writes the
 * outputs and moves the accepted K/V.
 */
dreams_status_t dreams_verify_step_speculative(const void *target_logits, const void *draft_logits,
                                               dreams_dtype_t dtype, int64_t V, int64_t row_stride,
                                               const dreams_tree_t *tree, const dreams_kv_cache_t *kv,
                                               int32_t max_path, float temperature, const float *u_accept,
                                               const float *u_resample, int32_t *accept_len, int32_t *path,
                                               int32_t *out_tokens, int32_t *new_kv_len, int32_t *status_word,
                                               dreams_stream_t stream);

/*
 * The LM head with its argmax fused: the target's greedy prediction per node
 * straight from its final hidden states (Sec. 2 "Speculative decoding" at
 * temperature 0), without writing the logits:
 *     logits[r][v] = sum_k hidden[r][k] * weight[v][k]     (f32 accumulation)
 *     out_idx[r]   = argmax_v logits[r][v]  (the order of dreams_vocab_argmax)
 *     out_max[r]   = logits[r][out_idx[r]]  (may be NULL)
 * hidden: bf16 [rows, hidden_dim] with row stride ld_hidden; weight: bf16
 * [V, hidden_dim] with row stride ld_weight (the usual [vocab, hidden] layout).
 * hidden_dim must be a multiple of 64, both strides multiples of 8 elements,
 * both pointers 16-byte aligned. The products of bf16 values are exact in
 * f32; the f32 sums run in the tensor cores' order, so a row whose two largest
 * logits lie within rounding of each other may get either index. Two launches:
 * a persistent tcgen05 GEMM (128 x 256 tiles, the argmax of each tile merged
 * into a 64-bit slot per row with atomicMax), then a small kernel that writes
 * the indices and resets the slots. The workspace holds the slots: zero-fill
 * it once when it is allocated; every call leaves it zero-filled. A wait that
 * times out inside the GEMM flags DREAMS_DATA_TIMEOUT in status_word (may be
 * NULL); the indices of such a call are then unreliable, except that rows no
 * tile reached are left untouched.
 */
size_t dreams_lm_head_argmax_workspace_size(int64_t rows);
dreams_status_t dreams_lm_head_argmax(const void *hidden, int64_t rows, int64_t hidden_dim, int64_t ld_hidden,
                                      const void *weight, int64_t V, int64_t ld_weight, int32_t *out_idx,
                                      float *out_max, void *workspace, size_t workspace_bytes,
                                      int32_t *status_word, dreams_stream_t stream);

/*
 * Visual-token importance and top-r selection (Sec. 3.2 "Visual Token
 * Compression", Eq. 2). attn: the target's final-layer prefill attention
 * weights, [B, H, Q, K] contiguous, f32 or bf16. The visual tokens are key
 * positions v0 .. v0 + n_vis - 1. For each sequence b:
 *     importance[b][j] = 1 / (H Q) * sum_h sum_i attn[b][h][i][v0 + j]
 *     keep[b][0..r)    = the positions v0 + j of the r largest importances
 *                        (equal values: the lower position first), in
 *                        increasing order
 * Sums are f32, in a fixed order (the result does not depend on scheduling).
 * 1 <= r <= n_vis <= 49152. Three launches: partial column sums over row
 * ranges (HBM-bound), their sum in a fixed tree, then one CTA per sequence
 * that selects. The workspace holds the partial sums and no state between
 * calls.
 */
size_t dreams_visual_importance_workspace_size(int64_t B, int64_t H, int64_t Q, int64_t n_vis);
dreams_status_t dreams_visual_importance(const void *attn, dreams_dtype_t dtype, int64_t B, int64_t H, int64_t Q,
                                         int64_t K, int64_t v0, int64_t n_vis, int32_t r, float *importance,
                                         int32_t *keep, void *workspace, size_t workspace_bytes,
                                         dreams_stream_t stream);

/*
 * Row-wise argmax for callers that cannot allocate device memory. The paper
 * has no counterpart to this call; it exists for integration. Some callers
 * cannot allocate, or cannot hand out a workspace, when the argmax runs: a
 * plugin inside an inference engine that owns and plans all device memory and
 * gives the plugin no way to ask for more at run time; a serving process that
 * reserves its whole memory budget at start-up and treats any later allocation
 * as an error; a latency-critical loop in which an allocation's implicit
 * synchronisation would stall other streams.
 *
 * Same result and arguments as dreams_vocab_argmax, without the workspace: the
 * scratch is a fixed device array inside this library (12 bytes per row for
 * DREAMS_NOALLOC_ARGMAX_MAX_ROWS rows, about 192 KiB), which every GPU that
 * loads the library holds until the process exits. The call allocates and
 * frees nothing; it clears the part of the scratch it uses with
 * cudaMemsetAsync on the given stream, then launches the argmax kernel.
 *  - rows > DREAMS_NOALLOC_ARGMAX_MAX_ROWS returns DREAMS_ERR_SCRATCH_LIMIT
 *    and launches nothing.
 *  - The first call on each device looks up the scratch's device address
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.
 *  - All calls share the one scratch array: calls that overlap on the GPU
 *    (different streams, or different host threads) race and may return
 *    wrong indices. Serialise them, e.g. on one stream.
 */
#define DREAMS_NOALLOC_ARGMAX_MAX_ROWS 16384
dreams_status_t dreams_vocab_argmax_noalloc(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V,
                                            int64_t row_stride, int32_t *out_idx, dreams_stream_t stream);

/*
 * Test hook for the bounded pipeline waits of the tcgen05 kernels; not for
 * production use. The paper has no counterpart: every wait of these kernels
 * on its own copy or MMA pipeline gives up after a limit instead of hanging
 * the GPU, and this hook lets a test make such a wait run out without any
 * fault. While stall_at >= 0, every later launch of the kernels selected by
 * `kernels` (DREAMS_TEST_ATTENTION: dreams_tree_verify_attn and
 * dreams_attention; DREAMS_TEST_LM_HEAD: dreams_lm_head_argmax) withholds the
 * TMA copies of each CTA from its stall_at-th K tile (attention) or k-block
 * (LM head, counted over the CTA's tiles) on, waiting instead on a barrier
 * that nothing arrives on, and every pipeline wait gives up after
 * wait_limit_ns (1 us .. 2 s) instead of 2 s. The kernels then flag
 * DREAMS_DATA_TIMEOUT, wait for the copies and MMAs they did issue, free
 * their tensor memory and exit; output rows they did not finish are left
 * untouched (attention), or unreliable (LM head; rows no tile reached are
 * untouched). stall_at < 0 restores normal operation (the other arguments
 * are then ignored). The setting is process-wide and read at launch, so a
 * CUDA graph keeps the setting it was captured with.
 */
#define DREAMS_TEST_ATTENTION 1
#define DREAMS_TEST_LM_HEAD 2
dreams_status_t dreams_test_set_stall(int32_t kernels, int32_t stall_at, int64_t wait_limit_ns);

const char *dreams_status_string(dreams_status_t status);
int32_t dreams_version(void);
int32_t dreams_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* DREAMS_H_ */
