/*
 * libsdsat -- the SDSAT block decode step on one GB300 (sm_103a).
 *
 * SDSAT ("Speculative Decoding with Semantic Adaptive Tokens", arXiv
 * 2403.18647) decodes with an unmodified Llama-architecture model in loops of
 * "two-step-draft-then-verify" (Sec. 2.1):
 *
 *   draft step 1 (Eq. 1)  block [last token, a_1 .. a_k]  -> y_{n+1} and k drafts
 *   draft step 2 (Eq. 2)  block [y_{n+1}, d_1 .. d_k]     -> targets t_0 .. t_k
 *   verification (Eq. 3)  accept t_0 .. t_m, m = leading matches d_i == t_{i-1}
 *
 * Each step is one pass of q = k + 1 positions through every layer
 * (sdsat_block_forward), then target selection, verification and KV commit
 * (sdsat_accept_greedy / sdsat_accept_nucleus).  The loop emits 2 + m tokens
 * for two passes (Sec. 2.1.1).
 *
 * Conventions for every entry point
 * ---------------------------------
 *  - Pointers named *_dev are CUDA device pointers owned by the caller; they
 *    must stay valid until the work queued on the context stream has run.
 *  - All compute calls are asynchronous on the context stream
 *    (sdsat_set_stream); only sdsat_create, sdsat_kv_create, sdsat_*_destroy
 *    and sdsat_get_error synchronise.  No compute call allocates memory, so
 *    compute calls may be captured into a CUDA graph.
 *  - Argument errors are detected on the host and returned synchronously
 *    (nothing is queued).  Errors only the device can see (a NaN logit, a
 *    row past the KV capacity, a timed-out wait) set bits in a device flag
 *    word read by sdsat_get_error.
 *  - Weights are bf16, row-major [out_features, in_features] (the layout of
 *    nn.Linear.weight), 16-byte aligned, in_features a multiple of 8.
 *  - Activations and logits are fp32; token ids int32.
 */
#ifndef SDSAT_H
#define SDSAT_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SDSAT_API __attribute__((visibility("default")))
#else
#define SDSAT_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SDSAT_OK = 0,
  SDSAT_EINVAL = 1,        /* bad argument: null/misaligned pointer, size out of range */
  SDSAT_ENOMEM = 2,        /* device allocation failed (create calls only) */
  SDSAT_ECAPACITY = 3,     /* batch, q, position or KV capacity limit exceeded */
  SDSAT_ECUDA = 4,         /* a CUDA runtime or driver call failed */
  SDSAT_EDEVICE = 5,       /* device-detected error bits were set (sdsat_get_error) */
  SDSAT_EUNSUPPORTED = 6   /* a configuration this library does not implement */
} sdsat_status;

/* device error bits reported by sdsat_get_error */
#define SDSAT_DEV_NAN_LOGITS 0x1u  /* NaN logit seen; it counted as -inf */
#define SDSAT_DEV_TIMEOUT 0x2u     /* a bounded in-kernel wait expired; results invalid */
#define SDSAT_DEV_CAPACITY 0x4u    /* a block row fell past the KV capacity; not written */
#define SDSAT_DEV_TOKEN 0x8u       /* a token id outside [0, vocab); id 0 used instead */
#define SDSAT_DEV_POSITION 0x10u   /* a RoPE position outside [0, max_position); clamped */
#define SDSAT_DEV_TREE 0x20u       /* a tree parent that is not an earlier row; read as the root */

#define SDSAT_MAX_Q 16           /* block rows per sequence (k <= 15 adaptive tokens) */
#define SDSAT_MAX_ROWS 64        /* batch * q rows per block forward */
#define SDSAT_MAX_ADAPTIVE 16

typedef struct sdsat_ctx sdsat_ctx;
typedef struct sdsat_kv sdsat_kv;

/* Model and decoding configuration (Llama architecture; Sec. 3 uses CodeLlama). */
typedef struct {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_heads;
  int32_t n_kv_heads;      /* must equal n_heads (this library has no grouped-query attention) */
  int32_t head_dim;        /* 64 or 128 */
  int32_t ffn_dim;         /* SwiGLU hidden size */
  int32_t vocab;           /* including the semantic adaptive tokens (Sec. 3.2: ordinary ids) */
  float rms_eps;
  float rope_theta;        /* RoPE base; rotate-half pairing (i, i + head_dim/2) */
  int32_t max_position;    /* RoPE table length: every position must be < max_position */
  int32_t n_adaptive;      /* 1: adaptive_ids[0] repeated k times (recommended, App. B);
                              >1: k distinct ids a_1..a_k (SDSAT-D, App. B) */
  int32_t adaptive_ids[SDSAT_MAX_ADAPTIVE];
} sdsat_config;

/* Per-layer weights (device pointers, borrowed: the caller keeps them alive). */
typedef struct {
  const void* attn_norm;   /* bf16 [d] */
  const void* wq;          /* bf16 [H*hd, d] */
  const void* wk;          /* bf16 [H*hd, d] */
  const void* wv;          /* bf16 [H*hd, d] */
  const void* wo;          /* bf16 [d, H*hd] */
  const void* ffn_norm;    /* bf16 [d] */
  const void* w_gate;      /* bf16 [F, d] */
  const void* w_up;        /* bf16 [F, d] */
  const void* w_down;      /* bf16 [d, F] */
} sdsat_layer_weights;

typedef struct {
  const void* embed;                    /* bf16 [V, d] */
  const void* final_norm;               /* bf16 [d] */
  const void* lm_head;                  /* bf16 [V, d] (untied) */
  const sdsat_layer_weights* layers;    /* host array of n_layers entries (copied) */
} sdsat_weights;

/* ---- lifetime ----------------------------------------------------------------- */

/* Validate `cfg`, record the weight pointers, build the TMA descriptors and the
 * RoPE table, allocate the library-owned workspaces.  The model is the unmodified
 * decoder the method runs (Abstract, Sec. 1: no structural change; Sec. 3.2: the
 * adaptive tokens are ordinary vocabulary ids), so the configuration is a plain
 * Llama configuration plus the adaptive ids; the paper prescribes no interface for
 * it.  `stream` is a cudaStream_t (NULL = legacy default stream).  Synchronous.  Errors: EINVAL (bad config or
 * pointer), EUNSUPPORTED (head_dim, GQA), ENOMEM, ECUDA.
 * Environment: SDSAT_NO_PDL=1 (read at each create) launches this context's kernels
 * without programmatic dependent launch, for tools that cannot follow it;
 * SDSAT_ATT_CLUSTER_MAX=n (read at the first create of the process) caps the
 * attention's thread-block cluster size at n in 1..16 for tuning sweeps (default
 * 16; the size itself is chosen per launch). */
SDSAT_API sdsat_status sdsat_create(const sdsat_config* cfg, const sdsat_weights* w, void* stream,
                          sdsat_ctx** out);
SDSAT_API void sdsat_destroy(sdsat_ctx* ctx);

/* Stream for all later compute calls on ctx (a cudaStream_t). */
SDSAT_API sdsat_status sdsat_set_stream(sdsat_ctx* ctx, void* stream);

/* Library-owned KV cache for `batch` sequences of up to `max_len` slots (the cache
 * that Eq. 1 and Eq. 2 extend by q positions per pass and that Sec. 2.1.1's
 * verification truncates to the accepted prefix; the paper states no layout):
 * K and V bf16 [n_layers][batch][n_heads][max_len][head_dim], and the committed
 * length len[batch] (int32, device, starts at 0).  Synchronous.
 * Errors: EINVAL, ENOMEM, ECAPACITY (max_len > max_position or > 32768). */
SDSAT_API sdsat_status sdsat_kv_create(sdsat_ctx* ctx, int batch, int max_len, sdsat_kv** out);
SDSAT_API void sdsat_kv_destroy(sdsat_kv* kv);

/* Device addresses and geometry of a KV cache (for tests and benches that fill
 * or inspect it).  Any output pointer may be NULL. */
SDSAT_API sdsat_status sdsat_kv_info(const sdsat_kv* kv, void** k_dev, void** v_dev, int32_t** len_dev,
                           int* batch, int* max_len);

/* Copy n rows into / out of the cache of one (layer, sequence), all heads:
 * src / dst are bf16 [n_heads][n][head_dim] device buffers; rows land at slots
 * slot0 .. slot0+n-1.  Asynchronous on the context stream.  Used to load a
 * snapshot (or synthetic contents) and to inspect what a block forward wrote.
 * Errors: EINVAL (null pointer, layer/seq/slot range). */
SDSAT_API sdsat_status sdsat_kv_write(sdsat_ctx* ctx, sdsat_kv* kv, int layer, int seq, int slot0, int n,
                                      const void* k_src_dev, const void* v_src_dev);
SDSAT_API sdsat_status sdsat_kv_read(sdsat_ctx* ctx, const sdsat_kv* kv, int layer, int seq, int slot0, int n,
                                     void* k_dst_dev, void* v_dst_dev);

/* ---- the block decode step ------------------------------------------------------- */

/* One pass of q new positions for sequences 0 .. b-1 through every layer
 * (Eq. 1 and Eq. 2 evaluate P_theta at all q positions of a block at once).
 *
 * tokens_dev     int32 [b*q], row j of sequence s at s*q + j.
 * positions_dev  int32 [b*q] RoPE positions, or NULL for len[s] + j.
 * logits_dev     fp32 [b*q][vocab], written.
 * Block rows are written to KV slots len[s] .. len[s]+q-1 (len is NOT advanced;
 * see the accept calls and sdsat_kv_commit).  Row j attends to slots [0, len[s])
 * and to block rows 0..j.
 * Errors: EINVAL (null pointer, b < 1, b > kv batch, q < 1, q > SDSAT_MAX_Q,
 * b*q > SDSAT_MAX_ROWS); device bit CAPACITY if len[s] + q > max_len. */
SDSAT_API sdsat_status sdsat_block_forward(sdsat_ctx* ctx, sdsat_kv* kv, const int32_t* tokens_dev,
                                 const int32_t* positions_dev, int b, int q, float* logits_dev);

/* Greedy target selection, Eq. 3 verification and KV commit (Sec. 2.1.1).
 *
 * logits_dev        fp32 [b*q][vocab] from sdsat_block_forward.
 * drafts_dev        int32 [b*q]: the block's input tokens; entry s*q + i (1 <= i < q)
 *                   is draft d_i.  Entry s*q is not read.
 * n_verify          number of drafts to verify (0 <= n_verify < q).  0 is draft
 *                   step 1: only t_0 is emitted and rows 1..q-1 return the drafts.
 * out_tokens_dev    int32 [b*q]: t_j = argmax of row j (lowest id on ties; NaN
 *                   counts as -inf and sets device bit NAN_LOGITS), for every j.
 * accepted_len_dev  int32 [b]: 1 + m, the number of emitted tokens t_0 .. t_m,
 *                   m = max{i <= n_verify : d_i' == t_{i'-1} for all i' <= i}.
 * commit            non-zero: len[s] += 1 + m on the device (rejected rows and
 *                   the adaptive positions are rolled back by not committing them).
 * Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_accept_greedy(sdsat_ctx* ctx, sdsat_kv* kv, const float* logits_dev,
                                 const int32_t* drafts_dev, int b, int q, int n_verify,
                                 int32_t* accepted_len_dev, int32_t* out_tokens_dev, int commit);

/* Nucleus (top-p) variant (Sec. 2.1.2, chain form: the accepted branch is the
 * longest verified prefix).  Each row's target is a sample defined exactly so
 * that any two implementations agree bit for bit:
 *   s_i = (l_i - max l) / temperature (fp32), w_i = exp(s_i) (fp32, Cody-Waite
 *   reduction + degree-7 polynomial, every step one rounded operation),
 *   W_i = floor(w_i * 2^24) (exact in 32 bits: the top weight is 2^24, and a
 *   token below 2^-24 of it gets 0);  candidates = the top_k heaviest by
 *   (W desc, id asc) (top_k = 0: all);  kept = the shortest prefix of the
 *   candidates in that order with C * 2^24 >= round(top_p * 2^24) * S;
 *   r = Philox4x32-10(key = rng_seed, counter = (position of the produced
 *   token, s, 0, 0)), 64-bit from its first two words;  tau = (r * S_kept) >> 64;
 *   the sample is the first kept id, ascending, whose inclusive cumulative
 *   weight exceeds tau.
 * The produced token of row j has position len[s] + j + 1.  temperature <= 0
 * selects greedy (Fig. 1: greedy is the special case).  Requires vocab <= 32768.
 * Other arguments as sdsat_accept_greedy.  Errors: EINVAL, EUNSUPPORTED. */
SDSAT_API sdsat_status sdsat_accept_nucleus(sdsat_ctx* ctx, sdsat_kv* kv, const float* logits_dev,
                                  const int32_t* drafts_dev, int b, int q, int n_verify,
                                  float top_p, float temperature, uint64_t rng_seed, int top_k,
                                  int32_t* accepted_len_dev, int32_t* out_tokens_dev, int commit);

/* Explicit commit / rollback (implied by Sec. 2.1.1: after Eq. 3 only the accepted
 * prefix stays in the context; the adaptive positions of draft step 1 and the rejected
 * drafts are dropped): len[s] = new_len_dev[s] for s < b (device values,
 * 0 <= new_len <= max_len; out-of-range values are clamped and set CAPACITY).
 * Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_kv_commit(sdsat_ctx* ctx, sdsat_kv* kv, const int32_t* new_len_dev, int b);

/* Copy the committed lengths len[0 .. b-1] into lens_dev (int32 [b], device),
 * asynchronously.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_kv_lengths(sdsat_ctx* ctx, const sdsat_kv* kv, int32_t* lens_dev, int b);

/* Tokens emitted so far per sequence: every accept call with commit != 0 adds
 * 1 + m to emitted[s] on the device.  Copies emitted[0 .. b-1] into
 * emitted_dev (int64 [b]) and, when reset != 0, zeroes the counters after the
 * copy.  Asynchronous.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_kv_emitted(sdsat_ctx* ctx, sdsat_kv* kv, int64_t* emitted_dev, int b, int reset);

/* Build the next block input on the device (the block inputs of Eq. 1 and Eq. 2),
 * so that a whole loop runs without the host:
 *   mode 1 (draft step 1): row 0 = prev_out[s*q + prev_acc[s] - 1] (the newest
 *     emitted token), rows 1..q-1 = the adaptive ids a_1 .. a_{q-1};
 *   mode 2 (draft step 2): row 0 = prev_out[s*q] (y_{n+1}), rows 1..q-1 = the drafts:
 *     prev_out[s*q + j] (the drafts draft step 1 produced), or, when
 *     draft_table_dev is given, draft_table_dev[s*table_stride + len[s] + j]
 *     (a per-position draft source, e.g. a test stub).
 * prev_out_dev / prev_acc_dev are the out_tokens / accepted_len of the previous
 * accept call; tokens_out_dev int32 [b*q] is written.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_build_block(sdsat_ctx* ctx, sdsat_kv* kv, int mode, const int32_t* prev_out_dev,
                               const int32_t* prev_acc_dev, const int32_t* draft_table_dev,
                               int table_stride, int b, int q, int32_t* tokens_out_dev);

/* ---- tree-structured draft step 2 (Sec. 2.1.2) ----------------------------------- */
/* A tree block holds q rows per sequence: the nodes of a draft tree in
 * topological order.  parent_dev int32 [b*q]: entry s*q + j is the parent row of
 * row j of sequence s; row 0 is the root (parent -1, the token y_{n+1} of draft
 * step 1) and every other row's parent is an earlier row (parent[j] < j).
 * Anything else sets device bit TREE and the row is read as a child of the root.
 * Row j has depth(j) = number of edges to the root, occupies KV slot len[s] + j
 * and sits at position len[s] + depth(j).  A chain (parent[j] = j - 1) is the
 * ordinary block of sdsat_block_forward / sdsat_accept_*. */

/* Tree block forward: as sdsat_block_forward, with RoPE positions
 * len[s] + depth(j) and the tree attention mask -- row j attends to the committed
 * slots [0, len[s]) and to the slots of its ancestors and itself only.
 * tokens_dev int32 [b*q]; logits_dev fp32 [b*q][vocab], written.  len is not
 * advanced.  Errors: EINVAL (null pointer, b < 1, b > kv batch, q < 1,
 * q > SDSAT_MAX_Q, b*q > SDSAT_MAX_ROWS); device bits TREE, CAPACITY. */
SDSAT_API sdsat_status sdsat_block_forward_tree(sdsat_ctx* ctx, sdsat_kv* kv, const int32_t* tokens_dev,
                                                const int32_t* parent_dev, int b, int q, float* logits_dev);

/* Tree verification and commit (Sec. 2.1.2: the longest branch of the tree that
 * is verified and accepted is the loop's result).
 *   targets  t_j = the selection of sdsat_accept_nucleus (temperature > 0) or
 *            argmax (temperature == 0) of row j's logits, the produced token at
 *            position len[s] + depth(j) + 1;
 *   accepted row 0 always; row j > 0 iff its parent p is accepted and
 *            tokens[s*q + j] == t_p (the chain test of Eq. 3 along each branch);
 *   path     n_0 = 0, n_1, ..., n_m: the root path of the deepest accepted row
 *            (the lowest row index among equally deep ones).
 * out_tokens_dev   int32 [b*q]: t_{n_0} .. t_{n_m}, then -1.
 * accepted_len_dev int32 [b]: 1 + m.
 * path_dev         int32 [b*q]: n_0 .. n_m, then -1; may be NULL.
 * The K and V rows of the path always move to slots len[s] + 1 .. len[s] + m
 * (slot len[s] + i receives row n_i's rows, which were rotated at position
 * len[s] + i already), so the cache holds the accepted branch contiguously;
 * commit != 0 then advances len[s] by 1 + m (with commit == 0, an explicit
 * sdsat_kv_commit of len[s] + 1 + m commits it later).
 * Other arguments as sdsat_accept_nucleus.  Errors: EINVAL (null parent_dev,
 * temperature < 0 or NaN, the sdsat_accept_nucleus conditions), EUNSUPPORTED
 * (temperature > 0 and vocab > 32768); device bit TREE. */
SDSAT_API sdsat_status sdsat_accept_tree(sdsat_ctx* ctx, sdsat_kv* kv, const float* logits_dev,
                                         const int32_t* tokens_dev, const int32_t* parent_dev, int b, int q,
                                         float temperature, float top_p, uint64_t rng_seed, int top_k,
                                         int32_t* accepted_len_dev, int32_t* out_tokens_dev, int32_t* path_dev,
                                         int commit);

/* Block building for tree loops, where consecutive blocks differ in size:
 *   mode 1 (draft step 1): q = k + 1 rows; row 0 = prev_out[s*prev_q + prev_acc[s] - 1],
 *     rows 1..k = the adaptive ids;
 *   mode 2 (draft step 2): the tree of `width` chains of k drafts below the root,
 *     q = 1 + width*k rows (parent of row 1 + w*k is 0, of row 1 + w*k + i is
 *     row w*k + i); row 0 = prev_out[s*prev_q]; row 1 + w*k + i - 1 (1 <= i <= k)
 *     = draft_tables_dev[(w*B + s)*table_stride + len[s] + i] with B the KV batch
 *     (branch w's draft for position len[s] + i).  Without tables (width 1 only)
 *     row i = prev_out[s*prev_q + i] (k < prev_q).
 * tokens_out_dev int32 [b*q].  Errors: EINVAL (q > SDSAT_MAX_Q, b*q > SDSAT_MAX_ROWS,
 * table_stride < max_len + SDSAT_MAX_Q, the sdsat_build_block conditions). */
SDSAT_API sdsat_status sdsat_build_tree_block(sdsat_ctx* ctx, sdsat_kv* kv, int mode, const int32_t* prev_out_dev,
                                              int prev_q, const int32_t* prev_acc_dev,
                                              const int32_t* draft_tables_dev, int width, int table_stride, int b,
                                              int k, int32_t* tokens_out_dev);

/* ---- pipelined variant (not a step of the paper) ---------------------------------- */
/* The verification block also carries the k adaptive tokens, so that a loop whose
 * drafts are all accepted needs no separate draft step 1.  Every block has
 * q = 2k + 1 rows [x_0, r_1 .. r_k, a_1 .. a_k] at slots len[s] .. len[s] + 2k:
 *   mode A (drafts known): r_i = the drafts for positions len[s] + i; Eq. 3 verifies
 *     them; if all k are accepted, the adaptive rows' targets are the next block's
 *     drafts and the next block is mode A again, otherwise it is mode S;
 *   mode S: r_i = a_i (the block is draft step 1 with k extra adaptive rows), nothing
 *     is verified, t_0 is emitted and t_1 .. t_k are the next block's drafts (mode A).
 * The emitted tokens are those of the two-step loop (and of plain decoding under greedy
 * selection or the position-keyed sampler). */

/* Build the next pipelined block on the device from the previous one's accept outputs:
 *   prev_out_dev int32 [b*(2k+1)], prev_acc_dev int32 [b]: the previous accept call's
 *     out_tokens and accepted_len (before the first block: out[s*(2k+1)] = the newest
 *     prompt token, acc = 1, mode = 1);
 *   mode_dev int32 [b], in: the previous block's mode (0 S, 1 A), out: this block's;
 *   n_verify_dev int32 [b], out: k for mode A, 0 for mode S (for sdsat_accept_pipelined);
 *   draft_table_dev: optional per-position drafts, [s*table_stride + len[s] + i] for
 *     row i of a mode-A block (the harness's stub); otherwise the previous targets.
 * x_0 = prev_out[s*(2k+1) + acc - 1]; mode A's drafts without a table are
 * prev_out[s*(2k+1) + acc .. + acc + k - 1].  tokens_out_dev int32 [b*(2k+1)].
 * Errors: EINVAL (null pointer, 2k + 1 > SDSAT_MAX_Q, b*(2k+1) > SDSAT_MAX_ROWS,
 * table_stride < max_len + SDSAT_MAX_Q). */
SDSAT_API sdsat_status sdsat_build_pipelined_block(sdsat_ctx* ctx, sdsat_kv* kv, const int32_t* prev_out_dev,
                                                   const int32_t* prev_acc_dev, int32_t* mode_dev,
                                                   int32_t* n_verify_dev, const int32_t* draft_table_dev,
                                                   int table_stride, int b, int k, int32_t* tokens_out_dev);

/* Target selection (argmax for temperature == 0, else the sampler of
 * sdsat_accept_nucleus), Eq. 3 verification of n_verify_dev[s] drafts per sequence
 * (device values, clamped to [0, q-1]) and the KV commit, as sdsat_accept_nucleus.
 * Errors: EINVAL (null n_verify_dev, temperature < 0 or NaN, q < 2, the
 * sdsat_accept_nucleus conditions), EUNSUPPORTED. */
SDSAT_API sdsat_status sdsat_accept_pipelined(sdsat_ctx* ctx, sdsat_kv* kv, const float* logits_dev,
                                              const int32_t* tokens_dev, const int32_t* n_verify_dev, int b, int q,
                                              float temperature, float top_p, uint64_t rng_seed, int top_k,
                                              int32_t* accepted_len_dev, int32_t* out_tokens_dev, int commit);

/* Run n prompt tokens of sequence `seq` through the model and commit them
 * (len[seq] += n): the step before the decode loop (Sec. 2.1.1 starts from a prompt
 * y_1 .. y_n already in the context; the paper gives the prefill no further detail).  Chunks of up to
 * SDSAT_MAX_ROWS positions go through one block forward each (the weights stream
 * once per chunk), position i attending to every earlier position; a tail shorter
 * than SDSAT_MAX_Q rows runs as one ordinary block.  No logits are produced.
 * Errors: EINVAL (null pointer, seq outside the KV batch, n < 0), ECAPACITY
 * (n > max_len); device bit CAPACITY if len[seq] + n > max_len. */
SDSAT_API sdsat_status sdsat_prefill(sdsat_ctx* ctx, sdsat_kv* kv, int seq, const int32_t* tokens_dev, int n);

/* Synchronise the context stream, return the accumulated device error bits in
 * *flags (SDSAT_DEV_*) and clear them.  Returns EDEVICE if any bit was set,
 * ECUDA if the stream reported a CUDA error. */
SDSAT_API sdsat_status sdsat_get_error(sdsat_ctx* ctx, uint32_t* flags);

/* A static, NUL-terminated English name of a status code ("ok", "invalid argument", ...;
 * unknown codes give "unknown status").  Host only, never fails.  The paper has no
 * counterpart: it is the error reporting of this library's boundary. */
SDSAT_API const char* sdsat_status_string(sdsat_status s);

/* ---- single kernels (unit parity tests and kernel sweeps) ------------------------- */

/* y[m][n] = sum_k x[m][k] * W[n][k] for m < M, n < N.  M <= SDSAT_MAX_ROWS runs the
 * weight-streaming skinny GEMM behind every projection of the block forward;
 * SDSAT_MAX_ROWS < M <= 512 runs the tiled GEMM of the prefill path (128 weight rows
 * x 128 positions per tile).  x fp32
 * [M][K] (row stride K), W bf16 [N][K], y fp32 [M][N]; x and W 16-byte aligned,
 * K a multiple of 8, K <= 32768.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_op_gemm(sdsat_ctx* ctx, const float* x_dev, int M, int K, const void* w_dev, int N,
                           float* y_dev);

/* Block-causal attention of q query rows per sequence against a bf16 cache:
 * out[s*q+j][h*hd+d] = sum_t softmax_t(q_j . k_t / sqrt(hd)) v_t[d] over slots
 * t < len[s] + j + 1.  q_dev fp32 [b*q][H*hd]; k_dev, v_dev bf16
 * [b][H][cap][hd]; len_dev int32 [b] (device); out_dev fp32 [b*q][H*hd].
 * hd must be 64 or 128; k_dev, v_dev and out_dev 16-byte aligned.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_op_attention(sdsat_ctx* ctx, const float* q_dev, const void* k_dev, const void* v_dev,
                                const int32_t* len_dev, int b, int q, int H, int hd, int cap,
                                float* out_dev);

/* Copy a context workspace of the last block forward into dst_dev (fp32,
 * rows x cols row-major, rows = b*q of that forward): which = 0 the residual
 * stream h [rows][d], 1 the RoPE'd queries [rows][H*hd], 2 the attention
 * output [rows][H*hd], 3 the SwiGLU activations [rows][F] -- of the last
 * layer.  For tests that check a forward stage by stage.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_debug_workspace(sdsat_ctx* ctx, int which, int rows, float* dst_dev);

/* The attention grid sdsat_block_forward and sdsat_op_attention launch for `pairs`
 * (sequence, head) pairs (host only, no GPU): one thread-block cluster of *cs CTAs per
 * pair, *nclusters = pairs, for the largest cs <= min(cs_cap, 16) with
 * max_clusters[cs] >= pairs and cs * (pairs + 8) <= max_clusters[1] (the CTAs resident
 * at once, else 2 * num_sms); otherwise *cs = 1 and *nclusters = min(pairs, resident),
 * each CTA taking several pairs.  max_clusters[c] (c = 1..16, host array of 17 entries,
 * [0] unused) = the most clusters of c CTAs the device holds at once, as
 * cudaOccupancyMaxActiveClusters reports it for the attention kernel.  Errors: EINVAL. */
SDSAT_API sdsat_status sdsat_attention_grid(int pairs, const int32_t* max_clusters, int cs_cap, int num_sms,
                                            int* cs, int* nclusters);

/* Test hook for failure detection: one kernel waits on a barrier that nothing
 * completes, through the bounded wait every kernel of the library uses.  After its
 * limit (2 s) it sets device bit TIMEOUT and returns; nothing faults and the
 * context stays usable.  Asynchronous (read the bit with sdsat_get_error).
 * Errors: EINVAL (null ctx), ECUDA. */
SDSAT_API sdsat_status sdsat_debug_wait_timeout(sdsat_ctx* ctx);

/* out[i] = the nucleus sampler's exp (see sdsat_accept_nucleus) of in[i] <= 0. */
SDSAT_API sdsat_status sdsat_op_exp(sdsat_ctx* ctx, const float* in_dev, float* out_dev, int n);

/* y[m][n] = sum_k x[m][k] * W[n][k] like sdsat_op_gemm, for callers that cannot
 * allocate device memory: no context, no cudaMalloc or other allocating call.
 * This entry point has no counterpart in the paper; it exists because a caller
 * may be capturing a CUDA graph (where allocation is not allowed), may run inside
 * a framework that owns all device memory through its own allocator, or may have
 * a fixed memory budget.  Its scratch -- the operand split, the split-K partial
 * sums and the tile counters -- is one fixed array in device memory (3 MiB +
 * 2 KiB, held by every GPU that loads the library until the process exits).
 *   x_dev fp32 [M][K] (16-byte aligned), W bf16 [N][K] (16-byte aligned),
 *   y_dev fp32 [M][N]; stream is a cudaStream_t (NULL = legacy default stream).
 *   Limits: 1 <= M <= 16, 8 <= K <= 16384 with K % 8 == 0, 1 <= N <= 65536;
 *   sizes past the limits return ECAPACITY, malformed arguments EINVAL.
 *   err_dev: optional caller-owned device word (NULL: not reported); a bounded
 *   in-kernel wait that runs out (2 s) ORs SDSAT_DEV_TIMEOUT into it and leaves
 *   y_dev incomplete.  The call never clears it.
 * The first call on a device (with that device current) looks up the array's
 * device address and prepares the kernels; make that first call before any
 * stream capture.  The set-up is redone when the device's context changes (after
 * cudaDeviceReset, for instance).  Every call shares the one array: calls whose
 * work overlaps on the GPU (different streams, or concurrent host threads) race
 * and must be serialised by the caller.  The call clears the tile counters it
 * uses; the other scratch contents are overwritten before they are read.
 * Asynchronous on `stream`. */
SDSAT_API sdsat_status sdsat_gemm_static(const float* x_dev, int M, int K, const void* w_dev, int N, float* y_dev,
                                         void* stream, uint32_t* err_dev);

/* ---- measurement ------------------------------------------------------------------ */

/* Per-kernel timing: between sdsat_profile_begin and sdsat_profile_end every
 * kernel the library launches on ctx is bracketed by CUDA events recorded on
 * the context stream (which serialises the launches: no overlap between
 * consecutive kernels while profiling).  begin creates a pool of events for
 * up to max_launches launches (call it outside any graph capture); launches
 * past the pool are not timed.  end synchronises and returns one record per
 * kernel class that ran: its name, launch count and summed duration. */
typedef struct {
  char name[32];
  int64_t launches;
  double total_ms;
} sdsat_kernel_stat;

SDSAT_API sdsat_status sdsat_profile_begin(sdsat_ctx* ctx, int max_launches);
SDSAT_API sdsat_status sdsat_profile_end(sdsat_ctx* ctx, sdsat_kernel_stat* out, int max_out, int* n_out);

/* Device timeline trace (does not serialise launches): between sdsat_trace_begin and
 * sdsat_trace_end, thread 0 of every CTA of the block forward's GEMM and attention kernels
 * appends one record of SDSAT_TRACE_WORDS uint64:
 *   [0] tag << 32 | block index, tag = kernel class << 24 | launch sequence number
 *       (sdsat_kernel_class_name names a class);
 *   [1] flags << 32 | SM id;
 *   [2] %globaltimer (ns) at kernel entry, [3] after the wait for the preceding kernel,
 *   [4], [5], [6] kernel-specific marks (0 = not reached), [7] at exit.
 * GEMM: marks = first MMA issued, accumulator of the CTA's last tile ready, that tile
 * reduced (or handed to another CTA); flags = 1 if this CTA reduced it | contributors << 8.
 * Attention: marks = first K/V tile usable, the CTA's partial of its last (sequence, head)
 * pair written, that pair's share of the merged output stored; flags = pairs taken |
 * units of 64 slots << 8.
 * begin allocates room for max_records records (call it outside any graph capture); end
 * synchronises, copies up to max_records records to host memory and frees the buffer. */
#define SDSAT_TRACE_WORDS 8
SDSAT_API sdsat_status sdsat_trace_begin(sdsat_ctx* ctx, int max_records);
SDSAT_API sdsat_status sdsat_trace_end(sdsat_ctx* ctx, uint64_t* records_host, int max_records, int* n_records);
SDSAT_API const char* sdsat_kernel_class_name(int kernel_class);

#ifdef __cplusplus
}
#endif
#endif /* SDSAT_H */
