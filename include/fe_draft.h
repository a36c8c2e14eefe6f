/*
 * fe_draft.h -- C ABI of the GB300 (sm_103a) FastEagle cascaded drafter.
 *
 * FastEagle (arXiv 2509.20416) drafts N tokens in one forward pass: the target's
 * multi-level features of the last verified position are fused by an FC layer,
 * joined with the next token's embedding and a second FC (Sec. 2.1, Eq. 1), and
 * pushed through N serially connected decoder layers h_i = L_i(h_{i-1}) (Eq. 2).
 * Every h_i goes through the target's frozen LM head to give the distribution
 * q_{t+i} (Sec. 2.1). The k most probable tokens per depth are then arranged into
 * the Backbone Expansion draft tree (Sec. 2.2) that the target verifies with tree
 * attention (Sec. 2.4).
 *
 * Conventions for every call:
 *  - Weight matrices are row-major [out, in] (y = W x). Storage type is the
 *    config's dtype (float32 or bfloat16) for weights, features and K/V caches;
 *    activations are float32 inside the library and all float outputs are float32.
 *  - "device" pointers are CUDA device (or managed) memory on the handle's device;
 *    "host" pointers are ordinary host memory. Memory passed to a call stays owned
 *    by the caller.
 *  - A handle belongs to the CUDA device that was current when fe_draft_init created it.
 *    Every later call on the handle (except fe_free) must be made with that device
 *    current; otherwise it returns FE_ERR_INVALID_ARG (fe_last_error_detail() names
 *    both devices) and enqueues nothing. fe_free switches to the handle's device itself.
 *  - Calls that take a stream enqueue work on it and return before it runs.
 *    Argument errors are detected on the host and returned synchronously, with
 *    nothing enqueued. Errors found while the kernels run (an out-of-range token,
 *    a prefix longer than the cache, a bad page id, a timed-out device wait) are
 *    recorded in a device status word and reported by fe_last_device_status();
 *    the offending work item is skipped, and no kernel traps.
 *  - No global state beyond two exceptions: the per-thread detail string of
 *    fe_last_error_detail() and the fixed scratch array of fe_lm_head_topk_noalloc().
 *    Several handles may coexist. One handle must not be used from two streams
 *    concurrently (its scratch buffers are shared by its calls).
 *  - No exceptions cross the ABI.
 */
#ifndef FE_DRAFT_H
#define FE_DRAFT_H

#include <stdint.h>

#if defined(__GNUC__)
#define FE_API __attribute__((visibility("default")))
#else
#define FE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FE_OK = 0,
    FE_ERR_INVALID_ARG = -1, /* a null pointer, a bad shape or an out-of-range scalar */
    FE_ERR_UNSUPPORTED = -2, /* a legal shape the library does not implement */
    FE_ERR_CUDA = -3,        /* a CUDA runtime call failed */
    FE_ERR_OOM = -4,         /* device allocation failed */
    FE_ERR_CAPACITY = -5,    /* a prefix does not fit its cache (P_b + 1 > max_seq) */
    FE_ERR_TIMEOUT = -6,     /* a bounded device-side wait ran out */
    FE_ERR_DEVICE = -7       /* a device-side range check failed (token, page id) */
} fe_status;

typedef enum { FE_F32 = 0, FE_BF16 = 1 } fe_dtype;

/* Shape of one drafter. Sec. 2.1 fixes the structure (N layers, shared frozen LM
 * head); the layer internals follow the LLaMA-style block EAGLE-3 uses. */
typedef struct {
    int32_t d;          /* hidden size of the drafter and the target */
    int32_t n_heads;    /* query heads H */
    int32_t n_kv_heads; /* key/value heads Hkv (H % Hkv == 0; Hkv == H is plain MHA) */
    int32_t head_dim;   /* hd: 64 or 128 */
    int32_t ffn;        /* SwiGLU intermediate size F */
    int32_t vocab;      /* V, rows of the embedding table and of the LM head */
    int32_t n_layers;   /* N, cascade depth (Eq. 2), 1..16 */
    int32_t top_k_max;  /* largest top_k any call will ask for, 1..32 */
    int32_t max_batch;  /* largest B any call will pass */
    int32_t max_seq;    /* cache rows per sequence: a call needs prefix_len[b] + 1 <= max_seq */
    int32_t page_size;  /* 0: contiguous caches; > 0: rows per page of paged caches */
    float rope_theta;   /* RoPE base */
    float rms_eps;      /* RMSNorm epsilon */
    fe_dtype dtype;     /* storage type of weights, features and caches */
    int32_t parallel_layers; /* 0: the cascade, L_i consumes h_{i-1} (Eq. 2); 1: every L_i
                                consumes x0 — the "w/o cascaded structure" ablation of
                                Sec. 3.2 (Table 2), parallel instead of serial layers */
} fe_config;

/* One cascade layer L_i (Eq. 2): RMSNorm gains [d]; w_qkv [(H + 2 Hkv) hd, d] with the
 * q rows first, then k, then v; w_o [d, H hd]; w_gate, w_up [F, d]; w_down [d, F]. */
typedef struct {
    const void *attn_norm, *w_qkv, *w_o, *mlp_norm, *w_gate, *w_up, *w_down;
} fe_layer_weights;

/* w_fuse [d, 3d] fuses concat(l, m, h) into g (Sec. 2.1); w_in [d, 2d] maps concat(g, e)
 * to the cascade input (Eq. 1); embed [V, d]; lm_head [V, d] and final_norm [d] are the
 * target's frozen LM head and its final RMSNorm; layers points to n_layers entries. */
typedef struct {
    const void *w_fuse, *w_in, *embed, *lm_head, *final_norm;
    const fe_layer_weights *layers;
} fe_weights;

/* Arguments of one draft (Sec. 2.4, "Non-Autoregressive Drafting").
 *
 *  feat       device [B, 3d] dtype   concat(l, m, h) of each sequence's last verified position
 *  next_tok   device [B] int32       the token t+1 whose embedding joins the fused feature
 *  prefix_len device [B] int32       P_b, rows already in each layer's cache; the drafted row
 *                                    takes sequence position P_b and cache slot P_b
 *  k_cache,   host arrays of n_layers device pointers, layer i's K and V cache:
 *  v_cache      page_size == 0: [max_batch, Hkv, max_seq, hd] dtype, row p of sequence b
 *                 and KV head g at ((b * Hkv + g) * max_seq + p) * hd
 *               page_size  > 0: a page pool [n_pages, Hkv, page_size, hd] dtype; row p of
 *                 sequence b lives in page page_table[b * max_pages + p / page_size],
 *                 slot p % page_size, with max_pages = ceil(max_seq / page_size)
 *               Cached keys are stored after RoPE. The call writes each layer's new key
 *               (rotated) and value into slot P_b and reads rows 0..P_b-1; it does not
 *               advance prefix_len (committing accepted rows is the caller's step).
 *  page_table device [B, max_pages] int32 (paged only; entries past the last used page
 *             are ignored), n_pages the pool size (paged only)
 *  top_k      candidates per depth, 1..top_k_max
 *  temperature  T > 0 scales the reported probabilities and lse as softmax(logit / T);
 *             T <= 0 (greedy) reports the T = 1 distribution. Unless sample is set, the
 *             candidates are the k largest logits, ties broken by the smaller token id.
 *  sample, seed  stochastic drafting (Sec. 2.2, "sample k candidates"). sample != 0 needs
 *             T > 0: depth i's candidates of sequence b are then k draws without replacement
 *             from softmax(logit / T), taken as the k largest keys logit_v / T + G_v
 *             (Gumbel-top-k), G_v = -log(-log U_v) and U_v = (floor(x / 2^41) + 1/2) / 2^23,
 *             where x is output n = (b N + i - 1) V + v + 1 of SplitMix64 seeded with `seed`
 *             (Steele, Lea and Flood 2014). The drawn set is reported ordered by logit like
 *             the greedy candidates (descending, ties to the smaller id), so the tree rule is
 *             unchanged: the most probable drawn token is the backbone.
 * Outputs (device, float32 unless stated):
 *  topk_id [B, N, top_k] int32, topk_logit [B, N, top_k], topk_prob [B, N, top_k], lse [B, N]
 *  topk_rank [B, N, top_k] int32 or NULL: each candidate's position in draw order (0 =
 *             drawn first, i.e. the largest key); r for the r-th greedy candidate
 *  dbg_logits [B, N, V] or NULL: full logits, for parity checks only (costs V floats a row)
 *  dbg_hidden [N, B, d] or NULL: the cascade's hidden states h_i
 */
typedef struct {
    int32_t B, top_k;
    float temperature;
    const void *feat;
    const int32_t *next_tok;
    const int32_t *prefix_len;
    void *const *k_cache;
    void *const *v_cache;
    const int32_t *page_table;
    int32_t n_pages;
    int32_t *topk_id;
    float *topk_logit, *topk_prob, *lse;
    float *dbg_logits, *dbg_hidden;
    int32_t sample;
    uint64_t seed;
    int32_t *topk_rank;
} fe_forward_args;

/* The draft tree of B sequences, device buffers with T = 1 + N * top_k nodes each:
 * tok [B, T] int32, parent [B, T] int32 (-1 for the root), depth [B, T] int32,
 * mask [B, T, T] uint8 (mask[b][a][c] = 1 iff node c is node a or one of its ancestors). */
typedef struct {
    int32_t *tok, *parent, *depth;
    uint8_t *mask;
} fe_tree;

typedef struct fe_handle fe_handle;

/* Create a drafter on the current CUDA device: the N cascade layers L_1..L_N of Eq. 2,
 * the two input FCs of Sec. 2.1 / Eq. 1 (feature fusion, then concat with the token
 * embedding) and the target's frozen LM head with its final norm (Sec. 2.1, shared by
 * every depth). Copies (and repacks) every weight into
 * memory the handle owns, so the caller may free its weights once the call returns.
 * Weight pointers may be host or device memory (any memory cudaMemcpyDefault reads).
 * Precomputes the RoPE table in double precision. `stream` orders the copies; the
 * call synchronises it before returning. Errors: FE_ERR_INVALID_ARG (null pointer,
 * inconsistent shape), FE_ERR_UNSUPPORTED, FE_ERR_OOM, FE_ERR_CUDA. *out is set only
 * on FE_OK. */
FE_API fe_status fe_draft_init(const fe_config *cfg, const fe_weights *w, void *stream, fe_handle **out);

/* One single-pass draft (Eq. 1, Eq. 2, Sec. 2.1): the cascade, the LM head for all
 * N hidden states at once, softmax statistics and top-k per depth. No full-vocab
 * logits reach memory unless dbg_logits is given. */
FE_API fe_status fe_draft_forward(fe_handle *h, const fe_forward_args *args, void *stream);

/* Backbone Expansion (Sec. 2.2) from fe_draft_forward's topk_id [B, N, top_k]: node 0 is
 * the root (next_tok[b]); level i = 1..N holds that depth's candidates in rank order at
 * nodes 1 + (i-1) top_k + r; level 1 hangs under the root and level i >= 2 under the
 * previous level's rank-0 node, the backbone. A token id outside [0, V) sets
 * FE_ERR_DEVICE in the status word. */
FE_API fe_status fe_build_tree(fe_handle *h, int32_t B, int32_t top_k, const int32_t *next_tok,
                        const int32_t *topk_id, fe_tree *out, void *stream);

/* One draft step from and to HOST memory (Sec. 2.4, the drafting step of the cycle): the
 * step's inputs go to the device, fe_draft_forward and fe_build_tree run, and the outputs
 * come back, all as one CUDA graph per argument set (the copies are graph nodes between the
 * handle's pinned staging buffers and its device buffers), so a step costs one launch.
 *
 *  feat [B, 3d] dtype, next_tok [B] int32, prefix_len [B] int32: HOST inputs, as in
 *    fe_forward_args (any host memory; copied into the handle's pinned staging before the
 *    launch, except page-locked features at a 16-byte boundary, which the graph copies
 *    from directly: keep such a buffer's address across calls to replay the graph)
 *  k_cache, v_cache, page_table, n_pages, top_k, temperature: as in fe_forward_args
 *    (the caches and the page table stay in device memory)
 *  topk_id [B, N, top_k] int32, topk_logit, topk_prob [B, N, top_k] float32, lse [B, N]
 *    float32, tree_tok, tree_parent, tree_depth [B, T] int32, tree_mask [B, T, T] uint8
 *    (T = 1 + N top_k): HOST outputs, as fe_draft_forward and fe_build_tree define them
 *  sample, seed: stochastic drafting, as in fe_forward_args; topk_rank [B, N, top_k] int32:
 *    HOST output of the draw positions, or NULL
 *
 * The call synchronises `stream` and returns once the outputs are in host memory. Errors:
 * FE_ERR_INVALID_ARG (null pointer, B or top_k out of range), FE_ERR_CUDA / FE_ERR_OOM;
 * device-side conditions are reported by fe_last_device_status as for fe_draft_forward. */
typedef struct {
    int32_t B, top_k;
    float temperature;
    const void *feat;
    const int32_t *next_tok;
    const int32_t *prefix_len;
    void *const *k_cache;
    void *const *v_cache;
    const int32_t *page_table;
    int32_t n_pages;
    int32_t *topk_id;
    float *topk_logit, *topk_prob, *lse;
    int32_t *tree_tok, *tree_parent, *tree_depth;
    uint8_t *tree_mask;
    int32_t sample;
    uint64_t seed;
    int32_t *topk_rank;
} fe_host_step_args;

FE_API fe_status fe_draft_step_host(fe_handle *h, const fe_host_step_args *args, void *stream);

/* Synchronise `stream`, return and clear the handle's device status word
 * (FE_OK, FE_ERR_CAPACITY, FE_ERR_DEVICE or FE_ERR_TIMEOUT). */
FE_API fe_status fe_last_device_status(fe_handle *h, void *stream);

/* Release everything the handle owns (synchronises the device first). NULL is a no-op. */
FE_API void fe_free(fe_handle *h);

/* A static, human-readable name of a status code. */
FE_API const char *fe_status_str(fe_status s);

/* The calling thread's description of the last failing CUDA call inside the library
 * (which call, where, and CUDA's error string); "" if none. Valid until the thread's next
 * failing call. */
FE_API const char *fe_last_error_detail(void);

/* Number of kernels fe_draft_forward (plus fe_build_tree when with_tree != 0) launches for
 * a batch of B, so a caller can count launches. Returns -1 for a bad handle. */
FE_API int32_t fe_launch_count(const fe_handle *h, int32_t B, int32_t with_tree);

/* Forward of the multi-level training objective (Sec. 2.3, Eq. 3-6) for one draft: runs
 * fe_draft_forward (args->dbg_logits [B, N, V] and args->dbg_hidden [N, B, d] are required:
 * the loss reads the full-vocabulary logits and hidden states from them), then, for each
 * sequence b and depth i = 1..N:
 *   ce [B, N]        = -sum_k p_k log q_k with q = softmax(logits) at temperature 1 (Eq. 4),
 *                      p = teacher_p [B, N, V] (the target's teacher distribution, float32)
 *   feat_loss [B, N] = sum_j SmoothL1(h_ij - f_ij), f = target_feat [N, B, d] float32 (Eq. 5-6)
 *   total [B]        = sum_i decay^(N - i) (alpha ce + beta feat_loss) (Eq. 3; the paper uses
 *                      decay 0.9, alpha 0.1, beta 1).
 * Device pointers, asynchronous on `stream`. Errors as fe_draft_forward, plus
 * FE_ERR_INVALID_ARG for a missing buffer or a NaN coefficient. Forward only (no gradients). */
FE_API fe_status fe_draft_loss(fe_handle *h, const fe_forward_args *args, const float *teacher_p,
                               const float *target_feat, float alpha, float beta, float decay, float *ce,
                               float *feat_loss, float *total, void *stream);

/* Verification side of a cycle (Sec. 2.4, "Parallel Verification"), after the target model
 * has scored the draft tree under tree attention. For each sequence b of a tree built by
 * fe_build_tree (top_k candidates per level, T = 1 + N top_k nodes):
 *   pos_ids [B, T] = prefix_len[b] + depth: the nodes' sequence positions for the target's
 *            tree-attention pass (the root, the token fed to the drafter, sits right after
 *            the P_b-token prefix);
 *   the greedy acceptance walk: from the root, the child (first in node order) whose token
 *   equals target_next[b, current] — the target's greedy token after the current node —
 *   is accepted and becomes current, until no child matches:
 *   n_accept [B] accepted draft tokens (0..N), path [B, N] their node ids (-1 after),
 *   bonus [B] = target_next at the last accepted node (or the root): the target's own
 *   next token, which a cycle emits in addition.
 * All pointers are device pointers (tree: tok, parent and depth are read; mask is not);
 * target_next [B, T] int32. Asynchronous on `stream`; FE_ERR_INVALID_ARG for bad arguments.
 * Stochastic (T > 0) verification of a sampled tree is fe_verify_sampled. */
FE_API fe_status fe_verify_greedy(fe_handle *h, int32_t B, int32_t top_k, const int32_t *prefix_len,
                                  const fe_tree *tree, const int32_t *target_next, int32_t *pos_ids,
                                  int32_t *path, int32_t *n_accept, int32_t *bonus, void *stream);

/* Lossless verification of a SAMPLED draft tree (Sec. 2.4: the target verifies the tree and
 * speculative sampling finds the longest accepted path; the paper names no variant), the
 * counterpart of fe_verify_greedy for stochastic drafting. Read as recursive rejection
 * sampling over each node's children in draw order (the multi-candidate form of
 * speculative sampling, matching candidates drawn without replacement). For each sequence
 * b, from the root: with r = the target's distribution after the current node and s = the
 * drafter's proposal of the next depth, the children are tested in draw order; child c
 * with token x is accepted iff u_acc[b, c] * s(x) <= r(x); on rejection r becomes
 * max(r - s, 0) renormalised and x leaves s (renormalised). An accepted child becomes the
 * current node (r its distribution); the walk ends when every child is rejected, the node
 * has none, or N tokens are accepted, and the bonus token is the smallest x with
 * u_bonus[b, current] < r(0) + ... + r(x) (the last token with r > 0 if rounding leaves the
 * sum below u). Every emitted token then has the target's law.
 *  tree      fe_build_tree's tree (tok, parent, depth read), T = 1 + N top_k nodes
 *  topk_rank device [B, N, top_k] int32, fe_draft_forward's draw positions: node c >= 1 of
 *            the tree has draw position topk_rank[b][c - 1] (nodes in level-major order)
 *  q         device [B, N, V] float32: the drafter's proposal at each depth, softmax(l_i / T)
 *  p         device [B, T, V] float32: the target's next-token distribution after each node
 *            (given its root path), at the same temperature
 *  u_acc, u_bonus  device [B, T] float32 uniform deviates in (0, 1)
 *  path      device [B, N] int32: accepted node ids, -1 after n_accept[b]
 *  n_accept  device [B] int32; bonus device [B] int32
 * Asynchronous on `stream`; FE_ERR_INVALID_ARG for bad host-side arguments; a token or depth
 * out of range in the tree ends that sequence's walk and sets FE_ERR_DEVICE in the status
 * word. The handle holds one V-float residual buffer per sequence for it. */
FE_API fe_status fe_verify_sampled(fe_handle *h, int32_t B, int32_t top_k, const fe_tree *tree,
                                   const int32_t *topk_rank, const float *q, const float *p, const float *u_acc,
                                   const float *u_bonus, int32_t *path, int32_t *n_accept, int32_t *bonus,
                                   void *stream);

/* The update step of a cycle (Sec. 2.4, "Update and Iterate"): before the next draft can
 * attend to the positions the target accepted, each layer's cache needs their rows. For
 * each sequence b, rows i = 0 .. n_rows[b]-1 sit at positions prefix_len[b] + i; row i has
 * inputs feat[b][i] (the target's concat(l, m, h) of the position before it) and tok[b][i]
 * (the token at its position). Each row runs through Eq. 1 and the cascade exactly like a
 * drafted row (no LM head): layer l attends to cache rows 0 .. prefix_len[b] + i - 1
 * (which include the rows committed before it in this call) plus its own key and value,
 * and stores its key (after RoPE) and value, rounded to the cache type, in slot
 * prefix_len[b] + i. The call does not advance prefix_len.
 *
 *  B, L        sequences (1..max_batch) and rows per sequence in feat / tok (1..n_layers)
 *  feat        device [B, L, 3d] dtype, 16-byte aligned
 *  tok         device [B, L] int32; entries at i >= n_rows[b] are ignored
 *  n_rows      device [B] int32 in 0..L
 *  prefix_len  device [B] int32; capacity: prefix_len[b] + n_rows[b] <= max_seq
 *  k_cache, v_cache, page_table, n_pages: as for fe_draft_forward
 * Asynchronous on `stream`; FE_ERR_INVALID_ARG for bad host-side arguments, device-side
 * range errors through fe_last_device_status (as fe_draft_forward). The rows of one call
 * share one stream of the weights when B * L <= 32 (in blocks of 32 rows otherwise). */
typedef struct {
    int32_t B, L;
    const void *feat;
    const int32_t *tok;
    const int32_t *n_rows;
    const int32_t *prefix_len;
    void *const *k_cache;
    void *const *v_cache;
    const int32_t *page_table;
    int32_t n_pages;
} fe_commit_args;

FE_API fe_status fe_commit(fe_handle *h, const fe_commit_args *args, void *stream);

/* Kernel families of one draft, as fe_profile_forward reports them. */
typedef enum {
    FE_KERNEL_LINEAR = 0,    /* weight-streaming linear phase (W_fuse, W_in, W_qkv, W_o, W_gate/up, W_down) */
    FE_KERNEL_ATTENTION = 1, /* RoPE + K/V append + decode attention of one layer */
    FE_KERNEL_LM_PREP = 2,   /* tensor-core LM head: RMSNorm of the hidden rows into its bf16 operand */
    FE_KERNEL_LM_HEAD = 3,   /* LM head + softmax statistics + top-k (and its merge) */
    FE_KERNEL_COPY = 4,      /* the dbg_hidden copy */
    FE_KERNEL_LINEAR_PREP = 5, /* tensor-core linear phase: prologue into its bf16 operand */
    FE_KERNEL_TREE = 6       /* the Backbone Expansion tree (fe_profile_graph with a tree) */
} fe_kernel_kind;

/* Measurement aid: runs one draft exactly as fe_draft_forward computes it, but launched
 * eagerly (no CUDA graph, no overlap of a kernel with its predecessor) with a CUDA event
 * recorded on `stream` before the first launch and after every launch. It then waits for
 * the stream and writes, for launch j < *n_launches, its family kinds[j] (fe_kernel_kind)
 * and its device time usec[j] in microseconds (event to event). Arguments and outputs are
 * those of fe_draft_forward; kinds and usec are HOST arrays of `cap` entries, and
 * cap >= fe_launch_count(h, B, 0) + 1 is enough. Returns FE_ERR_INVALID_ARG for bad
 * arguments or too small a cap. Not for use inside stream capture. */
FE_API fe_status fe_profile_forward(fe_handle *h, const fe_forward_args *args, void *stream, int32_t cap,
                                    int32_t *kinds, float *usec, int32_t *n_launches);

/* Measurement aid: the draft timed inside the CUDA graph it really runs as. Captures (once
 * per argument set, cached like fe_draft_forward's graph) the same launch sequence as
 * fe_draft_forward, with programmatic dependent launch, plus fe_build_tree's kernel when
 * `tree` is given (tree buffers as fe_build_tree's, built from args->topk_id), and runs it
 * once on `stream`. Each kernel records, with the GPU's global nanosecond timer, when its
 * first CTA started and when its last warp exited. The call then waits for the stream and
 * writes, for launch j < *n_launches in stream order, its family kinds[j] (fe_kernel_kind),
 * start_us[j] and end_us[j]: microseconds from the earliest start of the run (-1 for a
 * launch that records nothing, the dbg_hidden copy). Because a programmatic launch starts
 * while its predecessor finishes, consecutive spans overlap; end_us[j] - end_us[j - 1] is
 * the time launch j adds to the step, and these sum to end_us of the last launch. kinds,
 * start_us, end_us: HOST arrays of `cap` entries; cap >= fe_launch_count(h, B, tree != 0)
 * + 1 is enough. Errors as fe_draft_forward, and FE_ERR_INVALID_ARG for too small a cap.
 * The stamps cost two atomic operations per CTA and warp; fe_draft_forward's own graph has
 * none. Not for use inside stream capture. */
FE_API fe_status fe_profile_graph(fe_handle *h, const fe_forward_args *args, const fe_tree *tree, void *stream,
                                  int32_t cap, int32_t *kinds, double *start_us, double *end_us,
                                  int32_t *n_launches);

/* The LM head with its fused softmax statistics and top-k (the tail of fe_draft_forward)
 * over caller-provided hidden states, for callers that cannot allocate device memory at
 * the point they need it (a frozen memory pool or arena, a path that must not call
 * cudaMalloc, a serving loop whose memory was fixed at start-up). The paper has no
 * counterpart; this is a packaging of the same kernels.
 *   hidden     device [n_layers, B, d] float32, 16-byte aligned: the cascade's hidden
 *              states (the layout of fe_forward_args.dbg_hidden)
 *   outputs    device topk_id [B, N, top_k] int32, topk_logit / topk_prob [B, N, top_k],
 *              lse [B, N] float32, as fe_draft_forward; temperature as there
 * It allocates nothing: it reads the LM head and final norm the handle already holds and
 * keeps its working memory in one fixed ~2.1 MB device array, for the life of the process.
 * fe_draft_init looks that array up on its device (cudaGetSymbolAddress), which, under
 * CUDA's default lazy module loading, is when the array is reserved; so no call of this
 * entry point allocates or looks anything up. Limits: n_layers * B <= 16, d <= 16384,
 * top_k <= 32, at most 256 vocabulary slabs; larger requests return FE_ERR_INVALID_ARG
 * (reason in fe_last_error_detail()), as does a call made with another device current than
 * the handle's. All calls share that array and leave their data in it: calls that can
 * overlap on the GPU (several streams or host threads) race and must be serialised by the
 * caller. */
FE_API fe_status fe_lm_head_topk_noalloc(fe_handle *h, const float *hidden, int32_t B, int32_t top_k,
                                         float temperature, int32_t *topk_id, float *topk_logit,
                                         float *topk_prob, float *lse, void *stream);

/* Failure-detection self-test: launches one CTA whose bounded wait on a barrier that
 * nothing completes gives up after `timeout_ns` nanoseconds (1e3..1e9) and records
 * FE_ERR_TIMEOUT in the handle's status word. The GPU stays usable. */
FE_API fe_status fe_selftest_timeout(fe_handle *h, int64_t timeout_ns, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* FE_DRAFT_H */
