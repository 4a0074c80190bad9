/*
 * msd.h - C ABI of the GB300 (sm_103a) hot path of Multimodal Speculative
 * Decoding (MSD, arXiv 2505.14260): one draft -> verify -> accept -> compact
 * decode step of a LLaVA-style decoder, greedy (T = 0) or sampling (T > 0).
 *
 * Conventions shared by every call
 * --------------------------------
 * - All pointers named *_dev are device pointers on the device that was
 *   current when msd_create ran; *_host pointers are host memory. Sizes are
 *   element counts unless stated otherwise.
 * - Weight matrices are [out, in] row-major (in contiguous), in the dtype of
 *   msd_config.dtype; norm gains are [hidden] vectors of the same dtype.
 *   Weights are BORROWED: the caller keeps them alive and unchanged for the
 *   lifetime of the context. Exception: a bf16 context (MSD_BF16) packs every
 *   projection matrix -- the target layers' and the draft layer's wq, wk, wv,
 *   wo, w_gate, w_up and w_down, plus lm_head and draft_fc -- into
 *   context-owned tile-contiguous copies during msd_create and never reads
 *   those borrowed matrices again, so the caller may free them once
 *   msd_create has returned (the copies take as many bytes as the matrices).
 *   embed and the norm gains stay borrowed. An fp32 context reads every
 *   borrowed weight on every call.
 * - The context OWNS its KV caches, tree scratch and activations (allocated
 *   once in msd_create; no call allocates afterwards).
 * - Output buffers are caller-owned device memory.
 * - Every call is asynchronous on `stream` (a cudaStream_t, 0 = legacy default
 *   stream). Argument, shape and capacity errors are returned synchronously
 *   before anything is launched. Device-detected errors (bounded waits that
 *   timed out, failed in-kernel range checks) set a device status word; the
 *   first call that observes it returns MSD_ERR_DEVICE.
 * - One context is used from one host thread and one stream at a time.
 * - Token ids are int32 in [0, vocab). Trees are stored per request with a
 *   fixed stride of N = msd_config.tree_nodes nodes; node 0 is the root.
 *
 * Notation (paper): L = tokens in the target KV cache (positions 0..L-1); the
 * root token x_L sits at position L; N tree nodes including the root; depth D
 * (number of draft passes); top-k k.
 */
#ifndef MSD_H
#define MSD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct msd_ctx msd_ctx;

typedef enum {
    MSD_OK = 0,
    MSD_ERR_INVALID = -1,   /* bad argument, shape or state */
    MSD_ERR_CAPACITY = -2,  /* a request would exceed max_seq */
    MSD_ERR_OOM = -3,       /* device allocation failed in msd_create */
    MSD_ERR_CUDA = -4,      /* a CUDA runtime call failed */
    MSD_ERR_DEVICE = -5     /* the device status word was set by a kernel */
} msd_status;

enum { MSD_F32 = 0, MSD_BF16 = 1 };

/* Draft input of a VISUAL prefix position (the three strategies of the paper's
 * ablation of the input strategy, Sec. 5.3; text positions always take
 * f_down(Concat(h_i, e_{i+1}))). Decode-step positions are generated text, so
 * the strategy only changes the draft cache built by msd_prefill. */
enum {
    MSD_DRAFT_EMBEDDING = 0,  /* MSD (Sec. 4.1, Eq. 7): the raw visual embedding e_i */
    MSD_DRAFT_CONCAT = 1,     /* Baseline (Sec. 3.3): f_down(Concat(h_i, e_{i+1})) as text */
    MSD_DRAFT_FEATURE = 2     /* Visual Feature: the target's feature h_i, no concatenation */
};

/* Model and capacity. The target is a pre-norm LLaMA-style decoder (the LLM of
 * LLaVA-1.5, Sec. 3.1); the draft model is one decoder layer of the same shape
 * plus the fc projection f_down of Eq. 4 (Sec. 3.2). */
typedef struct {
    int32_t n_layers, hidden, n_heads, head_dim, ffn, vocab;
    float rms_eps, rope_base;
    int32_t dtype;          /* MSD_F32 or MSD_BF16: weights, KV cache, GEMM operands */
    int32_t max_batch;      /* B: requests decoded together */
    int32_t max_seq;        /* cache capacity per request, in positions */
    int32_t tree_nodes;     /* N, including the root; 1 <= N <= 256 */
    int32_t tree_depth;     /* D >= 1: draft passes per step */
    int32_t topk;           /* k >= 1; k + (D-1)k^2 >= N-1 */
    int32_t draft_input;    /* MSD_DRAFT_*; 0 (zero-initialised) = MSD's Eq. 7 */
} msd_config;

/* One decoder layer: RMSNorm gains [H]; wq, wk, wv, wo [H,H];
 * w_gate, w_up [F,H]; w_down [H,F]. */
typedef struct {
    const void *attn_norm, *wq, *wk, *wv, *wo, *mlp_norm, *w_gate, *w_up, *w_down;
} msd_layer;

/* All weights (device pointers). `layers` is a HOST array of n_layers entries
 * (copied by msd_create). embed and lm_head are [V,H] (untied); draft_fc is the
 * [H, 2H] f_down of Eq. 4, applied to Concat(h, e) in that order. */
typedef struct {
    const void *embed;
    const msd_layer *layers;
    const void *final_norm;
    const void *lm_head;
    msd_layer draft;
    const void *draft_fc;
} msd_weights;

/* A token tree, device memory, per request b at stride N:
 * tokens[b*N+i], parent[b*N+i] (-1 for the root, else < i), depth[b*N+i],
 * mask[(b*N+i)*W + w] with W = ceil(N/64): bit j%64 of word j/64 is set iff
 * node j is an ancestor of node i or j == i. n_nodes[b] (nullable: all N) is the
 * number of valid nodes of request b. */
typedef struct {
    int32_t *tokens, *parent, *depth;
    uint64_t *mask;
    int32_t *n_nodes;
} msd_tree;

/* Optional record of the draft passes (device, all nullable), for parity checks.
 * Pass p = 0 is the root slot (one row per request, row 0 used); passes
 * p = 1..D-1 have k rows per request (the expanded frontier, best first).
 *   logits    [B][D][k][V] fp32  draft LM-head logits of each row
 *   topk_ids  [B][D][k][k] int32 top-k token ids of each row (ties: lower id)
 *   topk_logp [B][D][k][k] fp32  their log-probabilities                   */
typedef struct {
    float *logits;
    int32_t *topk_ids;
    float *topk_logp;
} msd_draft_record;

/* Device-side view of the context state, for tests and tooling. Layouts:
 *   target_kv  [n_layers][2][B][n_heads][max_seq][head_dim]   (K then V, K after RoPE)
 *   draft_kv   [2][B][n_heads][max_seq][head_dim]
 *   seq_len    int32 [B]  L of each request
 *   n_pending  int32 [B]  draft rows still to be caught up (draft cache = L - n_pending)
 *   root       int32 [B]  current root token x_L
 * bf16 contexts keep every cache entry (and every activation that enters a
 * tensor-core product) as a pair of bf16 values hi + lo with hi = bf16(v) and
 * lo = bf16(v - hi), which carries v to about 2^-17 relative: the lo value of
 * the element at p sits lo_offset elements after it (lo_offset = 0 for fp32
 * contexts, whose caches hold the fp32 values).                               */
typedef struct {
    void *target_kv, *draft_kv;
    int32_t *seq_len, *n_pending, *root;
    int64_t elem_bytes;
    int64_t lo_offset;
} msd_state_view;

/* Creates a context on the current device: validates the configuration,
 * copies the weight pointer table, allocates caches and scratch.
 * Errors: MSD_ERR_INVALID (bad config or null weight), MSD_ERR_OOM. */
msd_status msd_create(const msd_config *cfg, const msd_weights *w, msd_ctx **out);

/* Frees everything the context owns. Safe on NULL. */
msd_status msd_destroy(msd_ctx *ctx);

/* Prefill (Sec. 3.1, Eq. 1-3; draft input of Eq. 7). For each request b <
 * batch: ids_dev[b*ids_stride + i], i < seq_len_host[b], is the interleaved
 * prompt, with -1 marking a visual slot; visual slots consume rows of
 * vis_dev ([rows][H], model dtype) in order starting at row vis_off_host[b].
 * Runs the target over the prompt (filling its KV cache), writes the root token
 * x_L = argmax of the last position's logits to root_out_dev[b], and builds the
 * draft cache over positions 0..L-2 with f = f_down(Concat(h, e_next)) at text
 * positions and, at visual positions, f = e (Eq. 7; or the strategy chosen by
 * msd_config.draft_input).
 * Errors: MSD_ERR_INVALID (batch out of range, empty prompt, prompt not ending
 * in a text token), MSD_ERR_CAPACITY (L + 1 + N > max_seq). Resets all state. */
msd_status msd_prefill(msd_ctx *ctx, int32_t batch, const int32_t *seq_len_host,
                       const int32_t *ids_dev, int32_t ids_stride,
                       const void *vis_dev, const int64_t *vis_off_host,
                       int32_t *root_out_dev, void *stream);

/* Draft tree (Sec. 3.2 feature-level draft phase, Eq. 4-5, with the MSD input
 * of Eq. 7). Pass 1 catches the draft cache up over the positions accepted by
 * the last step (root slot last) and gives the depth-1 candidates (top-k of the
 * root slot's distribution); passes 2..D expand the k best frontier nodes with
 * top-k children each, score = sum of log-probabilities; the N-1 best
 * candidates form the tree (index 1 + rank; ties: higher score, lower depth,
 * earlier creation). Writes the tree to *out (caller-owned device arrays of
 * the layout above; n_nodes, if given, is set to N). rec is nullable. */
msd_status msd_draft_tree(msd_ctx *ctx, const msd_tree *out,
                          const msd_draft_record *rec, void *stream);

/* Verify (Sec. 3.2 verification phase): one target forward over all tree
 * tokens, node i at position L + depth(i), attending to the whole prefix and to
 * its ancestors and itself. `tree` is the drafted tree or any caller-planted
 * tree with tokens[b*N] == the current root. Writes the target argmax of every
 * node to argmax_dev[b*N+i] (ties: lower id) and, if logits_dev is not NULL,
 * the fp32 logits [B][N][V]. Tree K/V are kept in context scratch for
 * msd_accept_compact. */
msd_status msd_verify(msd_ctx *ctx, const msd_tree *tree, int32_t *argmax_dev,
                      float *logits_dev, void *stream);

/* Completes a caller-planted tree (the draft-tree structure of Sec. 3.2: a
 * candidate is conditioned on its ancestors): for request b = `request` (or
 * every request b < max_batch if request is -1), from parent[b*N+i] of its n_nodes[b] nodes (all N if n_nodes is NULL) it
 * writes depth[b*N+i] (the number of ancestors) and the ancestor-or-self mask
 * words of the layout above; nodes at or past n_nodes[b] get depth 0 and an
 * empty mask. tokens are not read. A node whose parent does not precede it
 * (parent[b*N+i] outside [0, i) for i > 0, or a root with a parent) sets the
 * device status word (reported by the next call as MSD_ERR_DEVICE) and is
 * treated as a child of the root. Errors: MSD_ERR_INVALID (null arrays, request
 * outside [-1, max_batch)). */
msd_status msd_tree_complete(msd_ctx *ctx, const msd_tree *tree, int32_t request, void *stream);

/* Accept and compact (Eq. 6 at temperature 0, and the rule that rejected
 * drafts are discarded): from the root, follow the child whose token equals the
 * target argmax at the current node; path_dev[b*(D+1)+j] (j <= a, rest -1),
 * accept_len_dev[b] = a, bonus_dev[b] = argmax at the last accepted node. The
 * K/V of path[j] move to cache position L+j; L <- L + a + 1; the bonus becomes
 * the new root. index_map_dev (nullable) [b*(D+1)+j] = L_old + j for j <= a,
 * else -1. `tree` and `argmax_dev` must be those of the preceding msd_verify. */
msd_status msd_accept_compact(msd_ctx *ctx, const msd_tree *tree,
                              const int32_t *argmax_dev, int32_t *path_dev,
                              int32_t *accept_len_dev, int32_t *bonus_dev,
                              int32_t *index_map_dev, void *stream);

/* Accept and compact at temperature T > 0: speculative sampling over the tree
 * (Sec. 3.2, Eq. 6 and the adjusted distribution norm(max(0, p - q)) after it).
 * The target distribution at node i is p = softmax(logits[b][i] / T). The
 * tree's candidates are the draft's top-k choices, not draws from q, so the
 * proposal of a child -- given its siblings already rejected -- is a point mass
 * at its token x: Eq. 6 accepts it with probability p_adj(x), and the adjusted
 * distribution is p_adj with x removed and renormalised (p_adj = p at first).
 * From the root, the children of the current node are tried in tree order
 * (index order: best draft score first) with u_dev[(b*(D+1) + d)*(k+1) + j]
 * for the j-th child tried at depth d (d = drafts accepted so far); an accepted
 * child becomes the current node. When all of a node's children are rejected,
 * or it has none, the next token (the bonus) is drawn from p_adj by inverse CDF
 * in token-id order: the smallest token whose cumulative mass exceeds
 * u_dev[(b*(D+1) + d)*(k+1) + k] times the remaining mass.
 * logits_dev: the fp32 [B][N][V] logits of the preceding msd_verify -- the
 * same pointer that call was given, or NULL if it was given NULL (the context
 * keeps them then). u_dev: [B][D+1][k+1] fp32 uniforms in [0, 1), device,
 * caller-owned (the random numbers are inputs, so a step is reproducible).
 * temperature: finite, > 0. vocab <= 393216. A node with more than k children in a
 * caller-planted tree has only its first k tried and sets the device status.
 * Decisions are taken on the fp32 logits with fp32 exponentials and
 * error-free (fp32 pair / fp64) sums: they agree with an exact evaluation
 * except where a uniform lies within about 1e-6 (relative) of a boundary.
 * Launches two kernels (per-row statistics of all N rows, then the walk and
 * the draw, one CTA per request) and uses context scratch for the statistics.
 * Outputs, compaction and state update as msd_accept_compact (path, accepted
 * length a, bonus = the drawn token, index map). Errors: MSD_ERR_INVALID (null
 * tree or u_dev, bad temperature, no prefill), MSD_ERR_CAPACITY,
 * MSD_ERR_DEVICE, MSD_ERR_CUDA. */
msd_status msd_accept_sample(msd_ctx *ctx, const msd_tree *tree, const float *logits_dev,
                             float temperature, const float *u_dev, int32_t *path_dev,
                             int32_t *accept_len_dev, int32_t *bonus_dev, int32_t *index_map_dev,
                             void *stream);

/* One whole decode step: msd_draft_tree, msd_verify and msd_accept_compact in
 * sequence (Sec. 3.2; Eq. 6 at T = 0), with the same arguments and outputs as
 * those calls (the drafted tree is written to *tree and then verified). The
 * context records the sequence once into a CUDA graph per set of output
 * buffers and replays it, so a step is one graph launch (every kernel reads
 * the lengths it needs from device state; the first step with new buffers
 * records the graph, host work of a few milliseconds). While GEMM profiling
 * mode 1 is enabled the calls run without a graph; mode 2 replays graphs
 * recorded with launch stamps (msd_profile_enable). Errors: as for the three
 * calls, and MSD_ERR_CUDA if the graph cannot be recorded. */
msd_status msd_step(msd_ctx *ctx, const msd_tree *tree, int32_t *argmax_dev, int32_t *path_dev,
                    int32_t *accept_len_dev, int32_t *bonus_dev, void *stream);

/* One whole decode step at temperature T > 0: msd_draft_tree, msd_verify (its
 * logits kept in the context) and msd_accept_sample, recorded and replayed as a
 * CUDA graph exactly as msd_step (one graph per set of buffers, u_dev pointer,
 * and temperature). The caller refills u_dev
 * ([B][D+1][k+1] uniforms in [0, 1)) before each step; the graph reads it when
 * it runs. Errors: as msd_step, and MSD_ERR_INVALID for a null u_dev, a
 * temperature that is not finite and > 0, or vocab > 393216 (as
 * msd_accept_sample). */
msd_status msd_step_sample(msd_ctx *ctx, const msd_tree *tree, float temperature,
                           const float *u_dev, int32_t *argmax_dev, int32_t *path_dev,
                           int32_t *accept_len_dev, int32_t *bonus_dev, void *stream);

/* Plain greedy autoregressive decoding, the baseline against which the paper
 * measures its speedup ratio (Sec. 4.1, Eq. 9: T_p, the target's time per
 * generated token): one target forward over each request's current root token
 * at position L, its K/V appended to the cache at L, L <- L + 1, and the argmax
 * (ties: lower id) becomes the new root and is written to token_dev[b] (B int32,
 * device). The same kernels as msd_verify and msd_accept_compact run it (a
 * tree of the root alone), recorded once into a CUDA graph per token_dev and
 * replayed, as msd_step. A context created with
 * tree_nodes = 1 runs it on B token rows; with more tree nodes the other rows
 * are computed and ignored. The draft is not run, so after this call the draft
 * cache no longer follows the target's: msd_draft_tree and msd_step return
 * MSD_ERR_INVALID until the next msd_prefill. Errors: MSD_ERR_INVALID (null
 * token_dev, no prefill), MSD_ERR_CAPACITY, MSD_ERR_DEVICE, MSD_ERR_CUDA, as
 * for msd_step. */
msd_status msd_ar_step(msd_ctx *ctx, int32_t *token_dev, void *stream);

/* Building block used by every projection of the step (Sec. 3.1 decoder
 * layers, Eq. 4 f_down, Eq. 5 LM head), exposed for tests and kernel timing:
 * y[i][j] (= or, if accumulate != 0, +=) sum_t x[i][t] * w[j][t] for i < m,
 * j < o, t < k. x [m][ldx] and w [o][k] are in the context dtype (bf16 rows
 * 16-byte aligned: ldx and k multiples of 8), y [m][ldy] is fp32; all device.
 * bf16 runs on the tcgen05 tensor-core GEMM of the step: w is first re-laid
 * into the context's packing scratch (grown on demand, so this call may
 * allocate), then multiplied; fp32 runs on the CUDA-core GEMM.
 * Errors: MSD_ERR_INVALID on null pointers, non-positive sizes or bad strides,
 * MSD_ERR_OOM if the packing scratch cannot grow. */
msd_status msd_linear(msd_ctx *ctx, const void *x_dev, int32_t ldx, int32_t m, int32_t k,
                      const void *w_dev, int32_t o, float *y_dev, int32_t ldy,
                      int32_t accumulate, void *stream);

/* Allocation-free GEMM: the same y (=|+=) x w^T as msd_linear for bf16
 * operands, for callers that cannot allocate device memory (a host program
 * whose device memory is all owned by its own pool allocator, code running
 * where an allocation would synchronise the device or is not permitted, a
 * plug-in handed buffers but no allocator). It needs no context and allocates
 * nothing: its scratch is one static device array (a 256-byte status word,
 * 4096 int tile tickets and 16 MiB of fp32 split-K partials) which every GPU
 * that loads this library holds until the process exits. The paper has no
 * counterpart; this is a service of the library, not a step of the method.
 * Arguments are those of msd_linear (x [m][ldx], w [o][k] bf16 with ldx and k
 * multiples of 8, y [m][ldy] fp32, all device memory on the current device).
 * The split-K choice is limited to what the array holds: a shape whose best
 * split would need more partials or tickets runs with fewer splits (none at
 * worst), so no shape is refused for its scratch. The first call made on a
 * device looks up the array's device address on that device
 * (cudaGetSymbolAddress) and sets the kernel's shared-memory limit; make that
 * first call before any stream capture. Every call shares the array and it
 * keeps the last call's contents; the tile tickets are cleared on `stream`
 * before each launch that uses them. Calls that overlap on the GPU (other
 * streams, other host threads) race on the array: serialise them.
 * Device-side errors: a bounded wait of the kernel that runs out (2 s) sets the
 * array's status word. Each call first reads that word back on `stream` (so it
 * returns only after the work queued before it on `stream` has finished); if it
 * is set, the call clears it, launches nothing and returns MSD_ERR_DEVICE: the
 * failed call's y is not to be trusted.
 * Errors: MSD_ERR_INVALID (null pointer, non-positive size, bad stride or
 * alignment), MSD_ERR_CAPACITY (m > 65535 * 256, the token-tile grid limit),
 * MSD_ERR_DEVICE (see above), MSD_ERR_CUDA (a runtime call failed). */
msd_status msd_linear_noalloc(const void *x_dev, int32_t ldx, int32_t m, int32_t k,
                              const void *w_dev, int32_t o, float *y_dev, int32_t ldy,
                              int32_t accumulate, void *stream);

/* Test hook of the failure detection (no counterpart in the paper): launches
 * one CTA that waits, through the library's bounded mbarrier wait, on a
 * barrier that nothing ever arrives at; after limit_ns (1e3 .. 2e9) it gives up
 * and records a timeout in the device status word of ctx -- or, for ctx NULL,
 * in the status word of msd_linear_noalloc on the current device. No copy or
 * MMA is in flight during the wait, so nothing else is disturbed; the next call
 * on that context (or the next msd_linear_noalloc) reports MSD_ERR_DEVICE.
 * Errors: MSD_ERR_INVALID (limit out of range), MSD_ERR_CUDA. */
msd_status msd_test_wait_timeout(msd_ctx *ctx, int64_t limit_ns, void *stream);

/* Profiling counters (tracing subsystem). kernel_launches counts every kernel
 * the library has run in this process (kernels executed by step graphs
 * included, kernels merely recorded into graphs excluded).
 *
 * msd_profile_enable(ctx, mode) times the tensor-core GEMM launches of a bf16
 * context:
 *   mode 0  off.
 *   mode 1  each GEMM launch is bracketed by CUDA events on its own stream;
 *           step calls run as separate launches instead of their graphs.
 *           gemm_ms = the events' summed durations.
 *   mode 2  step calls replay graphs recorded with launch stamps: each CTA of
 *           a GEMM launch stamps a device slot with %globaltimer (earliest
 *           entry, earliest return from the wait on the previous kernel,
 *           latest exit) and the graph's last kernel adds the step's spans to
 *           a device sum, so the step runs as it does unprofiled (the same
 *           graph, programmatic dependent launches included) plus those atomics.
 *           gemm_ms = sum of exit - entry over launches; gemm_critical_ms =
 *           sum of exit - wait (these intervals are disjoint for the kernels of
 *           one stream, so their sum never exceeds the steps' time); windows =
 *           steps measured. Stamped graphs are cached apart from the others.
 * msd_profile_read synchronises the device, returns the launches timed since
 * the last read, their time and their algorithmic bytes (every weight element
 * once + activations read + output written, read too when accumulating), and
 * starts a new window. Enabling either mode also starts a new window.
 * The stamp buffers are made with the context; enabling allocates nothing.
 * Errors: MSD_ERR_INVALID (mode out of range), MSD_ERR_CUDA (the stamp reset failed). */
typedef struct {
    int64_t kernel_launches;
    int64_t gemm_launches;
    double gemm_ms;
    double gemm_bytes;
    double gemm_weight_bytes;
    double gemm_critical_ms;
    int64_t windows;
    double gemm_flops;       /* 2 x rows x outputs x inner size, summed */
    double gemm_mma_flops;   /* as issued to the tensor cores: twice gemm_flops
                                for launches whose token operand is a split pair */
    double gemm_prefetch_bytes; /* weight bytes the launches request before they
                                   wait for the previous kernel (part of gemm_bytes) */
} msd_profile;

msd_status msd_profile_enable(msd_ctx *ctx, int32_t mode);
msd_status msd_profile_read(msd_ctx *ctx, msd_profile *out);

/* Per-launch breakdown of mode 2 (the tracing subsystem's timeline of the
 * replayed step). Every launch of a stamped step graph owns a slot: its
 * tensor-core GEMMs in launch order, then its tree-attention launches (whose
 * CTAs stamp entry, wait and exit the same way). msd_profile_slots copies, for
 * each slot of the last stamped graph recorded, the sums over the steps
 * replayed since the last call of exit - wait (critical_ms) and exit - entry
 * (span_ms), with the launch's shape, then clears the sums. Slot i describes
 * the i-th stamped launch of that graph; graphs recorded with another launch
 * sequence (the sampling step) sum into the same slots, so read once per kind
 * of step. *n = slots written (at most max). Outside mode 2, *n = 0.
 * Errors: MSD_ERR_INVALID (null ctx or n, max < 0, null out with max > 0),
 * MSD_ERR_CUDA. */
typedef struct {
    int32_t kind;         /* 0 tensor-core GEMM, 1 tree attention */
    int32_t rows;         /* GEMM: token rows M; attention: query rows */
    int32_t outputs;      /* GEMM: output features O; attention: heads */
    int32_t inner;        /* GEMM: inner size K; attention: head dim */
    int64_t launches;     /* stamped launches summed (steps replayed) */
    double bytes;         /* GEMM: algorithmic bytes of one launch; attention: 0
                             (its bytes follow the visible prefix of each step) */
    double critical_ms;   /* sum of exit - wait */
    double span_ms;       /* sum of exit - entry */
} msd_kernel_slot;

msd_status msd_profile_slots(msd_ctx *ctx, msd_kernel_slot *out, int32_t max, int32_t *n);

/* Device pointers of the context state (see msd_state_view). */
msd_status msd_state(msd_ctx *ctx, msd_state_view *out);

/* Text of the last error on this context ("" if none). Never NULL. */
const char *msd_last_error(const msd_ctx *ctx);

#ifdef __cplusplus
}
#endif

#endif /* MSD_H */
