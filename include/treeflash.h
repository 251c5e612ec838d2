/*
 * treeflash.h - C ABI of the TreeFlash drafting hot path on one GB300 (sm_103a).
 *
 * TreeFlash ("Parallel AR-Approximation for Faster Speculative Decoding") drafts a tree of
 * B candidate tokens from the gamma hidden states h_{t+1..t+gamma} that a one-shot block
 * drafter produces in a single forward pass. Algorithm 1 (App. B, "AR-approximated OPT-Tree
 * construction") has two parts, and this library runs both on the GPU:
 *
 *   Part 1, stage 1  (tf_stage1_marginals)  q_{t+i} = LMHead(h_{t+i}); TopM per depth.
 *   Part 1, stage 2  (tf_stage2_ar_approx)  h' = h + SwiGLU(h~ :: e) (Eq. 1) on 1 + M(gamma-1)
 *                                           rows, each through the LM head, log-softmax, top-K2.
 *   Part 2           (tf_build_tree)        OPT-Tree best-first selection of B nodes (Sec. 3,
 *                                           "Inference"), the M-ary rule for non-leaves.
 *   verification     (tf_tree_mask)         ancestor mask and position ids for the verifier's
 *                                           single parallel pass over the tree (Sec. 1, Sec. 3).
 *   Part 2 + mask    (tf_build_tree_mask)   both of the above; one launch for B + 1 <= 128.
 *
 * Conventions shared by every call:
 *  - Pointers are DEVICE pointers owned by the caller unless a parameter says "host". The
 *    library allocates no memory and keeps no state between calls; scratch lives in the
 *    caller's workspace (tf_workspace_size). The one exception is the fixed scratch array of
 *    tf_stage1_marginals_static (end of this file). Calls are asynchronous on `stream` (NULL = the
 *    legacy default stream) and return once the work is queued.
 *  - Shapes are row-major. b = batch (independent sequences), d = hidden size, V = vocabulary,
 *    I = approximator width, gamma = block size, M = stage-1 candidates per depth, K2 =
 *    children kept per stage-2 row, B = draft budget (non-root nodes),
 *    R = 1 + M (gamma - 1) stage-2 rows per sequence (TF_APPROX_SWIGLU_2PREV: 1 + M +
 *    M^2 (gamma - 2) for gamma >= 2), K1 = max(M, K2).
 *  - Float tensors have the element type of dims->dtype (TF_BF16: __nv_bfloat16, TF_F32:
 *    float); log-probabilities are always float32, token ids int32.
 *  - Errors: a call that finds an invalid argument returns TF_ERR_INVALID_ARG,
 *    TF_ERR_UNSUPPORTED or TF_ERR_WORKSPACE before queueing anything; a failed launch returns
 *    TF_ERR_CUDA. Conditions only the GPU can see (an out-of-range token id, an underfull
 *    candidate universe, a bounded wait that gave up) are OR-ed into device status words
 *    (TF_DEV_* bits) that the caller reads after synchronising. No call aborts the process.
 *  - Ties (the paper is silent): inside a distribution the larger value comes first, then the
 *    smaller token id; in the queue the larger path score, then the smaller depth, then the
 *    smaller parent index, then the smaller token id.
 */
#ifndef TREEFLASH_H
#define TREEFLASH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t; declared here so the header needs no CUDA include. */
typedef struct CUstream_st* tf_stream_t;

typedef enum {
    TF_OK = 0,
    TF_ERR_INVALID_ARG = 1,   /* null pointer, inconsistent or out-of-range dimension */
    TF_ERR_UNSUPPORTED = 2,   /* valid but outside what the kernels implement (see limits) */
    TF_ERR_WORKSPACE = 3,     /* workspace null, too small or not 256-byte aligned */
    TF_ERR_CUDA = 4,          /* a CUDA runtime/driver call or a kernel launch failed */
    TF_ERR_DEVICE_STATUS = 5, /* tf_status_read found TF_DEV_* flags set */
    TF_ERR_TIMEOUT = 6        /* tf_status_read found TF_DEV_TIMEOUT set */
} tf_status;

typedef enum { TF_BF16 = 0, TF_F32 = 1 } tf_dtype;

typedef enum {
    TF_MODE_AR = 0,            /* TreeFlash: stage-2 conditional rows, M-ary rule (Alg. 1) */
    TF_MODE_MARGINAL = 1,      /* DDTree baseline: OPT-Tree on the stage-1 marginals, every
                                  node expandable (Sec. 4 "Baselines") */
    TF_MODE_MARGINAL_MARY = 2  /* stage-1 marginals under the M-ary rule: what TF_MODE_AR
                                  computes when the approximator is zero (Sec. 3 "Training") */
} tf_mode;

/* Which AR-approximator stage 2 runs (TF_MODE_AR only). */
typedef enum {
    TF_APPROX_SWIGLU = 0,      /* Eq. 1: h' = h + W_down (SiLU(W_gate x) * (W_up x)), x = [h~ ; e] */
    TF_APPROX_LINEAR = 1,      /* the "w/ Linear" ablation (Sec. 4 "Model Design", Table 3): the
                                  SwiGLU replaced by one linear layer on the same input,
                                  h' = h + W_lin x, W_lin [d, 2d], no bias */
    TF_APPROX_SWIGLU_2PREV = 2 /* the "w/ 2-prev" ablation (Sec. 4 "Model Design", Table 3): the
                                  SwiGLU of Eq. 1 on x = [h~ ; e(prev) ; e(token before prev)]
                                  (both embeddings normalised with norm_e), W_gate and W_up
                                  [I, 3d]. Stage 2 then has one row per pair of M-ary candidates
                                  (R = 1 + M + M^2 (gamma - 2), see tf_stage2_ar_approx), and
                                  root_tok holds TWO tokens per sequence, [b, 2] = (x_t, x_{t-1}),
                                  in every call that takes it */
} tf_approx;

/* Device status bits (int32 words written with atomic OR). */
enum {
    TF_DEV_BAD_TOKEN = 1,      /* a token id outside [0, V) was read; the row/node is skipped */
    TF_DEV_UNDERFULL = 2,      /* fewer than B candidates exist; missing nodes are marked */
    TF_DEV_NONFINITE = 4,      /* a non-finite logit or score was seen */
    TF_DEV_TIMEOUT = 8,        /* a bounded wait inside a kernel gave up; outputs invalid */
    TF_DEV_RECOMPUTED = 16     /* informational: a top-k list was recomputed exactly */
};

typedef struct {
    int32_t batch;        /* b >= 1 */
    int32_t d;            /* hidden size; TF_BF16 needs d % 64 == 0, TF_F32 d % 4 == 0 */
    int32_t V;            /* vocabulary size, K1 <= V < 2^31 */
    int32_t I;            /* approximator intermediate width; TF_BF16 needs I % 64 == 0 */
    int32_t gamma;        /* block size (max depth), 1..64 */
    int32_t M;            /* stage-1 candidates per depth (M-ary branching), 1..64 */
    int32_t K2;           /* children kept per distribution, 1..512; K2 >= B is exact */
    int32_t B;            /* draft budget (nodes besides the root), 1..1023 */
    float temperature;    /* logits are W_lm x / temperature, temperature > 0 */
    float rms_eps;        /* RMSNorm epsilon of Eq. 1's normalisations */
    int32_t dtype;        /* tf_dtype */
    int32_t mode;         /* tf_mode */
    int32_t approx;       /* tf_approx (0 = Eq. 1's SwiGLU); read only in TF_MODE_AR. With
                             TF_APPROX_LINEAR, I is ignored */
} tf_dims;

/* Model parameters (device, dims->dtype, row-major, read only, never copied). */
typedef struct {
    const void* lm_head;  /* [V, d]  verifier output embedding W_lm */
    const void* embed;    /* [V, d]  verifier input embedding Embd */
    const void* norm_h;   /* [d]     RMSNorm weight of the hidden-state half of Eq. 1 */
    const void* norm_e;   /* [d]     RMSNorm weight of the embedding half of Eq. 1 */
    const void* w_gate;   /* [I, 2d] SwiGLU gate projection, input [h~ ; e] ([I, 3d] with
                             TF_APPROX_SWIGLU_2PREV, input [h~ ; e ; e2]) */
    const void* w_up;     /* [I, 2d] SwiGLU up projection, input [h~ ; e] ([I, 3d] likewise) */
    const void* w_down;   /* [d, I]  SwiGLU down projection */
    const void* w_lin;    /* [d, 2d] linear approximator, input [h~ ; e] (TF_APPROX_LINEAR only;
                             w_gate, w_up and w_down are then not read and may be NULL) */
} tf_weights;

/* Human-readable name of a status code (static storage). */
const char* tf_status_string(tf_status status);

/* Library version as major*10000 + minor*100 + patch. */
int32_t tf_version(void);

/* Number of kernels this library has launched in the calling process since it was loaded, over
 * all devices and streams (a host-side counter; host only, no GPU work). Lets a caller count
 * the kernels of a timed region: read it before and after. */
uint64_t tf_kernel_launches(void);

/* Failure detection. Every wait inside the tensor-core kernels (a TMA copy landing, an MMA
 * finishing, an accumulator being drained) gives up after a time limit, 2 s by default: the
 * kernel then sets TF_DEV_TIMEOUT in the status word, waits (again bounded, always 2 s) for
 * its own copies and MMAs in flight, frees its tensor memory and returns, so the context stays
 * usable and tf_status_read reports TF_ERR_TIMEOUT. This sets the limit of those waits for
 * progress for every later launch in the process (ns = 0 restores the default); the waits that
 * drain in-flight work keep 2 s. A limit shorter than a copy's latency makes every call time
 * out, which is how the failure path is tested. Host only; returns TF_ERR_INVALID_ARG above
 * 60 s. It does not cover calls already enqueued. */
tf_status tf_set_wait_limit_ns(uint64_t ns);

/* Validate `dims` and return the workspace bytes every call below needs for these dims
 * (the maximum over all calls, so one buffer serves the whole step). Host only; no GPU
 * work. The workspace must be device memory, 256-byte aligned, and must not be used by two
 * calls that overlap on the GPU. */
tf_status tf_workspace_size(const tf_dims* dims, size_t* bytes);

/* Zero the workspace's status word (asynchronous). tf_stage1_marginals does this itself. */
tf_status tf_status_reset(void* ws, size_t ws_bytes, tf_stream_t stream);

/* Synchronise `stream`, copy the workspace's status word to *flags (host) and return
 * TF_ERR_TIMEOUT if TF_DEV_TIMEOUT is set, TF_ERR_DEVICE_STATUS if any other error bit is
 * set (TF_DEV_RECOMPUTED alone is not an error), TF_OK otherwise. */
tf_status tf_status_read(const void* ws, size_t ws_bytes, int32_t* flags, tf_stream_t stream);

/* Stage 1 of Algorithm 1 Part 1: for every sequence s and depth i,
 *   q_{t+i} = softmax(W_lm h_{t+i} / T) and its K1 largest entries.
 *  hidden   [b, gamma, d] dtype: the drafter's hidden states h_{t+1..t+gamma}.
 *  top_ids  [b, gamma, K1] int32 out: token ids in the tie order above; the first M are the
 *           candidates x^(1..M)_{t+i} of the M-ary tree.
 *  top_logp [b, gamma, K1] float out: log q_{t+i}(top_ids), exact log-softmax over all V.
 * Resets the workspace status word. */
tf_status tf_stage1_marginals(const tf_dims* dims, const tf_weights* w, const void* hidden,
                              int32_t* top_ids, float* top_logp,
                              void* ws, size_t ws_bytes, tf_stream_t stream);

/* Stage 2 of Algorithm 1 Part 1 (Eq. 1): for every sequence, R rows
 *   row 0:                 h' = h_{t+1} + SwiGLU(RMSNorm(h_{t+1}) :: RMSNorm(Embd(x_t)))
 *   row 1 + (i-2) M + m:   h' = h_{t+i} + SwiGLU(RMSNorm(h_{t+i}) :: RMSNorm(Embd(x^(m)_{t+i-1})))
 * for i = 2..gamma, m = 0..M-1, then q' = softmax(W_lm h' / T) and its K2 largest entries.
 * With dims->approx == TF_APPROX_LINEAR, W_lin (...) takes the place of SwiGLU(...).
 * With TF_APPROX_SWIGLU_2PREV the input also holds RMSNorm(Embd(token before prev)) and the
 * rows are (root_tok [b, 2] = (x_t, x_{t-1}))
 *   row 0:                          depth 1, tokens (x_t, x_{t-1})
 *   row 1 + m:                      depth 2, tokens (x^(m)_{t+1}, x_t)
 *   row 1 + M + (i-3) M^2 + m1 M + m2: depth i >= 3, tokens (x^(m1)_{t+i-1}, x^(m2)_{t+i-2}).
 *  hidden     [b, gamma, d] dtype (as in stage 1)
 *  root_tok   [b] int32: the last accepted token x_t of each sequence ([b, 2] = (x_t, x_{t-1})
 *             with TF_APPROX_SWIGLU_2PREV)
 *  top_ids    [b, gamma, K1] int32: stage-1 output (the first M per depth are used)
 *  child_ids  [b, R, K2] int32 out, child_logp [b, R, K2] float out (exact log-softmax).
 * h' is kept in the workspace (bf16 path: rounded to bf16, as the MLP's output type).
 * Requires dims->mode == TF_MODE_AR. */
tf_status tf_stage2_ar_approx(const tf_dims* dims, const tf_weights* w, const void* hidden,
                              const int32_t* root_tok, const int32_t* top_ids,
                              int32_t* child_ids, float* child_logp,
                              void* ws, size_t ws_bytes, tf_stream_t stream);

/* Algorithm 1 Part 2 (OPT-Tree selection, Sec. 3): one warp per sequence grows the tree by
 * popping the candidate of highest cumulative log-probability B times. The root's children
 * are row 0 of child_ids (TF_MODE_AR) or depth 1 of top_ids (marginal modes). A popped node
 * at depth i < gamma whose token is x^(m)_{t+i} (m < M) makes row 1 + (i-1) M + m available
 * (TF_MODE_AR); in TF_MODE_MARGINAL every node at depth i < gamma makes stage-1 depth i+1
 * available, in TF_MODE_MARGINAL_MARY only the M-ary ones do. Each distribution contributes
 * at most K2 children (exact when K2 >= B). With TF_APPROX_SWIGLU_2PREV a node of depth i whose
 * token is x^(m)_{t+i} and whose parent's token is x^(m')_{t+i-1} takes row
 * 1 + M + (i-2) M^2 + m M + m' (row 1 + m at depth 1), and root_tok is [b, 2] (x_t first).
 * child_ids/child_logp may be NULL in the marginal modes. Outputs [b, B+1]: node 0 is the
 * root (token x_t, parent -1, depth 0, score 0); nodes follow in pop order, so parent < child. Missing nodes (underfull universe) have
 * token/parent/depth -1 and score -inf, and set TF_DEV_UNDERFULL.
 *  dev_status [b] int32 out: TF_DEV_* bits per sequence (overwritten, not OR-ed). */
tf_status tf_build_tree(const tf_dims* dims, const int32_t* root_tok,
                        const int32_t* top_ids, const float* top_logp,
                        const int32_t* child_ids, const float* child_logp,
                        int32_t* node_tok, int32_t* node_parent, int32_t* node_depth,
                        float* node_score, int32_t* dev_status, tf_stream_t stream);

/* Tree-attention mask and position ids for verifying the tree in one forward pass:
 *  mask [b, B+1, B+1] uint8 out: mask[s][i][j] = 1 iff node j is node i or an ancestor.
 *  pos_ids [b, B+1] int32 out: root_pos[s] + depth; -1 for missing nodes (all-zero rows and
 *  columns in the mask).  root_pos [b] int32. */
tf_status tf_tree_mask(const tf_dims* dims, const int32_t* node_parent, const int32_t* node_depth,
                       const int32_t* root_pos, uint8_t* mask, int32_t* pos_ids,
                       tf_stream_t stream);

/* tf_build_tree followed by tf_tree_mask, with the same arguments and results: the two outputs
 * of both calls, bit for bit. When B + 1 <= 128 the mask and position ids are written by the
 * builder itself from the tree it holds (one launch instead of two); larger trees run both
 * launches. root_pos [b] int32; mask [b, B+1, B+1] uint8 and pos_ids [b, B+1] int32 out, as in
 * tf_tree_mask. */
tf_status tf_build_tree_mask(const tf_dims* dims, const int32_t* root_tok, const int32_t* root_pos,
                             const int32_t* top_ids, const float* top_logp,
                             const int32_t* child_ids, const float* child_logp,
                             int32_t* node_tok, int32_t* node_parent, int32_t* node_depth,
                             float* node_score, uint8_t* mask, int32_t* pos_ids,
                             int32_t* dev_status, tf_stream_t stream);

/* The whole drafting step for callers holding the step's inputs in HOST memory: copies hidden to
 * the device, runs stage 1, stage 2 (TF_MODE_AR) and tf_build_tree_mask, brings the tree, mask
 * and status back, and synchronises `stream`.
 * With page-locked host buffers (cudaHostAlloc, or torch's pin_memory) that the device can
 * address, the kernels read root_tok and root_pos and write every output in host memory
 * directly; other buffers go through the workspace and copies. On a created stream (not the
 * legacy default stream) with page-locked buffers, the first call with a given set of arguments
 * (dims, weight, buffer and workspace pointers, device, wait limit) captures the step as a CUDA
 * graph and later calls replay it: the buffers' contents may change between calls, their
 * addresses may not without a new capture. The library keeps the last 8 such graphs (the CUDA
 * driver instantiates them; the library itself allocates no memory); a capture that fails leaves
 * the step on plain launches. The call must not itself be made inside a stream capture (it
 * synchronises).
 * Host inputs: hidden [b, gamma, d] dtype, root_tok [b] ([b, 2] with TF_APPROX_SWIGLU_2PREV),
 * root_pos [b]. Host outputs:
 * node_tok, node_parent, node_depth [b, B+1] int32, node_score [b, B+1] float,
 * mask [b, B+1, B+1] uint8, pos_ids [b, B+1] int32, dev_status [b] int32 (per-sequence bits
 * OR-ed with the workspace status word). Weights stay on the device. The workspace size is
 * the same tf_workspace_size. Returns TF_ERR_TIMEOUT / TF_ERR_DEVICE_STATUS like
 * tf_status_read when an error bit is set. */
tf_status tf_draft_tree_host(const tf_dims* dims, const tf_weights* w, const void* hidden,
                             const int32_t* root_tok, const int32_t* root_pos,
                             int32_t* node_tok, int32_t* node_parent, int32_t* node_depth,
                             float* node_score, uint8_t* mask, int32_t* pos_ids,
                             int32_t* dev_status, void* ws, size_t ws_bytes, tf_stream_t stream);

/* The verification step that follows drafting (Sec. 3: token selection is deterministic, so
 * the verifier accepts a drafted token exactly when it equals its own next token at that
 * position; Sec. 4: block efficiency tau counts the accepted tokens plus the verifier's
 * residual token). For every sequence, from the root, move to the child of the current node
 * whose token equals the verifier's token at the current node, while one exists.
 *  node_tok, node_parent [b, B+1] int32: a drafted tree (as tf_build_tree writes it; missing
 *                nodes have parent -1 and are never accepted)
 *  verifier_tok [b, B+1] int32: the verifier's next token at each node's position, i.e. its
 *                choice after the path root..node (from the single parallel pass over the tree)
 *  accept_len  [b] int32 out: drafted tokens accepted, 0..gamma; the step gains accept_len + 1
 *  accept_path [b, gamma+1] int32 out: accepted node indices, root first, then -1: the tree rows
 *                whose KV-cache entries the verifier keeps, in order
 *  next_tok    [b] int32 out: the verifier's token at the last accepted node (the bonus token)
 * Children of one node carry distinct tokens; if an invalid tree repeats one, the smallest node
 * index is taken. At most gamma steps are taken, whatever the parent array holds. */
tf_status tf_accept_walk(const tf_dims* dims, const int32_t* node_tok, const int32_t* node_parent,
                         const int32_t* verifier_tok, int32_t* accept_len, int32_t* accept_path,
                         int32_t* next_tok, tf_stream_t stream);

/* ------------------------------------------------------------------------------------------
 * The pieces the stage calls are made of. tf_stage1_marginals is tf_lmhead_partials +
 * tf_lmhead_merge on the hidden states; tf_stage2_ar_approx is tf_ar_approx followed by the
 * same two on h'. They are exported so a caller (or a profiler) can run or time one kernel.
 * ---------------------------------------------------------------------------------------- */

/* The LM-head pass fused with log-softmax bookkeeping (Alg. 1 "LMHead" and "TopM"):
 * streams W_lm once and, for every row r of x [n_rows, d] (dtype) and every block of 256
 * vocabulary entries, leaves in the workspace per half block its max logit, sum of
 * exp(logit - max) and best (logit, id), and per 32-entry chunk its three largest logits with
 * the ids of the first two (TF_VIEW_HALVES, TF_VIEW_CHUNKS). Logits never reach memory.
 * n_rows <= the larger of b*gamma and b*R. */
tf_status tf_lmhead_partials(const tf_dims* dims, const void* lm_head, const void* x,
                             int32_t n_rows, void* ws, size_t ws_bytes, tf_stream_t stream);

/* Merge the partials of tf_lmhead_partials (same n_rows) into each row's log-sum-exp and exact
 * top-k (k <= 512): out_ids [n_rows, k] int32, out_logp [n_rows, k] float = logit - LSE. A chunk
 * whose third-largest logit could still be a member of the top-k has its 32 logits recomputed
 * exactly from lm_head and x (sets TF_DEV_RECOMPUTED), so the result never depends on keeping
 * only two entries per chunk. */
tf_status tf_lmhead_merge(const tf_dims* dims, const void* lm_head, const void* x,
                          int32_t n_rows, int32_t k, int32_t* out_ids, float* out_logp,
                          void* ws, size_t ws_bytes, tf_stream_t stream);

/* Eq. 1 on the R rows of every sequence (stage 2 before the LM head): gathers Embd rows,
 * normalises both halves, runs the SwiGLU MLP (or the linear layer of TF_APPROX_LINEAR) and
 * adds the residual.
 * h_prime [b, R, d] dtype out (may be NULL: then only the workspace copy is written). */
tf_status tf_ar_approx(const tf_dims* dims, const tf_weights* w, const void* hidden,
                       const int32_t* root_tok, const int32_t* top_ids, void* h_prime,
                       void* ws, size_t ws_bytes, tf_stream_t stream);

/* Device address of h' [b, R, d] (dims->dtype) inside a workspace laid out for `dims`: where
 * tf_ar_approx and tf_stage2_ar_approx leave the approximator's output. Host only; the address
 * is valid while the workspace is. Lets a caller run tf_lmhead_partials/tf_lmhead_merge on h'
 * as separate calls without a copy. */
tf_status tf_workspace_h_prime(const tf_dims* dims, void* ws, size_t ws_bytes, void** h_prime);

/* Regions of a workspace laid out for `dims` (for inspection, testing and for exchanging
 * LM-head partials between vocabulary shards; host only, no GPU work). *ptr receives the device
 * address and *bytes the region's size.
 * Intermediates of Eq. 1 left by the last tf_ar_approx / tf_stage2_ar_approx (TF_MODE_AR only):
 *   TF_VIEW_X        x = [RMSNorm(h)*w_h ; RMSNorm(Embd(prev))*w_e]   [b*R, 2d] dtype
 *   TF_VIEW_A        SiLU(W_gate x) * (W_up x)                         [b*R, I]  dtype
 *                    (0 bytes with TF_APPROX_LINEAR)
 *   TF_VIEW_H_PRIME  h' = h + W_down A  (or h + W_lin x)               [b*R, d]  dtype
 * The partials of the last tf_lmhead_partials over n_rows rows, n_tiles = ceil(V / 256), both
 * float4 tables indexed [block][part][row] with the call's n_rows as the row count:
 *   TF_VIEW_HALVES   [n_tiles][2][n_rows] per half block (128 entries): (max logit m,
 *                    sum of exp(z - m), best logit, best token id as int32 bits)
 *   TF_VIEW_CHUNKS   [n_tiles][8][n_rows] per 32-entry chunk: (largest, second, third largest
 *                    logit, offsets in the chunk of the first two in bits 0-7 and 8-15)
 * Logits are W_lm x / T; empty entries hold -inf, sum 0 and id -1. The merge reads token ids
 * of chunk entries from the block index, so partials of a vocabulary shard starting at token
 * v0 (a multiple of 256) join an unsharded table at block v0 / 256 once v0 is added to their
 * half-block ids. */
typedef enum {
    TF_VIEW_X = 0,
    TF_VIEW_A = 1,
    TF_VIEW_H_PRIME = 2,
    TF_VIEW_HALVES = 3,
    TF_VIEW_CHUNKS = 4
} tf_view;
tf_status tf_workspace_view(const tf_dims* dims, void* ws, size_t ws_bytes, int32_t view, void** ptr,
                            size_t* bytes);

/* ------------------------------------------------------------------------------------------
 * For callers that cannot allocate device memory. The paper has no counterpart to this call:
 * it serves callers that cannot provide a workspace, e.g. a plugin or custom operator inside a
 * host framework that owns all device memory and hands out none, or code on a latency-critical
 * path where cudaMalloc/cudaFree are ruled out because they can synchronise the device.
 * ---------------------------------------------------------------------------------------- */

/* Size of the library's own scratch array. Every GPU that loads the library holds this much
 * device memory until the process exits, whether or not the call below is used. */
#define TF_STATIC_SCRATCH_BYTES ((size_t)8 << 20)

/* tf_stage1_marginals without a workspace: the same kernels and the same results (top_ids,
 * top_logp as there), with the per-block partials and the status word in a fixed array inside
 * the library instead of the caller's workspace. Allocates nothing.
 *  dev_status [1] int32 out (device): the call's TF_DEV_* flags, overwritten (not OR-ed) when
 *             the call's work completes on `stream`; TF_DEV_RECOMPUTED alone is no error.
 * Limit: with n = b * gamma * ceil(V / 256), 256 + roundup(32 n, 256) + 128 n bytes must fit in
 * TF_STATIC_SCRATCH_BYTES, i.e. n <= 52426 (b * gamma <= 88 at V = 151936); larger requests
 * return TF_ERR_UNSUPPORTED before any GPU work. Other arguments are checked as in
 * tf_stage1_marginals (TF_ERR_INVALID_ARG, TF_ERR_UNSUPPORTED).
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress, with
 * that device current) and keeps it for that device's current CUDA context; make that first
 * call before any stream capture. A call in a new context of the device (after cudaDeviceReset,
 * or after the primary context was released and re-created) looks the address up again, so it
 * too should precede any capture.
 * Every call on a device shares the one array: calls that can overlap on the GPU (different
 * streams, or threads sharing a device without ordering) race and corrupt each other's results.
 * Issue them on one stream, or order them. */
tf_status tf_stage1_marginals_static(const tf_dims* dims, const tf_weights* w, const void* hidden,
                                     int32_t* top_ids, float* top_logp, int32_t* dev_status,
                                     tf_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* TREEFLASH_H */
