/*
 * prism.h -- C ABI of a GB300 (sm_103a) implementation of the PRISM draft round.
 *
 * PRISM (Parametrically Refactoring Inference for Speculative sampling draft
 * Models) drafts K tokens per round; draft step k runs its own processing
 * module (a fully connected fusion layer plus one transformer layer) chosen by
 * a surjection f_map from steps to modules, with a token embedding E and a
 * vocabulary head LM_head shared by all steps and one KV cache shared by all
 * modules (Sec. 3.2, Table 2).  The round is followed by verification; this
 * library implements its temperature-0 acceptance rule (Sec. 2).
 *
 * Conventions for every entry point:
 *   - All tensor arguments are DEVICE pointers on the context's device,
 *     row-major and densely packed, owned by the caller.  Weight, embedding,
 *     LM-head, hidden-state and cache pointers must be 16-byte aligned
 *     (checked: PRISM_ERR_INVALID_ARG).  Weight pointers are
 *     borrowed: they must stay valid until the context is destroyed or the
 *     weights are replaced.  The library owns only its workspace, allocated in
 *     prism_create and freed in prism_destroy.
 *   - "wtype" below is the configuration's dtype: PRISM_BF16 (bf16 bit
 *     patterns) or PRISM_F32 (float32).  Weights, E, LM head, target hidden
 *     states and the KV cache all use wtype.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t, passed as
 *     void*; NULL is the legacy default stream).  Nothing synchronises unless
 *     stated.
 *   - Every function returns a prism_status and never throws across the ABI.
 *     Conditions the host can check (null pointers, sizes, unloaded weights)
 *     are reported before anything is enqueued.  Conditions only the device
 *     can see (a token id outside [0, vocab), a cache position outside
 *     [0, max_ctx), n_new outside [1, max_new]) set a device error word; the
 *     kernels clamp and carry on without trapping, and prism_sync_status
 *     reports PRISM_ERR_DEVICE_FLAG.
 *   - prism_get_error returns a message for the last failing call on the
 *     context (valid until the next call).
 */
#ifndef PRISM_H_
#define PRISM_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PRISM_OK = 0,
    PRISM_ERR_INVALID_ARG = 1,  /* null pointer, bad enum, bad option */
    PRISM_ERR_SHAPE = 2,        /* sizes inconsistent with the configuration */
    PRISM_ERR_CAPACITY = 3,     /* batch above max_batch, and similar host-visible limits */
    PRISM_ERR_NOT_LOADED = 4,   /* shared or step weights missing */
    PRISM_ERR_CUDA = 5,         /* a CUDA runtime call failed; see prism_get_error */
    PRISM_ERR_OOM = 6,          /* workspace allocation failed */
    PRISM_ERR_DEVICE_FLAG = 7,  /* the device error word was set (see prism_sync_status) */
    PRISM_ERR_TIMEOUT = 8       /* a bounded device-side wait gave up */
} prism_status;

typedef enum { PRISM_F32 = 0, PRISM_BF16 = 1 } prism_dtype;

/* Device error word bits (reported by prism_sync_status). */
#define PRISM_DEVERR_TOKEN_RANGE 1   /* a token id outside [0, vocab) was clamped */
#define PRISM_DEVERR_CACHE_RANGE 2   /* a cache position outside [0, max_ctx) was skipped */
#define PRISM_DEVERR_NNEW_RANGE 4    /* n_new[b] outside [1, max_new] was clamped */
#define PRISM_DEVERR_TIMEOUT 8       /* a bounded wait expired */

/* Model and capacity description.  hidden = d, n_q_heads = Hq, n_kv_heads =
 * Hkv (Hq % Hkv == 0), head_dim = D (64 or 128), ffn = F, vocab = V,
 * n_steps = K (1..16) draft steps per round.  max_batch, max_ctx (cache
 * positions per sequence) and max_new (accepted tokens per sequence fed to
 * step 1) size the workspace.  topk in 1..8 candidates are reported per step
 * (the chained token is the first).  final_norm: 1 applies RMSNorm with the
 * step's g_final before the LM head.  rope_theta and rms_eps as in Llama.
 * max_tree_width: 0 (no tree rounds), or the largest width w (1..8) that
 * prism_draft_tree will be called with; the workspace then holds w rows per
 * sequence for the draft steps. */
typedef struct {
    int32_t hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab, n_steps;
    int32_t dtype;
    int32_t max_batch, max_ctx, max_new, topk;
    float rope_theta, rms_eps;
    int32_t final_norm;
    int32_t max_tree_width;
} prism_config;

/* One processing module (Sec. 3.2: a fully connected fusion layer and a
 * transformer layer), all wtype, row-major:
 *   w_fuse    [d, 2d]      fusion F(E(x), h) = w_fuse . [E(x); h]
 *   g_attn    [d]          RMSNorm gain before attention
 *   w_qkv     [(Hq + 2 Hkv) D, d]   q rows, then k rows, then v rows
 *   w_o       [d, Hq D]
 *   g_mlp     [d]          RMSNorm gain before the MLP
 *   w_gate_up [2F, d]      gate rows [0, F), up rows [F, 2F); SwiGLU
 *   w_down    [d, F]
 *   g_final   [d]          RMSNorm gain before the LM head (if final_norm) */
typedef struct {
    const void *w_fuse, *g_attn, *w_qkv, *w_o, *g_mlp, *w_gate_up, *w_down, *g_final;
} prism_step_weights;

typedef struct prism_ctx prism_ctx;

/* Create a context on CUDA device `device` and allocate its workspace.
 * Errors: INVALID_ARG (null out, unsupported sizes), OOM, CUDA. */
prism_status prism_create(const prism_config *cfg, int32_t device, prism_ctx **out);

/* Destroy a context; waits for its work to finish.  NULL is a no-op. */
prism_status prism_destroy(prism_ctx *ctx);

/* Token embedding E [V, d] and LM head [V, d] (both frozen and shared by all
 * steps, Table 2).  Borrowed.  Errors: INVALID_ARG (null). */
prism_status prism_load_shared_weights(prism_ctx *ctx, const void *embed, const void *lm_head);

/* Bind the module used by draft step `step` (0-based, 0..K-1).  The surjection
 * f_map of Table 2 is expressed by binding the same pointers to several steps.
 * Borrowed.  Errors: INVALID_ARG (null field, step out of range). */
prism_status prism_load_step_weights(prism_ctx *ctx, int32_t step, const prism_step_weights *w);

/* One draft round (Sec. 3.2 "Draft with PRISM") for `batch` independent
 * sequences:
 *   step 1: each sequence b's n_new[b] accepted tokens tokens[b, i] with
 *     their target hidden states hidden[b, i] (i < n_new[b]) are fused and
 *     run through step 1's transformer layer at cache positions
 *     kv_len[b] + i with causal attention; the last row is h^_0 and
 *     x^_1 = argmax LM_head(h^_0).
 *   step k = 2..K: fuse E(x^_{k-1}) with h^_{k-2}, run step k's layer at
 *     position kv_len[b] + n_new[b] + k - 2, x^_k = argmax LM_head(h^_{k-1}).
 * Arguments (device pointers):
 *   tokens      int32 [batch, max_new]        rows past n_new[b] are ignored
 *   hidden      wtype [batch, max_new, d]
 *   n_new       int32 [batch]                 1..max_new
 *   kv_len      int32 [batch]                 committed cache length L_b (read only)
 *   k_cache, v_cache  wtype [max_batch, Hkv, max_ctx, D]  read and written:
 *               rows kv_len[b] .. kv_len[b] + n_new[b] + K - 2 are written
 *   draft_ids   int32 [batch, K]              out
 *   topk_ids    int32 [batch, K, topk]        out, or NULL
 *   topk_logits float [batch, K, topk]        out, or NULL
 *   logits      float [batch, K, V]           out, or NULL
 *   hidden_out  float [batch, K, d]           out (h^_0 .. h^_{K-1}), or NULL
 * Ties in the argmax go to the lowest id; top-k is sorted by logit, then id.
 * The round is captured once per distinct argument set as a CUDA graph and
 * replayed (option "use_graph").  Errors: INVALID_ARG, CAPACITY
 * (batch > max_batch), NOT_LOADED, CUDA. */
prism_status prism_draft_round(prism_ctx *ctx, int32_t batch, const int32_t *tokens,
                               const void *hidden, const int32_t *n_new, const int32_t *kv_len,
                               void *k_cache, void *v_cache, int32_t *draft_ids,
                               int32_t *topk_ids, float *topk_logits, float *logits,
                               float *hidden_out, void *stream);

/* Greedy (temperature 0) acceptance, Sec. 2: accept_len[b] is the largest a
 * in [0, K] with draft[b, j] == target[b, j] for all j < a; out_tokens[b] is
 * draft[b, 0:a] followed by target[b, a] (the corrected or bonus token), then
 * -1 padding; kv_len[b] += n_new[b] commits the step-1 rows (draft rows are
 * scratch and are overwritten by the next round).
 *   draft int32 [batch, K], target int32 [batch, K+1], n_new int32 [batch],
 *   kv_len int32 [batch] in/out, accept_len int32 [batch] out,
 *   out_tokens int32 [batch, K+1] out.
 * Errors: INVALID_ARG, CAPACITY, CUDA. */
prism_status prism_accept_greedy(prism_ctx *ctx, int32_t batch, const int32_t *draft,
                                 const int32_t *target, const int32_t *n_new, int32_t *kv_len,
                                 int32_t *accept_len, int32_t *out_tokens, void *stream);

/* Steady-state draft loop: `rounds` greedy rounds back to back on the device,
 * each one prism_draft_round followed by prism_accept_greedy, where the
 * acceptance also writes the next round's input: the a accepted drafts and
 * the target's token at position a go to tokens[b, 0..a] and n_new[b] =
 * a + 1, and kv_len[b] += n_new[b] commits the rows the round prefilled
 * (Sec. 2 and Sec. 3.2: the next round re-fuses the accepted tokens with the
 * target's hidden states of its verification pass).  Nothing returns to the
 * host between rounds; the whole loop is one CUDA graph (cached per argument
 * set, like a round).
 *   tokens     int32 [batch, max_new] in/out (round 0's tokens; afterwards
 *              the next round's); max_new >= K + 1 is required
 *   hidden     wtype [rounds, batch, max_new, d]: the target hidden states
 *              paired with each round's tokens (row i of round r pairs with
 *              token i of that round)
 *   n_new      int32 [batch] in/out; kv_len int32 [batch] in/out
 *   k_cache, v_cache as prism_draft_round
 *   target     int32 [rounds, batch, K + 1]: the target's tokens per round
 *   draft_ids  int32 [rounds, batch, K] out; accept_len int32 [rounds, batch]
 *   out; out_tokens int32 [rounds, batch, K + 1] out (as prism_accept_greedy)
 * Errors: INVALID_ARG, SHAPE (rounds < 1), CAPACITY (batch > max_batch, or
 * max_new < K + 1), NOT_LOADED, CUDA. */
prism_status prism_draft_loop(prism_ctx *ctx, int32_t batch, int32_t rounds, int32_t *tokens, const void *hidden,
                              int32_t *n_new, int32_t *kv_len, void *k_cache, void *v_cache,
                              const int32_t *target, int32_t *draft_ids, int32_t *accept_len,
                              int32_t *out_tokens, void *stream);

/* Random numbers of the sampled calls below: the n-th output x of SplitMix64
 * (Steele, Lea and Flood, OOPSLA 2014) started from state *seed, with
 * n = (stream << 60) | (b << 40) | (k << 32) | i, taken as
 * ((x >> 41) + 1/2) / 2^23 in (0, 1).  Streams: 1 the draft draw of sequence
 * b at step k + 1 (i = token id), 2 the acceptance test of position k, 3 the
 * token drawn at position k (k = K: the extra token after a full accept).
 * `seed` is a device pointer, read when the kernels run, so a captured round
 * replays with a new seed written between rounds. */

/* One draft round with sampled drafting (Sec. 2: the draft model draws its
 * candidates from p_draft; here p_draft = softmax(z / temperature)): the same
 * round as prism_draft_round, except that x^_k is drawn from softmax(z / T)
 * of step k's logits (Gumbel-max rule, stream 1) and feeds step k + 1.
 *   temperature  > 0, finite
 *   seed         uint64 device word (8-byte aligned)
 *   logits       float [batch, K, V] out, required (the acceptance reads them)
 *   draft_lse    float [batch, K] out: log sum_i exp(z_i / T), so that
 *                p_draft(x) = exp(z_x / T - lse)
 *   draft_ids    the drawn tokens; topk_ids / topk_logits stay the argmax list
 * Other arguments as prism_draft_round.  Errors: INVALID_ARG (temperature,
 * null seed / logits / draft_lse, and as prism_draft_round), CAPACITY (also
 * max_batch >= 2^20 or K > 255, the counter's fields), NOT_LOADED, CUDA. */
prism_status prism_draft_round_sampled(prism_ctx *ctx, int32_t batch, const int32_t *tokens,
                                       const void *hidden, const int32_t *n_new, const int32_t *kv_len,
                                       void *k_cache, void *v_cache, float temperature, const uint64_t *seed,
                                       int32_t *draft_ids, int32_t *topk_ids, float *topk_logits,
                                       float *logits, float *draft_lse, float *hidden_out, void *stream);

/* Speculative-sampling acceptance (Sec. 2): for k = 0..K-1 in turn, the draft
 * token x = draft[b, k] is accepted when r < min(1, p_target(x) / p_draft(x))
 * (r from stream 2, evaluated as r * p_draft < p_target); the first rejected
 * position's replacement is drawn from max(0, p_target - p_draft) normalised
 * (stream 3; from p_target if that residual is zero everywhere); after a full
 * accept the extra token is drawn from p_target at position K.  p_draft(x) =
 * exp(logits[b, k, x] / T - draft_lse[b, k]).
 *   draft int32 [batch, K], logits float [batch, K, V], draft_lse float
 *   [batch, K] (as written by prism_draft_round_sampled), temperature the
 *   round's, target_probs float [batch, K+1, V] (rows sum to 1), seed uint64
 *   device word, n_new int32 [batch], kv_len int32 [batch] in/out (+= n_new),
 *   accept_len int32 [batch] out, out_tokens int32 [batch, K+1] out (the
 *   accepted drafts, the drawn token, then -1).
 * A draft id outside [0, V) sets the token bit of the device error word.
 * Errors: INVALID_ARG, CAPACITY (batch > max_batch), CUDA. */
prism_status prism_accept_sampled(prism_ctx *ctx, int32_t batch, const int32_t *draft, const float *logits,
                                  const float *draft_lse, float temperature, const float *target_probs,
                                  const uint64_t *seed, const int32_t *n_new, int32_t *kv_len,
                                  int32_t *accept_len, int32_t *out_tokens, void *stream);

/* Outputs of a tree round (prism_draft_tree), all device pointers:
 *   tokens, parents, depths  int32 [batch, n_nodes]  the verified tree in
 *                 candidate-pool order (parents before children); parents[i]
 *                 is the position of node i's parent in the list, -1 for a
 *                 child of the root (the last accepted token); depth 1..K
 *   scores        float [batch, n_nodes]  summed draft log-probabilities of
 *                 each node's path
 *   pool_tokens, pool_parents, pool_scores  [batch, P], P = w + (K - 1) w^2:
 *                 every candidate of the round (or NULL).  Depth-1 candidate
 *                 r sits at r; candidate r of frontier row j at step k at
 *                 w + (k - 2) w^2 + j w + r; parents are pool indices
 *   frontier      int32 [batch, K, w]  pool indices of the frontier chosen
 *                 after each step (or NULL)
 *   row_logits    float [K, batch, w, V]  every processed row's logits (or
 *                 NULL); step 1 has one row per sequence, written at j = 0 */
typedef struct {
    int32_t *tokens, *parents, *depths;
    float *scores;
    int32_t *pool_tokens, *pool_parents;
    float *pool_scores;
    int32_t *frontier;
    float *row_logits;
} prism_tree_outputs;

/* One tree-drafting round.  PRISM's step modules apply unchanged to
 * tree-shaped drafts (Sec. 3.2, after the recurrence), and the paper
 * evaluates a 6-step, 4-branch tree verifying at most 16 tokens (Sec. 4).
 * This is the dynamic top-w expansion of that tree:
 *   step 1: the prefill of prism_draft_round; the w best tokens of its
 *     logits are the depth-1 candidates and the first frontier;
 *   step k = 2..K: each of the w frontier nodes of a sequence is one row of
 *     step k's module: input [E(token); h^ of the row whose LM head proposed
 *     it], rotary position kv_len + n_new + k - 2, K/V stored at cache slot
 *     kv_len + n_new + (k - 2) w + j, attention over the rows
 *     [0, kv_len + n_new) and the slots of the node's ancestors and itself.
 *     Each row's w best tokens are candidates whose score is the parent's
 *     score plus the token's draft log-probability (logit - log-sum-exp);
 *     the next frontier is the w best of the w^2 new candidates;
 *   end: the verified tree is the n_nodes best candidates of the round.
 * Orders: top-w by logit, then id; frontiers and the tree by score
 * descending, then pool index ascending.
 *   width        1..max_tree_width; (K - 1) * width <= 64; P <= 1024
 *   n_nodes      1..P
 *   out          see prism_tree_outputs (tokens, parents, depths, scores
 *                required)
 * Other arguments as prism_draft_round; cache rows kv_len .. kv_len + n_new +
 * (K - 1) w - 1 are written (a row beyond max_ctx sets the cache-range bit
 * and is skipped).  With width 1 and n_nodes K the tree is the greedy chain.
 * Captured as a CUDA graph per argument set, like prism_draft_round.
 * Errors: INVALID_ARG (null or misaligned argument, width or n_nodes out of
 * range), CAPACITY (batch > max_batch, width > max_tree_width), NOT_LOADED,
 * CUDA. */
prism_status prism_draft_tree(prism_ctx *ctx, int32_t batch, const int32_t *tokens, const void *hidden,
                              const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                              int32_t width, int32_t n_nodes, const prism_tree_outputs *out, void *stream);

/* Greedy acceptance of a draft tree (Sec. 2's temperature-0 rule applied
 * along the tree, as in tree verification): starting at the root, accept the
 * child whose token equals the target's token at the current node, until no
 * child matches or K nodes are accepted.
 *   tree_tokens, tree_parents int32 [batch, n_nodes] (as prism_draft_tree
 *   writes them); target_next int32 [batch, n_nodes + 1]: entry 0 the
 *   target's token after the root, entry 1 + i its token after node i;
 *   n_new int32 [batch]; kv_len int32 [batch] in/out (+= n_new);
 *   accept_len int32 [batch] out; accept_nodes int32 [batch, K] out (the
 *   accepted nodes' positions, then -1); out_tokens int32 [batch, K+1] out
 *   (their tokens, the target's token at the last accepted node, then -1).
 * Errors: INVALID_ARG, CAPACITY, CUDA. */
prism_status prism_accept_tree(prism_ctx *ctx, int32_t batch, int32_t n_nodes, const int32_t *tree_tokens,
                               const int32_t *tree_parents, const int32_t *target_next, const int32_t *n_new,
                               int32_t *kv_len, int32_t *accept_len, int32_t *accept_nodes,
                               int32_t *out_tokens, void *stream);

/* LM-head selection that allocates nothing.  The paper has no counterpart to
 * this entry point; it serves callers that cannot call cudaMalloc, so cannot
 * own a prism_ctx workspace: an inference server whose caching allocator has
 * already reserved the device memory it may use, a plugin whose host
 * framework forbids allocation outside its own pool, or a process that fixes
 * its whole device-memory budget at start-up.
 * It computes what the last stage of a draft step computes (final RMSNorm with
 * gain g_final, logits = lm_head . norm(h), top-1 and top-k), using the same
 * kernel, and keeps that kernel's scratch (the per-CTA partial top-8 lists,
 * the last-CTA ticket and the device error word) in a static device array of
 * 1 MiB + 256 bytes inside the library, which every process that loads the
 * library holds on each device it uses until exit.
 *   dtype PRISM_F32 or PRISM_BF16 (the type of lm_head and g_final);
 *   h fp32 [batch, hidden] hidden rows before the final norm;
 *   g_final [hidden] or NULL (no final norm); lm_head [vocab, hidden];
 *   draft int32 [batch] out; topk_ids int32 [batch, topk], topk_logits fp32
 *   [batch, topk], logits fp32 [batch, vocab]: outputs, each may be NULL;
 *   dev_flags int32 [1] or NULL: receives the device error word of this call.
 * All pointers are device (or managed) memory of the current device; h,
 * lm_head and g_final 16-byte aligned.  A pointer to host memory or to
 * another device's memory returns PRISM_ERR_INVALID_ARG before any launch.
 * Limits: batch <= 64 rows; larger batches return PRISM_ERR_CAPACITY with a
 * message from prism_get_error(NULL): split them into several calls.
 * The first call on a device (the current one) does that device's set-up:
 * it resolves the array's device address with cudaGetSymbolAddress and sets
 * the kernel's shared-memory attribute; make that first call before any
 * stream capture.  Each call clears the ticket and the error word with a
 * stream-ordered memset, then launches the kernel on `stream`.  Every call
 * shares the one array, so calls that can overlap on the GPU (different
 * streams, or several host threads) race and corrupt each other's results:
 * keep them on one stream.  Calls no cudaMalloc, cudaFree or allocating
 * library routine.  Errors: INVALID_ARG, SHAPE, CAPACITY, CUDA. */
prism_status prism_lm_head_topk_static(int32_t dtype, int32_t hidden, int32_t vocab, int32_t batch,
                                       int32_t topk, float rms_eps, const float *h,
                                       const void *g_final, const void *lm_head, int32_t *draft,
                                       int32_t *topk_ids, float *topk_logits, float *logits,
                                       int32_t *dev_flags, void *stream);

/* Synchronise `stream`, read and clear the device error word.  Returns
 * PRISM_ERR_TIMEOUT when its timeout bit is set (a bounded device-side wait
 * gave up: the kernel wound down, every copy it had in flight landed, and
 * the outputs of the calls since the last check are not to be used),
 * PRISM_ERR_DEVICE_FLAG when only other bits are set (bits in *flags if
 * non-NULL in both cases), PRISM_ERR_CUDA when the stream reports an
 * error, PRISM_OK otherwise.  The context stays usable after either flag. */
prism_status prism_sync_status(prism_ctx *ctx, void *stream, int32_t *flags);

/* Options (name, value): "use_graph" (1: capture and replay, default 1),
 * "use_pdl" (1: programmatic dependent launch between kernels, default 1),
 * "gemv_chunk_kb" (target TMA stage size of the projection kernels, 0..128,
 * 0 = default), "gemv_smem_kb" (shared-memory budget of the projection
 * ring, 0..200, 0 = default), "gemv_groups" (consumer warp groups of the
 * projection kernels: 1, 2, 4, 8 or 16; 0 = default), "gemv_tcgen05"
 * (1, the default: bf16 projections run on the tcgen05 kernels, TMA tensor
 * loads into tensor-memory accumulators, except gate/up + SwiGLU with at
 * most 2 activation rows, which measures faster on the CUDA-core kernel;
 * 2: gate/up as well; 0: every projection on the kernels below),
 * "tc_stream_rows" (>= 1, default 1: a tcgen05 projection with at least
 * this many activation rows streams them through the TMA ring beside the
 * weights instead of staging them whole in shared memory, its split-K sums
 * added by a separate finish kernel that also writes the next projection's
 * rows; at most 16 rows can be staged, and a staged projection's last CTA
 * per tile adds the sums itself; an LM head other than that streamed top-1
 * below (lm_stream) streams from max(this, 8) rows outside tree rounds), "attn_ctas_per_sm" (1..64, default 2: the fused attention
 * kernel's cluster size halves while batch x KV heads x cluster size exceeds
 * this many CTAs per SM), "gemv_cuda_core" (for projections
 * not on the tcgen05 kernel: 1, the default, the CUDA-core TMA-ring kernel;
 * 0: the warp-level mma.sync kernel), "attn_fused" (1, the default: RoPE,
 * KV append and attention run as one kernel, a cluster of up to 8 CTAs per
 * sequence and KV head merging through distributed shared memory; 0: a
 * RoPE/append kernel, then split-KV attention with a last-CTA merge),
 * "attn_tc" (1, the default: the fused attention kernel of a bf16 context
 * with the tcgen05 projections loads cache chunks with TMA and computes QK^T
 * and PV with warp-level tensor-core MMAs; 0: the same fused computation on
 * CUDA cores), "attn_warps" (compute warps per CTA of that tensor-core
 * kernel: 8, stages of 128 keys, one CTA per SM; or 4, stages of 64 keys,
 * two CTAs per SM; 0, the default: 4 where one CTA per (sequence, KV head)
 * makes more CTAs than SMs but at most two per SM, else 8), "attn_lpt" (1,
 * the default: where that kernel's CTAs make more than one wave but at most
 * two, the CTAs take the sequences in order of decreasing context length;
 * 0: in index order),
 * "wait_polls" (0, the default: every wait between two roles of a kernel,
 * a consumer for a filled ring stage or accumulator, a producer for a
 * released one, gives up after a built-in bound of 2^22 polls; N > 0: after
 * N polls; N < 0: at once, so that every such wait fails: a setting for
 * testing the error path.  A wait that gives up sets the timeout bit and
 * the kernel winds down: it issues no more copies or MMAs, still waits
 * (with the built-in bound) for the copies and MMAs it has in flight, and
 * frees its tensor memory.  Covers the projection kernels and the fused
 * attention kernel),
 * "w_evict_first" (1, the default: the projection kernels load weight boxes
 * with an L2 evict-first cache policy, since each weight byte is read once
 * per step, so that the KV cache and the activations stay in L2; 0: the
 * default policy),
 * "lm_stream" (1, the default: the top-1 LM head of a greedy round with up
 * to 16 rows streams them through its ring beside the weights, leaving the
 * ring the shared memory staged rows would take, and joins the rows' best
 * through the packed top-1 in the kernel; 0: as the LM head of a sampled
 * round, it stages fewer than max(tc_stream_rows, 8) rows (a top-1 then
 * joins through the packed maximum) and streams more, selecting through
 * per-CTA lists and a merge kernel),
 * "tree_defer_merge" (1, the default: in tree rounds the LM head leaves its
 * per-CTA top-w lists unmerged and the log-sum-exp kernel merges them, one
 * CTA per row; 0: the LM head's last CTA merges them),
 * "lm_even_waves" (1, the default: the LM head launches the fewest CTAs
 * that stream its 128-row tiles in as many waves as one CTA per SM would, so
 * that every CTA streams the same number of tiles, e.g. 144 CTAs of 7 tiles
 * for a vocabulary of 128256 instead of 152 CTAs of 6 or 7; 0: one CTA per
 * SM), "prefetch_next_kb" (16384, the default: once a kernel's CTAs have
 * requested their last weight boxes, they request the first this many KB of
 * the next kernel's weights into L2, each CTA an even share, so that HBM
 * keeps streaming across the kernel boundary; 0: none),
 * "fuse_rows" (1, the default: a streamed projection's last kernel, the
 * split-K finish or the LM head's top-k merge, also writes the next
 * projection's bf16 activation rows, its RMSNorm or the next step's fusion
 * input, so that the next projection needs no row-preparation kernel; 0:
 * a preparation kernel before each projection).
 * Changing an option drops cached graphs.  Errors: INVALID_ARG (unknown name
 * or value out of range). */
prism_status prism_set_option(prism_ctx *ctx, const char *name, int32_t value);

/* Kernel launches of one round: the kernel nodes of the CUDA graph that the
 * most recent prism_draft_round call (with "use_graph" on) replayed.  The
 * count depends on the batch and the options (a projection may take one to
 * three kernels).  Errors: INVALID_ARG (null argument, or no round replayed
 * from a graph yet). */
prism_status prism_round_launches(prism_ctx *ctx, int32_t *n_launches);

/* Instrumented round for measurement: the same work as prism_draft_round
 * launched eagerly with a CUDA event recorded before and after every kernel.
 * kernel_ms[i] receives the duration of kernel i in launch order (capacity
 * max_kernels); *n_kernels receives the count; kernel_kind[i] (may be NULL)
 * receives a code: 0 fusion, 1 qkv, 2 rope/append, 3 attention (with the
 * fused option: RoPE, append and attention; no code-2 kernel then), 4 o-proj,
 * 5 gate/up, 6 down, 7 LM head + selection, 8 sampled draw (sampled rounds
 * only; this call profiles the greedy round).  Synchronises the stream. */
prism_status prism_profile_round(prism_ctx *ctx, int32_t batch, const int32_t *tokens,
                                 const void *hidden, const int32_t *n_new, const int32_t *kv_len,
                                 void *k_cache, void *v_cache, int32_t *draft_ids,
                                 int32_t *topk_ids, float *topk_logits, void *stream,
                                 float *kernel_ms, int32_t *kernel_kind, int32_t max_kernels,
                                 int32_t *n_kernels);

/* The same instrumentation for a tree round (prism_draft_tree's arguments);
 * kernel kinds add 9 tree gather and 10 tree log-sum-exp + selection (a tree
 * step's RoPE, KV append and attention are one kernel, reported as 3).
 * Synchronises the stream.  Errors: as prism_draft_tree and
 * prism_profile_round. */
prism_status prism_profile_tree(prism_ctx *ctx, int32_t batch, const int32_t *tokens, const void *hidden,
                                const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                                int32_t width, int32_t n_nodes, const prism_tree_outputs *out, void *stream,
                                float *kernel_ms, int32_t *kernel_kind, int32_t max_kernels, int32_t *n_kernels);

/* Message for the last failing call on ctx (or a global message when ctx is NULL). */
const char *prism_get_error(const prism_ctx *ctx);

/* Library version string. */
const char *prism_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PRISM_H_ */
