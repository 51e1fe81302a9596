// C ABI of the PRISM draft round: context, workspace, validation, the per-step
// launch sequence and CUDA-graph capture/replay.  See include/prism.h.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <utility>
#include <vector>

#include "../../include/prism.h"
#include "common.cuh"

using namespace prism;

namespace {

constexpr int kGraphCache = 8;
constexpr int kMaxProfileKernels = 12 * kMaxSteps + 8;

struct RoundArgs {
    int B;
    const int32_t *tokens;
    const void *hidden;
    const int32_t *n_new, *kv_len;
    void *k_cache, *v_cache;
    int32_t *draft;
    int32_t *topk_ids;
    float *topk_logits, *logits, *hidden_out;
    float temperature;             // > 0: sampled drafting (then logits, seed and lse are set)
    const uint64_t *seed;
    float *lse;
    int tree_w, tree_m;            // > 0: tree drafting of this width, verifying tree_m nodes
    prism_tree_outputs tree;
    bool operator==(const RoundArgs &o) const { return std::memcmp(this, &o, sizeof(RoundArgs)) == 0; }
};

// Zero-filled (padding included: graphs are looked up by memcmp of the arguments).
RoundArgs round_args(int B, const int32_t *tokens, const void *hidden, const int32_t *n_new, const int32_t *kv_len,
                     void *k_cache, void *v_cache, int32_t *draft, int32_t *topk_ids, float *topk_logits,
                     float *logits, float *hidden_out) {
    RoundArgs r;
    std::memset(&r, 0, sizeof r);
    r.B = B;
    r.tokens = tokens;
    r.hidden = hidden;
    r.n_new = n_new;
    r.kv_len = kv_len;
    r.k_cache = k_cache;
    r.v_cache = v_cache;
    r.draft = draft;
    r.topk_ids = topk_ids;
    r.topk_logits = topk_logits;
    r.logits = logits;
    r.hidden_out = hidden_out;
    return r;
}

// A multi-round loop: round 0's arguments, the round count and the
// acceptance arrays (per-round strides follow from the configuration).
struct LoopArgs {
    RoundArgs r0;
    int rounds;
    const int32_t *target;
    int32_t *accept_len, *out_tokens;
    bool operator==(const LoopArgs &o) const { return std::memcmp(this, &o, sizeof(LoopArgs)) == 0; }
};

struct LoopGraph {
    LoopArgs key;
    bool pdl;
    cudaGraphExec_t exec;
};

struct GraphEntry {
    RoundArgs key;
    bool pdl;
    cudaGraphExec_t exec;
    unsigned long long used;
    int kernels;        // kernel nodes of the captured round
};

thread_local std::string g_error;

}  // namespace

void prism::set_global_error(const char *msg) { g_error = msg; }

struct prism_ctx {
    prism_config cfg{};
    int device = 0;
    int sms = 0;
    bool bf16 = true;
    int qkv_rows = 0;
    int lm_grid = 0;
    int attn_chunk = 64;
    int attn_splits = 0;
    // weights (borrowed)
    const void *embed = nullptr, *lm_head = nullptr;
    prism_step_weights steps[kMaxSteps]{};
    bool step_loaded[kMaxSteps]{};
    // workspace (owned)
    void *ws = nullptr;
    size_t ws_bytes = 0;
    float *rope_cos = nullptr, *rope_sin = nullptr;
    float *x0 = nullptr, *qkv = nullptr, *q = nullptr, *attn_part = nullptr, *a = nullptr, *hhat = nullptr;
    void *o_buf = nullptr, *m_buf = nullptr;
    float *lm_val = nullptr;
    int *lm_id = nullptr;
    int *counters = nullptr;  // [max_batch * Hkv] attention + [1] LM head
    unsigned long long *lm_best = nullptr;  // [max_batch] LM head top-1 keys (left at zero)
    float *sample_part = nullptr;           // [max_batch, kSampleMaxBlocks, 4] sampled-draft partials
    int *sample_ctr = nullptr;              // [max_batch] sampled-draft tickets (left at zero)
    // tree drafting (max_tree_width > 0): w rows per sequence, frontier and candidate pool
    int tree_rows = 0;                      // max_batch * max(1, max_tree_width)
    void *tree_u = nullptr;                 // [rows, 2d] wtype fusion inputs
    float *tree_logits = nullptr;           // [rows, V]
    int32_t *tree_top_ids = nullptr;        // [rows, 8]
    float *tree_top_vals = nullptr;         // [rows, 8]
    int32_t *tree_draft = nullptr;          // [rows] (LM-head top-1, unused by the tree)
    float *tree_lse = nullptr;              // [rows]
    float *tree_lse_part = nullptr;         // [rows, kSampleMaxBlocks, 2]
    int *tree_lse_ctr = nullptr;            // [rows] (left at zero)
    int32_t *front_tok = nullptr, *front_row = nullptr, *front_pool = nullptr;  // [rows]
    float *front_score = nullptr;           // [rows]
    unsigned long long *front_mask = nullptr;  // [rows]
    int32_t *pool_tok = nullptr, *pool_par = nullptr;  // [max_batch, P_max]
    float *pool_score = nullptr;
    int *err = nullptr;
    // execution
    cudaStream_t cap_stream = nullptr;
    bool use_graph = true, use_pdl = true;
    int gemv_chunk = 0, gemv_smem = 0, gemv_groups = 0;   // projection ring knobs (0 = built-in default)
    int gemv_cuda_core = 1;                               // 1: bf16 projections on CUDA cores
    int gemv_tcgen05 = 1;                                 // 1: bf16 projections on tcgen05 where they fit
    int attn_fused = 1;                                   // 1: fused RoPE/append/attention cluster kernel
    int attn_ctas_per_sm = 2;                             // fused attention: clusters shrink until B*Hkv*cs <= this * SMs
    int tc_stream_rows = 1;                               // tcgen05 projections with this many rows or more stream X
    int attn_max_cs = 8;                                  // largest cluster the device co-schedules
    int fuse_rows = 1;                                    // streamed projections write the next one's activation rows
    int wait_polls = 0;                                   // role-to-role wait bound (0: built in, < 0: none)
    int w_evict_first = 1;                                // weight streams with an L2 evict-first policy
    int attn_tc = 1;                                      // fused attention on tensor cores (0: CUDA cores)
    int prefetch_next_kb = 16384;                         // KB of the next kernel's weights requested into L2
    int lm_even_waves = 1;                                // LM head: the fewest CTAs with the same tile waves
    int tree_defer_merge = 1;                             // tree: the lse kernel merges the LM head's lists
    int lm_stream = 1;                                    // top-1 LM head: rows streamed beside the weights
    int attn_warps = 0;                                   // tensor-core attention warps per CTA: 0 auto, 4 or 8
    int attn_lpt = 1;                                     // several waves of attention CTAs: longest sequences first
    // tensor-core path: TMA tensor maps of the weights, split-K workspace
    bool tc_ready = false;
    CUtensorMap tm_lm;
    CUtensorMap tm_step[kMaxSteps][5];                    // fusion, QKV, O, gate/up, down
    bool tm_lm_ok = false;
    bool tm_step_ok[kMaxSteps]{};
    float *tc_part = nullptr;
    size_t tc_part_floats = 0;
    int *tc_ctr = nullptr;
    int tc_ctr_n = 0;
    uint16_t *xbuf = nullptr;                             // bf16 activation rows of the streamed kernel
    std::vector<GraphEntry> graphs;
    std::vector<LoopGraph> loop_graphs;
    int last_round_kernels = -1;                          // kernel launches of the last replayed round
    unsigned long long tick = 0;
    std::string error;
};

namespace {

prism_status fail(prism_ctx *c, prism_status s, const std::string &msg) {
    if (c) c->error = msg;
    g_error = msg;
    return s;
}

prism_status cuda_fail(prism_ctx *c, cudaError_t e, const char *what) {
    return fail(c, PRISM_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// 16-byte vector loads need 16-byte aligned bases.
bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

void drop_graphs(prism_ctx *c) {
    for (auto &g : c->graphs) cudaGraphExecDestroy(g.exec);
    c->graphs.clear();
    for (auto &g : c->loop_graphs) cudaGraphExecDestroy(g.exec);
    c->loop_graphs.clear();
}

// Persistent projection grid: one CTA per SM (never more CTAs than units).
int gemv_grid(const prism_ctx *c, int units) {
    return units < c->sms ? (units < 1 ? 1 : units) : c->sms;
}

// Enqueue one round.  prof_ev != null: record an event before the first and
// after every kernel (eager launches, no programmatic dependencies).
cudaError_t enqueue_round(prism_ctx *c, const RoundArgs &r, cudaStream_t s, bool pdl,
                          cudaEvent_t *prof_ev, int32_t *kinds, int *n_kernels) {
    const prism_config &f = c->cfg;
    const int d = f.hidden, Hq = f.n_q_heads, Hkv = f.n_kv_heads, D = f.head_dim, F = f.ffn;
    const int V = f.vocab, K = f.n_steps;
    cudaError_t e = cudaSuccess;
    int nk = 0;
    bool first = true;
    auto after = [&](int kind) {
#ifdef PRISM_CHECKED
        // checked builds run eagerly: localise a failing kernel
        cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
        cudaStreamIsCapturing(s, &cap);
        if (e == cudaSuccess && cap == cudaStreamCaptureStatusNone) {
            cudaError_t se = cudaStreamSynchronize(s);
            if (se != cudaSuccess) {
                std::fprintf(stderr, "prism checked: kernel #%d (kind %d) failed: %s\n", nk, kind, cudaGetErrorString(se));
                e = se;
            }
            int w[5] = {0};
            if (cudaMemcpy(w, c->err, sizeof(w), cudaMemcpyDeviceToHost) == cudaSuccess && (w[0] || w[1]))
                std::fprintf(stderr, "prism checked: after kernel #%d (kind %d): err 0x%x check %d block %d values %d %d\n",
                             nk, kind, w[0], w[1], w[2], w[3], w[4]);
        }
#endif
        if (prof_ev) {
            if (nk < kMaxProfileKernels) {
                cudaEventRecord(prof_ev[nk + 1], s);
                if (kinds) kinds[nk] = kind;
            }
        }
        ++nk;
        first = false;
    };
    if (prof_ev) cudaEventRecord(prof_ev[0], s);

    GemvArgs base{};
    base.embed = c->embed;
    base.tokens = r.tokens;
    base.hidden_in = r.hidden;
    base.draft = r.draft;
    base.eps = f.rms_eps;
    base.n_new = r.n_new;
    base.max_new = f.max_new;
    base.K = K;
    base.vocab = V;
    base.d = d;
    base.err = c->err;
    base.topk = f.topk;
    base.chunk_target = c->gemv_chunk;
    base.smem_budget = c->gemv_smem;
    base.groups = c->gemv_groups;
    base.force_cuda_core = c->gemv_cuda_core;
    base.wait_polls = c->wait_polls;
    base.w_evict_first = c->w_evict_first;

    // a projection on the tensor-core kernel when enabled and it fits, else on
    // the CUDA-core ring kernel
    // (gate/up + SwiGLU with one activation row stays on the CUDA-core kernel
    // unless gemv_tcgen05 = 2: with 112 unit tiles it needs split-K on the
    // tensor-core kernel, and measured slower there; from two rows on the
    // CUDA-core kernel's issue cost doubles and the tensor cores win)
    auto want_tc = [&](const GemvArgs &g) {
        return c->gemv_tcgen05 == 2 || (c->gemv_tcgen05 == 1 && (g.epi != kEpiSwiGLU || g.T > 1));
    };
    // the streamed tcgen05 kernel takes g (its activation rows in the bf16 buffer)
    auto on_tcs = [&](const GemvArgs &g, const CUtensorMap *tm) -> bool {
        // the top-1 LM head streams its rows from one row on with lm_stream
        // (not in sampled rounds, whose draw reads the logits it writes)
        const bool lm1 = c->lm_stream && g.stream_top1 && g.epi == kEpiTopK && g.topk == 1 && g.best;
        // any other LM head outside tree rounds (sampled rounds; greedy ones with
        // lm_stream off) keeps fewer than 8 rows staged:
        // at batch 1 a sampled round took 1371 us with every row streamed against
        // 1360 us with every row staged, while streaming the other projections
        // alone saves 17 us in a greedy round
        const int rows_min = g.epi == kEpiTopK && !lm1 && !(r.tree_w > 0) ? std::max(c->tc_stream_rows, 8)
                                                                            : c->tc_stream_rows;
        if (!(tm && want_tc(g) && c->tc_ready && c->bf16 && (g.T >= rows_min || lm1) &&
              gemv_tcs_supported(g, c->sms)))
            return false;
        const size_t ws = gemv_tcs_workspace_floats(g, c->sms);
        return ws == 0 || (ws <= c->tc_part_floats && gemv_tc_tiles(g) <= c->tc_ctr_n);
    };
    // the staged tcgen05 kernel takes g (when the streamed one does not)
    auto on_tc_staged = [&](const GemvArgs &g, const CUtensorMap *tm) -> bool {
        return tm && want_tc(g) && c->tc_ready && c->bf16 && gemv_tc_supported(g, c->sms);
    };
    // x_ready: the bf16 buffer already holds the rows of the next projection,
    // written by the previous projection's last kernel
    bool x_ready = false;
    auto proj = [&](GemvArgs g, const CUtensorMap *tm, int grid, bool pdl_here, const GemvArgs *next = nullptr,
                    const CUtensorMap *ntm = nullptr) -> cudaError_t {
        if (on_tcs(g, tm)) {
            if (x_ready) {
                g.pro = kProCopy;
                g.act = c->xbuf;
            }
            x_ready = false;
            if (c->fuse_rows && next && next->T == g.T && on_tcs(*next, ntm)) {
                if (g.epi == kEpiTopK && next->pro == kProFuseDecode) {
                    g.next_fuse = 1;
                    g.next_x = c->xbuf;
                } else if ((g.epi == kEpiStore || g.epi == kEpiResid) && next->pro == kProNorm &&
                           next->kin == g.n_units) {
                    g.next_norm = 1;
                    g.next_gain = next->gain;
                    g.next_x = c->xbuf;
                }
            }
            bool done = false;
            const cudaError_t le = launch_gemv_tcs(g, *tm, c->sms, c->tc_part, c->tc_ctr, c->xbuf, s, pdl_here, &done);
            x_ready = le == cudaSuccess && done;
            return le;
        }
        x_ready = false;
        if (on_tc_staged(g, tm)) {
            // split-K launches need the partial-sum workspace and one ticket per tile
            const size_t ws = gemv_tc_workspace_floats(g, c->sms);
            if (ws == 0 || (ws <= c->tc_part_floats && gemv_tc_tiles(g) <= c->tc_ctr_n))
                return launch_gemv_tc(g, *tm, c->sms, c->tc_part, c->tc_ctr, s, pdl_here);
        }
        return launch_gemv(g, c->bf16, grid, s, pdl_here);
    };

    // the caches as TMA tensor maps for the tensor-core attention kernel
    CUtensorMap tmk, tmv;
    const bool cache_maps = c->attn_fused && c->attn_tc && c->bf16 && c->tc_ready &&
                            make_cache_map(&tmk, r.k_cache, r.B * Hkv, f.max_ctx, D, fused_attention_chunk()) == cudaSuccess &&
                            make_cache_map(&tmv, r.v_cache, r.B * Hkv, f.max_ctx, D, fused_attention_chunk()) == cudaSuccess;

    // tree drafting: w rows per sequence from step 2 on
    const bool tree = r.tree_w > 0;
    const int tw = tree ? r.tree_w : 1;
    TreeArgs ta{};
    if (tree) {
        ta.B = r.B;
        ta.w = tw;
        ta.K = K;
        ta.d = d;
        ta.V = V;
        ta.Hq = Hq;
        ta.Hkv = Hkv;
        ta.D = D;
        ta.max_ctx = f.max_ctx;
        ta.max_new = f.max_new;
        ta.n_nodes = r.tree_m;
        ta.P = tw + (K - 1) * tw * tw;
        ta.n_new = r.n_new;
        ta.kv_len = r.kv_len;
        ta.err = c->err;
        ta.embed = c->embed;
        ta.hhat = c->hhat;
        ta.u_out = c->tree_u;
        ta.front_tok = c->front_tok;
        ta.front_row = c->front_row;
        ta.front_pool = c->front_pool;
        ta.front_score = c->front_score;
        ta.front_mask = c->front_mask;
        ta.pool_tok = c->pool_tok;
        ta.pool_par = c->pool_par;
        ta.pool_score = c->pool_score;
        ta.top_ids = c->tree_top_ids;
        ta.top_vals = c->tree_top_vals;
        ta.lse = c->tree_lse;
        ta.lse_part = c->tree_lse_part;
        ta.lse_ctr = c->tree_lse_ctr;
        ta.seq_ctr = c->tree_lse_ctr + c->tree_rows;
        ta.qkv = c->qkv;
        ta.k_cache = r.k_cache;
        ta.v_cache = r.v_cache;
        ta.rope_cos = c->rope_cos;
        ta.rope_sin = c->rope_sin;
        ta.attn_part = c->attn_part;
        ta.attn_ctr = c->counters;
        ta.o_out = c->o_buf;
        ta.chunk = c->attn_chunk;
        ta.splits = c->attn_splits;
        ta.tree_tokens = r.tree.tokens;
        ta.tree_parents = r.tree.parents;
        ta.tree_depths = r.tree.depths;
        ta.tree_scores = r.tree.scores;
        ta.out_pool_tokens = r.tree.pool_tokens;
        ta.out_pool_parents = r.tree.pool_parents;
        ta.out_pool_scores = r.tree.pool_scores;
        ta.out_frontier = r.tree.frontier;
    }

    // the projections of step k (rows: T1 for the fusion and QKV, which see
    // every prefill row at step 1; Trow from the O projection on)
    auto step_tm = [&](int k, int i) -> const CUtensorMap * {
        return c->tm_step_ok[k - 1] ? &c->tm_step[k - 1][i] : nullptr;
    };
    auto rows_trow = [&](int k) { return tree && k > 1 ? r.B * tw : r.B; };
    auto rows_t1 = [&](int k) { return k == 1 ? r.B * f.max_new : rows_trow(k); };
    auto fusion_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->steps[k - 1].w_fuse;
        g.n_units = d;
        g.kin = 2 * d;
        g.T = rows_t1(k);
        g.pro = k == 1 ? kProFusePrefill : (tree ? kProCopy : kProFuseDecode);
        g.src = c->hhat;
        g.act = c->tree_u;
        g.epi = kEpiStore;
        g.out = c->x0;
        g.out_ld = d;
        return g;
    };
    auto qkv_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->steps[k - 1].w_qkv;
        g.n_units = c->qkv_rows;
        g.kin = d;
        g.T = rows_t1(k);
        g.pro = kProNorm;
        g.src = c->x0;
        g.gain = c->steps[k - 1].g_attn;
        g.epi = kEpiStore;
        g.out = c->qkv;
        g.out_ld = c->qkv_rows;
        return g;
    };
    auto o_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->steps[k - 1].w_o;
        g.n_units = d;
        g.kin = Hq * D;
        g.T = rows_trow(k);
        g.pro = kProCopy;
        g.act = c->o_buf;
        g.epi = kEpiResid;
        g.resid = c->x0;
        g.resid_prefill_rows = k == 1;
        g.out = c->a;
        g.out_ld = d;
        return g;
    };
    auto gate_up_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->steps[k - 1].w_gate_up;
        g.n_units = F;
        g.pair_offset = F;
        g.kin = d;
        g.T = rows_trow(k);
        g.pro = kProNorm;
        g.src = c->a;
        g.gain = c->steps[k - 1].g_mlp;
        g.epi = kEpiSwiGLU;
        g.out_act = c->m_buf;
        g.out_ld = F;
        return g;
    };
    auto down_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->steps[k - 1].w_down;
        g.n_units = d;
        g.kin = F;
        g.T = rows_trow(k);
        g.pro = kProCopy;
        g.act = c->m_buf;
        g.epi = kEpiResid;
        g.resid = c->a;
        g.out = c->hhat;
        g.out_ld = d;
        g.hidden_out = tree ? nullptr : r.hidden_out;
        return g;
    };
    auto lm_args = [&](int k) {
        GemvArgs g = base;
        g.step = k;
        g.W = c->lm_head;
        g.even_waves = c->lm_even_waves;
        g.stream_top1 = c->lm_stream && !(r.temperature > 0.f);
        g.n_units = V;
        g.kin = d;
        g.T = rows_trow(k);
        g.pro = kProNorm;
        g.src = c->hhat;
        g.gain = f.final_norm ? c->steps[k - 1].g_final : nullptr;
        g.epi = kEpiTopK;
        g.logits = r.logits;
        g.lm_part = c->lm_val;
        g.lm_part_id = c->lm_id;
        g.counter = c->counters + (size_t)f.max_batch * Hkv;
        g.best = c->lm_best;
        g.draft_out = r.draft;
        g.topk_ids = r.topk_ids;
        g.topk_logits = r.topk_logits;
        if (tree) {
            // rows b * w + j of [B * w, .] buffers: at step 1 (one row per
            // sequence) K = w puts row b at b * w; later steps index by row
            float *lg = r.tree.row_logits ? r.tree.row_logits + (size_t)(k - 1) * r.B * tw * V : c->tree_logits;
            g.K = k == 1 ? tw : 1;
            g.step = 1;
            g.topk = tw;
            g.logits = lg;
            g.draft_out = c->tree_draft;
            g.topk_ids = c->tree_top_ids;
            g.topk_logits = c->tree_top_vals;
            g.best = nullptr;           // the list path, which also yields the log-sum-exp partials
            // on a tcgen05 kernel the LM head also writes each row's per-CTA
            // log-sum-exp partials, and the logits only when the caller wants them
            const CUtensorMap *ltm = c->tm_lm_ok ? &c->tm_lm : nullptr;
            if (on_tcs(g, ltm) || on_tc_staged(g, ltm)) {
                g.lse_part = c->tree_lse_part;
                if (!r.tree.row_logits) g.logits = nullptr;
                // the per-CTA lists are merged by the tree's lse kernel, one CTA per row
                g.defer_merge = c->tree_defer_merge;
            }
        }
        return g;
    };
    const CUtensorMap *lm_tm = c->tm_lm_ok ? &c->tm_lm : nullptr;
    // a kernel's CTAs, once their own weights are requested, request the next
    // kernel's first bytes into L2
    const size_t wes = c->bf16 ? 2 : 4;
    auto pf = [&](const void *w, size_t elems) -> std::pair<const void *, long long> {
        const long long cap = (long long)c->prefetch_next_kb * 1024;
        if (!w || cap <= 0) return {nullptr, 0};
        return {w, std::min(cap, (long long)(elems * wes))};
    };
    auto with_pf = [&](GemvArgs g, std::pair<const void *, long long> n) {
        g.pf_next = n.first;
        g.pf_next_bytes = n.second;
        return g;
    };

    for (int k = 1; k <= K && e == cudaSuccess; ++k) {
        const bool prefill = k == 1;
        const bool tstep = tree && !prefill;       // a tree step: w rows per sequence
        const int Trow = tstep ? r.B * tw : r.B;   // rows from attention on
        const int T1 = prefill ? r.B * f.max_new : Trow;
        const bool p = pdl && !first;
        ta.step = k;
        ta.R = prefill ? 1 : tw;

        if (tstep) {
            // fusion input rows [E(token); round(h^ of the emitting row)]
            e = launch_tree_gather(ta, c->bf16, s, p);
            after(9);
            if (e != cudaSuccess) break;
        }

        // fusion F(E(x), h), then the attention pre-norm + QKV, whose rows the
        // fusion's last kernel can write
        const GemvArgs gq = qkv_args(k);
        e = proj(with_pf(fusion_args(k), pf(c->steps[k - 1].w_qkv, (size_t)c->qkv_rows * d)), step_tm(k, 0),
                 gemv_grid(c, d), tstep ? pdl : p, &gq, step_tm(k, 1));
        after(0);
        if (e != cudaSuccess) break;
        e = proj(gq, step_tm(k, 1), gemv_grid(c, c->qkv_rows), pdl);
        after(1);
        if (e != cudaSuccess) break;

        if (tstep) {
            // RoPE at the node's depth, K/V appended at its own slot, attention
            // over the committed rows and the node's ancestors: one kernel
            const auto n = pf(c->steps[k - 1].w_o, (size_t)d * Hq * D);
            ta.pf_next = n.first;
            ta.pf_next_bytes = n.second;
            e = launch_tree_attention(ta, c->bf16, s, pdl);
            after(3);
            if (e != cudaSuccess) break;
        } else if (c->attn_fused) {
            // RoPE + KV append + attention in one cluster launch per (sequence, KV head)
            FusedAttnArgs fa{};
            fa.qkv = c->qkv;
            fa.k_cache = r.k_cache;
            fa.v_cache = r.v_cache;
            fa.o_out = c->o_buf;
            fa.rope_cos = c->rope_cos;
            fa.rope_sin = c->rope_sin;
            fa.n_new = r.n_new;
            fa.kv_len = r.kv_len;
            fa.B = r.B;
            fa.max_new = f.max_new;
            fa.prefill = prefill;
            fa.step = k;
            fa.Hq = Hq;
            fa.Hkv = Hkv;
            fa.D = D;
            fa.max_ctx = f.max_ctx;
            fa.cs = c->attn_max_cs;
            while (fa.cs > 1 && (long long)r.B * Hkv * fa.cs > (long long)c->attn_ctas_per_sm * c->sms) fa.cs /= 2;
            fa.err = c->err;
            fa.wait_polls = c->wait_polls;
            {
                const auto n = pf(c->steps[k - 1].w_o, (size_t)d * Hq * D);
                fa.pf_next = n.first;
                fa.pf_next_bytes = n.second;
            }
            // more CTAs than SMs but no more than two per SM: 4-warp CTAs, two per
            // SM, run as one wave instead of two
            const long long ctas = (long long)r.B * Hkv * fa.cs;
            fa.warps = c->attn_warps ? c->attn_warps : fa.cs == 1 && ctas > c->sms && ctas <= 2LL * c->sms ? 4 : 8;
            if (fa.warps == 4 && fa.cs > 8) fa.cs = 8;   // clusters of 16 are checked for the 8-warp kernel only
            // more than one wave of CTAs but at most two: the longest sequences
            // first (with more waves the hardware's scheduling already evens
            // them out and each CTA's ranking of the sequences costs more than
            // the order gains: batch 16, 1498 -> 1488 us; batch 64, 2111 ->
            // 2141 us)
            const long long per_wave = (long long)c->sms * (fa.warps == 4 ? 2 : 1);
            const long long n_ctas = (long long)r.B * Hkv * fa.cs;
            fa.lpt = c->attn_lpt && r.B > 1 && r.B <= 256 && n_ctas > per_wave && n_ctas <= 2 * per_wave;
            e = launch_fused_attention(fa, c->bf16, s, pdl, cache_maps ? &tmk : nullptr, cache_maps ? &tmv : nullptr);
            after(3);
            if (e != cudaSuccess) break;
        } else {
        // RoPE + KV append (+ rotated q of the query rows)
        RopeArgs ra{};
        ra.qkv = c->qkv;
        ra.k_cache = r.k_cache;
        ra.v_cache = r.v_cache;
        ra.q_out = c->q;
        ra.rope_cos = c->rope_cos;
        ra.rope_sin = c->rope_sin;
        ra.n_new = r.n_new;
        ra.kv_len = r.kv_len;
        ra.B = r.B;
        ra.max_new = f.max_new;
        ra.rows = T1;
        ra.prefill = prefill;
        ra.step = k;
        ra.K = K;
        ra.Hq = Hq;
        ra.Hkv = Hkv;
        ra.D = D;
        ra.max_ctx = f.max_ctx;
        ra.err = c->err;
        e = launch_rope_append(ra, c->bf16, s, pdl);
        after(2);
        if (e != cudaSuccess) break;

        // split-KV attention with last-CTA combine
        AttnArgs aa{};
        aa.q = c->q;
        aa.k_cache = r.k_cache;
        aa.v_cache = r.v_cache;
        aa.part = c->attn_part;
        aa.counter = c->counters;
        aa.o_out = c->o_buf;
        aa.n_new = r.n_new;
        aa.kv_len = r.kv_len;
        aa.B = r.B;
        aa.max_new = f.max_new;
        aa.prefill = prefill;
        aa.step = k;
        aa.Hq = Hq;
        aa.Hkv = Hkv;
        aa.D = D;
        aa.max_ctx = f.max_ctx;
        aa.chunk = c->attn_chunk;
        aa.splits = c->attn_splits;
        aa.err = c->err;
        e = launch_attention(aa, c->bf16, s, pdl);
        after(3);
        if (e != cudaSuccess) break;
        }

        // O projection + residual; MLP pre-norm + gate/up + SwiGLU; down
        // projection + residual -> h^_{k-1}; final norm + LM head + top-8
        // selection -> x^_k.  Each hands its rows to the next where it can;
        // the LM head to the next step's fusion in a greedy chain.
        const GemvArgs gg = gate_up_args(k), gl = lm_args(k);
        e = proj(with_pf(o_args(k), pf(c->steps[k - 1].w_gate_up, (size_t)2 * F * d)), step_tm(k, 2),
                 gemv_grid(c, d), pdl, &gg, step_tm(k, 3));
        after(4);
        if (e != cudaSuccess) break;
        e = proj(with_pf(gg, pf(c->steps[k - 1].w_down, (size_t)d * F)), step_tm(k, 3), gemv_grid(c, F), pdl);
        after(5);
        if (e != cudaSuccess) break;
        e = proj(with_pf(down_args(k), pf(c->lm_head, (size_t)V * d)), step_tm(k, 4), gemv_grid(c, d), pdl, &gl,
                 lm_tm);
        after(6);
        if (e != cudaSuccess) break;
        const bool chain_next = k < K && !tree && !(r.temperature > 0.f);
        const GemvArgs gn = chain_next ? fusion_args(k + 1) : GemvArgs{};
        e = proj(with_pf(gl, pf(k < K ? c->steps[k].w_fuse : nullptr, (size_t)d * 2 * d)), lm_tm, c->lm_grid, pdl,
                 chain_next ? &gn : nullptr, chain_next ? step_tm(k + 1, 0) : nullptr);
        if (tree) {
            ta.logits = gl.logits;
            // the LM head's grid (one log-sum-exp partial per CTA and row): one
            // CTA per SM, or with even waves the fewest CTAs for as many waves
            const int lm_tiles = (V + 127) / 128;
            int lm_ctas = lm_tiles < c->sms ? lm_tiles : c->sms;
            if (c->lm_even_waves) lm_ctas = (lm_tiles + (lm_tiles + lm_ctas - 1) / lm_ctas - 1) / ((lm_tiles + lm_ctas - 1) / lm_ctas);
            ta.lm_lse_grid = gl.lse_part ? lm_ctas : 0;
            ta.lm_val = gl.defer_merge ? c->lm_val : nullptr;
            ta.lm_id = gl.defer_merge ? c->lm_id : nullptr;
        }
        after(7);
        if (e != cudaSuccess) break;

        if (tree) {
            // draft log-probabilities; the last row of each sequence then scores
            // the candidates and picks the next frontier (and the tree after step K)
            e = launch_tree_lse(ta, s, pdl);
            after(10);
            if (e != cudaSuccess) break;
            continue;
        }

        if (r.temperature > 0.f) {
            // x^_k drawn from softmax(z / T): replaces the argmax before the next step reads it
            SampleArgs sa{};
            sa.logits = r.logits;
            sa.seed = r.seed;
            sa.draft = r.draft;
            sa.lse = r.lse;
            sa.part = c->sample_part;
            sa.counter = c->sample_ctr;
            sa.temperature = r.temperature;
            sa.V = V;
            sa.K = K;
            sa.step = k;
            e = launch_sample(sa, r.B, s, pdl);
            after(8);
        }
    }
    if (n_kernels) *n_kernels = nk;
    return e;
}

prism_status check_round_args(prism_ctx *c, const RoundArgs &r) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (r.B < 1) return fail(c, PRISM_ERR_SHAPE, "batch must be >= 1");
    if (r.B > c->cfg.max_batch) return fail(c, PRISM_ERR_CAPACITY, "batch exceeds max_batch");
    if (!r.tokens || !r.hidden || !r.n_new || !r.kv_len || !r.k_cache || !r.v_cache || !r.draft)
        return fail(c, PRISM_ERR_INVALID_ARG, "null tensor argument");
    if (!aligned16(r.hidden) || !aligned16(r.k_cache) || !aligned16(r.v_cache))
        return fail(c, PRISM_ERR_INVALID_ARG, "hidden, k_cache and v_cache must be 16-byte aligned");
    if (!c->embed || !c->lm_head) return fail(c, PRISM_ERR_NOT_LOADED, "shared weights not loaded");
    for (int k = 0; k < c->cfg.n_steps; ++k)
        if (!c->step_loaded[k]) return fail(c, PRISM_ERR_NOT_LOADED, "weights of step " + std::to_string(k) + " not loaded");
    return PRISM_OK;
}

}  // namespace

extern "C" {

const char *prism_version(void) { return "prism-gb300 0.1 (sm_103a)"; }

const char *prism_get_error(const prism_ctx *ctx) {
    return ctx ? ctx->error.c_str() : g_error.c_str();
}

prism_status prism_create(const prism_config *cfg, int32_t device, prism_ctx **out) {
    if (!cfg || !out) return fail(nullptr, PRISM_ERR_INVALID_ARG, "null argument");
    *out = nullptr;
    const prism_config &f = *cfg;
    if (f.hidden < 8 || f.hidden % 8 || f.n_q_heads < 1 || f.n_kv_heads < 1 || f.n_q_heads % f.n_kv_heads ||
        (f.head_dim != 64 && f.head_dim != 128) || f.ffn < 8 || f.ffn % 8 || f.vocab < kTopK ||
        f.n_steps < 1 || f.n_steps > kMaxSteps || f.max_batch < 1 || f.max_ctx < 2 || f.max_new < 1 ||
        f.topk < 1 || f.topk > kTopK || (f.dtype != PRISM_F32 && f.dtype != PRISM_BF16) ||
        f.n_q_heads / f.n_kv_heads > 16 || !(f.rms_eps >= 0.f) || !(f.rope_theta > 0.f) ||
        f.max_tree_width < 0 || f.max_tree_width > kTreeMaxWidth)
        return fail(nullptr, PRISM_ERR_INVALID_ARG, "unsupported configuration");
    prism_ctx *c = new prism_ctx();
    c->cfg = f;
    c->device = device;
    c->bf16 = f.dtype == PRISM_BF16;
    cudaError_t e = cudaSetDevice(device);
    if (e != cudaSuccess) { delete c; return cuda_fail(nullptr, e, "cudaSetDevice"); }
    cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, device);
    const int d = f.hidden, Hq = f.n_q_heads, Hkv = f.n_kv_heads, D = f.head_dim, F = f.ffn;
    const size_t es = c->bf16 ? 2 : 4;
    c->qkv_rows = (Hq + 2 * Hkv) * D;
    c->lm_grid = f.vocab < c->sms ? f.vocab : c->sms;
    // attention split size: 64 keys, larger when the split count would exceed
    // what the last-CTA combine reads per lane (256 splits)
    c->attn_chunk = 64;
    while ((f.max_ctx + c->attn_chunk - 1) / c->attn_chunk > 256) c->attn_chunk *= 2;
    c->attn_splits = (f.max_ctx + c->attn_chunk - 1) / c->attn_chunk;

    // rows per sequence after step 1: w for tree rounds, else 1
    const size_t TW = f.max_tree_width > 0 ? (size_t)f.max_tree_width : 1;
    const size_t Bw = (size_t)f.max_batch * TW;
    const size_t T1 = std::max((size_t)f.max_batch * f.max_new, Bw), B = Bw, Bseq = f.max_batch;
    const size_t tree_on = f.max_tree_width > 0 ? 1 : 0;
    const size_t P_max = TW + (size_t)(f.n_steps - 1) * TW * TW;
    // split-K workspace of the tensor-core projections: the largest need of
    // any projection of this shape
    size_t tc_floats = 0;
    int tc_tiles = 0;
    if (c->bf16) {
        const int units[] = {d, c->qkv_rows, d, F, d};
        const int kins[] = {2 * d, d, Hq * D, d, F};
        const int epis[] = {kEpiStore, kEpiStore, kEpiResid, kEpiSwiGLU, kEpiResid};
        const int pros[] = {kProFuseDecode, kProNorm, kProCopy, kProNorm, kProCopy};
        for (int i = 0; i < 5; ++i)
            for (int T : {(int)T1, (int)B, (int)Bseq}) {
                GemvArgs g{};
                g.n_units = units[i];
                g.kin = kins[i];
                g.epi = epis[i];
                g.pro = pros[i];
                g.T = T;
                size_t need = gemv_tc_workspace_floats(g, c->sms);
                if (need > tc_floats) tc_floats = need;
                need = gemv_tcs_workspace_floats(g, c->sms);
                if (need > tc_floats) tc_floats = need;
                if (gemv_tc_tiles(g) > tc_tiles) tc_tiles = gemv_tc_tiles(g);
            }
    }
    size_t sizes[] = {
        (size_t)f.max_ctx * (D / 2) * 4,                           // rope cos
        (size_t)f.max_ctx * (D / 2) * 4,                           // rope sin
        T1 * d * 4,                                                // x0
        T1 * c->qkv_rows * 4,                                      // qkv
        B * Hq * D * 4,                                            // q
        B * Hq * (size_t)c->attn_splits * (D + 4) * 4,             // attention partials
        B * d * 4,                                                 // a
        B * d * 4,                                                 // h^
        B * Hq * D * es,                                           // o
        B * F * es,                                                // m
        B * (size_t)c->lm_grid * kTopK * 4,                        // LM partial values
        B * (size_t)c->lm_grid * kTopK * 4,                        // LM partial ids
        (Bseq * Hkv + 1) * 4,                                      // counters
        B * 8,                                                     // LM head packed top-1 keys
        32,                                                        // error word (+ checked-build record)
        tc_floats * 4,                                             // tensor-core split-K partials
        (size_t)tc_tiles * 4,                                      // tensor-core tile tickets
        T1 * 2 * d * es,                                           // streamed-kernel activation rows
        B * (size_t)kSampleMaxBlocks * 4 * 4,                      // sampled-draft partials
        B * 4,                                                     // sampled-draft tickets
        tree_on * Bw * 2 * d * es,                                 // tree fusion inputs
        tree_on * Bw * f.vocab * 4,                                // tree row logits
        tree_on * Bw * kTopK * 4,                                  // tree top-w ids
        tree_on * Bw * kTopK * 4,                                  // tree top-w logits
        tree_on * Bw * 4,                                          // tree LM-head top-1 (unused)
        tree_on * Bw * 4,                                          // tree row lse
        tree_on * Bw * (size_t)(c->lm_grid > kSampleMaxBlocks ? c->lm_grid : kSampleMaxBlocks) * 2 * 4,  // tree lse partials
        tree_on * (Bw + Bseq) * 4,                                 // tree lse tickets, sequence tickets
        tree_on * Bw * 4 * 4,                                      // frontier token, row, pool index, score
        tree_on * Bw * 8,                                          // frontier ancestor masks
        tree_on * Bseq * P_max * 4 * 3,                            // pool tokens, parents, scores
    };
    size_t total = 0;
    for (size_t s : sizes) total += align256(s);
    void *ws = nullptr;
    e = cudaMalloc(&ws, total);
    if (e != cudaSuccess) { delete c; return fail(nullptr, PRISM_ERR_OOM, std::string("workspace: ") + cudaGetErrorString(e)); }
    cudaMemset(ws, 0, total);
    c->ws = ws;
    c->ws_bytes = total;
    uint8_t *p = (uint8_t *)ws;
    void *slot[sizeof(sizes) / sizeof(sizes[0])];
    for (size_t i = 0; i < sizeof(sizes) / sizeof(sizes[0]); ++i) { slot[i] = p; p += align256(sizes[i]); }
    c->rope_cos = (float *)slot[0];
    c->rope_sin = (float *)slot[1];
    c->x0 = (float *)slot[2];
    c->qkv = (float *)slot[3];
    c->q = (float *)slot[4];
    c->attn_part = (float *)slot[5];
    c->a = (float *)slot[6];
    c->hhat = (float *)slot[7];
    c->o_buf = slot[8];
    c->m_buf = slot[9];
    c->lm_val = (float *)slot[10];
    c->lm_id = (int *)slot[11];
    c->counters = (int *)slot[12];
    c->lm_best = (unsigned long long *)slot[13];
    c->err = (int *)slot[14];
    c->tc_part = (float *)slot[15];
    c->tc_part_floats = tc_floats;
    c->tc_ctr = (int *)slot[16];
    c->tc_ctr_n = tc_tiles;
    c->xbuf = (uint16_t *)slot[17];
    c->sample_part = (float *)slot[18];
    c->sample_ctr = (int *)slot[19];
    c->tree_rows = (int)Bw;
    c->tree_u = slot[20];
    c->tree_logits = (float *)slot[21];
    c->tree_top_ids = (int32_t *)slot[22];
    c->tree_top_vals = (float *)slot[23];
    c->tree_draft = (int32_t *)slot[24];
    c->tree_lse = (float *)slot[25];
    c->tree_lse_part = (float *)slot[26];
    c->tree_lse_ctr = (int *)slot[27];
    c->front_tok = (int32_t *)slot[28];
    c->front_row = c->front_tok + Bw;
    c->front_pool = c->front_row + Bw;
    c->front_score = (float *)(c->front_pool + Bw);
    c->front_mask = (unsigned long long *)slot[29];
    c->pool_tok = (int32_t *)slot[30];
    c->pool_par = c->pool_tok + Bseq * P_max;
    c->pool_score = (float *)(c->pool_par + Bseq * P_max);

    // rotary tables: angle p * theta^(-2j/D), computed in double, stored as float
    std::vector<float> cs((size_t)f.max_ctx * (D / 2)), sn((size_t)f.max_ctx * (D / 2));
    for (int pos = 0; pos < f.max_ctx; ++pos)
        for (int j = 0; j < D / 2; ++j) {
            const double inv = std::pow((double)f.rope_theta, -2.0 * j / (double)D);
            const double ang = (double)pos * inv;
            cs[(size_t)pos * (D / 2) + j] = (float)std::cos(ang);
            sn[(size_t)pos * (D / 2) + j] = (float)std::sin(ang);
        }
    e = cudaMemcpy(c->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = prepare_gemv_kernels();
    if (e == cudaSuccess && c->bf16) {
        // the tensor-core path is optional: without a tensor-map encoder the
        // CUDA-core kernels run everything
        c->tc_ready = prepare_gemv_tc_kernels() == cudaSuccess;
        cudaGetLastError();
    }
    if (e == cudaSuccess) {
        // every projection shape must fit the shared-memory ring
        const int T1 = f.max_batch * f.max_new;
        const int kins[] = {2 * d, d, Hq * D, d, F, d};
        const int epis[] = {kEpiStore, kEpiStore, kEpiResid, kEpiSwiGLU, kEpiResid, kEpiTopK};
        for (int i = 0; i < 6; ++i) {
            GemvArgs g{};
            g.kin = kins[i];
            g.epi = epis[i];
            g.T = i < 2 ? (int)T1 : (int)B;
            if (!gemv_supported(g, c->bf16)) {
                cudaFree(ws);
                delete c;
                return fail(nullptr, PRISM_ERR_INVALID_ARG, "a projection row does not fit shared memory");
            }
        }
    }
    if (e == cudaSuccess && attention_smem_bytes(c->bf16, D, c->attn_chunk, Hq / Hkv, c->attn_splits) > 200 * 1024) {
        cudaFree(ws);
        delete c;
        return fail(nullptr, PRISM_ERR_INVALID_ARG, "max_ctx too large for the attention combine");
    }
    if (e == cudaSuccess) e = prepare_attention_kernel(c->bf16, D, c->attn_chunk, Hq / Hkv, c->attn_splits);
    if (e == cudaSuccess) e = prepare_fused_attention(c->bf16, D, Hq / Hkv, Hkv, &c->attn_max_cs);
    if (e == cudaSuccess && tree_on) {
        if (tree_attention_smem_bytes(c->bf16, D, c->attn_chunk, Hq / Hkv, (int)TW, c->attn_splits) > 200 * 1024) {
            cudaFree(ws);
            delete c;
            return fail(nullptr, PRISM_ERR_INVALID_ARG, "max_ctx too large for the tree attention combine");
        }
        e = prepare_tree_kernels(c->bf16, D, c->attn_chunk, Hq / Hkv, (int)TW, c->attn_splits, f.max_ctx);
    }
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking);
    if (e != cudaSuccess) {
        prism_status st = cuda_fail(nullptr, e, "context setup");
        cudaFree(ws);
        delete c;
        return st;
    }
    *out = c;
    return PRISM_OK;
}

prism_status prism_destroy(prism_ctx *c) {
    if (!c) return PRISM_OK;
    cudaSetDevice(c->device);
    cudaDeviceSynchronize();
    drop_graphs(c);
    if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
    if (c->ws) cudaFree(c->ws);
    delete c;
    return PRISM_OK;
}

prism_status prism_load_shared_weights(prism_ctx *c, const void *embed, const void *lm_head) {
    if (!c || !embed || !lm_head) return fail(c, PRISM_ERR_INVALID_ARG, "null argument");
    if (!aligned16(embed) || !aligned16(lm_head))
        return fail(c, PRISM_ERR_INVALID_ARG, "embed and lm_head must be 16-byte aligned");
    c->embed = embed;
    c->lm_head = lm_head;
    c->tm_lm_ok = c->tc_ready && make_weight_map(&c->tm_lm, lm_head, c->cfg.vocab, c->cfg.hidden) == cudaSuccess;
    drop_graphs(c);
    return PRISM_OK;
}

prism_status prism_load_step_weights(prism_ctx *c, int32_t step, const prism_step_weights *w) {
    if (!c || !w) return fail(c, PRISM_ERR_INVALID_ARG, "null argument");
    if (step < 0 || step >= c->cfg.n_steps) return fail(c, PRISM_ERR_INVALID_ARG, "step out of range");
    if (!w->w_fuse || !w->g_attn || !w->w_qkv || !w->w_o || !w->g_mlp || !w->w_gate_up || !w->w_down ||
        (c->cfg.final_norm && !w->g_final))
        return fail(c, PRISM_ERR_INVALID_ARG, "null weight pointer");
    for (const void *p : {w->w_fuse, w->g_attn, w->w_qkv, w->w_o, w->g_mlp, w->w_gate_up, w->w_down, w->g_final})
        if (p && !aligned16(p)) return fail(c, PRISM_ERR_INVALID_ARG, "weight pointers must be 16-byte aligned");
    c->steps[step] = *w;
    c->step_loaded[step] = true;
    if (c->tc_ready) {
        const prism_config &f = c->cfg;
        const int d = f.hidden, F = f.ffn;
        CUtensorMap *m = c->tm_step[step];
        c->tm_step_ok[step] = make_weight_map(&m[0], w->w_fuse, d, 2 * d) == cudaSuccess &&
                              make_weight_map(&m[1], w->w_qkv, c->qkv_rows, d) == cudaSuccess &&
                              make_weight_map(&m[2], w->w_o, d, f.n_q_heads * f.head_dim) == cudaSuccess &&
                              make_weight_map(&m[3], w->w_gate_up, 2 * F, d) == cudaSuccess &&
                              make_weight_map(&m[4], w->w_down, d, F) == cudaSuccess;
    }
    drop_graphs(c);
    return PRISM_OK;
}

prism_status prism_set_option(prism_ctx *c, const char *name, int32_t value) {
    if (!c || !name) return fail(c, PRISM_ERR_INVALID_ARG, "null argument");
    if (!std::strcmp(name, "use_graph")) c->use_graph = value != 0;
    else if (!std::strcmp(name, "use_pdl")) c->use_pdl = value != 0;
    else if (!std::strcmp(name, "gemv_chunk_kb") && value >= 0 && value <= 128) c->gemv_chunk = value * 1024;
    else if (!std::strcmp(name, "gemv_smem_kb") && value >= 0 && value <= 200) c->gemv_smem = value * 1024;
    else if (!std::strcmp(name, "gemv_groups") && (value == 0 || value == 1 || value == 2 || value == 4 ||
                                                   value == 8 || value == 16)) c->gemv_groups = value;
    else if (!std::strcmp(name, "gemv_cuda_core")) c->gemv_cuda_core = value != 0;
    else if (!std::strcmp(name, "gemv_tcgen05") && value >= 0 && value <= 2) c->gemv_tcgen05 = value;
    else if (!std::strcmp(name, "attn_fused")) c->attn_fused = value != 0;
    else if (!std::strcmp(name, "tc_stream_rows") && value >= 1) c->tc_stream_rows = value;
    else if (!std::strcmp(name, "attn_ctas_per_sm") && value >= 1 && value <= 64) c->attn_ctas_per_sm = value;
    else if (!std::strcmp(name, "fuse_rows")) c->fuse_rows = value != 0;
    else if (!std::strcmp(name, "wait_polls")) c->wait_polls = value;
    else if (!std::strcmp(name, "w_evict_first")) c->w_evict_first = value != 0;
    else if (!std::strcmp(name, "attn_tc")) c->attn_tc = value != 0;
    else if (!std::strcmp(name, "prefetch_next_kb")) {
        if (value < 0) return fail(c, PRISM_ERR_INVALID_ARG, "prefetch_next_kb must be >= 0");
        c->prefetch_next_kb = value;
    } else if (!std::strcmp(name, "lm_stream")) {
        c->lm_stream = value != 0;
    } else if (!std::strcmp(name, "tree_defer_merge")) {
        c->tree_defer_merge = value != 0;
    } else if (!std::strcmp(name, "lm_even_waves")) {
        c->lm_even_waves = value != 0;
    } else if (!std::strcmp(name, "attn_lpt")) {
        c->attn_lpt = value != 0;
    } else if (!std::strcmp(name, "attn_warps")) {
        if (value != 0 && value != 4 && value != 8) return fail(c, PRISM_ERR_INVALID_ARG, "attn_warps must be 0, 4 or 8");
        c->attn_warps = value;
    }
    else return fail(c, PRISM_ERR_INVALID_ARG, std::string("unknown option ") + name);
    drop_graphs(c);
    return PRISM_OK;
}

}  // extern "C"

namespace {

// One round, as a replayed graph (captured on first use per argument set) or eagerly.
prism_status run_round(prism_ctx *c, const RoundArgs &r, void *stream) {
    prism_status st = check_round_args(c, r);
    if (st != PRISM_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaSetDevice(c->device);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaSetDevice");
    if (!c->use_graph) {
        e = enqueue_round(c, r, s, c->use_pdl, nullptr, nullptr, nullptr);
        return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "kernel launch");
    }
    GraphEntry *hit = nullptr;
    for (auto &g : c->graphs)
        if (g.key == r && g.pdl == c->use_pdl) hit = &g;
    if (!hit) {
        if ((int)c->graphs.size() >= kGraphCache) {
            size_t old = 0;
            for (size_t i = 1; i < c->graphs.size(); ++i)
                if (c->graphs[i].used < c->graphs[old].used) old = i;
            cudaGraphExecDestroy(c->graphs[old].exec);
            c->graphs.erase(c->graphs.begin() + old);
        }
        cudaGraph_t graph = nullptr;
        e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamBeginCapture");
        cudaError_t le = enqueue_round(c, r, c->cap_stream, c->use_pdl, nullptr, nullptr, nullptr);
        e = cudaStreamEndCapture(c->cap_stream, &graph);
        if (le != cudaSuccess) {
            if (graph) cudaGraphDestroy(graph);
            return cuda_fail(c, le, "kernel launch during capture");
        }
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamEndCapture");
        // the round's kernel launches, as the graph holds them
        int kernels = 0;
        size_t n_nodes = 0;
        if (cudaGraphGetNodes(graph, nullptr, &n_nodes) == cudaSuccess && n_nodes > 0) {
            std::vector<cudaGraphNode_t> nodes(n_nodes);
            if (cudaGraphGetNodes(graph, nodes.data(), &n_nodes) == cudaSuccess)
                for (size_t i = 0; i < n_nodes; ++i) {
                    cudaGraphNodeType t;
                    if (cudaGraphNodeGetType(nodes[i], &t) == cudaSuccess && t == cudaGraphNodeTypeKernel) ++kernels;
                }
        }
        cudaGraphExec_t exec = nullptr;
        e = cudaGraphInstantiate(&exec, graph, 0);
        cudaGraphDestroy(graph);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaGraphInstantiate");
        c->graphs.push_back(GraphEntry{r, c->use_pdl, exec, 0, kernels});
        hit = &c->graphs.back();
    }
    hit->used = ++c->tick;
    c->last_round_kernels = hit->kernels;
    e = cudaGraphLaunch(hit->exec, s);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "cudaGraphLaunch");
}

}  // namespace

extern "C" {

prism_status prism_draft_round(prism_ctx *c, int32_t batch, const int32_t *tokens, const void *hidden,
                               const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                               int32_t *draft_ids, int32_t *topk_ids, float *topk_logits, float *logits,
                               float *hidden_out, void *stream) {
    return run_round(c, round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids, topk_ids,
                                   topk_logits, logits, hidden_out), stream);
}

prism_status prism_draft_round_sampled(prism_ctx *c, int32_t batch, const int32_t *tokens, const void *hidden,
                                       const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                                       float temperature, const uint64_t *seed, int32_t *draft_ids,
                                       int32_t *topk_ids, float *topk_logits, float *logits, float *draft_lse,
                                       float *hidden_out, void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!(temperature > 0.f) || !std::isfinite(temperature))
        return fail(c, PRISM_ERR_INVALID_ARG, "temperature must be a finite value > 0");
    if (!seed || ((uintptr_t)seed & 7) || !logits || !draft_lse)
        return fail(c, PRISM_ERR_INVALID_ARG, "sampled rounds need seed (8-byte aligned), logits and draft_lse");
    if (c->cfg.max_batch >= (1 << 20) || c->cfg.n_steps > 255)
        return fail(c, PRISM_ERR_CAPACITY, "random-stream counter: batch below 2^20, steps below 256");
    RoundArgs r = round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids, topk_ids,
                             topk_logits, logits, hidden_out);
    r.temperature = temperature;
    r.seed = seed;
    r.lse = draft_lse;
    return run_round(c, r, stream);
}

prism_status prism_draft_tree(prism_ctx *c, int32_t batch, const int32_t *tokens, const void *hidden,
                              const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                              int32_t width, int32_t n_nodes, const prism_tree_outputs *out, void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!out || !out->tokens || !out->parents || !out->depths || !out->scores)
        return fail(c, PRISM_ERR_INVALID_ARG, "tree outputs: tokens, parents, depths and scores are required");
    if (width < 1 || width > kTreeMaxWidth || width > c->cfg.vocab)
        return fail(c, PRISM_ERR_INVALID_ARG, "tree width must be in 1..8");
    if (width > c->cfg.max_tree_width)
        return fail(c, PRISM_ERR_CAPACITY, "tree width exceeds the context's max_tree_width");
    const long K = c->cfg.n_steps;
    const long P = width + (K - 1) * width * width;
    if ((K - 1) * width > kTreeMaskBits || P > kTreeMaxPool)
        return fail(c, PRISM_ERR_INVALID_ARG, "tree too large: (K - 1) * width must be <= 64 and the pool <= 1024");
    if (n_nodes < 1 || n_nodes > P) return fail(c, PRISM_ERR_INVALID_ARG, "n_nodes must be in 1..w + (K - 1) w^2");
    RoundArgs r = round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, c->tree_draft, nullptr,
                             nullptr, nullptr, nullptr);
    r.tree_w = width;
    r.tree_m = n_nodes;
    r.tree = *out;
    return run_round(c, r, stream);
}

prism_status prism_accept_tree(prism_ctx *c, int32_t batch, int32_t n_nodes, const int32_t *tree_tokens,
                               const int32_t *tree_parents, const int32_t *target_next, const int32_t *n_new,
                               int32_t *kv_len, int32_t *accept_len, int32_t *accept_nodes, int32_t *out_tokens,
                               void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!tree_tokens || !tree_parents || !target_next || !n_new || !kv_len || !accept_len || !accept_nodes ||
        !out_tokens)
        return fail(c, PRISM_ERR_INVALID_ARG, "null tensor argument");
    if (batch < 1 || n_nodes < 1) return fail(c, PRISM_ERR_SHAPE, "batch and n_nodes must be >= 1");
    if (batch > c->cfg.max_batch) return fail(c, PRISM_ERR_CAPACITY, "batch exceeds max_batch");
    cudaSetDevice(c->device);
    AcceptTreeArgs a{tree_tokens, tree_parents, target_next, n_new, kv_len, accept_len, accept_nodes, out_tokens,
                     batch, n_nodes, c->cfg.n_steps};
    cudaError_t e = launch_accept_tree(a, (cudaStream_t)stream);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "tree accept kernel launch");
}

}  // extern "C"

namespace {

// rounds x (draft round, acceptance that also writes the next round's tokens
// and n_new), all on the device
cudaError_t enqueue_loop(prism_ctx *c, const LoopArgs &L, cudaStream_t s, bool pdl) {
    const prism_config &f = c->cfg;
    const int B = L.r0.B, K = f.n_steps;
    const size_t es = c->bf16 ? 2 : 4;
    const size_t hid_stride = (size_t)B * f.max_new * f.hidden * es;
    cudaError_t e = cudaSuccess;
    for (int i = 0; i < L.rounds && e == cudaSuccess; ++i) {
        RoundArgs r = L.r0;
        r.hidden = (const uint8_t *)L.r0.hidden + i * hid_stride;
        r.draft = L.r0.draft + (size_t)i * B * K;
        e = enqueue_round(c, r, s, pdl, nullptr, nullptr, nullptr);
        if (e != cudaSuccess) break;
        AcceptArgs a{r.draft, L.target + (size_t)i * B * (K + 1), r.n_new, const_cast<int32_t *>(r.kv_len),
                     L.accept_len + (size_t)i * B, L.out_tokens + (size_t)i * B * (K + 1), B, K,
                     const_cast<int32_t *>(r.tokens), const_cast<int32_t *>(r.n_new), f.max_new};
        e = launch_accept(a, s);
    }
    return e;
}

}  // namespace

extern "C" {

prism_status prism_draft_loop(prism_ctx *c, int32_t batch, int32_t rounds, int32_t *tokens, const void *hidden,
                              int32_t *n_new, int32_t *kv_len, void *k_cache, void *v_cache, const int32_t *target,
                              int32_t *draft_ids, int32_t *accept_len, int32_t *out_tokens, void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (rounds < 1) return fail(c, PRISM_ERR_SHAPE, "rounds must be >= 1");
    if (!target || !accept_len || !out_tokens) return fail(c, PRISM_ERR_INVALID_ARG, "null tensor argument");
    if (c->cfg.max_new < c->cfg.n_steps + 1)
        return fail(c, PRISM_ERR_CAPACITY, "a loop needs max_new >= K + 1 (the next round prefills up to K + 1 tokens)");
    LoopArgs L;
    std::memset(&L, 0, sizeof L);
    L.r0 = round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids, nullptr, nullptr, nullptr,
                      nullptr);
    L.rounds = rounds;
    L.target = target;
    L.accept_len = accept_len;
    L.out_tokens = out_tokens;
    prism_status st = check_round_args(c, L.r0);
    if (st != PRISM_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaSetDevice(c->device);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaSetDevice");
    if (!c->use_graph) {
        e = enqueue_loop(c, L, s, c->use_pdl);
        return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "kernel launch");
    }
    LoopGraph *hit = nullptr;
    for (auto &g : c->loop_graphs)
        if (g.key == L && g.pdl == c->use_pdl) hit = &g;
    if (!hit) {
        if ((int)c->loop_graphs.size() >= kGraphCache) {
            cudaGraphExecDestroy(c->loop_graphs.front().exec);
            c->loop_graphs.erase(c->loop_graphs.begin());
        }
        cudaGraph_t graph = nullptr;
        e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamBeginCapture");
        cudaError_t le = enqueue_loop(c, L, c->cap_stream, c->use_pdl);
        e = cudaStreamEndCapture(c->cap_stream, &graph);
        if (le != cudaSuccess) {
            if (graph) cudaGraphDestroy(graph);
            return cuda_fail(c, le, "kernel launch during capture");
        }
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamEndCapture");
        cudaGraphExec_t exec = nullptr;
        e = cudaGraphInstantiate(&exec, graph, 0);
        cudaGraphDestroy(graph);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaGraphInstantiate");
        c->loop_graphs.push_back(LoopGraph{L, c->use_pdl, exec});
        hit = &c->loop_graphs.back();
    }
    e = cudaGraphLaunch(hit->exec, s);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "cudaGraphLaunch");
}

prism_status prism_round_launches(prism_ctx *c, int32_t *n_launches) {
    if (!c || !n_launches) return fail(c, PRISM_ERR_INVALID_ARG, "null argument");
    if (c->last_round_kernels < 0) return fail(c, PRISM_ERR_INVALID_ARG, "no round has been replayed from a graph");
    *n_launches = c->last_round_kernels;
    return PRISM_OK;
}

namespace {
prism_status profile_round(prism_ctx *c, const RoundArgs &r, void *stream, float *kernel_ms, int32_t *kernel_kind,
                           int32_t max_kernels, int32_t *n_kernels);
}

prism_status prism_profile_round(prism_ctx *c, int32_t batch, const int32_t *tokens, const void *hidden,
                                 const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                                 int32_t *draft_ids, int32_t *topk_ids, float *topk_logits, void *stream,
                                 float *kernel_ms, int32_t *kernel_kind, int32_t max_kernels,
                                 int32_t *n_kernels) {
    const RoundArgs r = round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids, topk_ids,
                                   topk_logits, nullptr, nullptr);
    return profile_round(c, r, stream, kernel_ms, kernel_kind, max_kernels, n_kernels);
}

prism_status prism_profile_tree(prism_ctx *c, int32_t batch, const int32_t *tokens, const void *hidden,
                                const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                                int32_t width, int32_t n_nodes, const prism_tree_outputs *out, void *stream,
                                float *kernel_ms, int32_t *kernel_kind, int32_t max_kernels, int32_t *n_kernels) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!out || !out->tokens || !out->parents || !out->depths || !out->scores)
        return fail(c, PRISM_ERR_INVALID_ARG, "tree outputs: tokens, parents, depths and scores are required");
    const long K = c->cfg.n_steps;
    const long P = width + (K - 1) * (long)width * width;
    if (width < 1 || width > c->cfg.max_tree_width || width > c->cfg.vocab || (K - 1) * width > kTreeMaskBits ||
        P > kTreeMaxPool || n_nodes < 1 || n_nodes > P)
        return fail(c, PRISM_ERR_INVALID_ARG, "tree width or n_nodes out of range");
    RoundArgs r = round_args(batch, tokens, hidden, n_new, kv_len, k_cache, v_cache, c->tree_draft, nullptr,
                             nullptr, nullptr, nullptr);
    r.tree_w = width;
    r.tree_m = n_nodes;
    r.tree = *out;
    return profile_round(c, r, stream, kernel_ms, kernel_kind, max_kernels, n_kernels);
}

}  // extern "C"

namespace {
prism_status profile_round(prism_ctx *c, const RoundArgs &r, void *stream, float *kernel_ms, int32_t *kernel_kind,
                           int32_t max_kernels, int32_t *n_kernels) {
    prism_status st = check_round_args(c, r);
    if (st != PRISM_OK) return st;
    if (!kernel_ms || !n_kernels || max_kernels < 1) return fail(c, PRISM_ERR_INVALID_ARG, "null output");
    cudaStream_t s = (cudaStream_t)stream;
    cudaSetDevice(c->device);
    cudaEvent_t ev[kMaxProfileKernels + 1];
    for (auto &x : ev) cudaEventCreate(&x);
    int32_t kinds[kMaxProfileKernels];
    int nk = 0;
    cudaError_t e = enqueue_round(c, r, s, false, ev, kinds, &nk);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    const int n = nk < max_kernels ? nk : max_kernels;
    for (int i = 0; i < n && e == cudaSuccess && i < kMaxProfileKernels; ++i) {
        float ms = 0.f;
        cudaEventElapsedTime(&ms, ev[i], ev[i + 1]);
        kernel_ms[i] = ms;
        if (kernel_kind) kernel_kind[i] = kinds[i];
    }
    *n_kernels = n;
    for (auto &x : ev) cudaEventDestroy(x);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "profiled round");
}
}  // namespace

extern "C" {

prism_status prism_accept_greedy(prism_ctx *c, int32_t batch, const int32_t *draft, const int32_t *target,
                                 const int32_t *n_new, int32_t *kv_len, int32_t *accept_len,
                                 int32_t *out_tokens, void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!draft || !target || !n_new || !kv_len || !accept_len || !out_tokens)
        return fail(c, PRISM_ERR_INVALID_ARG, "null tensor argument");
    if (batch < 1) return fail(c, PRISM_ERR_SHAPE, "batch must be >= 1");
    if (batch > c->cfg.max_batch) return fail(c, PRISM_ERR_CAPACITY, "batch exceeds max_batch");
    cudaSetDevice(c->device);
    AcceptArgs a{draft, target, n_new, kv_len, accept_len, out_tokens, batch, c->cfg.n_steps, nullptr, nullptr, 0};
    cudaError_t e = launch_accept(a, (cudaStream_t)stream);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "accept kernel launch");
}

prism_status prism_accept_sampled(prism_ctx *c, int32_t batch, const int32_t *draft, const float *logits,
                                  const float *draft_lse, float temperature, const float *target_probs,
                                  const uint64_t *seed, const int32_t *n_new, int32_t *kv_len, int32_t *accept_len,
                                  int32_t *out_tokens, void *stream) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (!draft || !logits || !draft_lse || !target_probs || !seed || !n_new || !kv_len || !accept_len || !out_tokens)
        return fail(c, PRISM_ERR_INVALID_ARG, "null tensor argument");
    if ((uintptr_t)seed & 7) return fail(c, PRISM_ERR_INVALID_ARG, "seed must be 8-byte aligned");
    if (!(temperature > 0.f) || !std::isfinite(temperature))
        return fail(c, PRISM_ERR_INVALID_ARG, "temperature must be a finite value > 0");
    if (batch < 1) return fail(c, PRISM_ERR_SHAPE, "batch must be >= 1");
    if (batch > c->cfg.max_batch) return fail(c, PRISM_ERR_CAPACITY, "batch exceeds max_batch");
    cudaSetDevice(c->device);
    AcceptSampledArgs a{};
    a.draft = draft;
    a.logits = logits;
    a.lse = draft_lse;
    a.target = target_probs;
    a.seed = seed;
    a.n_new = n_new;
    a.kv_len = kv_len;
    a.accept_len = accept_len;
    a.out_tokens = out_tokens;
    a.err = c->err;
    a.temperature = temperature;
    a.B = batch;
    a.K = c->cfg.n_steps;
    a.V = c->cfg.vocab;
    cudaError_t e = launch_accept_sampled(a, (cudaStream_t)stream);
    return e == cudaSuccess ? PRISM_OK : cuda_fail(c, e, "sampled accept kernel launch");
}

prism_status prism_sync_status(prism_ctx *c, void *stream, int32_t *flags) {
    if (!c) return fail(c, PRISM_ERR_INVALID_ARG, "null context");
    if (flags) *flags = 0;
    cudaSetDevice(c->device);
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "stream synchronize");
    int w = 0;
    e = cudaMemcpy(&w, c->err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "error word read");
    if (w) {
        cudaMemset(c->err, 0, sizeof(int));
        if (flags) *flags = w;
        char buf[160];
        std::snprintf(buf, sizeof(buf), "device error word 0x%x (token range %d, cache range %d, n_new range %d, timeout %d)",
                      w, !!(w & 1), !!(w & 2), !!(w & 4), !!(w & 8));
        // a wait that gave up means the results are not to be trusted at all
        return fail(c, (w & kErrTimeout) ? PRISM_ERR_TIMEOUT : PRISM_ERR_DEVICE_FLAG, buf);
    }
    return PRISM_OK;
}

}  // extern "C"
