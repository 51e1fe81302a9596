// Device helpers and launch interfaces shared by the PRISM draft-round kernels
// (sm_103a).  Internal to the library; the public ABI is include/prism.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace prism {

constexpr int kMaxSteps = 16;
constexpr int kTopK = 8;          // every selection keeps a sorted top-8 list
constexpr int kGemvThreads = 512; // 16 warps per projection CTA
constexpr int kGemvWarps = kGemvThreads / 32;
constexpr int kAttnThreads = 128;

enum DevErr : int {
    kErrToken = 1,
    kErrCache = 2,
    kErrNNew = 4,
    kErrTimeout = 8,
};

// ----------------------------------------------------------------- PTX helpers

// Programmatic dependent launch: let the next kernel in the stream start its
// independent prologue (weight prefetch) while this one runs; and wait until
// every prerequisite grid has completed and its writes are visible.
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// 128-bit streaming load of read-only data: not kept in L1.
__device__ __forceinline__ uint4 ldg_stream(const uint4 *p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

// ----------------------------------------------------------------- bf16

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

// float -> bf16 bits, round to nearest even (finite inputs).
__device__ __forceinline__ uint16_t f32_to_bf16(float f) {
    uint32_t u = __float_as_uint(f);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}
// Two floats as adjacent bf16 values in one word (the first at the lower address).
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    return (uint32_t)f32_to_bf16(lo) | ((uint32_t)f32_to_bf16(hi) << 16);
}
__device__ __forceinline__ float round_bf16(float f) {
    return __uint_as_float((uint32_t)f32_to_bf16(f) << 16);
}

// Element access for the two storage types (uint16_t = bf16 bits, float).
template <typename T> struct Elem;
template <> struct Elem<uint16_t> {
    static constexpr int kPerVec = 8;  // elements per 16-byte vector
    __device__ static float load(const uint16_t *p, int64_t i) { return bf16_to_f32(p[i]); }
    __device__ static void store(uint16_t *p, int64_t i, float v) { p[i] = f32_to_bf16(v); }
    __device__ static float round(float v) { return round_bf16(v); }
};
template <> struct Elem<float> {
    static constexpr int kPerVec = 4;
    __device__ static float load(const float *p, int64_t i) { return p[i]; }
    __device__ static void store(float *p, int64_t i, float v) { p[i] = v; }
    __device__ static float round(float v) { return v; }
};

__device__ __forceinline__ void set_err(int *err, int bit) {
    if (err) atomicOr(err, bit);
}

// Polls a wait between two roles of a kernel (a consumer for a filled stage
// or accumulator, a producer for a released one) makes before it gives up,
// sets the timeout bit and lets the kernel wind down: wait_polls > 0 is that
// count, 0 the built-in bound `dflt`, < 0 none (every such wait gives up at
// once; used to test the error path).  The drain waits (a producer for its
// own copies in flight, the MMA lane for its own MMAs) always use `dflt`,
// so that nothing is in flight when a CTA exits.
// An L2 cache policy under which the lines a load brings in are evicted
// first (for data read once, such as a weight stream).
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// Share `part` of `parts` of the byte range [base, base + bytes), cut at
// 16-byte boundaries, requested into L2 with bulk prefetches of up to 32 KB.
// A prefetch changes no data; base must be 16-byte aligned.
__device__ __forceinline__ void prefetch_l2_share(const void *base, long long bytes, int part, int parts) {
    if (!base || bytes < 16 || parts < 1) return;
    const long long lo = (bytes * part / parts) & ~15LL;
    const long long hi = part + 1 == parts ? (bytes & ~15LL) : (bytes * (part + 1) / parts) & ~15LL;
    for (long long o = lo; o < hi; o += 32768) {
        const uint32_t n = (uint32_t)(hi - o < 32768 ? hi - o : 32768);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"((const char *)base + o), "r"(n) : "memory");
    }
}

// Running log-sum-exp as (max m, sum s of exp(z - m)): add one logit, and
// combine two partial pairs.
__device__ __forceinline__ void lse_add(float &m, float &s, float z) {
    if (z > m) {
        s = s * expf(m - z) + 1.f;
        m = z;
    } else {
        s += expf(z - m);
    }
}
__device__ __forceinline__ void lse_combine(float &m, float &s, float m2, float s2) {
    if (m2 == -INFINITY) return;
    if (m == -INFINITY) { m = m2; s = s2; return; }
    if (m2 > m) { s = s * expf(m - m2) + s2; m = m2; }
    else s += s2 * expf(m2 - m);
}

__device__ __forceinline__ long wait_bound(int wait_polls, long dflt) {
    return wait_polls > 0 ? (long)wait_polls : (wait_polls < 0 ? 0L : dflt);
}

// Checked builds (-DPRISM_CHECKED): record the first failed bounds or
// alignment check (code, block, two values) in the four words after the
// device error word, and skip the access.  Compiled out otherwise.
#ifdef PRISM_CHECKED
__device__ __forceinline__ bool dbg_fail(int *err, int code, long v1, long v2) {
    if (err && atomicCAS(err + 1, 0, code) == 0) {
        err[2] = (int)blockIdx.x;
        err[3] = (int)v1;
        err[4] = (int)v2;
    }
    return true;
}
#define PRISM_CHECK(err, cond, code, v1, v2) (!(cond) && dbg_fail((err), (code), (long)(v1), (long)(v2)))
#else
#define PRISM_CHECK(err, cond, code, v1, v2) false
#endif

// Top-8 ordering: larger logit first, then lower id.
__device__ __forceinline__ bool better(float a, int ia, float b, int ib) {
    return a > b || (a == b && ia < ib);
}

// Insert (v, id) into a descending top-8 list held in registers.
__device__ __forceinline__ void top8_insert(float (&vals)[kTopK], int (&ids)[kTopK], float v, int id) {
    if (!better(v, id, vals[kTopK - 1], ids[kTopK - 1])) return;
    vals[kTopK - 1] = v;
    ids[kTopK - 1] = id;
#pragma unroll
    for (int i = kTopK - 1; i > 0; --i) {
        if (better(vals[i], ids[i], vals[i - 1], ids[i - 1])) {
            float tv = vals[i]; vals[i] = vals[i - 1]; vals[i - 1] = tv;
            int ti = ids[i]; ids[i] = ids[i - 1]; ids[i - 1] = ti;
        }
    }
}

__device__ __forceinline__ void top8_init(float (&vals)[kTopK], int (&ids)[kTopK]) {
#pragma unroll
    for (int i = 0; i < kTopK; ++i) { vals[i] = -INFINITY; ids[i] = 0x7FFFFFFF; }
}

// Top-1 as one 64-bit key: an order-preserving image of the fp32 logit in
// the high word and the inverted id in the low word, so that the numeric
// maximum is the best candidate under `better` (larger logit, then lower id).
__device__ __forceinline__ unsigned long long pack_best(float v, int id) {
    const uint32_t b = __float_as_uint(v);
    const uint32_t k = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return ((unsigned long long)k << 32) | (uint32_t)(0xFFFFFFFFu - (uint32_t)id);
}
__device__ __forceinline__ void unpack_best(unsigned long long key, float &v, int &id) {
    const uint32_t k = (uint32_t)(key >> 32);
    v = __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
    id = (int)(0xFFFFFFFFu - (uint32_t)key);
}

using Key = unsigned long long;

__device__ __forceinline__ void key_clear(Key (&l)[kTopK]) {
#pragma unroll
    for (int i = 0; i < kTopK; ++i) l[i] = 0ull;
}

// Insert k into the sorted list l (static indices: l stays in registers).
__device__ __forceinline__ void key_insert(Key (&l)[kTopK], Key k) {
    if (k <= l[kTopK - 1]) return;
    l[kTopK - 1] = k;
#pragma unroll
    for (int s = kTopK - 1; s > 0; --s) {
        const Key x = l[s - 1], y = l[s];
        l[s - 1] = x > y ? x : y;
        l[s] = x > y ? y : x;
    }
}

// Lanes lane and lane ^ m both end with the best kTopK keys of their two
// lists: the element-wise maximum of one list and the other reversed is that
// set as a bitonic sequence, sorted by three half-cleaner stages.  Every lane
// of the warp takes part.
__device__ __forceinline__ void key_merge_xor(Key (&l)[kTopK], int m) {
    Key c[kTopK];
#pragma unroll
    for (int i = 0; i < kTopK; ++i) {
        const Key o = __shfl_xor_sync(0xFFFFFFFFu, l[kTopK - 1 - i], m);
        c[i] = l[i] > o ? l[i] : o;
    }
#pragma unroll
    for (int d = kTopK / 2; d > 0; d >>= 1)
#pragma unroll
        for (int i = 0; i < kTopK; ++i)
            if ((i & d) == 0) {
                const Key x = c[i], y = c[i + d];
                c[i] = x > y ? x : y;
                c[i + d] = x > y ? y : x;
            }
#pragma unroll
    for (int i = 0; i < kTopK; ++i) l[i] = c[i];
}

// Entry r of a register list without a dynamic index.
__device__ __forceinline__ Key key_at(const Key (&l)[kTopK], int r) {
    Key k = l[0];
#pragma unroll
    for (int i = 1; i < kTopK; ++i)
        if (r == i) k = l[i];
    return k;
}

// ----------------------------------------------------------------- launches

// Projection kinds (weight-streaming GEMV family).
enum ProKind : int {
    kProFusePrefill = 0,  // X[t] = [E(tokens[b,i]); hidden[b,i]]
    kProFuseDecode = 1,   // X[b] = [E(draft[b,k-2]); round(h^[b])]
    kProNorm = 2,         // X[t] = round(RMSNorm(src[t]) * g) (or round(src[t]) without norm)
    kProCopy = 3,         // X[t] = act[t] (already rounded, wtype)
};
enum EpiKind : int {
    kEpiStore = 0,   // out[t, r] = acc
    kEpiResid = 1,   // out[t, r] = resid[row(t), r] + acc
    kEpiSwiGLU = 2,  // out_act[t, j] = round(silu(acc_gate) * acc_up)
    kEpiTopK = 3,    // logits (optional) + top-8 selection
};

struct GemvArgs {
    const void *W;        // [rows, kin] wtype
    int n_units;          // output units (rows; gate/up pairs for SwiGLU)
    int kin;              // contraction length
    int pair_offset;      // row offset of the second row of a unit (SwiGLU: F)
    int T;                // activation rows
    int pro, epi;
    // prologue sources
    const void *embed;       // [V, d]
    const int32_t *tokens;   // [B, max_new]
    const void *hidden_in;   // [B, max_new, d] wtype
    const int32_t *draft;    // [B, K]
    const float *src;        // fp32 rows [*, d] (norm source, or h^ for decode fusion)
    int src_prefill_rows;    // norm source rows are the last prefill row of each sequence
    const void *act;         // [T, kin] wtype (copy source)
    const void *gain;        // [d] wtype, or null (no norm)
    float eps;
    const int32_t *n_new;
    int max_new, K, step, vocab, d;
    // epilogue
    float *out;              // fp32 [T, out_ld]
    int out_ld;
    void *out_act;           // wtype [T, out_ld] (SwiGLU)
    const float *resid;      // fp32 residual rows
    int resid_prefill_rows;  // residual row = b*max_new + n_new[b]-1
    float *hidden_out;       // [B, K, d] or null (down projection)
    float *logits;           // [B, K, V] or null (LM head)
    float *lm_part;          // [T, grid, 8] values (LM head)
    int *lm_part_id;         // [T, grid, 8] ids
    int *counter;            // LM head last-CTA counter
    unsigned long long *best;  // [T] packed (value, id) of the best logit so far, for top-1 (zero: none)
    int32_t *draft_out;      // [B, K]
    int32_t *topk_ids;       // [B, K, topk] or null
    float *topk_logits;      // [B, K, topk] or null
    int topk;
    int *err;
    // ring plan knobs: target stage bytes, smem budget bytes, consumer groups;
    // force_cuda_core selects the CUDA-core kernel for bf16 too
    int chunk_target, smem_budget, groups, force_cuda_core;
    // streamed projections: the next projection's bf16 activation rows
    // [T][kin of the next projection], written by this projection's last
    // kernel so that the next one needs no row preparation.  next_norm: the
    // split-K finish writes RMSNorm(out row) * next_gain (next_gain null: the
    // row as it is), rounded.  next_fuse: the LM head's top-k merge writes the
    // next decode step's fusion row [E(chosen token); round(src row)].
    uint16_t *next_x;
    const void *next_gain;
    int next_norm, next_fuse;
    int wait_polls;          // see wait_bound
    // 1: weight boxes are loaded with an L2 evict-first policy (each weight
    // byte is read once per step; other data then stays in L2)
    int w_evict_first;
    // LM head with top-k lists: per row and CTA, (max, sum of exp(z - max))
    // of the logits the CTA produced, [T][gridDim.x][2]; null: not computed
    float *lse_part;
    // the next kernel's weights: once a CTA has requested its last weight
    // box it requests its share of these bytes into L2; null / 0: none
    const void *pf_next;
    long long pf_next_bytes;
    // 1: a selection (LM head) launch takes the fewest CTAs that keep its
    // number of tile waves, so that every CTA streams as many tiles
    int even_waves;
    // 1: top-k lists are only published per CTA ([T][grid][8] in lm_part /
    // lm_part_id); the kernel that reads the selection merges them
    int defer_merge;
    // 1: a streamed top-1 selection of up to 16 rows joins through the packed
    // atomic maximum in the kernel itself (no list merge kernel)
    int stream_top1;
};

struct RopeArgs {
    const float *qkv;       // [rows, (Hq + 2Hkv) D]
    void *k_cache, *v_cache;
    float *q_out;           // [B, Hq, D]
    const float *rope_cos, *rope_sin;  // [max_ctx, D/2]
    const int32_t *n_new, *kv_len;
    int B, max_new, rows, prefill, step, K;
    int Hq, Hkv, D, max_ctx;
    int *err;
};

struct AttnArgs {
    const float *q;          // [B, Hq, D] (rotated)
    const void *k_cache, *v_cache;
    float *part;             // [B, Hq, splits, D + 4]
    int *counter;            // [B * Hkv]
    void *o_out;             // [B, Hq * D] wtype (rounded operand of the O projection)
    const int32_t *n_new, *kv_len;
    int B, max_new, prefill, step, Hq, Hkv, D, max_ctx, chunk, splits;
    int *err;
};

// Fused RoPE + KV append + attention (one cluster of `cs` CTAs per sequence
// and KV head).
struct FusedAttnArgs {
    const float *qkv;                  // [rows, (Hq + 2Hkv) D]
    void *k_cache, *v_cache;           // [B, Hkv, max_ctx, D]
    void *o_out;                       // [B, Hq * D] wtype
    const float *rope_cos, *rope_sin;  // [max_ctx, D/2]
    const int32_t *n_new, *kv_len;
    int B, max_new, prefill, step, Hq, Hkv, D, max_ctx, cs;
    int *err;
    int wait_polls;                    // see wait_bound
    int warps;                         // tensor-core kernel: compute warps per CTA, 8 (0) or 4 (two CTAs per SM)
    int lpt;                           // 1: longest sequences first (B <= 256)
    // the next kernel's weights, requested into L2 as in GemvArgs
    const void *pf_next;
    long long pf_next_bytes;
};

struct AcceptArgs {
    const int32_t *draft, *target, *n_new;
    int32_t *kv_len, *accept_len, *out_tokens;
    int B, K;
    // multi-round loop (optional): the next round's accepted tokens
    // [B, max_new] and their count (a + 1); next_n may alias n_new
    int32_t *next_tokens, *next_n;
    int max_new;
};

// Sampled drafting (Sec. 2 at a temperature T > 0): the draw of step `step`
// from the logits that step's LM head wrote.
constexpr int kSampleMaxBlocks = 128;   // CTAs per row of logits
struct SampleArgs {
    const float *logits;       // [B, K, V] fp32
    const uint64_t *seed;      // device word: the round's random-stream seed
    int32_t *draft;            // [B, K]: the drawn token replaces the argmax
    float *lse;                // [B, K]: log sum exp(z / T)
    float *part;               // [B, kSampleMaxBlocks, 4] per-CTA partials
    int *counter;              // [B] last-CTA tickets (left at zero)
    float temperature;
    int V, K, step, chunk, max_blocks;
};
// Speculative-sampling acceptance of B sequences with K drafted tokens each.
struct AcceptSampledArgs {
    const int32_t *draft;      // [B, K]
    const float *logits;       // [B, K, V] draft logits
    const float *lse;          // [B, K]
    const float *target;       // [B, K + 1, V] target probabilities
    const uint64_t *seed;
    const int32_t *n_new;
    int32_t *kv_len, *accept_len, *out_tokens;
    int *err;
    float temperature;
    int B, K, V;
};
int sample_blocks(int V, int *chunk);

// Tree drafting (tree.cu): the frontier of each sequence is w rows b * w + j.
constexpr int kTreeMaxWidth = 8;      // branches per node (the top-k lists hold 8)
constexpr int kTreeMaxPool = 1024;    // candidates per sequence and round
constexpr int kTreeMaskBits = 64;     // draft slots a row's ancestor mask can name
struct TreeArgs {
    int B, w, K, step, R;             // R: rows per sequence this step (1 at step 1, else w)
    int d, V, Hq, Hkv, D, max_ctx, max_new, n_nodes, P;
    const int32_t *n_new, *kv_len;
    int *err;
    // fusion input rows
    const void *embed;                // [V, d] wtype
    const float *hhat;                // h^ rows [*, d]
    void *u_out;                      // [B*w, 2d] wtype
    // frontier (rows b*w + j): token, h^ row that emitted it, pool index,
    // score, ancestor slot mask of the row that will process it
    int32_t *front_tok, *front_row, *front_pool;
    float *front_score;
    unsigned long long *front_mask;
    // candidate pool [B, P]
    int32_t *pool_tok, *pool_par;
    float *pool_score;
    // this step's LM-head outputs (rows b*w + j)
    const float *logits;              // [B*w, V]
    int32_t *top_ids;                 // [B*w, w] (written by the lse kernel when the LM head defers its merge)
    float *top_vals;                  // [B*w, w]
    float *lse;                       // [B*w]
    float *lse_part;                  // [B*w, kSampleMaxBlocks, 2]
    int *lse_ctr;                     // [B*w] (left at zero)
    int *seq_ctr;                     // [B] rows of each sequence with their lse (left at zero)
    int lse_chunk, lse_blocks;
    // > 0: the LM head wrote per-CTA (max, sum exp) partials of every row,
    // lm_lse_grid of them, into lse_part ([LM-head row][lm_lse_grid][2])
    int lm_lse_grid;
    // non-null: the LM head left its per-CTA top-8 lists unmerged
    // ([LM-head row][lm_lse_grid][8] values and ids); the lse kernel merges them
    const float *lm_val;
    const int *lm_id;
    // RoPE / append / attention (one kernel)
    const float *qkv;                 // [B*w, (Hq + 2Hkv) D]
    void *k_cache, *v_cache;          // [B, Hkv, max_ctx, D]
    const float *rope_cos, *rope_sin;
    float *attn_part;                 // [B*w, Hq, splits, D + 4]
    int *attn_ctr;                    // [B, Hkv] (left at zero)
    void *o_out;                      // [B*w, Hq*D] wtype
    int chunk, splits;
    // the O projection's weights, requested into L2 as in GemvArgs
    const void *pf_next;
    long long pf_next_bytes;
    // caller outputs: the verified tree [B, n_nodes]; optional pool [B, P] and frontier [B, K, w]
    int32_t *tree_tokens, *tree_parents, *tree_depths;
    float *tree_scores;
    int32_t *out_pool_tokens, *out_pool_parents, *out_frontier;
    float *out_pool_scores;
};
struct AcceptTreeArgs {
    const int32_t *tree_tokens, *tree_parents, *target_next, *n_new;  // [B, m], [B, m], [B, m+1], [B]
    int32_t *kv_len, *accept_len, *accept_nodes, *out_tokens;         // [B], [B], [B, K], [B, K+1]
    int B, n_nodes, K;
};
size_t tree_attention_smem_bytes(bool bf16, int D, int chunk, int G, int w, int splits);
cudaError_t prepare_tree_kernels(bool bf16, int D, int chunk, int G, int w, int splits, int max_ctx);
cudaError_t launch_tree_gather(const TreeArgs &a, bool bf16, cudaStream_t s, bool pdl);
cudaError_t launch_tree_attention(const TreeArgs &a, bool bf16, cudaStream_t s, bool pdl);
cudaError_t launch_tree_lse(const TreeArgs &a, cudaStream_t s, bool pdl);
cudaError_t launch_accept_tree(const AcceptTreeArgs &a, cudaStream_t s);

// Host launchers (return cudaGetLastError of the launch).
cudaError_t launch_gemv(const GemvArgs &a, bool bf16, int grid, cudaStream_t s, bool pdl);
size_t gemv_smem_bytes(const GemvArgs &a, bool bf16, int tc);
int gemv_rows_per_pass(const GemvArgs &a, bool bf16);
cudaError_t launch_rope_append(const RopeArgs &a, bool bf16, cudaStream_t s, bool pdl);
cudaError_t launch_attention(const AttnArgs &a, bool bf16, cudaStream_t s, bool pdl);
cudaError_t launch_accept(const AcceptArgs &a, cudaStream_t s);
cudaError_t launch_sample(const SampleArgs &a, int B, cudaStream_t s, bool pdl);
cudaError_t launch_accept_sampled(const AcceptSampledArgs &a, cudaStream_t s);
// One-time kernel attribute setup (maximum dynamic shared memory); must run
// before any stream capture.
cudaError_t prepare_gemv_kernels();
// Message returned by prism_get_error(NULL) (host, thread-local).
void set_global_error(const char *msg);
bool gemv_supported(const GemvArgs &a, bool bf16);
bool gemv_mma_supported(const GemvArgs &a);
cudaError_t prepare_gemv_mma_kernels();
cudaError_t launch_gemv_mma(const GemvArgs &a, int grid, cudaStream_t s, bool pdl);
// Tensor-core projections (gemv_tc.cu): tensor-map encoder and kernel
// attributes (before any capture); a weight matrix [rows, kin] bf16 as a TMA
// tensor map of 128 x 64 boxes; plan check, split-K workspace need, launch.
cudaError_t prepare_gemv_tc_kernels();
cudaError_t make_weight_map(CUtensorMap *m, const void *W, int rows, int kin);
bool gemv_tc_supported(const GemvArgs &a, int sms);
size_t gemv_tc_workspace_floats(const GemvArgs &a, int sms);
int gemv_tc_tiles(const GemvArgs &a);
cudaError_t launch_gemv_tc(const GemvArgs &a, const CUtensorMap &m, int sms, float *part, int *tile_ctr,
                           cudaStream_t s, bool pdl);
// Streamed variant for many activation rows (up to 256; 128 for SwiGLU, 64
// for top-k): prep kernel for the activation rows (into xbuf, bf16
// [T][kin], unless the prologue is a copy), the projection, and for top-k
// the cross-CTA merge kernel.
bool gemv_tcs_supported(const GemvArgs &a, int sms);
size_t gemv_tcs_workspace_floats(const GemvArgs &a, int sms);
// *next_done (may be null) reports whether the launch also wrote the next
// projection's rows (a.next_norm or a.next_fuse) into a.next_x.
cudaError_t launch_gemv_tcs(const GemvArgs &a, const CUtensorMap &mw, int sms, float *part, int *tile_ctr,
                            uint16_t *xbuf, cudaStream_t s, bool pdl, bool *next_done = nullptr);
cudaError_t prepare_attention_kernel(bool bf16, int D, int chunk, int G, int splits);
// Sets kernel attributes; *max_cs receives the largest cluster size (8 or 16)
// for which `need` clusters can be resident at once.
cudaError_t prepare_fused_attention(bool bf16, int D, int G, int need, int *max_cs);
size_t fused_attention_smem_bytes(bool bf16, int D, int G);
// K or V cache [heads, max_ctx, D] bf16 as a TMA tensor map of
// rows_per_box x 64-column boxes in the 128-byte swizzle (D a multiple of 64).
cudaError_t make_cache_map(CUtensorMap *m, const void *cache, int heads, int max_ctx, int D, int rows_per_box);
// Keys per chunk of the tensor-core attention kernel (the box height it needs).
int fused_attention_chunk();
// tk / tv: cache tensor maps; the bf16 tensor-core kernel runs when both are
// given, the CUDA-core kernel otherwise.
cudaError_t launch_fused_attention(const FusedAttnArgs &a, bool bf16, cudaStream_t s, bool pdl,
                                   const CUtensorMap *tk, const CUtensorMap *tv);
size_t attention_smem_bytes(bool bf16, int D, int chunk, int G, int splits);

// Launch with optional programmatic stream serialization.
template <typename Kern, typename... Args>
cudaError_t launch_k(Kern k, dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k, args...);
}

}  // namespace prism
