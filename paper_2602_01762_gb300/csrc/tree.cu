// Tree drafting for the PRISM draft round (sm_103a).
//
// PRISM's step-wise modules work unchanged with tree-shaped drafts (Sec. 3.2,
// after the recurrence); the paper evaluates a 6-step, 4-branch tree that
// verifies at most 16 tokens (Sec. 4).  The tree is read as the dynamic top-w
// expansion: step 1 (the chain's prefill) yields the w best tokens as depth-1
// candidates; at step k >= 2 every frontier node is processed by step k's
// module as its own activation row, so the projections and the LM head run on
// T = B * w rows through the chain's kernels.  A candidate's score is the sum
// of draft log-probabilities along its path; the next frontier is the w best
// new candidates, and after step K the verified tree is the n best candidates
// of the round.  The kernels this file adds:
//   tree_gather_kernel     fusion input row [E(token); round(h^ of the row
//                          that emitted the token)];
//   tree_attention_tc_kernel / tree_attention_kernel
//                          rotary embedding at the node's depth, K/V appended
//                          at the node's own cache slot L + n + (k - 2) w + j,
//                          and split-KV attention over the committed rows
//                          [0, L+n) plus the draft slots in the row's 64-bit
//                          ancestor mask, all w rows of a sequence against one
//                          staged chunk of keys, last-CTA merge in split order
//                          (tensor cores for bf16 caches with w * G <= 16
//                          row-head pairs, CUDA cores otherwise);
//   tree_lse_kernel        log-sum-exp of every row's logits; the last row of
//                          each sequence to finish then scores the candidates,
//                          picks the next frontier and, after the last step,
//                          the verified tree;
//   accept_tree_kernel     greedy acceptance along the tree (Sec. 2's
//                          temperature-0 rule applied from the root).
#include "common.cuh"

namespace prism {

namespace {

__device__ __forceinline__ int tree_n(const TreeArgs &a, int b) {
    int n = a.n_new[b];
    if (n < 1 || n > a.max_new) {
        set_err(a.err, kErrNNew);
        n = n < 1 ? 1 : a.max_new;
    }
    return n;
}

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

// (max, sum of exp(v - max)) of two parts, combined.
__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2) {
    if (m2 == -INFINITY) return;
    if (m == -INFINITY) { m = m2; s = s2; return; }
    if (m2 > m) { s = s * expf(m - m2) + s2; m = m2; }
    else s += s2 * expf(m2 - m);
}

// ------------------------------------------------------------------ gather

constexpr int kGatherThreads = 128;

// Grid (rows, ceil(d / (VEC * 128))): thread i of CTA (t, c) moves VEC
// consecutive elements (16 bytes of the embedding row) of both halves of
// row t, issuing its loads before its stores.
template <typename WT>
__global__ void __launch_bounds__(kGatherThreads) tree_gather_kernel(const TreeArgs a) {
    constexpr int VEC = Elem<WT>::kPerVec;
    pdl_trigger();
    pdl_wait();
    const int t = blockIdx.x;              // row b * w + j
    const int i0 = (blockIdx.y * kGatherThreads + threadIdx.x) * VEC;
    if (i0 >= a.d) return;
    int tok = a.front_tok[t];
    if (tok < 0 || tok >= a.V) {
        set_err(a.err, kErrToken);
        tok = tok < 0 ? 0 : a.V - 1;
    }
    const uint4 ev = *(const uint4 *)((const WT *)a.embed + (size_t)tok * a.d + i0);
    const float *h = a.hhat + (size_t)a.front_row[t] * a.d + i0;
    float hv[VEC];
#pragma unroll
    for (int q = 0; q < VEC; q += 4) {
        const float4 f = *(const float4 *)(h + q);
        hv[q] = f.x; hv[q + 1] = f.y; hv[q + 2] = f.z; hv[q + 3] = f.w;
    }
    WT *u = (WT *)a.u_out + (size_t)t * 2 * a.d;
    *(uint4 *)(u + i0) = ev;
    alignas(16) WT r[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) Elem<WT>::store(r, q, hv[q]);   // the fusion input's operand rounding
    *(uint4 *)(u + a.d + i0) = *(const uint4 *)r;
}

// ------------------------------------------------------------------ attention

// q . k for one key row in shared memory (16-byte vector reads of both).
template <typename WT, int D>
__device__ __forceinline__ float dot_row(const float *q, const WT *k) {
    float acc = 0.f;
    if constexpr (sizeof(WT) == 2) {
#pragma unroll 4
        for (int c = 0; c < D; c += 8) {
            const uint4 kv = *(const uint4 *)(k + c);
            const float4 q0 = *(const float4 *)(q + c), q1 = *(const float4 *)(q + c + 4);
            acc = fmaf(q0.x, bf16lo(kv.x), acc);
            acc = fmaf(q0.y, bf16hi(kv.x), acc);
            acc = fmaf(q0.z, bf16lo(kv.y), acc);
            acc = fmaf(q0.w, bf16hi(kv.y), acc);
            acc = fmaf(q1.x, bf16lo(kv.z), acc);
            acc = fmaf(q1.y, bf16hi(kv.z), acc);
            acc = fmaf(q1.z, bf16lo(kv.w), acc);
            acc = fmaf(q1.w, bf16hi(kv.w), acc);
        }
    } else {
#pragma unroll 4
        for (int c = 0; c < D; c += 4) {
            const float4 kv = *(const float4 *)(k + c), q0 = *(const float4 *)(q + c);
            acc = fmaf(q0.x, kv.x, acc);
            acc = fmaf(q0.y, kv.y, acc);
            acc = fmaf(q0.z, kv.z, acc);
            acc = fmaf(q0.w, kv.w, acc);
        }
    }
    return acc;
}

// The DPL consecutive values a lane owns in one V row.
template <typename WT, int DPL>
__device__ __forceinline__ void load_run(const WT *p, float (&out)[DPL]) {
    if constexpr (sizeof(WT) == 2 && DPL == 4) {
        const uint2 v = *(const uint2 *)p;
        out[0] = bf16lo(v.x); out[1] = bf16hi(v.x); out[2] = bf16lo(v.y); out[3] = bf16hi(v.y);
    } else if constexpr (sizeof(WT) == 2 && DPL == 2) {
        const uint32_t v = *(const uint32_t *)p;
        out[0] = bf16lo(v); out[1] = bf16hi(v);
    } else {
#pragma unroll
        for (int u = 0; u < DPL; ++u) out[u] = Elem<WT>::load(p, u);
    }
}

// Stage keys [j0, j0 + nk) of KV head g of sequence b and the queries of its
// G heads in all w rows.  Rows written before this step come from the cache
// (cp.async); this step's rows (slots new0 + j) are rotated at the node's
// depth and written to the cache and the stage; queries are rotated,
// multiplied by q_scale and stored QS floats apart.  Callers wait for the
// copies and synchronise.
// Rows [j0, j0 + done) were requested earlier (tree_stage_committed).
template <typename WT, int D, int RS, int QS>
__device__ __forceinline__ void tree_stage(const TreeArgs &a, int b, int g, int j0, int nk, int base, WT *Ks,
                                           WT *Vs, float *qs, float q_scale, int done) {
    constexpr int VEC = Elem<WT>::kPerVec;
    const int G = a.Hq / a.Hkv, NQ = a.w * G;
    const int new0 = base + (a.step - 2) * a.w;
    const int pos = base + a.step - 2;
    const int H = a.Hq + 2 * a.Hkv, half = D / 2;
    const int nold = new0 - j0 < 0 ? 0 : (new0 - j0 < nk ? new0 - j0 : nk);
    WT *kc = (WT *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D;
    WT *vc = (WT *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D;
    constexpr int VPR = D / VEC;
    for (int e = threadIdx.x + done * VPR; e < nold * VPR; e += blockDim.x) {
        const int r = e / VPR, c = e % VPR;
        cp_async16(Ks + (size_t)r * RS + c * VEC, (const uint4 *)kc + e);
        cp_async16(Vs + (size_t)r * RS + c * VEC, (const uint4 *)vc + e);
    }
    const int pc = pos < a.max_ctx ? pos : 0;
    const float *cs_row = a.rope_cos + (size_t)pc * half, *sn_row = a.rope_sin + (size_t)pc * half;
    for (int e = threadIdx.x; e < NQ * half; e += blockDim.x) {
        const int pr = e / half, c = e % half, j = pr / G, hl = pr % G;
        const float *x = a.qkv + ((size_t)b * a.w + j) * H * D + (size_t)(g * G + hl) * D;
        const float cs = cs_row[c], sn = sn_row[c], x0 = x[c], x1 = x[c + half];
        qs[(size_t)pr * QS + c] = (x0 * cs - x1 * sn) * q_scale;
        qs[(size_t)pr * QS + c + half] = (x1 * cs + x0 * sn) * q_scale;
    }
    // this step's rows in the chunk (each slot lies in exactly one chunk)
    for (int e = threadIdx.x; e < (nk - nold) * half; e += blockDim.x) {
        const int r = nold + e / half, c = e % half, j = j0 + r - new0;
        const float *x = a.qkv + ((size_t)b * a.w + j) * H * D + (size_t)(a.Hq + g) * D;
        const float cs = cs_row[c], sn = sn_row[c], x0 = x[c], x1 = x[c + half];
        const float k0 = x0 * cs - x1 * sn, k1 = x1 * cs + x0 * sn;
        Elem<WT>::store(kc + (size_t)r * D, c, k0);
        Elem<WT>::store(kc + (size_t)r * D, c + half, k1);
        Elem<WT>::store(Ks + (size_t)r * RS, c, k0);
        Elem<WT>::store(Ks + (size_t)r * RS, c + half, k1);
    }
    for (int e = threadIdx.x; e < (nk - nold) * D; e += blockDim.x) {
        const int r = nold + e / D, c = e % D, j = j0 + r - new0;
        const float v = a.qkv[((size_t)b * a.w + j) * H * D + (size_t)(a.Hq + a.Hkv + g) * D + c];
        Elem<WT>::store(vc + (size_t)r * D, c, v);
        Elem<WT>::store(Vs + (size_t)r * RS, c, v);
    }
}

// The chunk's rows that were committed before the round (below kv_len): they
// do not depend on any kernel of this round, so they are requested before
// the dependency wait.  Returns how many rows that is.
template <typename WT, int D, int RS>
__device__ __forceinline__ int tree_stage_committed(const TreeArgs &a, int b, int g, int j0, int nk, int L, WT *Ks,
                                                    WT *Vs) {
    constexpr int VEC = Elem<WT>::kPerVec;
    constexpr int VPR = D / VEC;
    const int ncom = L - j0 < 0 ? 0 : (L - j0 < nk ? L - j0 : nk);
    const WT *kc = (const WT *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D;
    const WT *vc = (const WT *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D;
    for (int e = threadIdx.x; e < ncom * VPR; e += blockDim.x) {
        const int r = e / VPR, c = e % VPR;
        cp_async16(Ks + (size_t)r * RS + c * VEC, (const uint4 *)kc + e);
        cp_async16(Vs + (size_t)r * RS + c * VEC, (const uint4 *)vc + e);
    }
    return ncom;
}

// The last CTA of (b, g) to finish merges every pair's split partials in
// split order (log-sum-exp rule, eight splits' loads in flight at a time) and
// writes the rounded attention output.  ws: [NQ][splits] shared floats.
template <typename WT, int D>
__device__ __forceinline__ void tree_merge_splits(const TreeArgs &a, int b, int g, float *ws, int *s_last) {
    constexpr int DPL = D / 32;
    constexpr int PS = D + 4;
    const int G = a.Hq / a.Hkv, NQ = a.w * G;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
    __threadfence();
    __syncthreads();
    int *ctr = a.attn_ctr + (size_t)b * a.Hkv + g;
    if (threadIdx.x == 0) *s_last = (atomicAdd(ctr, 1) == a.splits - 1);
    __syncthreads();
    if (!*s_last) return;
    __threadfence();
    for (int pr = warp; pr < NQ; pr += nwarp) {
        const int j = pr / G, hl = pr % G, t = b * a.w + j, h = g * G + hl;
        const float *part = a.attn_part + ((size_t)t * a.Hq + h) * a.splits * PS;
        float *wh = ws + (size_t)pr * a.splits;
        constexpr int kMaxPerLane = 8;           // splits <= 256
        float mv[kMaxPerLane], lv[kMaxPerLane];
#pragma unroll
        for (int k = 0; k < kMaxPerLane; ++k) {
            const int sp = lane + 32 * k;
            const bool in = sp < a.splits;
            mv[k] = in ? __ldcg(part + (size_t)sp * PS + D) : -INFINITY;
            lv[k] = in ? __ldcg(part + (size_t)sp * PS + D + 1) : 0.f;
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxPerLane; ++k) M = fmaxf(M, mv[k]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
        float den = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxPerLane; ++k) {
            const int sp = lane + 32 * k;
            const float wgt = lv[k] > 0.f ? expf(mv[k] - M) : 0.f;
            if (sp < a.splits) wh[sp] = wgt;
            den = fmaf(wgt, lv[k], den);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) den += __shfl_xor_sync(0xFFFFFFFFu, den, o);
        __syncwarp();
        float acc[DPL];
#pragma unroll
        for (int u = 0; u < DPL; ++u) acc[u] = 0.f;
        // a split with no visible key has weight 0 and zero sums
        constexpr int kBatch = 8;
        for (int sp0 = 0; sp0 < a.splits; sp0 += kBatch) {
            float v[kBatch][DPL], wv[kBatch];
#pragma unroll
            for (int i = 0; i < kBatch; ++i) {
                const int sp = sp0 + i;
                const bool in = sp < a.splits;
                wv[i] = in ? wh[sp] : 0.f;
                const float *src = part + (size_t)(in ? sp : 0) * PS + lane * DPL;
#pragma unroll
                for (int u = 0; u < DPL; ++u) v[i][u] = in ? __ldcg(src + u) : 0.f;
            }
#pragma unroll
            for (int i = 0; i < kBatch; ++i)
#pragma unroll
                for (int u = 0; u < DPL; ++u) acc[u] = fmaf(wv[i], v[i][u], acc[u]);
        }
        WT *o = (WT *)a.o_out + ((size_t)t * a.Hq + h) * D;
        const float inv = den > 0.f ? 1.0f / den : 0.f;
#pragma unroll
        for (int u = 0; u < DPL; ++u) Elem<WT>::store(o, lane * DPL + u, acc[u] * inv);
    }
    if (threadIdx.x == 0) *ctr = 0;
}

// Key slot p of sequence b is visible to a row with ancestor mask msk when it
// is committed or a step-1 row (p < base) or its draft-slot bit is set.
__device__ __forceinline__ bool tree_visible(int p, int base, unsigned long long msk) {
    const int off = p - base;
    return off < 0 || (off < kTreeMaskBits && ((msk >> off) & 1ull));
}

constexpr int kTreeAttnThreads = 512;   // 16 warps: one (row, query head) pair each when w * G = 16

// CUDA-core kernel (fp32 caches, or more than 16 row-head pairs).  Grid
// (splits, Hkv, B); CTA (s, g, b) stages keys [s C, s C + C) of KV head g once
// and each warp scores them against one (row, query head) pair at a time.
template <typename WT, int D>
__global__ void __launch_bounds__(kTreeAttnThreads) tree_attention_kernel(const TreeArgs a) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ int s_last;
    constexpr int VEC = Elem<WT>::kPerVec;
    constexpr int RS = D + VEC;              // padded row stride (elements)
    constexpr int DPL = D / 32;
    constexpr int PS = D + 4;                // partial record: D sums, max, sum, 2 pad
    const int C = a.chunk, G = a.Hq / a.Hkv, NQ = a.w * G;
    WT *Ks = (WT *)smem_raw;
    WT *Vs = Ks + (size_t)C * RS;
    float *qs = (float *)(Vs + (size_t)C * RS);  // [NQ][D], pair (j, hl) at j * G + hl
    float *ps = qs + (size_t)NQ * D;             // [NQ][C]
    float *ws = ps + (size_t)NQ * C;             // [NQ][splits]
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;

    pdl_trigger();

    const int n = tree_n(a, b), L = a.kv_len[b];
    const int base = L + n;
    int PE = base + (a.step - 1) * a.w;          // keys [0, PE)
    if (PE > a.max_ctx) PE = a.max_ctx;
    const int j0 = s * C;
    const int nk = PE - j0 < C ? PE - j0 : C;
    const float scale = 1.0f / sqrtf((float)D);
    const int ncom = nk > 0 && L >= 0 ? tree_stage_committed<WT, D, RS>(a, b, g, j0, nk, L, Ks, Vs) : 0;
    pdl_wait();
    if (s == 0 && g == 0 && threadIdx.x == 0 && (L < 0 || base + (a.step - 1) * a.w > a.max_ctx))
        set_err(a.err, kErrCache);

    if (nk > 0 && L >= 0) {
        tree_stage<WT, D, RS, D>(a, b, g, j0, nk, base, Ks, Vs, qs, 1.0f, ncom);
        cp_async_wait_all();
        __syncthreads();
        for (int pr = warp; pr < NQ; pr += nwarp) {
            const int j = pr / G, hl = pr % G, t = b * a.w + j;
            const unsigned long long msk = a.front_mask[t];
            const float *q = qs + (size_t)pr * D;
            float *pp = ps + (size_t)pr * C;
            float mloc = -INFINITY;
            for (int jj = lane; jj < nk; jj += 32) {
                float sc = -INFINITY;
                if (tree_visible(j0 + jj, base, msk)) sc = dot_row<WT, D>(q, Ks + (size_t)jj * RS) * scale;
                pp[jj] = sc;
                mloc = fmaxf(mloc, sc);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xFFFFFFFFu, mloc, o));
            float lsum = 0.f;
            for (int jj = lane; jj < nk; jj += 32) {
                const float p = mloc == -INFINITY ? 0.f : expf(pp[jj] - mloc);
                pp[jj] = p;
                lsum += p;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xFFFFFFFFu, lsum, o);
            __syncwarp();
            float acc[DPL];
#pragma unroll
            for (int u = 0; u < DPL; ++u) acc[u] = 0.f;
            for (int jj = 0; jj < nk; ++jj) {
                const float p = pp[jj];
                if (p == 0.f) continue;
                float vv[DPL];
                load_run<WT, DPL>(Vs + (size_t)jj * RS + lane * DPL, vv);
#pragma unroll
                for (int u = 0; u < DPL; ++u) acc[u] = fmaf(p, vv[u], acc[u]);
            }
            float *part = a.attn_part + (((size_t)t * a.Hq + (size_t)g * G + hl) * a.splits + s) * PS;
#pragma unroll
            for (int u = 0; u < DPL; ++u) part[lane * DPL + u] = acc[u];
            if (lane == 0) { part[D] = mloc; part[D + 1] = lsum; }
        }
    } else {
        for (int pr = warp; pr < NQ; pr += nwarp) {
            const int j = pr / G, hl = pr % G, t = b * a.w + j;
            float *part = a.attn_part + (((size_t)t * a.Hq + (size_t)g * G + hl) * a.splits + s) * PS;
#pragma unroll
            for (int u = 0; u < DPL; ++u) part[lane * DPL + u] = 0.f;
            if (lane == 0) { part[D] = -INFINITY; part[D + 1] = 0.f; }
        }
    }
    tree_merge_splits<WT, D>(a, b, g, ws, &s_last);
}

// ------------------------------------------------------------------ attention on tensor cores

// bf16 caches with at most 16 row-head pairs (w * G <= 16).  CTA (s, g, b)
// stages kTcChunk keys as above; compute warp w takes keys 16w .. 16w + 15 in
// the M dimension of mma.sync.m16n8k16 with the pairs in N (one or two n8
// tiles).  S^T = K q^T with each query (rotated, times 1/sqrt(D)) split into a
// bf16 hi + lo pair (two MMAs: operand error near 2^-17, K exact); the warp's
// softmax per pair over its 16 keys; P^T from the S^T tile by movmatrix (the
// accumulator layout of S^T is the B-fragment layout of P^T, transposed), also
// split hi + lo; O^T += V^T P^T with V^T read by a transposing ldmatrix.  The
// warps' (max, sum, O) merge in shared memory into the CTA's split partial;
// the splits then merge as in the CUDA-core kernel.
constexpr int kTcWarps = 8;
constexpr int kTcChunk = kTcWarps * 16;
constexpr int kTcMaxPairs = 16;

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}
__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
                 "{%8, %9}, {%0, %1, %2, %3};"
                 : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// bf16 hi / lo parts of two floats, packed (low half = first element).
__device__ __forceinline__ void split2(float x, float y, uint32_t &hi, uint32_t &lo) {
    const uint16_t hx = f32_to_bf16(x), hy = f32_to_bf16(y);
    hi = (uint32_t)hx | ((uint32_t)hy << 16);
    lo = (uint32_t)f32_to_bf16(x - bf16_to_f32(hx)) | ((uint32_t)f32_to_bf16(y - bf16_to_f32(hy)) << 16);
}

template <int D>
__global__ void __launch_bounds__(kTcWarps * 32) tree_attention_tc_kernel(const TreeArgs a) {
    constexpr int RS = D + 8;                 // bf16 row stride: 16-byte rows, conflict-free ldmatrix
    constexpr int NT = D / 16;                // 16-dim tiles
    constexpr int PS = D + 4;
    constexpr int QS = D + 8;                 // query row stride: at most 2-way bank conflicts in the B loads
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ int s_last;
    __shared__ unsigned long long s_mask[kTreeMaxWidth];
    uint16_t *Ks = (uint16_t *)smem_raw;
    uint16_t *Vs = Ks + (size_t)kTcChunk * RS;
    float *qs = (float *)(Vs + (size_t)kTcChunk * RS);  // [16][QS] scaled queries, pairs >= NQ zero
    float *wm = qs + kTcMaxPairs * QS;                  // [warp][16]
    float *wl = wm + kTcWarps * kTcMaxPairs;            // [warp][16]
    float *ws = wl + kTcWarps * kTcMaxPairs;            // [16][splits]
    float *wo = (float *)smem_raw;                      // [warp][16][D], after the keys are consumed
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = a.Hq / a.Hkv, NQ = a.w * G;

    pdl_trigger();

    const int n = tree_n(a, b), L = a.kv_len[b];
    const int base = L + n;
    int PE = base + (a.step - 1) * a.w;
    if (PE > a.max_ctx) PE = a.max_ctx;
    const int j0 = s * kTcChunk;
    int nk = PE - j0 < kTcChunk ? PE - j0 : kTcChunk;
    if (L < 0) nk = 0;
    const int ncom = nk > 0 ? tree_stage_committed<uint16_t, D, RS>(a, b, g, j0, nk, L, Ks, Vs) : 0;
    pdl_wait();
    if (s == 0 && g == 0 && tid == 0 && (L < 0 || base + (a.step - 1) * a.w > a.max_ctx)) set_err(a.err, kErrCache);
    if (tid < a.w) s_mask[tid] = a.front_mask[b * a.w + tid];
    for (int e = tid; e < (kTcMaxPairs - NQ) * QS; e += blockDim.x) qs[NQ * QS + e] = 0.f;
    if (nk > 0) {
        tree_stage<uint16_t, D, RS, QS>(a, b, g, j0, nk, base, Ks, Vs, qs, 1.0f / sqrtf((float)D), ncom);
        // rows past the chunk's keys: zero (their probabilities are 0, and 0 * NaN would not be)
        for (int e = tid; e < (kTcChunk - nk) * (D / 8); e += blockDim.x) {
            const int r = nk + e / (D / 8), c = e % (D / 8);
            *(uint4 *)(Ks + (size_t)r * RS + c * 8) = make_uint4(0, 0, 0, 0);
            *(uint4 *)(Vs + (size_t)r * RS + c * 8) = make_uint4(0, 0, 0, 0);
        }
    }
    cp_async_wait_all();
    __syncthreads();
    // this CTA's keys are in: its share of the next kernel's weights into L2
    if (tid == 0)
        prefetch_l2_share(a.pf_next, a.pf_next_bytes, s + a.splits * (g + a.Hkv * b), a.splits * a.Hkv * a.B);

    // warp state: pairs nt * 8 + 2 (lane % 4) + {0, 1}; O^T dims 16 t + lane / 4 (+ 8)
    const int kr = 16 * warp;
    const int cnt = nk - kr;                  // keys of this warp (may be <= 0)
    const int ntn = (NQ + 7) / 8;
    float mx[2][2], sm[2][2], o[2][NT][4];
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        mx[nt][0] = mx[nt][1] = -INFINITY;
        sm[nt][0] = sm[nt][1] = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) o[nt][t][0] = o[nt][t][1] = o[nt][t][2] = o[nt][t][3] = 0.f;
    }
    if (cnt > 0) {
        const uint32_t kb = (uint32_t)__cvta_generic_to_shared(Ks), vb = (uint32_t)__cvta_generic_to_shared(Vs);
        const int mi = lane >> 3;
        float sh[2][4], sl[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int q = 0; q < 4; ++q) sh[nt][q] = sl[nt][q] = 0.f;
#pragma unroll
        for (int ks = 0; ks < NT; ++ks) {
            uint32_t ka[4];
            ldsm_x4(kb + (uint32_t)(((kr + (mi & 1) * 8 + (lane & 7)) * RS + 16 * ks + (mi >> 1) * 8) * 2), ka);
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                if (nt >= ntn) break;
                uint32_t qh[2], ql[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const float *src = qs + (nt * 8 + (lane >> 2)) * QS + 16 * ks + 2 * (lane & 3) + 8 * u;
                    split2(src[0], src[1], qh[u], ql[u]);
                }
                mma16816(sh[nt], ka, qh[0], qh[1]);
                mma16816(sl[nt], ka, ql[0], ql[1]);
            }
        }
        uint32_t pbh[2][2], pbl[2][2];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            float sv[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int key = (lane >> 2) + (q >> 1) * 8, pr = nt * 8 + 2 * (lane & 3) + (q & 1);
                const bool vis = key < cnt && pr < NQ && tree_visible(j0 + kr + key, base, s_mask[pr / G]);
                sv[q] = vis ? sh[nt][q] + sl[nt][q] : -INFINITY;
            }
            // softmax per pair over the warp's 16 keys: lanes with equal lane % 4 share pairs
            float c0 = fmaxf(sv[0], sv[2]), c1 = fmaxf(sv[1], sv[3]);
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                c0 = fmaxf(c0, __shfl_xor_sync(0xFFFFFFFFu, c0, off));
                c1 = fmaxf(c1, __shfl_xor_sync(0xFFFFFFFFu, c1, off));
            }
            mx[nt][0] = c0;
            mx[nt][1] = c1;
            float p[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float mq = (q & 1) ? c1 : c0;
                p[q] = sv[q] == -INFINITY ? 0.f : expf(sv[q] - mq);
            }
            sm[nt][0] = p[0] + p[2];
            sm[nt][1] = p[1] + p[3];
            uint32_t h01, l01, h23, l23;
            split2(p[0], p[1], h01, l01);
            split2(p[2], p[3], h23, l23);
            pbh[nt][0] = movm_t(h01);
            pbh[nt][1] = movm_t(h23);
            pbl[nt][0] = movm_t(l01);
            pbl[nt][1] = movm_t(l23);
        }
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            uint32_t va[4];
            ldsm_x4_t(vb + (uint32_t)(((kr + (mi >> 1) * 8 + (lane & 7)) * RS + 16 * t + (mi & 1) * 8) * 2), va);
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                if (nt >= ntn) break;
                mma16816(o[nt][t], va, pbh[nt][0], pbh[nt][1]);
                mma16816(o[nt][t], va, pbl[nt][0], pbl[nt][1]);
            }
        }
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                sm[nt][0] += __shfl_xor_sync(0xFFFFFFFFu, sm[nt][0], off);
                sm[nt][1] += __shfl_xor_sync(0xFFFFFFFFu, sm[nt][1], off);
            }
    }
    __syncthreads();                          // every warp is done with K and V: wo may overwrite them
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        const int p0 = nt * 8 + 2 * (lane & 3);
        if (lane < 4) {
            wm[warp * kTcMaxPairs + p0] = mx[nt][0];
            wm[warp * kTcMaxPairs + p0 + 1] = mx[nt][1];
            wl[warp * kTcMaxPairs + p0] = sm[nt][0];
            wl[warp * kTcMaxPairs + p0 + 1] = sm[nt][1];
        }
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int d = 16 * t + (lane >> 2) + (q >> 1) * 8, pr = p0 + (q & 1);
                wo[((size_t)warp * kTcMaxPairs + pr) * D + d] = o[nt][t][q];
            }
    }
    __syncthreads();
    // the CTA's partial of each pair: warps merged in warp order
    for (int e = tid; e < NQ * D; e += blockDim.x) {
        const int pr = e / D, d = e % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kTcWarps; ++w) M = fmaxf(M, wm[w * kTcMaxPairs + pr]);
        float acc = 0.f, den = 0.f;
#pragma unroll
        for (int w = 0; w < kTcWarps; ++w) {
            const float lw = wl[w * kTcMaxPairs + pr];
            const float wt = lw > 0.f ? expf(wm[w * kTcMaxPairs + pr] - M) : 0.f;
            acc = fmaf(wt, wo[((size_t)w * kTcMaxPairs + pr) * D + d], acc);
            den = fmaf(wt, lw, den);
        }
        const int j = pr / G, hl = pr % G, t = b * a.w + j;
        float *part = a.attn_part + (((size_t)t * a.Hq + (size_t)g * G + hl) * a.splits + s) * PS;
        part[d] = acc;
        if (d == 0) { part[D] = M; part[D + 1] = den; }
    }
    tree_merge_splits<uint16_t, D>(a, b, g, ws, &s_last);
}

// ------------------------------------------------------------------ selection

constexpr int kSelectThreads = 256;

// One CTA per sequence.  Candidate c = j * w + r of step k (row j's r-th best
// token) has pool index base + c and score = frontier score of row j +
// logit - lse.  Frontier and tree orders: score descending, then pool index
// ascending (a parent always ranks before its children).
struct SelectSmem {
    unsigned long long fmask[kTreeMaxWidth];
    float fscore[kTreeMaxWidth];
    int fpool[kTreeMaxWidth];
    float cs[kTreeMaxWidth * kTreeMaxWidth];
    float ps[kTreeMaxPool];
    int sel[kTreeMaxPool];
    int pos[kTreeMaxPool];
};

// Run by all kSelectThreads threads of one CTA for sequence b, once every row
// of b has its log-sum-exp (read through L2: other CTAs wrote them).
__device__ void select_sequence(const TreeArgs &a, int b, SelectSmem &sm) {
    float *s_fscore = sm.fscore, *s_cs = sm.cs, *s_ps = sm.ps;
    int *s_fpool = sm.fpool, *s_sel = sm.sel, *s_pos = sm.pos;
    unsigned long long *s_fmask = sm.fmask;
    const int tid = threadIdx.x, w = a.w, k = a.step, R = a.R;
    const int base = k == 1 ? 0 : w + (k - 2) * w * w;
    const int nc = R * w;
    if (tid < R) {
        s_fscore[tid] = k == 1 ? 0.f : a.front_score[b * w + tid];
        s_fpool[tid] = k == 1 ? -1 : a.front_pool[b * w + tid];
        s_fmask[tid] = k == 1 ? 0ull : a.front_mask[b * w + tid];
    }
    __syncthreads();
    int tok = 0;
    float sc = 0.f;
    if (tid < nc) {
        const int j = tid / w, r = tid % w, t = b * w + j;
        tok = a.top_ids[(size_t)t * w + r];
        sc = s_fscore[j] + (a.top_vals[(size_t)t * w + r] - __ldcg(a.lse + t));
        s_cs[tid] = sc;
        const size_t e = (size_t)b * a.P + base + tid;
        a.pool_tok[e] = tok;
        a.pool_par[e] = s_fpool[j];
        a.pool_score[e] = sc;
    }
    __syncthreads();
    if (tid < nc) {
        int rank = 0;
        for (int c = 0; c < nc; ++c) rank += (s_cs[c] > sc) || (s_cs[c] == sc && c < tid);
        if (rank < w) {
            const int j = tid / w, o = b * w + rank;
            a.front_tok[o] = tok;
            a.front_row[o] = k == 1 ? b : b * w + j;   // the h^ row that emitted the token
            a.front_pool[o] = base + tid;
            a.front_score[o] = sc;
            const int bit = (k - 1) * w + rank;     // the slot offset of the row that processes it next
            a.front_mask[o] = s_fmask[j] | (bit < kTreeMaskBits ? 1ull << bit : 0ull);
            if (a.out_frontier) a.out_frontier[((size_t)b * a.K + k - 1) * w + rank] = base + tid;
        }
    }
    if (k < a.K) return;                           // uniform over the CTA

    // the verified tree: the n_nodes best of the pool, listed in pool order
    __syncthreads();
    const int P = a.P;
    const size_t pb = (size_t)b * P;
    for (int e = tid; e < P; e += kSelectThreads) s_ps[e] = __ldcg(a.pool_score + pb + e);
    __syncthreads();
    for (int e = tid; e < P; e += kSelectThreads) {
        const float se = s_ps[e];
        int rank = 0;
        for (int c = 0; c < P; ++c) {
            const float x = s_ps[c];
            rank += (x > se) || (x == se && c < e);
        }
        s_sel[e] = rank < a.n_nodes;
    }
    __syncthreads();
    for (int e = tid; e < P; e += kSelectThreads) {
        int p = -1;
        if (s_sel[e]) {
            p = 0;
            for (int c = 0; c < e; ++c) p += s_sel[c];
        }
        s_pos[e] = p;
    }
    __syncthreads();
    for (int e = tid; e < P; e += kSelectThreads) {
        const int tk = __ldcg(a.pool_tok + pb + e), par = __ldcg(a.pool_par + pb + e);
        if (a.out_pool_tokens) a.out_pool_tokens[pb + e] = tk;
        if (a.out_pool_parents) a.out_pool_parents[pb + e] = par;
        if (a.out_pool_scores) a.out_pool_scores[pb + e] = s_ps[e];
        const int p = s_pos[e];
        if (p < 0) continue;
        const size_t o = (size_t)b * a.n_nodes + p;
        a.tree_tokens[o] = tk;
        a.tree_depths[o] = e < w ? 1 : 2 + (e - w) / (w * w);
        a.tree_scores[o] = s_ps[e];
        a.tree_parents[o] = par < 0 ? -1 : s_pos[par];
    }
}

// ------------------------------------------------------------------ log-sum-exp

// Grid (blocks per row, B * R): row t = b * w + j.  Its log-sum-exp comes
// either from the LM head's per-CTA partials (lm_lse_grid > 0: one CTA per
// row merges them) or from the logits the LM head wrote (chunks of the row
// per CTA, the row's last CTA merging the chunks' partials).  The last row
// of a sequence to finish then scores the candidates and picks the frontier.
constexpr int kLseMaxParts = 256;
__global__ void __launch_bounds__(256) tree_lse_kernel(const TreeArgs a) {
    __shared__ float s_m[8], s_s[8];
    __shared__ int s_last, s_seq;
    __shared__ Key s_k[4][kTopK];
    __shared__ SelectSmem sm;
    pdl_trigger();
    pdl_wait();
    const int blk = blockIdx.x, nblk = gridDim.x;
    const int b = blockIdx.y / a.R, j = blockIdx.y % a.R, t = b * a.w + j;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float *parts;
    int nparts;
    if (a.lm_lse_grid > 0) {
        // the LM head's row of this tree row: b at step 1 (one row per sequence), t after
        const int lm_row = a.step == 1 ? b : t;
        parts = a.lse_part + (size_t)lm_row * a.lm_lse_grid * 2;
        nparts = a.lm_lse_grid;
    } else {
        const float *z = a.logits + (size_t)t * a.V;
        const int lo = blk * a.lse_chunk, hi = min(a.V, lo + a.lse_chunk);
        float m = -INFINITY, s = 0.f;
        constexpr int kBatch = 8;                  // loads in flight per thread before any use
        for (int i0 = lo + tid; i0 < hi; i0 += kBatch * 256) {
            float v[kBatch];
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                const int i = i0 + q * 256;
                v[q] = i < hi ? z[i] : -INFINITY;
            }
#pragma unroll
            for (int q = 0; q < kBatch; ++q)
                if (v[q] != -INFINITY) lse_merge(m, s, v[q], 1.f);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o), s2 = __shfl_xor_sync(0xFFFFFFFFu, s, o);
            lse_merge(m, s, m2, s2);
        }
        if (lane == 0) { s_m[warp] = m; s_s[warp] = s; }
        __syncthreads();
        if (tid == 0) {
            for (int q = 1; q < (int)(blockDim.x >> 5); ++q) lse_merge(m, s, s_m[q], s_s[q]);
            float *part = a.lse_part + ((size_t)t * kSampleMaxBlocks + blk) * 2;
            part[0] = m;
            part[1] = s;
            __threadfence();
            s_last = atomicAdd(a.lse_ctr + t, 1) == nblk - 1;
        }
        __syncthreads();
        if (!s_last) return;                       // uniform over the CTA
        __threadfence();
        if (tid == 0) a.lse_ctr[t] = 0;
        parts = a.lse_part + (size_t)t * kSampleMaxBlocks * 2;
        nparts = nblk;
    }
    // lane l of warp 0 merges partials l, l + 32, ... (all loads issued
    // first), then the lanes merge in a fixed butterfly order
    if (warp == 0) {
        constexpr int kPer = kLseMaxParts / 32;
        float pm[kPer], ps[kPer];
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            const int q = lane + 32 * i;
            pm[i] = q < nparts ? __ldcg(parts + 2 * q) : -INFINITY;
            ps[i] = q < nparts ? __ldcg(parts + 2 * q + 1) : 0.f;
        }
        float M = -INFINITY, S = 0.f;
#pragma unroll
        for (int i = 0; i < kPer; ++i) lse_merge(M, S, pm[i], ps[i]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xFFFFFFFFu, M, o), s2 = __shfl_xor_sync(0xFFFFFFFFu, S, o);
            lse_merge(M, S, m2, s2);
        }
        if (lane == 0) a.lse[t] = M + logf(S);
    } else if (a.lm_val && a.lm_lse_grid > 0 && warp <= 4) {
        // warps 1-4: the LM head's per-CTA top-8 lists of this row, merged
        // (every load of a thread's share first, then its insertions, then
        // each warp's lists across lanes)
        const int lm_row = a.step == 1 ? b : t;
        const int nc = a.lm_lse_grid * kTopK, e = tid - 32;
        const float *pv = a.lm_val + (size_t)lm_row * nc;
        const int *pi = a.lm_id + (size_t)lm_row * nc;
        constexpr int kB = 16;
        float v[kB];
        int id[kB];
#pragma unroll
        for (int q = 0; q < kB; ++q) {
            const int c = e + q * 128;
            v[q] = c < nc ? __ldcg(pv + c) : 0.f;
            id[q] = c < nc ? __ldcg(pi + c) : -1;
        }
        Key l[kTopK];
        key_clear(l);
#pragma unroll 1
        for (int q = 0; q < kB; ++q)
            if (id[q] >= 0) key_insert(l, pack_best(v[q], id[q]));
#pragma unroll 1
        for (int c = e + kB * 128; c < nc; c += 128)
            if (__ldcg(pi + c) >= 0) key_insert(l, pack_best(__ldcg(pv + c), __ldcg(pi + c)));
#pragma unroll 1
        for (int m = 1; m < 32; m <<= 1) key_merge_xor(l, m);
        if (lane == 0)
#pragma unroll
            for (int i = 0; i < kTopK; ++i) s_k[warp - 1][i] = l[i];
    }
    __syncthreads();
    if (a.lm_val && a.lm_lse_grid > 0 && warp == 1) {
        // the row's top-w candidates, ranked (logit descending, then id ascending)
        Key l[kTopK];
#pragma unroll
        for (int i = 0; i < kTopK; ++i) l[i] = lane < 4 ? s_k[lane][i] : 0ull;
#pragma unroll 1
        for (int m = 1; m < 32; m <<= 1) key_merge_xor(l, m);
        if (lane < a.w) {
            float v;
            int id;
            unpack_best(key_at(l, lane), v, id);
            a.top_ids[(size_t)t * a.w + lane] = id;
            a.top_vals[(size_t)t * a.w + lane] = v;
        }
    }
    // the row's results before its ticket
    __threadfence();
    __syncthreads();
    if (tid == 0) s_seq = atomicAdd(a.seq_ctr + b, 1) == a.R - 1;
    __syncthreads();
    if (!s_seq) return;                        // uniform over the CTA
    // the last row of sequence b to finish: candidates, frontier (and the tree)
    __threadfence();
    if (threadIdx.x == 0) a.seq_ctr[b] = 0;
    select_sequence(a, b, sm);
}

// ------------------------------------------------------------------ acceptance

__global__ void accept_tree_kernel(const AcceptTreeArgs a) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= a.B) return;
    const int m = a.n_nodes, K = a.K;
    const int32_t *tok = a.tree_tokens + (size_t)b * m, *par = a.tree_parents + (size_t)b * m;
    const int32_t *tn = a.target_next + (size_t)b * (m + 1);
    for (int j = 0; j < K; ++j) a.accept_nodes[b * K + j] = -1;
    for (int j = 0; j <= K; ++j) a.out_tokens[b * (K + 1) + j] = -1;
    int cur = -1, acc = 0;
    while (acc < K) {
        const int want = tn[cur + 1];
        int next = -1;
        for (int i = 0; i < m; ++i)
            if (par[i] == cur && tok[i] == want) { next = i; break; }
        if (next < 0) break;
        a.accept_nodes[b * K + acc] = next;
        a.out_tokens[b * (K + 1) + acc] = tok[next];
        ++acc;
        cur = next;
    }
    a.out_tokens[b * (K + 1) + acc] = tn[cur + 1];
    a.accept_len[b] = acc;
    a.kv_len[b] += a.n_new[b];
}

template <typename WT, int D>
size_t tree_attn_smem(int chunk, int G, int w, int splits) {
    constexpr int RS = D + Elem<WT>::kPerVec;
    const int NQ = w * G;
    return 2 * (size_t)chunk * RS * sizeof(WT) + ((size_t)NQ * D + (size_t)NQ * chunk + (size_t)NQ * splits) * 4;
}

template <int D>
size_t tree_attn_tc_smem(int splits) {
    return 2 * (size_t)kTcChunk * (D + 8) * 2 + ((size_t)kTcMaxPairs * (D + 8) + 2 * kTcWarps * kTcMaxPairs +
                                                 (size_t)kTcMaxPairs * splits) * 4;
}

// the tensor-core kernel's split count (kTcChunk keys per CTA)
int tc_splits(int max_ctx) { return (max_ctx + kTcChunk - 1) / kTcChunk; }

template <typename WT, int D>
cudaError_t launch_tree_attn_t(const TreeArgs &args, cudaStream_t s, bool pdl) {
    if (sizeof(WT) == 2 && args.w * (args.Hq / args.Hkv) <= kTcMaxPairs && tc_splits(args.max_ctx) <= 256) {
        TreeArgs a = args;
        a.chunk = kTcChunk;
        a.splits = tc_splits(a.max_ctx);
        return launch_k(tree_attention_tc_kernel<D>, dim3(a.splits, a.Hkv, a.B), dim3(kTcWarps * 32),
                        tree_attn_tc_smem<D>(a.splits), s, pdl, a);
    }
    const size_t smem = tree_attn_smem<WT, D>(args.chunk, args.Hq / args.Hkv, args.w, args.splits);
    return launch_k(tree_attention_kernel<WT, D>, dim3(args.splits, args.Hkv, args.B), dim3(kTreeAttnThreads), smem,
                    s, pdl, args);
}

template <typename WT, int D>
cudaError_t prepare_tree_attn_t(int chunk, int G, int w, int splits, int max_ctx) {
    if (sizeof(WT) == 2 && tc_splits(max_ctx) <= 256) {
        cudaError_t e = cudaFuncSetAttribute(tree_attention_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)tree_attn_tc_smem<D>(tc_splits(max_ctx)));
        if (e != cudaSuccess) return e;
    }
    const size_t smem = tree_attn_smem<WT, D>(chunk, G, w, splits);
    return cudaFuncSetAttribute(tree_attention_kernel<WT, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

}  // namespace

size_t tree_attention_smem_bytes(bool bf16, int D, int chunk, int G, int w, int splits) {
    if (bf16) return D == 64 ? tree_attn_smem<uint16_t, 64>(chunk, G, w, splits) : tree_attn_smem<uint16_t, 128>(chunk, G, w, splits);
    return D == 64 ? tree_attn_smem<float, 64>(chunk, G, w, splits) : tree_attn_smem<float, 128>(chunk, G, w, splits);
}

cudaError_t prepare_tree_kernels(bool bf16, int D, int chunk, int G, int w, int splits, int max_ctx) {
    if (bf16) return D == 64 ? prepare_tree_attn_t<uint16_t, 64>(chunk, G, w, splits, max_ctx)
                             : prepare_tree_attn_t<uint16_t, 128>(chunk, G, w, splits, max_ctx);
    return D == 64 ? prepare_tree_attn_t<float, 64>(chunk, G, w, splits, max_ctx)
                   : prepare_tree_attn_t<float, 128>(chunk, G, w, splits, max_ctx);
}

cudaError_t launch_tree_gather(const TreeArgs &a, bool bf16, cudaStream_t s, bool pdl) {
    const int vec = bf16 ? 8 : 4;
    const dim3 grid(a.B * a.w, (a.d / vec + kGatherThreads - 1) / kGatherThreads);
    if (bf16) return launch_k(tree_gather_kernel<uint16_t>, grid, dim3(kGatherThreads), 0, s, pdl, a);
    return launch_k(tree_gather_kernel<float>, grid, dim3(kGatherThreads), 0, s, pdl, a);
}

cudaError_t launch_tree_attention(const TreeArgs &a, bool bf16, cudaStream_t s, bool pdl) {
    if (bf16) return a.D == 64 ? launch_tree_attn_t<uint16_t, 64>(a, s, pdl) : launch_tree_attn_t<uint16_t, 128>(a, s, pdl);
    return a.D == 64 ? launch_tree_attn_t<float, 64>(a, s, pdl) : launch_tree_attn_t<float, 128>(a, s, pdl);
}

cudaError_t launch_tree_lse(const TreeArgs &args, cudaStream_t s, bool pdl) {
    TreeArgs a = args;
    a.lse_blocks = a.lm_lse_grid > 0 ? 1 : sample_blocks(a.V, &a.lse_chunk);
    if (a.lm_lse_grid > kLseMaxParts) return cudaErrorInvalidValue;
    return launch_k(tree_lse_kernel, dim3(a.lse_blocks, a.B * a.R), dim3(256), 0, s, pdl, a);
}

cudaError_t launch_accept_tree(const AcceptTreeArgs &a, cudaStream_t s) {
    return launch_k(accept_tree_kernel, dim3((a.B + 127) / 128), dim3(128), 0, s, false, a);
}

}  // namespace prism
