// Rotary embedding + KV append, split-KV decode attention and greedy
// acceptance for the PRISM draft round (sm_103a).
//
// All draft modules append to and attend over ONE shared draft KV cache
// (Sec. 3.2): step 1 writes the rows of the n accepted tokens at positions
// L..L+n-1, decode step k writes position L+n+k-2.  Only the last prefill row
// of each sequence feeds h^_0, so attention runs for one query row per
// sequence: the causal window of that row is [0, p].
//
// Attention is flash-decode style: CTA (split s, KV head g, sequence b) scores
// the chunk [s*C, (s+1)*C) of g's keys against the Hq/Hkv query heads that
// share g (grouped-query attention), keeps an fp32 running max / sum / output,
// and writes a partial.  The last CTA of (b, g) to finish (atomic ticket)
// merges the partials in split order with the log-sum-exp rule and writes the
// bf16-rounded attention output that the O projection consumes.
#include "common.cuh"

namespace prism {

namespace {

__device__ __forceinline__ int clamp_n(const int32_t *n_new, int b, int max_new, int *err) {
    int n = n_new[b];
    if (n < 1 || n > max_new) {
        set_err(err, kErrNNew);
        n = n < 1 ? 1 : max_new;
    }
    return n;
}

// Position of the query row of sequence b in this step.
__device__ __forceinline__ int query_pos(int prefill, int L, int n, int step) {
    return prefill ? L + n - 1 : L + n + step - 2;
}

// Asynchronous 16-byte global -> shared copy (no register staging) and the
// wait for all of this thread's outstanding copies.
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

// Partial record of one (sequence, head, split): D output sums, running max,
// running sum, two pad words (16-byte aligned records).
template <int D> struct Part {
    static constexpr int kStride = D + 4;
};

// acc += q[0..VEC) . k-vector (16 bytes of keys)
template <typename WT>
__device__ __forceinline__ void dot_qk(float &acc, const float *q, const uint4 &k);
template <>
__device__ __forceinline__ void dot_qk<uint16_t>(float &acc, const float *q, const uint4 &k) {
    const float4 q0 = *(const float4 *)q, q1 = *(const float4 *)(q + 4);
    acc = fmaf(q0.x, bf16lo(k.x), acc);
    acc = fmaf(q0.y, bf16hi(k.x), acc);
    acc = fmaf(q0.z, bf16lo(k.y), acc);
    acc = fmaf(q0.w, bf16hi(k.y), acc);
    acc = fmaf(q1.x, bf16lo(k.z), acc);
    acc = fmaf(q1.y, bf16hi(k.z), acc);
    acc = fmaf(q1.z, bf16lo(k.w), acc);
    acc = fmaf(q1.w, bf16hi(k.w), acc);
}
template <>
__device__ __forceinline__ void dot_qk<float>(float &acc, const float *q, const uint4 &k) {
    const float4 q0 = *(const float4 *)q;
    acc = fmaf(q0.x, __uint_as_float(k.x), acc);
    acc = fmaf(q0.y, __uint_as_float(k.y), acc);
    acc = fmaf(q0.z, __uint_as_float(k.z), acc);
    acc = fmaf(q0.w, __uint_as_float(k.w), acc);
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

template <typename WT>
__global__ void __launch_bounds__(128) rope_append_kernel(const RopeArgs a) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int H = a.Hq + 2 * a.Hkv;
    if (gw >= a.rows * H) return;
    const int row = gw / H, h = gw % H;
    const int b = a.prefill ? row / a.max_new : row;
    const int i = a.prefill ? row % a.max_new : 0;
    const int n = clamp_n(a.n_new, b, a.max_new, a.err);
    if (a.prefill && i >= n) return;
    const int L = a.kv_len[b];
    const int pos = a.prefill ? L + i : L + n + a.step - 2;
    const bool is_last = !a.prefill || i == n - 1;
    const int D = a.D, half = D / 2;
    const float *x = a.qkv + (size_t)row * H * D + (size_t)h * D;
    const bool in_range = pos >= 0 && pos < a.max_ctx;
    if (h >= a.Hq && !in_range) {
        if (lane == 0) set_err(a.err, kErrCache);
        return;
    }
    const int pc = in_range ? pos : 0;
    if (h < a.Hq) {
        if (!is_last) return;
        float *q = a.q_out + ((size_t)b * a.Hq + h) * D;
        for (int j = lane; j < half; j += 32) {
            const float c = a.rope_cos[(size_t)pc * half + j], s = a.rope_sin[(size_t)pc * half + j];
            const float x0 = x[j], x1 = x[j + half];
            q[j] = x0 * c - x1 * s;
            q[j + half] = x1 * c + x0 * s;
        }
    } else if (h < a.Hq + a.Hkv) {
        const int g = h - a.Hq;
        WT *k = (WT *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        for (int j = lane; j < half; j += 32) {
            const float c = a.rope_cos[(size_t)pos * half + j], s = a.rope_sin[(size_t)pos * half + j];
            const float x0 = x[j], x1 = x[j + half];
            Elem<WT>::store(k, j, x0 * c - x1 * s);
            Elem<WT>::store(k, j + half, x1 * c + x0 * s);
        }
    } else {
        const int g = h - a.Hq - a.Hkv;
        WT *v = (WT *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        for (int j = lane; j < D; j += 32) Elem<WT>::store(v, j, x[j]);
    }
}

template <typename WT, int D>
__global__ void __launch_bounds__(kAttnThreads) attention_kernel(const AttnArgs a) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ int s_last;
    constexpr int VEC = Elem<WT>::kPerVec;
    constexpr int PAD = VEC;                 // one 16-byte vector of padding per row
    constexpr int RS = D + PAD;              // row stride in elements
    constexpr int DPL = D / 32;              // output dims per lane
    const int C = a.chunk;
    const int G = a.Hq / a.Hkv;
    WT *Ks = (WT *)smem_raw;
    WT *Vs = Ks + (size_t)C * RS;
    float *qs = (float *)(Vs + (size_t)C * RS);   // [G][D]
    float *ps = qs + (size_t)G * D;               // [G][C]
    float *ws = ps + (size_t)G * C;               // [G][splits] combine weights
    constexpr int PS = Part<D>::kStride;

    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;

    pdl_trigger();
    pdl_wait();

    const int n = clamp_n(a.n_new, b, a.max_new, a.err);
    const int L = a.kv_len[b];
    int P = query_pos(a.prefill, L, n, a.step) + 1;   // keys [0, P)
    if (P > a.max_ctx) P = a.max_ctx;
    if (P < 1) P = 1;
    const int j0 = s * C;
    const int nk = P - j0 < C ? P - j0 : C;
    if (PRISM_CHECK(a.err, (((uintptr_t)a.k_cache | (uintptr_t)a.v_cache) & 15) == 0, 201, 0, 0) ||
        PRISM_CHECK(a.err, j0 + (nk > 0 ? nk : 0) <= a.max_ctx, 202, j0, nk))
        return;
    const float scale = 1.0f / sqrtf((float)D);

    if (nk > 0) {
        const uint4 *kg = (const uint4 *)((const WT *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D);
        const uint4 *vg = (const uint4 *)((const WT *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + j0) * D);
        constexpr int VPR = D / VEC;   // vectors per row
        for (int e = threadIdx.x; e < nk * VPR; e += blockDim.x) {
            const int r = e / VPR, c = e % VPR;
            cp_async16(Ks + (size_t)r * RS + c * VEC, kg + e);
            cp_async16(Vs + (size_t)r * RS + c * VEC, vg + e);
        }
        for (int e = threadIdx.x; e < G * D; e += blockDim.x)
            qs[e] = a.q[((size_t)b * a.Hq + (size_t)g * G) * D + e];
        cp_async_wait_all();
        __syncthreads();

        for (int hl = warp; hl < G; hl += nwarp) {
            const float *q = qs + (size_t)hl * D;
            float mloc = -INFINITY;
            for (int jj = lane; jj < nk; jj += 32) {
                const WT *kr = Ks + (size_t)jj * RS;
                float dot = 0.f;
#pragma unroll 4
                for (int c = 0; c < D; c += VEC) dot_qk<WT>(dot, q + c, *(const uint4 *)(kr + c));
                dot *= scale;
                ps[(size_t)hl * C + jj] = dot;
                mloc = fmaxf(mloc, dot);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xFFFFFFFFu, mloc, o));
            float lsum = 0.f;
            for (int jj = lane; jj < nk; jj += 32) {
                const float p = expf(ps[(size_t)hl * C + jj] - mloc);
                ps[(size_t)hl * C + jj] = p;
                lsum += p;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xFFFFFFFFu, lsum, o);
            __syncwarp();
            float acc[DPL];
#pragma unroll
            for (int u = 0; u < DPL; ++u) acc[u] = 0.f;
            for (int jj = 0; jj < nk; ++jj) {
                const float p = ps[(size_t)hl * C + jj];
                float vv[DPL];
                load_run<WT, DPL>(Vs + (size_t)jj * RS + lane * DPL, vv);
#pragma unroll
                for (int u = 0; u < DPL; ++u) acc[u] = fmaf(p, vv[u], acc[u]);
            }
            const int h = g * G + hl;
            float *part = a.part + (((size_t)b * a.Hq + h) * a.splits + s) * PS;
#pragma unroll
            for (int u = 0; u < DPL; ++u) part[lane * DPL + u] = acc[u];
            if (lane == 0) { part[D] = mloc; part[D + 1] = lsum; }
        }
    } else {
        for (int hl = warp; hl < G; hl += nwarp) {
            const int h = g * G + hl;
            float *part = a.part + (((size_t)b * a.Hq + h) * a.splits + s) * PS;
#pragma unroll
            for (int u = 0; u < DPL; ++u) part[lane * DPL + u] = 0.f;
            if (lane == 0) { part[D] = -INFINITY; part[D + 1] = 0.f; }
        }
    }

    // last CTA of (b, g): log-sum-exp merge of the splits in split order
    __threadfence();
    __syncthreads();
    int *ctr = a.counter + (size_t)b * a.Hkv + g;
    if (threadIdx.x == 0) s_last = (atomicAdd(ctr, 1) == a.splits - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int hl = warp; hl < G; hl += nwarp) {
        const int h = g * G + hl;
        const float *part = a.part + ((size_t)b * a.Hq + h) * a.splits * PS;
        float *wh = ws + (size_t)hl * a.splits;
        // lanes over splits: global max, split weights exp(m_s - M), denominator
        // (each lane issues all its loads before using any of them)
        constexpr int kMaxPerLane = 8;                 // splits <= 256
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
            const float w = lv[k] > 0.f ? expf(mv[k] - M) : 0.f;
            if (sp < a.splits) wh[sp] = w;
            den = fmaf(w, lv[k], den);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) den += __shfl_xor_sync(0xFFFFFFFFu, den, o);
        __syncwarp();
        // lanes over output dims: weighted sum of the split outputs in split order
        float acc[DPL];
#pragma unroll
        for (int u = 0; u < DPL; ++u) acc[u] = 0.f;
#pragma unroll 16
        for (int sp = 0; sp < a.splits; ++sp) {
            const float w = wh[sp];
            float v[DPL];
            const float *src = part + (size_t)sp * PS + lane * DPL;
            if constexpr (DPL == 4) {
                const float4 t = __ldcg((const float4 *)src);
                v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
            } else {
                const float2 t = __ldcg((const float2 *)src);
                v[0] = t.x; v[1] = t.y;
            }
#pragma unroll
            for (int u = 0; u < DPL; ++u) acc[u] = fmaf(w, v[u], acc[u]);
        }
        WT *o = (WT *)a.o_out + (size_t)b * a.Hq * D + (size_t)h * D;
        const float inv = 1.0f / den;
#pragma unroll
        for (int u = 0; u < DPL; ++u) Elem<WT>::store(o, lane * DPL + u, acc[u] * inv);
    }
    if (threadIdx.x == 0) *ctr = 0;
}

__global__ void accept_kernel(const AcceptArgs a) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= a.B) return;
    const int K = a.K;
    int acc = 0;
    while (acc < K && a.draft[b * K + acc] == a.target[b * (K + 1) + acc]) ++acc;
    a.accept_len[b] = acc;
    for (int j = 0; j <= K; ++j) {
        int v = -1;
        if (j < acc) v = a.draft[b * K + j];
        else if (j == acc) v = a.target[b * (K + 1) + acc];
        a.out_tokens[b * (K + 1) + j] = v;
    }
    a.kv_len[b] += a.n_new[b];
    if (a.next_tokens) {
        // the next round prefills the accepted drafts and the target's token
        for (int j = 0; j <= acc; ++j) a.next_tokens[b * a.max_new + j] = a.out_tokens[b * (K + 1) + j];
        a.next_n[b] = acc + 1;
    }
}

// ------------------------------------------------------------------ fused
// RoPE + KV append + attention for one query row per sequence, one thread-
// block cluster of CS CTAs per (sequence b, KV head g).  CTA rank r owns the
// key range [r P / CS, (r+1) P / CS) of the causal window [0, P):
//   * cache rows below the committed length L are never written during a
//     round, so the first two chunks of them are requested (cp.async) before
//     griddepcontrol.wait, overlapping the QKV projection's tail;
//   * after the wait, the CTA whose range holds a new position rotates that
//     row's key and stores key and value in the cache; every CTA rotates the
//     query heads of g (scaled by 1/sqrt(D)) into shared memory;
//   * keys stream in chunks of C rows through two shared-memory buffers, K
//     stored transposed (16-byte vector v of key j at [v][j]) so that a warp
//     reads 32 consecutive keys without bank conflicts while every lane reads
//     the same query element; V stays row-major (a warp reads consecutive
//     dims of one row).  An online softmax keeps the running max, sum and
//     unnormalised output of each head;
//   * the CS partial results are merged through distributed shared memory:
//     after a cluster barrier, rank r combines its slice of the (head, dim)
//     outputs from every rank, in rank order, and writes the bf16-rounded
//     attention output.  A second cluster barrier keeps every rank's shared
//     memory alive until all reads are done.
constexpr int kFusedThreads = 512;
constexpr int kMaxCluster = 16;
constexpr long kAttnWaitLimit = 1L << 22;

template <typename WT, int D> struct FusedCfg {
    static constexpr int C = sizeof(WT) * D <= 256 ? 128 : 64;   // keys per chunk
    static constexpr int kVecs = D * (int)sizeof(WT) / 16;       // 16-byte vectors per row
    static constexpr int kPerVec = 16 / (int)sizeof(WT);         // elements per vector
};

__device__ __forceinline__ uint32_t sa(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ float dsmem_ld(const float *local, uint32_t rank) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(sa(local)), "r"(rank));
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
    return v;
}
__device__ __forceinline__ bool fa_try(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                 : "=r"(ok) : "r"(sa(b)), "r"(parity) : "memory");
    return ok != 0;
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Request chunk [j, j + cnt) of head (b, g): K transposed into kt, V row-major
// into vb (16-byte pieces, one per thread in turn).  The caller commits.
template <typename WT, int D>
__device__ __forceinline__ void fa_load(const FusedAttnArgs &a, int b, int g, int j, int cnt, uint4 *kt, WT *vb) {
    using Cf = FusedCfg<WT, D>;
    constexpr int C = Cf::C, NV = Cf::kVecs;
    const size_t off = (((size_t)b * a.Hkv + g) * a.max_ctx + j) * D;
    const uint4 *ks = (const uint4 *)((const WT *)a.k_cache + off);
    const uint4 *vs = (const uint4 *)((const WT *)a.v_cache + off);
    for (int e = threadIdx.x; e < cnt * NV; e += kFusedThreads) {
        const int jj = e / NV, v = e % NV;
        cp_async16(kt + v * C + jj, ks + e);
        cp_async16((uint4 *)vb + e, vs + e);
    }
}

// p4[i % 4] += q[i] * k[i] over one 16-byte vector of keys (q broadcast).
template <typename WT>
__device__ __forceinline__ void dot4(float (&p4)[4], const float *q, const uint4 &k);
template <>
__device__ __forceinline__ void dot4<uint16_t>(float (&p4)[4], const float *q, const uint4 &k) {
    const float4 q0 = *(const float4 *)q, q1 = *(const float4 *)(q + 4);
    p4[0] = fmaf(q0.x, bf16lo(k.x), p4[0]);
    p4[1] = fmaf(q0.y, bf16hi(k.x), p4[1]);
    p4[2] = fmaf(q0.z, bf16lo(k.y), p4[2]);
    p4[3] = fmaf(q0.w, bf16hi(k.y), p4[3]);
    p4[0] = fmaf(q1.x, bf16lo(k.z), p4[0]);
    p4[1] = fmaf(q1.y, bf16hi(k.z), p4[1]);
    p4[2] = fmaf(q1.z, bf16lo(k.w), p4[2]);
    p4[3] = fmaf(q1.w, bf16hi(k.w), p4[3]);
}
template <>
__device__ __forceinline__ void dot4<float>(float (&p4)[4], const float *q, const uint4 &k) {
    const float4 q0 = *(const float4 *)q;
    p4[0] = fmaf(q0.x, __uint_as_float(k.x), p4[0]);
    p4[1] = fmaf(q0.y, __uint_as_float(k.y), p4[1]);
    p4[2] = fmaf(q0.z, __uint_as_float(k.z), p4[2]);
    p4[3] = fmaf(q0.w, __uint_as_float(k.w), p4[3]);
}

template <typename WT, int D>
__global__ void __launch_bounds__(kFusedThreads, 1) fused_attention_kernel(const FusedAttnArgs a) {
    using Cf = FusedCfg<WT, D>;
    constexpr int C = Cf::C, NV = Cf::kVecs;
    extern __shared__ __align__(128) uint8_t smem_raw[];
    __shared__ float s_m[16], s_l[16], s_alpha[16];
    const int G = a.Hq / a.Hkv;
    uint4 *kt = (uint4 *)smem_raw;                   // [2][NV][C] transposed keys
    WT *vbuf = (WT *)(kt + 2 * NV * C);              // [2][C][D]
    float *qs = (float *)(vbuf + 2 * C * D);         // [G][D] rotated, scaled queries
    float *ps = qs + G * D;                          // [G][C] scores, then probabilities
    float *po = ps + G * C;                          // [G][D] this rank's unnormalised output
    float *pm = po + G * D;                          // [16] this rank's running max
    float *pl = pm + 16;                             // [16] this rank's running sum

    const int r = blockIdx.x, g = blockIdx.y, b = blockIdx.z, CS = a.cs;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int half = D / 2, H = a.Hq + 2 * a.Hkv;
    pdl_trigger();

    // ranges (n_new and kv_len are inputs of the round, stable throughout it)
    const int n = clamp_n(a.n_new, b, a.max_new, a.err);
    const int L = a.kv_len[b];
    const int qp = query_pos(a.prefill, L, n, a.step);
    int P = qp + 1;
    if (P > a.max_ctx) P = a.max_ctx;
    if (P < 1) P = 1;
    const int j0 = (int)((long)r * P / CS), j1 = (int)((long)(r + 1) * P / CS);
    const int nch = (j1 - j0 + C - 1) / C;
    const int L_old = L < P ? (L > 0 ? L : 0) : P;   // rows below L_old are immutable
    auto chunk = [&](int i, int &j, int &cnt) {
        j = j0 + i * C;
        cnt = j1 - j < C ? j1 - j : C;
    };
    // chunk 1 holds later positions than chunk 0, so "chunk 1 old" implies "chunk 0 old"
    int pre = 0;                                      // chunks requested before the wait
    for (int i = 0; i < 2 && i < nch; ++i) {
        int j, cnt;
        chunk(i, j, cnt);
        if (j + cnt > L_old) break;
        fa_load<WT, D>(a, b, g, j, cnt, kt + i * NV * C, vbuf + i * C * D);
        cp_commit();
        ++pre;
    }
    pdl_wait();

    // append the new rows this rank owns: positions L .. L+n-1 (prefill) or qp
    const int first_new = a.prefill ? L : qp, n_rows = a.prefill ? n : 1;
    for (int i = 0; i < n_rows; ++i) {
        const int pos = first_new + i;
        if (pos < 0 || pos >= a.max_ctx) {              // no rank owns it: rank 0 reports
            if (r == 0 && tid == 0) set_err(a.err, kErrCache);
            continue;
        }
        if (pos < j0 || pos >= j1) continue;
        const int row = a.prefill ? b * a.max_new + i : b;
        const float *xk = a.qkv + (size_t)row * H * D + (size_t)(a.Hq + g) * D;
        const float *xv = a.qkv + (size_t)row * H * D + (size_t)(a.Hq + a.Hkv + g) * D;
        WT *kc = (WT *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        WT *vc = (WT *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        for (int j = tid; j < half; j += kFusedThreads) {
            const float c = a.rope_cos[(size_t)pos * half + j], sn = a.rope_sin[(size_t)pos * half + j];
            const float x0 = xk[j], x1 = xk[j + half];
            Elem<WT>::store(kc, j, x0 * c - x1 * sn);
            Elem<WT>::store(kc, j + half, x1 * c + x0 * sn);
        }
        for (int j = tid; j < D; j += kFusedThreads) Elem<WT>::store(vc, j, xv[j]);
    }
    // rotated queries of the heads sharing g, at qp, scaled by 1/sqrt(D)
    {
        const int row = a.prefill ? b * a.max_new + n - 1 : b;
        const int pc = qp >= 0 && qp < a.max_ctx ? qp : 0;
        const float scale = 1.0f / sqrtf((float)D);
        for (int e = tid; e < G * half; e += kFusedThreads) {
            const int h = e / half, j = e % half;
            const float *xq = a.qkv + (size_t)row * H * D + (size_t)(g * G + h) * D;
            const float c = a.rope_cos[(size_t)pc * half + j], sn = a.rope_sin[(size_t)pc * half + j];
            const float x0 = xq[j], x1 = xq[j + half];
            qs[h * D + j] = (x0 * c - x1 * sn) * scale;
            qs[h * D + j + half] = (x1 * c + x0 * sn) * scale;
        }
    }
    if (tid < 16) { s_m[tid] = -INFINITY; s_l[tid] = 0.f; }
    __syncthreads();                                  // new cache rows written, queries ready
    for (int i = pre; i < 2 && i < nch; ++i) {
        int j, cnt;
        chunk(i, j, cnt);
        fa_load<WT, D>(a, b, g, j, cnt, kt + i * NV * C, vbuf + i * C * D);
        cp_commit();
    }

    // per-thread outputs: e = tid + 512 i  ->  (head e / D, dim e % D)
    constexpr int kMaxOut = (16 * D + kFusedThreads - 1) / kFusedThreads;
    float acc[kMaxOut];
#pragma unroll
    for (int i = 0; i < kMaxOut; ++i) acc[i] = 0.f;
    const int n_out = G * D;
    constexpr int NHG = kFusedThreads / C;            // head groups in the score pass

    for (int ci = 0; ci < nch; ++ci) {
        const int bi = ci & 1;
        int j, cnt;
        chunk(ci, j, cnt);
        const uint4 *kb = kt + bi * NV * C;
        const WT *vb = vbuf + bi * C * D;
        // this chunk's copies are the oldest outstanding group
        if (ci + 1 < nch) cp_wait<1>(); else cp_wait<0>();
        __syncthreads();
        // scores: thread -> key jl = tid % C, heads tid / C + NHG i; four partial sums
        {
            const int jl = tid % C;
            for (int h = tid / C; h < G; h += NHG) {
                float dot = -INFINITY;
                if (jl < cnt) {
                    float p4[4] = {0.f, 0.f, 0.f, 0.f};
                    const float *q = qs + h * D;
#pragma unroll 4
                    for (int v = 0; v < NV; ++v) dot4<WT>(p4, q + v * Cf::kPerVec, kb[v * C + jl]);
                    dot = (p4[0] + p4[1]) + (p4[2] + p4[3]);
                }
                ps[h * C + jl] = dot;
            }
        }
        __syncthreads();
        // online softmax: warp w takes heads w, w + 16
        for (int h = warp; h < G; h += kFusedThreads / 32) {
            float mx = -INFINITY;
            for (int jl = lane; jl < cnt; jl += 32) mx = fmaxf(mx, ps[h * C + jl]);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
            const float m_old = s_m[h];
            const float m_new = fmaxf(m_old, mx);
            float sum = 0.f;
            for (int jl = lane; jl < cnt; jl += 32) {
                const float pv = m_new == -INFINITY ? 0.f : expf(ps[h * C + jl] - m_new);
                ps[h * C + jl] = pv;
                sum += pv;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
            if (lane == 0) {
                const float alpha = m_old == -INFINITY ? 0.f : expf(m_old - m_new);
                s_alpha[h] = alpha;
                s_l[h] = s_l[h] * alpha + sum;
                s_m[h] = m_new;
            }
        }
        __syncthreads();
        // PV: acc(h, d) = acc * alpha_h + sum_j p_hj V_jd; keys unrolled by 8 in two chains
#pragma unroll
        for (int i = 0; i < kMaxOut; ++i) {
            const int e = tid + kFusedThreads * i;
            if (e >= n_out) break;
            const int h = e / D, d = e % D;
            const float *ph = ps + h * C;
            float x0 = acc[i] * s_alpha[h], x1 = 0.f;
            int jl = 0;
            for (; jl + 8 <= cnt; jl += 8) {
#pragma unroll
                for (int u = 0; u < 8; u += 2) {
                    x0 = fmaf(ph[jl + u], Elem<WT>::load(vb, (size_t)(jl + u) * D + d), x0);
                    x1 = fmaf(ph[jl + u + 1], Elem<WT>::load(vb, (size_t)(jl + u + 1) * D + d), x1);
                }
            }
            for (; jl < cnt; ++jl) x0 = fmaf(ph[jl], Elem<WT>::load(vb, (size_t)jl * D + d), x0);
            acc[i] = x0 + x1;
        }
        __syncthreads();                              // buffer bi and ps free
        if (ci + 2 < nch) {
            int jn, cn;
            chunk(ci + 2, jn, cn);
            fa_load<WT, D>(a, b, g, jn, cn, kt + bi * NV * C, vbuf + bi * C * D);
            cp_commit();
        }
    }
    cp_wait<0>();

    // publish this rank's partial, then merge across the cluster
#pragma unroll
    for (int i = 0; i < kMaxOut; ++i) {
        const int e = tid + kFusedThreads * i;
        if (e < n_out) po[e] = acc[i];
    }
    if (tid < G) { pm[tid] = s_m[tid]; pl[tid] = s_l[tid]; }
    cluster_sync_all();
    {
        const int e0 = (int)((long)r * n_out / CS), e1 = (int)((long)(r + 1) * n_out / CS);
        for (int e = e0 + tid; e < e1; e += kFusedThreads) {
            const int h = e / D;
            // every remote load of this output issued before any is used
            float mq[kMaxCluster], lq[kMaxCluster], oq[kMaxCluster];
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) {
                if (q < CS) {
                    mq[q] = dsmem_ld(pm + h, (uint32_t)q);
                    lq[q] = dsmem_ld(pl + h, (uint32_t)q);
                    oq[q] = dsmem_ld(po + e, (uint32_t)q);
                } else {
                    mq[q] = -INFINITY;
                    lq[q] = oq[q] = 0.f;
                }
            }
            float M = -INFINITY;
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) M = fmaxf(M, mq[q]);
            float num = 0.f, den = 0.f;
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) {
                const float w = mq[q] == -INFINITY ? 0.f : expf(mq[q] - M);
                den = fmaf(w, lq[q], den);
                num = fmaf(w, oq[q], num);
            }
            WT *o = (WT *)a.o_out + (size_t)b * a.Hq * D + (size_t)g * G * D;
            Elem<WT>::store(o, e, den > 0.f ? num / den : 0.f);
        }
    }
    cluster_sync_all();
}

// Tensor-core variant for bf16 caches, with the products transposed so that
// keys fill the MMA's 16-row M dimension and the G <= 8 query heads of g its
// 8-column N dimension:
//   S^T[key][h]  = K[key][:] . q[h][:]       A = 16 keys of K (ldmatrix),
//                                            B = q^T, held in registers;
//   O^T[d][h]   += V^T[d][keys] P^T[keys][h]  A = V^T (transposing ldmatrix),
//                                            B = P^T (movmatrix of the S^T tile).
// The contract keeps q and the probabilities in fp32, so each enters a product
// as a bf16 pair hi + lo (hi = bf16(x), lo = bf16(x - hi)): two MMAs per tile,
// an error near 2^-17 of the operand, with K and V exact.  Shared memory holds
// only K and V as TMA wrote them (128-byte swizzle), and each of their bytes is
// read once.
//   * Keys stream through a ring of kTaStages stages of 16 W rows, filled by
//     one producer warp with TMA tensor loads; stages made only of rows
//     committed before the round are requested before griddepcontrol.wait;
//   * compute warp w owns keys 16w .. 16w + 15 of every stage and keeps its own
//     online softmax (running max, sum and O^T per head), so a stage needs no
//     block-wide barrier: each warp releases it through an mbarrier;
//   * at the end the warps' states merge in shared memory (log-sum-exp rule,
//     warp order), then the cluster's ranks merge through distributed shared
//     memory as in the CUDA-core kernel.
constexpr int kTaStages = 3;
constexpr int kTaBoxRows = 64;                        // rows of one TMA box of the caches
// W compute warps (one more warp issues loads), 16 W keys per stage; with 4
// warps two CTAs share an SM
template <int W> struct TaCfg {
    static constexpr int kThreads = (W + 1) * 32;
    static constexpr int kC = 16 * W;
    static constexpr int kMinBlocks = W <= 4 ? 2 : 1;
    static_assert(W == 4 || W == 8, "4 or 8 compute warps");
};

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
// bf16 hi/lo split of two floats, packed (low half = first element).
__device__ __forceinline__ void split2(float x, float y, uint32_t &hi, uint32_t &lo) {
    const uint16_t hx = f32_to_bf16(x), hy = f32_to_bf16(y);
    hi = (uint32_t)hx | ((uint32_t)hy << 16);
    lo = (uint32_t)f32_to_bf16(x - bf16_to_f32(hx)) | ((uint32_t)f32_to_bf16(y - bf16_to_f32(hy)) << 16);
}
// Whole-warp bounded wait on an mbarrier phase: lane 0 polls, every lane then
// observes the completed phase itself.  Warp-uniform result.
__device__ __forceinline__ bool ta_wait_warp(uint64_t *bar, uint32_t parity, long limit) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) {
        ok = false;
        for (long it = 0; it < limit && !ok; ++it) ok = fa_try(bar, parity);
    }
    ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
    if (ok) fa_try(bar, parity);
    return ok;
}
// Shared-memory address of 16-byte piece `chunk` (8 dims) of row `row` of a
// stage buffer of C rows: D / 64 column blocks of C rows x 128 bytes (each
// loaded as C / 64 boxes), pieces XOR-swizzled by row (the TMA 128-byte
// swizzle).
template <int C>
__device__ __forceinline__ uint32_t ta_piece(uint32_t buf, int row, int chunk) {
    return buf + (uint32_t)(chunk >> 3) * (C * 128) + (uint32_t)row * 128 + ((uint32_t)((chunk & 7) ^ (row & 7)) << 4);
}

// A compute warp's online-softmax state: entries for keys lane / 4 (+ 8) of
// the warp's 16 and heads h0 = 2 (lane % 4), h1 = h0 + 1; O^T for dims
// 16 t + lane / 4 (+ 8) of those heads.
template <int NT> struct TaWarpState {
    float m0, m1, l0, l1;
    float o[NT][4];
    __device__ __forceinline__ void reset() {
        m0 = m1 = -INFINITY;
        l0 = l1 = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
    }
};

// q^T as B fragments from the rotated, scaled queries qs ([8][D], heads past
// G zero): b0 = q[h][16 ks + 2 (lane % 4) + {0, 1}], b1 the same dims + 8,
// h = lane / 4, each as a bf16 pair hi + lo.
template <int NT>
__device__ __forceinline__ void ta_q_frags(const float *qs, uint32_t (&qh)[NT][2], uint32_t (&ql)[NT][2]) {
    constexpr int D = NT * 16;
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int ks = 0; ks < NT; ++ks)
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const float *src = qs + (lane >> 2) * D + 16 * ks + 2 * (lane & 3) + 8 * u;
            split2(src[0], src[1], qh[ks][u], ql[ks][u]);
        }
}

// One stage for one compute warp: its keys kr .. kr + 15 of the stage whose
// K boxes start at kb and V boxes at vb, the first cnt of them valid (cnt in
// 1 .. 16), folded into the warp's state.
template <int NT, int C>
__device__ __forceinline__ void ta_stage(TaWarpState<NT> &st, uint32_t kb, uint32_t vb, int kr, int cnt,
                                         const uint32_t (&qh)[NT][2], const uint32_t (&ql)[NT][2]) {
    constexpr int NH = NT / 4;                        // 64-column boxes per row
    const int lane = threadIdx.x & 31;
    // value rows past the range hold other positions' data: zero them
    // (their probabilities are zero, and 0 * NaN would not be)
    if (cnt < 16) {
        for (int e = lane; e < (16 - cnt) * NH * 8; e += 32) {
            const int row = kr + cnt + e / (NH * 8), piece = e % (NH * 8);
            asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(ta_piece<C>(vb, row, piece)), "r"(0) : "memory");
        }
        __syncwarp();
    }
    // S^T for 16 keys x 8 heads: hi and lo queries, even and odd 16-dim
    // tiles in four independent accumulation chains (half the dependent depth)
    float sh[2][4] = {}, sl[2][4] = {};
#pragma unroll
    for (int ks = 0; ks < NT; ++ks) {
        uint32_t ka[4];
        const int mi = lane >> 3;
        ldsm_x4(ta_piece<C>(kb, kr + (mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), ka);
        mma16816(sh[ks & 1], ka, qh[ks][0], qh[ks][1]);
        mma16816(sl[ks & 1], ka, ql[ks][0], ql[ks][1]);
    }
    float sv[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int key = (lane >> 2) + (q >> 1) * 8;
        sv[q] = key < cnt ? (sh[0][q] + sh[1][q]) + (sl[0][q] + sl[1][q]) : -INFINITY;
    }
    // online softmax of this warp: heads h0 = 2 (lane % 4) (entries 0, 2), h1 (1, 3)
    float c0 = fmaxf(sv[0], sv[2]), c1 = fmaxf(sv[1], sv[3]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        c0 = fmaxf(c0, __shfl_xor_sync(0xFFFFFFFFu, c0, off));
        c1 = fmaxf(c1, __shfl_xor_sync(0xFFFFFFFFu, c1, off));
    }
    // scores are in log2 units (the queries carry log2(e) / sqrt(D)): exp2
    const float n0 = fmaxf(st.m0, c0), n1 = fmaxf(st.m1, c1);
    float p[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float mq = (q & 1) ? n1 : n0;
        p[q] = (sv[q] == -INFINITY || mq == -INFINITY) ? 0.f : exp2f(sv[q] - mq);
    }
    // the running sums rescale only where a lane's maximum moved (rarely,
    // after the first stages)
    if (__any_sync(0xFFFFFFFFu, n0 != st.m0 || n1 != st.m1)) {
        const float al0 = st.m0 == -INFINITY ? 0.f : exp2f(st.m0 - n0);
        const float al1 = st.m1 == -INFINITY ? 0.f : exp2f(st.m1 - n1);
        st.l0 *= al0;
        st.l1 *= al1;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            st.o[t][0] *= al0;
            st.o[t][1] *= al1;
            st.o[t][2] *= al0;
            st.o[t][3] *= al1;
        }
    }
    st.l0 += p[0] + p[2];
    st.l1 += p[1] + p[3];
    st.m0 = n0;
    st.m1 = n1;
    // P^T as B fragments: the S^T tile's 8 x 8 halves, transposed in registers
    uint32_t h01, l01, h23, l23;
    split2(p[0], p[1], h01, l01);
    split2(p[2], p[3], h23, l23);
    const uint32_t pb_h0 = movm_t(h01), pb_h1 = movm_t(h23), pb_l0 = movm_t(l01), pb_l1 = movm_t(l23);
    // O^T += V^T P^T, one 16-dim tile at a time
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        uint32_t va[4];
        const int mi = lane >> 3;
        ldsm_x4_t(ta_piece<C>(vb, kr + (mi >> 1) * 8 + (lane & 7), 2 * t + (mi & 1)), va);
        mma16816(st.o[t], va, pb_h0, pb_h1);
        mma16816(st.o[t], va, pb_l0, pb_l1);
    }
    // zeros written above precede the next TMA write of this slot
    if (cnt < 16) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// With two waves of CTAs the order in which they start decides the tail:
// clusters start roughly in the order of their linear index, so the one with
// sequence index z takes the sequence of rank z in decreasing key count (ties
// by index), and the longest contexts run first.  Every CTA ranks the
// sequences itself from the round's inputs (no kernel of the round writes
// them), before the dependency wait.
constexpr int kLptMaxB = 256;
__device__ __forceinline__ int lpt_sequence(const FusedAttnArgs &a, int z) {
    __shared__ int s_p[kLptMaxB];
    __shared__ int s_b;
    const int B = a.B;
    for (int t = threadIdx.x; t < B; t += blockDim.x) {
        const int n = clamp_n(a.n_new, t, a.max_new, a.err);
        s_p[t] = min(query_pos(a.prefill, a.kv_len[t], n, a.step) + 1, a.max_ctx);
    }
    if (threadIdx.x == 0) s_b = z;
    __syncthreads();
    for (int t = threadIdx.x; t < B; t += blockDim.x) {
        const int p = s_p[t];
        int rank = 0;
        for (int u = 0; u < B; ++u) rank += s_p[u] > p || (s_p[u] == p && u < t);
        if (rank == z) s_b = t;
    }
    __syncthreads();
    return s_b;
}

template <int D, int W>
__global__ void __launch_bounds__(TaCfg<W>::kThreads, TaCfg<W>::kMinBlocks)
    fused_attention_tc_kernel(const FusedAttnArgs a, const __grid_constant__ CUtensorMap tk,
                              const __grid_constant__ CUtensorMap tv) {
    constexpr int kTaWarps = W, kTaThreads = TaCfg<W>::kThreads, kTaC = TaCfg<W>::kC;
    constexpr int NH = D / 64;                        // 64-column boxes per row
    constexpr uint32_t kBox = kTaC * 128;
    constexpr uint32_t kStage = 2 * NH * kBox;        // K boxes, then V boxes
    constexpr int NT = D / 16;                        // 16-dim tiles
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kTaStages], empty[kTaStages];
    uint8_t *ring = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float *qs = (float *)(ring + kTaStages * kStage);  // [8][D] rotated, scaled queries (heads >= G zero)
    float *po = qs + 8 * D;                            // [G][D] this rank's unnormalised output
    float *pm = po + 8 * D;                            // [8]
    float *pl = pm + 8;                                // [8]
    // after the key loop the ring holds the warps' states
    float *wo = (float *)ring;                         // [warp][8][D]
    float *wm = wo + kTaWarps * 8 * D;                 // [warp][8]
    float *wl = wm + kTaWarps * 8;                     // [warp][8]

    const int r = blockIdx.x, g = blockIdx.y, CS = a.cs;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int half = D / 2, H = a.Hq + 2 * a.Hkv, G = a.Hq / a.Hkv;
    const long lim = wait_bound(a.wait_polls, kAttnWaitLimit);
    pdl_trigger();
    const int b = a.lpt ? lpt_sequence(a, blockIdx.z) : blockIdx.z;

    const int n = clamp_n(a.n_new, b, a.max_new, a.err);
    const int L = a.kv_len[b];
    const int qp = query_pos(a.prefill, L, n, a.step);
    int P = qp + 1;
    if (P > a.max_ctx) P = a.max_ctx;
    if (P < 1) P = 1;
    const int j0 = (int)((long)r * P / CS), j1 = (int)((long)(r + 1) * P / CS);
    const int nst = (j1 - j0 + kTaC - 1) / kTaC;
    const int L_old = L < P ? (L > 0 ? L : 0) : P;
    const uint32_t ring_s = sa(ring);

    // stage i -> ring slot i % kTaStages: NH boxes of K and NH of V from row
    // j0 + i * kTaC of head (b, g); rows past max_ctx arrive as zeros
    auto load = [&](int i) {
        const int s = i % kTaStages, j = j0 + i * kTaC, z = b * a.Hkv + g;
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sa(&full[s])), "r"(kStage)
                     : "memory");
        const uint32_t kd = ring_s + (uint32_t)s * kStage, vd = kd + NH * kBox;
#pragma unroll
        for (int h = 0; h < NH; ++h)
#pragma unroll
            for (int q = 0; q < kTaC / kTaBoxRows; ++q) {
                const uint32_t o = h * kBox + q * kTaBoxRows * 128;
                asm volatile(
                    "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
                    "%3, %4}], [%5];" ::"r"(kd + o), "l"((uint64_t)&tk), "r"(h * 64), "r"(j + q * kTaBoxRows), "r"(z),
                    "r"(sa(&full[s]))
                    : "memory");
                asm volatile(
                    "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
                    "%3, %4}], [%5];" ::"r"(vd + o), "l"((uint64_t)&tv), "r"(h * 64), "r"(j + q * kTaBoxRows), "r"(z),
                    "r"(sa(&full[s]))
                    : "memory");
            }
    };
    const bool producer = tid == kTaWarps * 32;
    if (producer) {
        for (int s = 0; s < kTaStages; ++s) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(sa(&full[s])));
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(sa(&empty[s])), "r"(kTaWarps));
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tk) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tv) : "memory");
    }
    __syncthreads();
    // stages made only of committed rows do not wait for the QKV projection
    int pre = 0;
    while (pre < kTaStages && pre < nst && min(j0 + (pre + 1) * kTaC, j1) <= L_old) ++pre;
    if (producer)
        for (int i = 0; i < pre; ++i) load(i);
    pdl_wait();

    // append the new rows this rank owns
    const int first_new = a.prefill ? L : qp, n_rows = a.prefill ? n : 1;
    for (int i = 0; i < n_rows; ++i) {
        const int pos = first_new + i;
        if (pos < 0 || pos >= a.max_ctx) {
            if (r == 0 && tid == 0) set_err(a.err, kErrCache);
            continue;
        }
        if (pos < j0 || pos >= j1) continue;
        const int row = a.prefill ? b * a.max_new + i : b;
        const float *xk = a.qkv + (size_t)row * H * D + (size_t)(a.Hq + g) * D;
        const float *xv = a.qkv + (size_t)row * H * D + (size_t)(a.Hq + a.Hkv + g) * D;
        uint16_t *kc = (uint16_t *)a.k_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        uint16_t *vc = (uint16_t *)a.v_cache + (((size_t)b * a.Hkv + g) * a.max_ctx + pos) * D;
        for (int j = tid; j < half; j += kTaThreads) {
            const float c = a.rope_cos[(size_t)pos * half + j], sn = a.rope_sin[(size_t)pos * half + j];
            const float x0 = xk[j], x1 = xk[j + half];
            kc[j] = f32_to_bf16(x0 * c - x1 * sn);
            kc[j + half] = f32_to_bf16(x1 * c + x0 * sn);
        }
        for (int j = tid; j < D; j += kTaThreads) vc[j] = f32_to_bf16(xv[j]);
    }
    // queries (heads >= G zero), rotated and scaled by 1/sqrt(D)
    {
        const int row = a.prefill ? b * a.max_new + n - 1 : b;
        const int pc = qp >= 0 && qp < a.max_ctx ? qp : 0;
        // 1/sqrt(D), times log2(e): the scores come out in log2 units
        const float scale = 1.4426950408889634f / sqrtf((float)D);
        for (int e = tid; e < 8 * half; e += kTaThreads) {
            const int h = e / half, j = e % half;
            float y0 = 0.f, y1 = 0.f;
            if (h < G) {
                const float *xq = a.qkv + (size_t)row * H * D + (size_t)(g * G + h) * D;
                const float c = a.rope_cos[(size_t)pc * half + j], sn = a.rope_sin[(size_t)pc * half + j];
                const float x0 = xq[j], x1 = xq[j + half];
                y0 = (x0 * c - x1 * sn) * scale;
                y1 = (x1 * c + x0 * sn) * scale;
            }
            qs[h * D + j] = y0;
            qs[h * D + j + half] = y1;
        }
    }
    // the async proxy reads rows this kernel just wrote: order those writes first
    asm volatile("fence.proxy.async.global;" ::: "memory");
    __syncthreads();

    bool dead = false;
    TaWarpState<NT> st;
    st.reset();
    if (warp == kTaWarps) {
        // ---------------------------------------------------------------- producer
        if (producer) {
            int issued = pre;
            for (int i = pre; i < nst && !dead; ++i) {
                if (i >= kTaStages) {
                    // slot i % S is free once every warp has released stage i - S
                    bool ok = false;
                    const uint32_t par = (uint32_t)((i / kTaStages - 1) & 1);
                    for (long it = 0; it < lim && !ok; ++it) ok = fa_try(&empty[i % kTaStages], par);
                    if (!ok) {
                        set_err(a.err, kErrTimeout);
                        dead = true;
                        break;
                    }
                }
                load(i);
                issued = i + 1;
            }
            if (!dead) prefetch_l2_share(a.pf_next, a.pf_next_bytes, r + CS * (g + a.Hkv * b), CS * a.Hkv * a.B);
            // every copy issued lands before the ring is reused or the CTA exits
            for (int i = issued > kTaStages ? issued - kTaStages : 0; i < issued; ++i) {
                bool ok = false;
                for (long it = 0; it < kAttnWaitLimit && !ok; ++it)
                    ok = fa_try(&full[i % kTaStages], (uint32_t)((i / kTaStages) & 1));
                if (!ok) set_err(a.err, kErrTimeout);
            }
        }
    } else {
        // ---------------------------------------------------------------- compute warps
        uint32_t qh[NT][2], ql[NT][2];
        ta_q_frags<NT>(qs, qh, ql);
        const int kr = 16 * warp;                     // this warp's first row in a stage
        for (int i = 0; i < nst; ++i) {
            const int s = i % kTaStages;
            if (!dead && !ta_wait_warp(&full[s], (uint32_t)((i / kTaStages) & 1), lim)) {
                if (lane == 0) set_err(a.err, kErrTimeout);
                dead = true;
            }
            const int key0 = j0 + i * kTaC + kr;     // position of the warp's first key
            const int cnt = min(16, j1 - key0);       // valid keys of the warp (may be <= 0)
            if (!dead && cnt > 0) {
                const uint32_t kb = ring_s + (uint32_t)s * kStage;
                ta_stage<NT, kTaC>(st, kb, kb + NH * kBox, kr, cnt, qh, ql);
            }
            __syncwarp();
            // a warp that gave up on this stage does not release it (its copy may
            // still be in flight); the producer's wait for the slot then gives up
            if (lane == 0 && !dead)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(sa(&empty[s])) : "memory");
        }
        // the warp's sums over its lanes' keys
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            st.l0 += __shfl_xor_sync(0xFFFFFFFFu, st.l0, off);
            st.l1 += __shfl_xor_sync(0xFFFFFFFFu, st.l1, off);
        }
    }
    __syncthreads();                                  // every copy landed, every warp done with the ring
    if (warp < kTaWarps) {
        const int h0 = 2 * (lane & 3), d0 = lane >> 2;
        if (lane < 4) {
            wm[warp * 8 + h0] = st.m0;
            wm[warp * 8 + h0 + 1] = st.m1;
            wl[warp * 8 + h0] = st.l0;
            wl[warp * 8 + h0 + 1] = st.l1;
        }
        float *w0 = wo + (size_t)(warp * 8 + h0) * D, *w1 = w0 + D;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            w0[16 * t + d0] = st.o[t][0];
            w1[16 * t + d0] = st.o[t][1];
            w0[16 * t + d0 + 8] = st.o[t][2];
            w1[16 * t + d0 + 8] = st.o[t][3];
        }
    }
    __syncthreads();
    // this rank's partial: the warps' states merged in warp order
    for (int e = tid; e < G * D; e += kTaThreads) {
        const int h = e / D, d = e % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kTaWarps; ++w) M = fmaxf(M, wm[w * 8 + h]);
        float num = 0.f, den = 0.f;
#pragma unroll
        for (int w = 0; w < kTaWarps; ++w) {
            const float mw = wm[w * 8 + h];
            const float f = mw == -INFINITY ? 0.f : exp2f(mw - M);
            den = fmaf(f, wl[w * 8 + h], den);
            num = fmaf(f, wo[(size_t)(w * 8 + h) * D + d], num);
        }
        po[h * D + d] = num;
        if (d == 0) {
            pm[h] = M;
            pl[h] = den;
        }
    }
    cluster_sync_all();
    // rank r combines its slice of the (head, dim) outputs from every rank, in rank order
    {
        const int n_out = G * D;
        const int e0 = (int)((long)r * n_out / CS), e1 = (int)((long)(r + 1) * n_out / CS);
        for (int e = e0 + tid; e < e1; e += kTaThreads) {
            const int h = e / D;
            float mq[kMaxCluster], lq[kMaxCluster], oq[kMaxCluster];
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) {
                if (q < CS) {
                    mq[q] = dsmem_ld(pm + h, (uint32_t)q);
                    lq[q] = dsmem_ld(pl + h, (uint32_t)q);
                    oq[q] = dsmem_ld(po + e, (uint32_t)q);
                } else {
                    mq[q] = -INFINITY;
                    lq[q] = oq[q] = 0.f;
                }
            }
            float M = -INFINITY;
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) M = fmaxf(M, mq[q]);
            float num = 0.f, den = 0.f;
#pragma unroll
            for (int q = 0; q < kMaxCluster; ++q) {
                const float w = mq[q] == -INFINITY ? 0.f : exp2f(mq[q] - M);
                den = fmaf(w, lq[q], den);
                num = fmaf(w, oq[q], num);
            }
            uint16_t *out = (uint16_t *)a.o_out + (size_t)b * a.Hq * D + (size_t)g * G * D;
            out[e] = f32_to_bf16(den > 0.f ? num / den : 0.f);
        }
    }
    cluster_sync_all();
}

template <int D, int W>
constexpr size_t fused_tc_smem() {
    return 1024 + (size_t)kTaStages * 2 * (D / 64) * TaCfg<W>::kC * 128 + (size_t)2 * 8 * D * 4 + 16 * 4;
}
static_assert((size_t)8 * 8 * 128 * 4 + 2 * 8 * 8 * 4 <= (size_t)kTaStages * 2 * 2 * TaCfg<8>::kC * 128 &&
                  (size_t)4 * 8 * 128 * 4 + 2 * 4 * 8 * 4 <= (size_t)kTaStages * 2 * 2 * TaCfg<4>::kC * 128,
              "the warps' states fit in the ring");
static_assert(2 * (fused_tc_smem<128, 4>() + 1024 + 64 + (kLptMaxB + 1) * 4) <= (size_t)228 * 1024,
              "two 4-warp CTAs per SM");

template <typename WT, int D>
size_t fused_smem(int G) {
    using Cf = FusedCfg<WT, D>;
    return (size_t)4 * Cf::C * D * sizeof(WT) + (size_t)G * D * 4 * 2 + (size_t)G * Cf::C * 4 + 32 * 4;
}
static_assert(kFusedThreads % 128 == 0, "score pass maps threads to (key, head group)");

template <typename Kern, typename... Args>
cudaError_t launch_cluster(Kern k, size_t smem, int threads, const FusedAttnArgs &a, cudaStream_t s, bool pdl,
                           Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.cs, a.Hkv, a.B);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = a.cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, k, args...);
}

template <typename WT, int D>
cudaError_t launch_fused_t(const FusedAttnArgs &a, cudaStream_t s, bool pdl, const CUtensorMap *tk,
                           const CUtensorMap *tv) {
    if constexpr (sizeof(WT) == 2) {
        if (tk && tv && a.Hq / a.Hkv <= 8) {
            if (a.warps == 4)
                return launch_cluster(fused_attention_tc_kernel<D, 4>, fused_tc_smem<D, 4>(), TaCfg<4>::kThreads, a, s,
                                      pdl, a, *tk, *tv);
            return launch_cluster(fused_attention_tc_kernel<D, 8>, fused_tc_smem<D, 8>(), TaCfg<8>::kThreads, a, s,
                                  pdl, a, *tk, *tv);
        }
    }
    return launch_cluster(fused_attention_kernel<WT, D>, fused_smem<WT, D>(a.Hq / a.Hkv), kFusedThreads, a, s, pdl, a);
}

// Clusters of 16 are a non-portable size: allowed only where the occupancy
// query confirms that `need` of them can be resident at once.
template <typename Kern>
int max_cluster_for(Kern k, size_t smem, int threads, int need) {
    if (cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        return 8;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(16, 1, 1);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 16;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 8;
    }
    return n >= need ? 16 : 8;
}

template <typename WT, int D>
cudaError_t prepare_fused_t(int G, int need, int *max_cs) {
    // the CUDA-core kernel serves every cache type (and bf16 caches without
    // tensor maps); the tensor-core kernel bf16 caches with G <= 8
    if (G > 16 || fused_smem<WT, D>(G) > (size_t)200 * 1024) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(fused_attention_kernel<WT, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         200 * 1024);
    if (e == cudaSuccess && max_cs)
        *max_cs = max_cluster_for(fused_attention_kernel<WT, D>, fused_smem<WT, D>(G), kFusedThreads, need);
    if constexpr (sizeof(WT) == 2) {
        if (e == cudaSuccess && G <= 8) {
            static_assert(fused_tc_smem<D, 8>() <= (size_t)227 * 1024, "tensor-core attention shared memory");
            e = cudaFuncSetAttribute(fused_attention_tc_kernel<D, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)fused_tc_smem<D, 8>());
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(fused_attention_tc_kernel<D, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)fused_tc_smem<D, 4>());
            if (e == cudaSuccess && max_cs)
                *max_cs = max_cluster_for(fused_attention_tc_kernel<D, 8>, fused_tc_smem<D, 8>(), TaCfg<8>::kThreads,
                                          need);
        }
    }
    return e;
}

template <typename WT, int D>
size_t attn_smem(int chunk, int G, int splits) {
    constexpr int RS = D + Elem<WT>::kPerVec;
    return (size_t)2 * chunk * RS * sizeof(WT) + (size_t)G * D * 4 + (size_t)G * chunk * 4 + (size_t)G * splits * 4;
}

template <typename WT, int D>
cudaError_t launch_attn_t(const AttnArgs &a, cudaStream_t s, bool pdl) {
    const size_t smem = attn_smem<WT, D>(a.chunk, a.Hq / a.Hkv, a.splits);
    return launch_k(attention_kernel<WT, D>, dim3(a.splits, a.Hkv, a.B), dim3(kAttnThreads), smem, s, pdl, a);
}

// The attribute is a per-function ceiling shared by every context, so it is
// set to the cap that prism_create validates against, never lowered.
constexpr int kAttnSmemCap = 200 * 1024;
template <typename WT, int D>
cudaError_t prepare_attn_t(int chunk, int G, int splits) {
    if (attn_smem<WT, D>(chunk, G, splits) > (size_t)kAttnSmemCap) return cudaErrorInvalidValue;
    return cudaFuncSetAttribute(attention_kernel<WT, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmemCap);
}

}  // namespace

cudaError_t launch_rope_append(const RopeArgs &a, bool bf16, cudaStream_t s, bool pdl) {
    const int warps = a.rows * (a.Hq + 2 * a.Hkv);
    const int grid = (warps + 3) / 4;
    if (bf16) return launch_k(rope_append_kernel<uint16_t>, dim3(grid), dim3(128), 0, s, pdl, a);
    return launch_k(rope_append_kernel<float>, dim3(grid), dim3(128), 0, s, pdl, a);
}

cudaError_t launch_attention(const AttnArgs &a, bool bf16, cudaStream_t s, bool pdl) {
    if (bf16) return a.D == 64 ? launch_attn_t<uint16_t, 64>(a, s, pdl) : launch_attn_t<uint16_t, 128>(a, s, pdl);
    return a.D == 64 ? launch_attn_t<float, 64>(a, s, pdl) : launch_attn_t<float, 128>(a, s, pdl);
}

cudaError_t prepare_attention_kernel(bool bf16, int D, int chunk, int G, int splits) {
    if (bf16) return D == 64 ? prepare_attn_t<uint16_t, 64>(chunk, G, splits) : prepare_attn_t<uint16_t, 128>(chunk, G, splits);
    return D == 64 ? prepare_attn_t<float, 64>(chunk, G, splits) : prepare_attn_t<float, 128>(chunk, G, splits);
}

size_t attention_smem_bytes(bool bf16, int D, int chunk, int G, int splits) {
    if (bf16) return D == 64 ? attn_smem<uint16_t, 64>(chunk, G, splits) : attn_smem<uint16_t, 128>(chunk, G, splits);
    return D == 64 ? attn_smem<float, 64>(chunk, G, splits) : attn_smem<float, 128>(chunk, G, splits);
}

int fused_attention_chunk() { return kTaBoxRows; }

cudaError_t launch_fused_attention(const FusedAttnArgs &a, bool bf16, cudaStream_t s, bool pdl,
                                   const CUtensorMap *tk, const CUtensorMap *tv) {
    if (a.cs < 1 || a.cs > kMaxCluster || a.Hq / a.Hkv > 16) return cudaErrorInvalidValue;
    if (bf16)
        return a.D == 64 ? launch_fused_t<uint16_t, 64>(a, s, pdl, tk, tv)
                         : launch_fused_t<uint16_t, 128>(a, s, pdl, tk, tv);
    return a.D == 64 ? launch_fused_t<float, 64>(a, s, pdl, nullptr, nullptr)
                     : launch_fused_t<float, 128>(a, s, pdl, nullptr, nullptr);
}

cudaError_t prepare_fused_attention(bool bf16, int D, int G, int need, int *max_cs) {
    if (bf16) return D == 64 ? prepare_fused_t<uint16_t, 64>(G, need, max_cs) : prepare_fused_t<uint16_t, 128>(G, need, max_cs);
    return D == 64 ? prepare_fused_t<float, 64>(G, need, max_cs) : prepare_fused_t<float, 128>(G, need, max_cs);
}

size_t fused_attention_smem_bytes(bool bf16, int D, int G) {
    if (bf16 && G <= 8) return D == 64 ? fused_tc_smem<64, 8>() : fused_tc_smem<128, 8>();
    if (bf16) return D == 64 ? fused_smem<uint16_t, 64>(G) : fused_smem<uint16_t, 128>(G);
    return D == 64 ? fused_smem<float, 64>(G) : fused_smem<float, 128>(G);
}

cudaError_t launch_accept(const AcceptArgs &a, cudaStream_t s) {
    accept_kernel<<<(a.B + 127) / 128, 128, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace prism
