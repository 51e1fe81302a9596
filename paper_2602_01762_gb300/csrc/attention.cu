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

cudaError_t launch_accept(const AcceptArgs &a, cudaStream_t s) {
    accept_kernel<<<(a.B + 127) / 128, 128, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace prism
