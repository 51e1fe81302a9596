// Weight-streaming projections of the PRISM draft step (sm_103a).
//
// Every projection of a draft step (fusion F, QKV, O, gate/up, down, LM head;
// Sec. 3.2 and the Llama block) is y[t] = W x[t] for a handful of activation
// rows t, so the kernel is bound by reading W once from HBM.  Design:
//   * persistent grid (2 CTAs of 16 warps per SM); CTA c owns a contiguous,
//     balanced range of output units; its warps take units round-robin;
//   * one warp computes whole rows: each lane streams 16-byte vectors of the
//     weight row (ld.global.nc, no L1 allocation, U vectors in flight) and
//     multiplies them with the activation rows staged in shared memory; a
//     butterfly shuffle finishes each dot product (no atomics: deterministic);
//   * the activation rows are built in the prologue (embedding gather +
//     concatenation, RMSNorm with its gain, bf16 rounding) from the previous
//     kernel's fp32 output, so no separate norm/concat kernels run;
//   * the epilogue fuses the residual add, SwiGLU, or (LM head) the logits
//     write and a top-8 selection whose per-CTA partials are merged by the
//     last CTA to finish (a two-pass vocabulary argmax without a second launch);
//   * programmatic dependent launch: before griddepcontrol.wait each CTA asks
//     the TMA engine to prefetch the start of its weight range into L2, so the
//     weight stream overlaps the previous kernel's tail.
#include "common.cuh"

namespace prism {

namespace {

constexpr int kPrefetchBytes = 64 * 1024;
constexpr int kPrefetchPiece = 16 * 1024;

template <typename WT>
__device__ __forceinline__ void fma_vec(float &acc, const uint4 &w, const uint4 &x);

template <>
__device__ __forceinline__ void fma_vec<uint16_t>(float &acc, const uint4 &w, const uint4 &x) {
    acc = fmaf(bf16lo(w.x), bf16lo(x.x), acc);
    acc = fmaf(bf16hi(w.x), bf16hi(x.x), acc);
    acc = fmaf(bf16lo(w.y), bf16lo(x.y), acc);
    acc = fmaf(bf16hi(w.y), bf16hi(x.y), acc);
    acc = fmaf(bf16lo(w.z), bf16lo(x.z), acc);
    acc = fmaf(bf16hi(w.z), bf16hi(x.z), acc);
    acc = fmaf(bf16lo(w.w), bf16lo(x.w), acc);
    acc = fmaf(bf16hi(w.w), bf16hi(x.w), acc);
}

template <>
__device__ __forceinline__ void fma_vec<float>(float &acc, const uint4 &w, const uint4 &x) {
    acc = fmaf(__uint_as_float(w.x), __uint_as_float(x.x), acc);
    acc = fmaf(__uint_as_float(w.y), __uint_as_float(x.y), acc);
    acc = fmaf(__uint_as_float(w.z), __uint_as_float(x.z), acc);
    acc = fmaf(__uint_as_float(w.w), __uint_as_float(x.w), acc);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

// Deterministic block-wide sum (same tree in every CTA).
__device__ float block_sum(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float s = 0.f;
    if (threadIdx.x == 0) {
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
        red[32] = s;
    }
    __syncthreads();
    return red[32];
}

__device__ __forceinline__ int clamp_nnew(const GemvArgs &a, int b) {
    int n = a.n_new[b];
    if (n < 1 || n > a.max_new) {
        set_err(a.err, kErrNNew);
        n = n < 1 ? 1 : a.max_new;
    }
    return n;
}

__device__ __forceinline__ int checked_token(const GemvArgs &a, int tok) {
    if (tok < 0 || tok >= a.vocab) {
        set_err(a.err, kErrToken);
        return 0;
    }
    return tok;
}

// Build activation rows [t0, t0 + tc) in shared memory X ([TC][kin] WT);
// rows tc..TC-1 are zeroed.
template <typename WT, int TC>
__device__ void stage_x(const GemvArgs &a, int t0, int tc, WT *X, float *red) {
    const int NT = blockDim.x, tid = threadIdx.x;
    const int kin = a.kin, d = a.d;
    const WT *E = (const WT *)a.embed;
    for (int t = 0; t < TC; ++t) {
        WT *xr = X + (size_t)t * kin;
        if (t >= tc) {
            for (int c = tid; c < kin; c += NT) xr[c] = (WT)0;
            continue;
        }
        const int row = t0 + t;
        if (a.pro == kProFusePrefill) {
            const int b = row / a.max_new, i = row % a.max_new;
            const int n = clamp_nnew(a, b);
            const bool valid = i < n;
            const int tok = valid ? checked_token(a, a.tokens[b * a.max_new + i]) : 0;
            const WT *hid = (const WT *)a.hidden_in + ((size_t)b * a.max_new + i) * d;
            const WT *er = E + (size_t)tok * d;
            for (int c = tid; c < d; c += NT) {
                xr[c] = valid ? er[c] : (WT)0;
                xr[d + c] = valid ? hid[c] : (WT)0;
            }
        } else if (a.pro == kProFuseDecode) {
            const int b = row;
            const int tok = checked_token(a, a.draft[b * a.K + a.step - 2]);
            const WT *er = E + (size_t)tok * d;
            const float *h = a.src + (size_t)b * d;
            for (int c = tid; c < d; c += NT) {
                xr[c] = er[c];
                float v = Elem<WT>::round(h[c]);
                if constexpr (sizeof(WT) == 2) xr[d + c] = f32_to_bf16(v); else xr[d + c] = v;
            }
        } else if (a.pro == kProNorm) {
            const int sr = a.src_prefill_rows ? (row * a.max_new + clamp_nnew(a, row) - 1) : row;
            const float *s = a.src + (size_t)sr * d;
            float inv = 1.f;
            if (a.gain) {
                float ss = 0.f;
                for (int c = tid; c < d; c += NT) ss = fmaf(s[c], s[c], ss);
                ss = block_sum(ss, red);
                inv = 1.0f / sqrtf(ss / (float)d + a.eps);
            }
            const WT *g = (const WT *)a.gain;
            for (int c = tid; c < d; c += NT) {
                float v = a.gain ? s[c] * inv * Elem<WT>::load(g, c) : s[c];
                v = Elem<WT>::round(v);
                if constexpr (sizeof(WT) == 2) xr[c] = f32_to_bf16(v); else xr[c] = v;
            }
        } else {  // kProCopy
            const WT *src = (const WT *)a.act + (size_t)row * kin;
            for (int c = tid; c < kin; c += NT) xr[c] = src[c];
        }
    }
}

// Warp-level merge of per-lane top-8 lists; lane 0 ends with the merged list.
__device__ void warp_merge_top8(float (&v)[kTopK], int (&id)[kTopK]) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        float pv[kTopK];
        int pi[kTopK];
#pragma unroll
        for (int i = 0; i < kTopK; ++i) {
            pv[i] = __shfl_down_sync(0xFFFFFFFFu, v[i], o);
            pi[i] = __shfl_down_sync(0xFFFFFFFFu, id[i], o);
        }
        if ((threadIdx.x & 31) < o) {
#pragma unroll
            for (int i = 0; i < kTopK; ++i) top8_insert(v, id, pv[i], pi[i]);
        }
    }
}

template <typename WT, int TC, int RPW, bool TOPK>
__global__ void __launch_bounds__(kGemvThreads, 2) gemv_kernel(const GemvArgs a) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ float red[33];
    __shared__ float s_val[TOPK ? kGemvWarps : 1][TOPK ? TC : 1][kTopK];
    __shared__ int s_id[TOPK ? kGemvWarps : 1][TOPK ? TC : 1][kTopK];
    __shared__ int s_last;

    constexpr int VEC = Elem<WT>::kPerVec;
    constexpr int U0 = TC == 1 ? 8 : (TC == 4 ? 4 : 2);
    constexpr int U = U0 / RPW > 0 ? U0 / RPW : 1;
    WT *X = (WT *)smem_raw;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int u_begin = (int)((long long)blockIdx.x * a.n_units / gridDim.x);
    const int u_end = (int)((long long)(blockIdx.x + 1) * a.n_units / gridDim.x);
    const size_t row_bytes = (size_t)a.kin * sizeof(WT);

    pdl_trigger();
    if (threadIdx.x == 0 && u_end > u_begin) {
        // prefetch the start of this CTA's weight range (RPW ranges)
        for (int r = 0; r < RPW; ++r) {
            const uint8_t *base = (const uint8_t *)a.W + ((size_t)u_begin + (size_t)r * a.pair_offset) * row_bytes;
            size_t total = (size_t)(u_end - u_begin) * row_bytes;
            size_t lim = total < (size_t)(kPrefetchBytes / RPW) ? total : (size_t)(kPrefetchBytes / RPW);
            for (size_t off = 0; off < lim; off += kPrefetchPiece) {
                size_t n = lim - off < (size_t)kPrefetchPiece ? lim - off : (size_t)kPrefetchPiece;
                prefetch_l2_bulk(base + off, (uint32_t)(n & ~(size_t)15));
            }
        }
    }
    pdl_wait();

    const int nvec = a.kin / VEC;
    const uint4 *X4 = (const uint4 *)X;

    for (int t0 = 0; t0 < a.T; t0 += TC) {
        const int tc = a.T - t0 < TC ? a.T - t0 : TC;
        stage_x<WT, TC>(a, t0, tc, X, red);
        __syncthreads();

        // LM head: lane t keeps the top-8 list of activation row t0 + t in
        // shared memory (s_val/s_id[warp][t]) and only its current 8th-best
        // entry in registers; a logit that beats it is inserted (rare).
        float thr_v = -INFINITY;
        int thr_i = 0x7FFFFFFF;
        if constexpr (TOPK) {
            if (lane < TC) {
#pragma unroll
                for (int i = 0; i < kTopK; ++i) { s_val[warp][lane][i] = -INFINITY; s_id[warp][lane][i] = 0x7FFFFFFF; }
            }
        }

        for (int u = u_begin + warp; u < u_end; u += kGemvWarps) {
            const uint4 *wr[RPW];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
                wr[r] = (const uint4 *)((const uint8_t *)a.W + ((size_t)u + (size_t)r * a.pair_offset) * row_bytes);
            float acc[RPW][TC];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int t = 0; t < TC; ++t) acc[r][t] = 0.f;

            for (int v0 = lane; v0 < nvec; v0 += 32 * U) {
                uint4 wv[RPW][U];
#pragma unroll
                for (int j = 0; j < U; ++j) {
                    const int v = v0 + 32 * j;
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
                        wv[r][j] = v < nvec ? ldg_stream(wr[r] + v) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int j = 0; j < U; ++j) {
                    const int v = v0 + 32 * j;
                    if (v < nvec) {
#pragma unroll
                        for (int t = 0; t < TC; ++t) {
                            const uint4 xv = X4[(size_t)t * nvec + v];
#pragma unroll
                            for (int r = 0; r < RPW; ++r) fma_vec<WT>(acc[r][t], wv[r][j], xv);
                        }
                    }
                }
            }
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int t = 0; t < TC; ++t) acc[r][t] = warp_sum(acc[r][t]);

            // epilogue: lane t handles activation row t0 + t
#pragma unroll
            for (int t = 0; t < TC; ++t) {
                if (lane != t || t >= tc) continue;
                const int row = t0 + t;
                if constexpr (TOPK) {
                    const float z = acc[0][t];
                    if (a.logits) a.logits[((size_t)row * a.K + a.step - 1) * a.vocab + u] = z;
                    if (better(z, u, thr_v, thr_i)) {
                        float *lv = s_val[warp][t];
                        int *li = s_id[warp][t];
                        int pos = kTopK - 1;
                        while (pos > 0 && better(z, u, lv[pos - 1], li[pos - 1])) {
                            lv[pos] = lv[pos - 1];
                            li[pos] = li[pos - 1];
                            --pos;
                        }
                        lv[pos] = z;
                        li[pos] = u;
                        thr_v = lv[kTopK - 1];
                        thr_i = li[kTopK - 1];
                    }
                } else if constexpr (RPW == 2) {
                    const float g = acc[0][t], up = acc[1][t];
                    const float m = g / (1.0f + expf(-g)) * up;
                    Elem<WT>::store((WT *)a.out_act, (size_t)row * a.out_ld + u, m);
                } else {
                    float val = acc[0][t];
                    if (a.epi == kEpiResid) {
                        const int rr = a.resid_prefill_rows ? (row * a.max_new + clamp_nnew(a, row) - 1) : row;
                        val += a.resid[(size_t)rr * a.out_ld + u];
                        if (a.hidden_out) a.hidden_out[((size_t)row * a.K + a.step - 1) * a.d + u] = val;
                    }
                    a.out[(size_t)row * a.out_ld + u] = val;
                }
            }
        }

        if constexpr (TOPK) {
            // per-CTA merge of the warps' lists, one warp per activation row
            __syncthreads();
            for (int t = warp; t < tc; t += kGemvWarps) {
                float v[kTopK];
                int id[kTopK];
                top8_init(v, id);
                for (int c = lane; c < kGemvWarps * kTopK; c += 32)
                    top8_insert(v, id, s_val[c / kTopK][t][c % kTopK], s_id[c / kTopK][t][c % kTopK]);
                warp_merge_top8(v, id);
                if (lane == 0) {
                    const size_t base = (((size_t)(t0 + t)) * gridDim.x + blockIdx.x) * kTopK;
#pragma unroll
                    for (int i = 0; i < kTopK; ++i) { a.lm_part[base + i] = v[i]; a.lm_part_id[base + i] = id[i]; }
                }
            }
        }
        __syncthreads();
    }

    if constexpr (TOPK) {
        // the last CTA to finish merges every CTA's partial lists
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) s_last = (atomicAdd(a.counter, 1) == (int)gridDim.x - 1);
        __syncthreads();
        if (!s_last) return;
        __threadfence();
        const int G = gridDim.x;
        for (int t = warp; t < a.T; t += kGemvWarps) {
            float v[kTopK];
            int id[kTopK];
            top8_init(v, id);
            const size_t base = (size_t)t * G * kTopK;
            for (int c = lane; c < G * kTopK; c += 32)
                top8_insert(v, id, __ldcg(a.lm_part + base + c), __ldcg(a.lm_part_id + base + c));
            warp_merge_top8(v, id);
            if (lane == 0) {
                const size_t o = (size_t)t * a.K + a.step - 1;
                a.draft_out[o] = id[0];
#pragma unroll
                for (int i = 0; i < kTopK; ++i) {
                    if (i < a.topk) {
                        if (a.topk_ids) a.topk_ids[o * a.topk + i] = id[i];
                        if (a.topk_logits) a.topk_logits[o * a.topk + i] = v[i];
                    }
                }
            }
        }
        if (threadIdx.x == 0) *a.counter = 0;
    }
}

template <typename WT, int TC>
cudaError_t dispatch_kind(const GemvArgs &a, int grid, size_t smem, cudaStream_t s, bool pdl) {
    if (a.epi == kEpiTopK)
        return launch_k(gemv_kernel<WT, TC, 1, true>, dim3(grid), dim3(kGemvThreads), smem, s, pdl, a);
    if (a.epi == kEpiSwiGLU)
        return launch_k(gemv_kernel<WT, TC, 2, false>, dim3(grid), dim3(kGemvThreads), smem, s, pdl, a);
    return launch_k(gemv_kernel<WT, TC, 1, false>, dim3(grid), dim3(kGemvThreads), smem, s, pdl, a);
}

template <typename WT>
cudaError_t set_smem_attrs(int bytes) {
    cudaError_t e = cudaSuccess;
#define PRISM_SET(TC, RPW, TK)                                                                   \
    if (e == cudaSuccess)                                                                        \
        e = cudaFuncSetAttribute(gemv_kernel<WT, TC, RPW, TK>,                                   \
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    PRISM_SET(1, 1, true) PRISM_SET(1, 2, false) PRISM_SET(1, 1, false)
    PRISM_SET(4, 1, true) PRISM_SET(4, 2, false) PRISM_SET(4, 1, false)
    PRISM_SET(8, 1, true) PRISM_SET(8, 2, false) PRISM_SET(8, 1, false)
#undef PRISM_SET
    return e;
}

}  // namespace

// Shared-memory budget of the activation rows per CTA (two CTAs per SM).
constexpr size_t kXBudget = 100 * 1024;

int gemv_rows_per_pass(const GemvArgs &a, bool bf16) {
    const size_t row = (size_t)a.kin * (bf16 ? 2 : 4);
    int tc = a.T <= 1 ? 1 : (a.T <= 4 ? 4 : 8);
    while (tc > 1 && (size_t)tc * row > kXBudget) tc = tc == 8 ? 4 : 1;
    return tc;
}

size_t gemv_smem_bytes(const GemvArgs &a, bool bf16, int tc) {
    return (size_t)tc * a.kin * (bf16 ? 2 : 4);
}

cudaError_t prepare_gemv_kernels() {
    cudaError_t e = set_smem_attrs<uint16_t>((int)kXBudget);
    if (e == cudaSuccess) e = set_smem_attrs<float>((int)kXBudget);
    return e;
}

cudaError_t launch_gemv(const GemvArgs &a, bool bf16, int grid, cudaStream_t s, bool pdl) {
    const int tc = gemv_rows_per_pass(a, bf16);
    const size_t smem = gemv_smem_bytes(a, bf16, tc);
    if (bf16) {
        if (tc == 1) return dispatch_kind<uint16_t, 1>(a, grid, smem, s, pdl);
        if (tc == 4) return dispatch_kind<uint16_t, 4>(a, grid, smem, s, pdl);
        return dispatch_kind<uint16_t, 8>(a, grid, smem, s, pdl);
    }
    if (tc == 1) return dispatch_kind<float, 1>(a, grid, smem, s, pdl);
    if (tc == 4) return dispatch_kind<float, 4>(a, grid, smem, s, pdl);
    return dispatch_kind<float, 8>(a, grid, smem, s, pdl);
}

}  // namespace prism
