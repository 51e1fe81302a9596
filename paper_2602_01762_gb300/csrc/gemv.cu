// Weight-streaming projections of the PRISM draft step (sm_103a).
//
// Every projection of a draft step (fusion F, QKV, O, gate/up, down, LM head;
// Sec. 3.2 and the Llama block) is y[t] = W x[t] for a handful of activation
// rows t, so the kernel is bound by reading W once from HBM.  Design:
//   * persistent grid, one CTA per SM; CTA c owns a contiguous, balanced range
//     of output rows, i.e. one contiguous byte range of W;
//   * a producer lane streams that range through a ring of shared-memory
//     stages with TMA bulk copies (cp.async.bulk, mbarrier complete_tx), each
//     stage holding R whole rows.  It starts before griddepcontrol.wait, so
//     under programmatic dependent launch the ring fills while the previous
//     kernel finishes;
//   * sixteen consumer warps form G groups; group g owns the stages s with
//     s % G == g (the stage count is a multiple of G) and takes them in
//     order, so every stage has exactly one consumer group and no waiter can
//     run two ring phases ahead of a barrier (parity waits stay
//     unambiguous); G groups work on G stages at once.  Warps compute whole
//     rows, or with fewer rows than warps per group, column segments whose
//     partial sums are added in fixed segment order after a group barrier:
//     no atomics, deterministic;
//   * the prologue builds the activation rows (embedding gather +
//     concatenation, RMSNorm with its gain, bf16 rounding) from the previous
//     kernel's fp32 output; the epilogue fuses the residual add, SwiGLU, or
//     (LM head) the logits write and a top-8 selection whose per-CTA partials
//     are merged by the last CTA to finish (two-pass vocabulary argmax without
//     a second launch);
//   * every mbarrier wait is bounded; on expiry the kernel sets the timeout bit
//     of the device error word, skips the rest of its work (still reaching
//     every named barrier), drains its copies in flight and returns.
#include "common.cuh"

namespace prism {

namespace {

constexpr int kConsumers = 16;
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kMaxStages = 16;
constexpr long kWaitLimit = 1L << 22;
constexpr size_t kChunkTarget = 32 * 1024;
constexpr size_t kSmemAlone = 200 * 1024;

__device__ __forceinline__ uint32_t saddr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(saddr(b)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive(uint64_t *b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(saddr(b)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t *b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                 : "=r"(ok) : "r"(saddr(b)), "r"(parity) : "memory");
    return ok != 0;
}
// Bounded wait for the completion of the phase with the given parity.
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity, long limit = kWaitLimit) {
    for (long i = 0; i < limit; ++i)
        if (mbar_try(b, parity)) return true;
    return false;
}
// 1-D TMA bulk copy global -> shared, completing on mbarrier b.
__device__ __forceinline__ void tma_load(void *dst, const void *src, uint32_t bytes, uint64_t *b, uint64_t pol = 0) {
    if (pol == 0) {
        asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                     ::"r"(saddr(dst)), "l"(src), "r"(bytes), "r"(saddr(b)) : "memory");
        return;
    }
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
                 ::"r"(saddr(dst)), "l"(src), "r"(bytes), "r"(saddr(b)), "l"(pol) : "memory");
}
// Barrier among the consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumers_sync() {
    asm volatile("bar.sync 1, %0;" ::"r"(kConsumers * 32) : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}
// Packed pair of fp32 lanes: acc += a * b on both halves (one FFMA2).
__device__ __forceinline__ void ffma2(unsigned long long &acc, unsigned long long a, unsigned long long b) {
    asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc) : "l"(a), "l"(b));
}
__device__ __forceinline__ unsigned long long pack2(uint32_t lo, uint32_t hi) {
    return ((unsigned long long)hi << 32) | lo;
}
__device__ __forceinline__ float sum2(unsigned long long v) {
    return __uint_as_float((uint32_t)v) + __uint_as_float((uint32_t)(v >> 32));
}
// Two packed accumulators += 8 weights times 8 activations, both given as
// one 16-byte vector of the storage type (bf16 pairs are widened exactly).
template <typename WT>
__device__ __forceinline__ void dot16B(unsigned long long &a0, unsigned long long &a1, const uint4 &w,
                                       const uint4 &x);
template <>
__device__ __forceinline__ void dot16B<uint16_t>(unsigned long long &a0, unsigned long long &a1, const uint4 &w,
                                                 const uint4 &x) {
    ffma2(a0, pack2(w.x << 16, w.x & 0xFFFF0000u), pack2(x.x << 16, x.x & 0xFFFF0000u));
    ffma2(a1, pack2(w.y << 16, w.y & 0xFFFF0000u), pack2(x.y << 16, x.y & 0xFFFF0000u));
    ffma2(a0, pack2(w.z << 16, w.z & 0xFFFF0000u), pack2(x.z << 16, x.z & 0xFFFF0000u));
    ffma2(a1, pack2(w.w << 16, w.w & 0xFFFF0000u), pack2(x.w << 16, x.w & 0xFFFF0000u));
}
template <>
__device__ __forceinline__ void dot16B<float>(unsigned long long &a0, unsigned long long &a1, const uint4 &w,
                                              const uint4 &x) {
    ffma2(a0, pack2(w.x, w.y), pack2(x.x, x.y));
    ffma2(a1, pack2(w.z, w.w), pack2(x.z, x.w));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

// Deterministic sum over the consumer threads (same tree in every CTA).
__device__ float consumers_sum(float v, float *red) {
    const int lane = threadIdx.x & 31, w = (threadIdx.x >> 5) - 1;
    v = warp_sum(v);
    consumers_sync();
    if (lane == 0) red[w] = v;
    consumers_sync();
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kConsumers; ++i) s += red[i];
    return s;
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

template <typename WT>
__device__ __forceinline__ void put(WT *x, int i, float v) {
    if constexpr (sizeof(WT) == 2) x[i] = f32_to_bf16(v); else x[i] = v;
}

// Build activation rows [t0, t0 + tc) in shared memory X ([TC][kin] in the
// weight type, rounded per the numeric contract), rows tc..TC-1 zeroed.
// Consumer threads only.
template <typename WT, int TC>
__device__ void stage_x(const GemvArgs &a, int t0, int tc, WT *X, float *red) {
    const int NT = kConsumers * 32, tid = threadIdx.x - 32;
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
                put<WT>(xr, d + c, Elem<WT>::round(h[c]));
            }
        } else if (a.pro == kProNorm) {
            const int sr = a.src_prefill_rows ? (row * a.max_new + clamp_nnew(a, row) - 1) : row;
            const float *s = a.src + (size_t)sr * d;
            float inv = 1.f;
            if (a.gain) {
                float ss = 0.f;
                for (int c = tid; c < d; c += NT) ss = fmaf(s[c], s[c], ss);
                ss = consumers_sum(ss, red);
                inv = 1.0f / sqrtf(ss / (float)d + a.eps);
            }
            const WT *g = (const WT *)a.gain;
            for (int c = tid; c < d; c += NT) {
                float v = a.gain ? s[c] * inv * Elem<WT>::load(g, c) : s[c];
                put<WT>(xr, c, Elem<WT>::round(v));
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

struct RingPlan {
    int R;          // rows (units) per stage
    int stages;     // a multiple of G
    int G;          // consumer warp groups
    size_t stage_bytes, x_bytes;
};

template <typename WT, int TC, int RPW, bool TOPK>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const GemvArgs a, const RingPlan plan) {
    extern __shared__ __align__(128) uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kMaxStages], empty[kMaxStages];
    __shared__ float red[kConsumers];
    __shared__ float s_val[TOPK ? kConsumers : 1][TOPK ? TC : 1][kTopK];
    __shared__ int s_id[TOPK ? kConsumers : 1][TOPK ? TC : 1][kTopK];
    __shared__ int s_last;
    // per-chunk partial sums of the column segments, double-buffered by chunk
    __shared__ float s_part[2][kConsumers][RPW][TC];   // column-segment partials

    constexpr int VEC = Elem<WT>::kPerVec;
    constexpr int U = TC <= 2 ? 4 : (TC == 4 ? 2 : 1);
    static_assert(sizeof(WT) == 2 || sizeof(WT) == 4, "weight type");
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int R = plan.R, S = plan.stages;
    const size_t row_bytes = (size_t)a.kin * sizeof(WT);
    const int u0 = (int)((long long)blockIdx.x * a.n_units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * a.n_units / gridDim.x);
    const int n_chunks = (u1 - u0 + R - 1) / R;
    const int n_pass = (a.T + TC - 1) / TC;
    uint8_t *ring = smem_raw;
    WT *X = (WT *)(smem_raw + (size_t)S * plan.stage_bytes);

    pdl_trigger();
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumers / plan.G);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane != 0) return;
        const int total = n_pass * n_chunks;
        const uint64_t wpol = a.w_evict_first ? l2_evict_first_policy() : 0ull;
        int issued = 0;
        int s = 0, c = 0;
        uint32_t ph = 0;                                      // phase parity of stage s
        for (int i = 0; i < total; ++i) {
            if (!mbar_wait(&empty[s], ph ^ 1, wait_bound(a.wait_polls, kWaitLimit))) {
                set_err(a.err, kErrTimeout);
                break;
            }
            const int first = u0 + c * R;
            const int rows = u1 - first < R ? u1 - first : R;
            const uint32_t bytes = (uint32_t)(rows * row_bytes);
            if (PRISM_CHECK(a.err, (size_t)s * plan.stage_bytes + (size_t)(RPW - 1) * R * row_bytes + bytes <=
                                       (size_t)S * plan.stage_bytes, 101, s, bytes) ||
                PRISM_CHECK(a.err, first + rows <= a.n_units && first >= 0, 102, first, rows) ||
                PRISM_CHECK(a.err, (((uintptr_t)a.W) & 15) == 0 && (row_bytes & 15) == 0, 103, 0, row_bytes))
                break;
            mbar_arrive_tx(&full[s], bytes * RPW);
            uint8_t *st = ring + (size_t)s * plan.stage_bytes;
#pragma unroll
            for (int r = 0; r < RPW; ++r)
                tma_load(st + (size_t)r * R * row_bytes,
                         (const uint8_t *)a.W + ((size_t)first + (size_t)r * a.pair_offset) * row_bytes, bytes,
                         &full[s], wpol);
            issued = i + 1;
            if (++c == n_chunks) c = 0;
            if (++s == S) { s = 0; ph ^= 1; }
        }
        if (issued == total) prefetch_l2_share(a.pf_next, a.pf_next_bytes, blockIdx.x, gridDim.x);
        // drain: the last stages' copies land before this CTA may exit
        for (int i = issued > S ? issued - S : 0; i < issued; ++i)
            if (!mbar_wait(&full[i % S], (uint32_t)((i / S) & 1))) set_err(a.err, kErrTimeout);
        return;
    }

    // ---------------------------------------------------------------- consumers
    const int cw = warp - 1;
    const int G = plan.G, Wg = kConsumers / G;                // groups, warps per group
    const int grp = cw / Wg, gw = cw % Wg;
    const int SEG = R >= Wg ? 1 : Wg / R;                     // column segments per row
    const int seg = gw % SEG;
    const int nvec = a.kin / VEC;
    const int v_lo = (int)((long)seg * nvec / SEG), v_hi = (int)((long)(seg + 1) * nvec / SEG);
    const int rr0 = SEG == 1 ? gw : gw / SEG, rstep = SEG == 1 ? Wg : R;
    const uint32_t x_base = saddr(X);
    const uint32_t ring_base = saddr(ring);
    bool dead = false;
    int lc = 0;                                               // chunks this group has taken
    // Ring items are numbered i = pass * n_chunks + chunk in issue order; group
    // g takes the items i = g, g + G, ... across all passes, so with G dividing
    // S it only ever waits on stages s = g (mod G), each in fill order.
    int item = grp, s = grp;
    uint32_t ph = 0;                                          // phase parity of stage s
    pdl_wait();

    for (int p = 0; p < n_pass; ++p) {
        const int t0 = p * TC;
        const int tc = a.T - t0 < TC ? a.T - t0 : TC;
        stage_x<WT, TC>(a, t0, tc, X, red);
        if constexpr (TOPK) {
            if (lane < TC) {
#pragma unroll
                for (int i = 0; i < kTopK; ++i) { s_val[cw][lane][i] = -INFINITY; s_id[cw][lane][i] = 0x7FFFFFFF; }
            }
        }
        consumers_sync();
        float thr_v = -INFINITY;
        int thr_i = 0x7FFFFFFF;

        for (; item < (p + 1) * n_chunks; item += G, ++lc) {
            const int c = item - p * n_chunks;
            if (!dead && !mbar_wait(&full[s], ph, wait_bound(a.wait_polls, kWaitLimit))) {
                set_err(a.err, kErrTimeout);
                dead = true;
            }
            const int first = u0 + c * R;
            const int rows = u1 - first < R ? u1 - first : R;
            for (int rr = rr0; rr < R; rr += rstep) {
                bool live = !dead && rr < rows;
                if (live && (PRISM_CHECK(a.err, ((size_t)(RPW - 1) * R + rr + 1) * nvec * 16 <= plan.stage_bytes, 104, rr, nvec) ||
                             PRISM_CHECK(a.err, (size_t)TC * a.kin * sizeof(WT) <= plan.x_bytes, 105, TC, a.kin)))
                    live = false;   // skip the access, keep the barrier sequence
                unsigned long long p0[RPW][TC], p1[RPW][TC];
#pragma unroll
                for (int r = 0; r < RPW; ++r)
#pragma unroll
                    for (int t = 0; t < TC; ++t) p0[r][t] = p1[r][t] = 0ull;
                if (live) {
                    uint32_t wa[RPW];
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
                        wa[r] = ring_base + (uint32_t)(s * plan.stage_bytes) + (uint32_t)(((r * R + rr) * nvec) * 16);
                    const int vb = SEG == 1 ? 0 : v_lo, ve = SEG == 1 ? nvec : v_hi;
                    int v = vb + lane;
                    for (; v + 32 * (U - 1) < ve; v += 32 * U) {
                        uint4 wv[RPW][U];
#pragma unroll
                        for (int j = 0; j < U; ++j)
#pragma unroll
                            for (int r = 0; r < RPW; ++r) wv[r][j] = lds128(wa[r] + (uint32_t)(v + 32 * j) * 16u);
#pragma unroll
                        for (int j = 0; j < U; ++j) {
#pragma unroll
                            for (int t = 0; t < TC; ++t) {
                                const uint4 xv = lds128(x_base + (uint32_t)(t * nvec + v + 32 * j) * 16u);
#pragma unroll
                                for (int r = 0; r < RPW; ++r) dot16B<WT>(p0[r][t], p1[r][t], wv[r][j], xv);
                            }
                        }
                    }
                    for (; v < ve; v += 32) {
#pragma unroll
                        for (int t = 0; t < TC; ++t) {
                            const uint4 xv = lds128(x_base + (uint32_t)(t * nvec + v) * 16u);
#pragma unroll
                            for (int r = 0; r < RPW; ++r)
                                dot16B<WT>(p0[r][t], p1[r][t], lds128(wa[r] + (uint32_t)v * 16u), xv);
                        }
                    }
                }
                float acc[RPW][TC];
#pragma unroll
                for (int r = 0; r < RPW; ++r)
#pragma unroll
                    for (int t = 0; t < TC; ++t) acc[r][t] = warp_sum(sum2(p0[r][t]) + sum2(p1[r][t]));
                if (SEG > 1) {
                    // add the row's column segments in segment order (group barrier)
                    const int buf = lc & 1;
                    if (lane == 0) {
#pragma unroll
                        for (int r = 0; r < RPW; ++r)
#pragma unroll
                            for (int t = 0; t < TC; ++t) s_part[buf][cw][r][t] = acc[r][t];
                    }
                    asm volatile("bar.sync %0, %1;" ::"r"(2 + grp), "r"(Wg * 32) : "memory");
                    if (seg != 0) continue;
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
#pragma unroll
                        for (int t = 0; t < TC; ++t) {
                            float v2 = 0.f;
                            for (int q = 0; q < SEG; ++q) v2 += s_part[buf][cw + q][r][t];
                            acc[r][t] = v2;
                        }
                }
                if (!live) continue;
                const int u = first + rr;
#pragma unroll
                for (int t = 0; t < TC; ++t) {
                    if (lane != t || t >= tc) continue;
                    const int row = t0 + t;
                    if constexpr (TOPK) {
                        const float z = acc[0][t];
                        if (a.logits) a.logits[((size_t)row * a.K + a.step - 1) * a.vocab + u] = z;
                        if (better(z, u, thr_v, thr_i)) {
                            float *lv = s_val[cw][t];
                            int *li = s_id[cw][t];
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
                        Elem<WT>::store((WT *)a.out_act, (size_t)row * a.out_ld + u, g / (1.0f + expf(-g)) * up);
                    } else {
                        float val = acc[0][t];
                        if (a.epi == kEpiResid) {
                            const int rrow = a.resid_prefill_rows ? (row * a.max_new + clamp_nnew(a, row) - 1) : row;
                            val += a.resid[(size_t)rrow * a.out_ld + u];
                            if (a.hidden_out) a.hidden_out[((size_t)row * a.K + a.step - 1) * a.d + u] = val;
                        }
                        a.out[(size_t)row * a.out_ld + u] = val;
                    }
                }
            }
            __syncwarp();
            // a warp that gave up on this stage does not release it: its copy
            // may still be in flight, and the producer must not reuse the slot
            // (the producer's own wait then gives up and it drains)
            if (lane == 0 && !dead) mbar_arrive(&empty[s]);
            s += G;
            if (s >= S) { s -= S; ph ^= 1; }
        }

        if constexpr (TOPK) {
            // per-CTA merge of the consumer warps' lists, one warp per activation row
            consumers_sync();
            for (int t = cw; t < tc; t += kConsumers) {
                float v[kTopK];
                int id[kTopK];
                top8_init(v, id);
                for (int c2 = lane; c2 < kConsumers * kTopK; c2 += 32)
                    top8_insert(v, id, s_val[c2 / kTopK][t][c2 % kTopK], s_id[c2 / kTopK][t][c2 % kTopK]);
                warp_merge_top8(v, id);
                if (lane == 0) {
                    const size_t base = (((size_t)(t0 + t)) * gridDim.x + blockIdx.x) * kTopK;
#pragma unroll
                    for (int i = 0; i < kTopK; ++i) { a.lm_part[base + i] = v[i]; a.lm_part_id[base + i] = id[i]; }
                }
            }
        }
        consumers_sync();
    }

    if constexpr (TOPK) {
        // the last CTA to finish merges every CTA's partial lists
        __threadfence();
        consumers_sync();
        if (threadIdx.x == 32) s_last = (atomicAdd(a.counter, 1) == (int)gridDim.x - 1);
        consumers_sync();
        if (!s_last) return;
        __threadfence();
        const int Gd = gridDim.x;
        for (int t = cw; t < a.T; t += kConsumers) {
            float v[kTopK];
            int id[kTopK];
            top8_init(v, id);
            const size_t base = (size_t)t * Gd * kTopK;
            for (int c2 = lane; c2 < Gd * kTopK; c2 += 32)
                top8_insert(v, id, __ldcg(a.lm_part + base + c2), __ldcg(a.lm_part_id + base + c2));
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
        if (threadIdx.x == 32) *a.counter = 0;
    }
}

template <typename WT, int TC>
cudaError_t dispatch_kind(const GemvArgs &a, const RingPlan &pl, int grid, size_t smem, cudaStream_t s,
                          bool pdl) {
    if (a.epi == kEpiTopK)
        return launch_k(gemv_kernel<WT, TC, 1, true>, dim3(grid), dim3(kThreads), smem, s, pdl, a, pl);
    if (a.epi == kEpiSwiGLU)
        return launch_k(gemv_kernel<WT, TC, 2, false>, dim3(grid), dim3(kThreads), smem, s, pdl, a, pl);
    return launch_k(gemv_kernel<WT, TC, 1, false>, dim3(grid), dim3(kThreads), smem, s, pdl, a, pl);
}

template <typename WT>
cudaError_t set_smem_attrs(int bytes) {
    cudaError_t e = cudaSuccess;
#define PRISM_SET(TC, RPW, TK)                                                                   \
    if (e == cudaSuccess)                                                                        \
        e = cudaFuncSetAttribute(gemv_kernel<WT, TC, RPW, TK>,                                   \
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    PRISM_SET(1, 1, true) PRISM_SET(1, 2, false) PRISM_SET(1, 1, false)
    PRISM_SET(2, 1, true) PRISM_SET(2, 2, false) PRISM_SET(2, 1, false)
    PRISM_SET(4, 1, true) PRISM_SET(4, 2, false) PRISM_SET(4, 1, false)
    PRISM_SET(8, 1, true) PRISM_SET(8, 2, false) PRISM_SET(8, 1, false)
#undef PRISM_SET
    return e;
}

int rows_per_pass(int T) { return T <= 1 ? 1 : (T <= 2 ? 2 : (T <= 4 ? 4 : 8)); }

// Ring plan: stage = R whole rows (R a power of two), G consumer groups, S
// stages (a multiple of G).  Chosen for the fewest passes over W (largest
// activation block), then the most bytes in flight within the budget, then
// the preferred group count.
bool make_plan(const GemvArgs &a, bool bf16, int &tc, RingPlan &pl, size_t &smem) {
    const size_t es = bf16 ? 2 : 4;
    const int RPW = a.epi == kEpiSwiGLU ? 2 : 1;
    const size_t row = (size_t)a.kin * es;
    const size_t target = a.chunk_target > 0 ? (size_t)a.chunk_target : kChunkTarget;
    const size_t budget = a.smem_budget > 0 ? (size_t)a.smem_budget : kSmemAlone;
    const int g_pref = a.groups > 0 ? a.groups : 4;
    int R0 = 1;
    while ((size_t)(R0 * 2) * row * RPW <= target && R0 < 64) R0 *= 2;
    for (tc = rows_per_pass(a.T); tc >= 1; tc = tc == 1 ? 0 : tc / 2) {
        const size_t x = (size_t)tc * row;
        bool found = false;
        size_t best_inflight = 0;
        RingPlan best{};
        for (int G : {g_pref, 4, 2, 8, 1, 16}) {
            for (int R = R0; R >= 1; R /= 2) {
                const size_t stage = (size_t)R * row * RPW;
                if (x + (size_t)G * stage > budget) continue;
                int S = (int)((budget - x) / stage);
                if (S > kMaxStages) S = kMaxStages;
                S = S / G * G;
                if (S < 2) continue;
                const size_t inflight = (size_t)S * stage;
                if (!found || inflight > best_inflight + 16 * 1024) {
                    found = true;
                    best_inflight = inflight;
                    best = RingPlan{R, S, G, stage, x};
                }
                break;   // largest R that fits for this G
            }
        }
        if (found) {
            pl = best;
            smem = (size_t)pl.stages * pl.stage_bytes + pl.x_bytes;
            return true;
        }
    }
    return false;
}

}  // namespace

cudaError_t prepare_gemv_kernels() {
    cudaError_t e = set_smem_attrs<uint16_t>((int)kSmemAlone);
    if (e == cudaSuccess) e = set_smem_attrs<float>((int)kSmemAlone);
    if (e == cudaSuccess) e = prepare_gemv_mma_kernels();
    return e;
}

bool gemv_supported(const GemvArgs &a, bool bf16) {
    // launch_gemv takes the mma.sync kernel only when the CUDA-core one is not forced
    if (bf16 && !a.force_cuda_core && gemv_mma_supported(a)) return true;
    int tc;
    RingPlan pl;
    size_t smem;
    return make_plan(a, bf16, tc, pl, smem);
}

// bf16 projections whose contraction length is a multiple of 32 run on the
// tensor-core kernel (gemv_mma.cu); the rest on the CUDA-core ring kernel.
cudaError_t launch_gemv(const GemvArgs &a, bool bf16, int grid, cudaStream_t s, bool pdl) {
    if (bf16 && !a.force_cuda_core && gemv_mma_supported(a)) return launch_gemv_mma(a, grid, s, pdl);
    int tc;
    RingPlan pl;
    size_t smem;
    if (!make_plan(a, bf16, tc, pl, smem)) return cudaErrorInvalidValue;
    if (bf16) {
        if (tc == 1) return dispatch_kind<uint16_t, 1>(a, pl, grid, smem, s, pdl);
        if (tc == 2) return dispatch_kind<uint16_t, 2>(a, pl, grid, smem, s, pdl);
        if (tc == 4) return dispatch_kind<uint16_t, 4>(a, pl, grid, smem, s, pdl);
        return dispatch_kind<uint16_t, 8>(a, pl, grid, smem, s, pdl);
    }
    if (tc == 1) return dispatch_kind<float, 1>(a, pl, grid, smem, s, pdl);
    if (tc == 2) return dispatch_kind<float, 2>(a, pl, grid, smem, s, pdl);
    if (tc == 4) return dispatch_kind<float, 4>(a, pl, grid, smem, s, pdl);
    return dispatch_kind<float, 8>(a, pl, grid, smem, s, pdl);
}

}  // namespace prism
