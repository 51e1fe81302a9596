// Tensor-core weight-streaming projections for bf16 drafters (sm_103a).
//
// Same contract as the CUDA-core ring kernel in gemv.cu (y[t] = W x[t] for a
// few activation rows, fused prologue/epilogue), built so that the consumer
// side costs a handful of instructions per 512 bytes of weights:
//   * the contraction runs on warp-level tensor-core MMAs (m16n8k16, bf16 x
//     bf16 -> fp32): the 16 MMA rows are activation rows (T <= 16 per pass,
//     padded with zeros), the 8 MMA columns are 8 weight rows, K = 16;
//   * the weight rows are cut into 8-row tiles (RPW = 2: 8 gate + 8 up rows);
//     a ring stage holds one tile's K slice of KC columns, filled by one TMA
//     bulk copy per row issued in parallel by the producer warp's lanes
//     (copies of >= 2 KB, which the bulk-copy engine needs for full rate),
//     into padded rows (pitch KC*2 + 16 bytes, bank-conflict free);
//   * all 8 consumer warps take every stage in order (sound parity waits);
//     warp w contracts columns [w*KC/8, (w+1)*KC/8) of the slice and keeps
//     its partial sums in registers across the tile's slices; at the end of
//     the tile the 8 partials are added in warp order through shared memory
//     (deterministic) and one thread per (activation row, weight row) runs
//     the epilogue;
//   * fragments: lane (g, t) loads 16 bytes of weight row g at columns
//     8t..8t+7 of a 32-column group and the same columns of activation rows
//     g and g+8; words {0,1} form the k-step pairing MMA k-slots (2t, 2t+1)
//     and (2t+8, 2t+9) with columns 8t+{0,1} and 8t+{2,3}, words {2,3} the
//     second k-step with 8t+{4,5}, 8t+{6,7}.  The pairing depends on t only,
//     so A and B agree on every k-slot and each column is used exactly once;
//   * the prologue/epilogue, PDL behaviour and bounded waits are those of
//     gemv.cu.
#include "common.cuh"

namespace prism {

namespace {

constexpr int kW = 8;                  // consumer warps
constexpr int kThreadsM = (kW + 1) * 32;
constexpr int kStagesM = 8;            // maximum ring depth
constexpr long kWaitLimitM = 1L << 22;
constexpr size_t kSmemM = 200 * 1024;

__device__ __forceinline__ uint32_t sa(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void bar_init(uint64_t *b, uint32_t n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(sa(b)), "r"(n));
}
__device__ __forceinline__ void bar_arrive(uint64_t *b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(sa(b)) : "memory");
}
__device__ __forceinline__ void bar_arrive_tx(uint64_t *b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sa(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool bar_wait(uint64_t *b, uint32_t parity, long limit = kWaitLimitM) {
    for (long i = 0; i < limit; ++i) {
        uint32_t ok;
        asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                     : "=r"(ok) : "r"(sa(b)), "r"(parity) : "memory");
        if (ok) return true;
    }
    return false;
}
__device__ __forceinline__ bool bar_test(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile("{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                 : "=r"(ok) : "r"(sa(b)), "r"(parity) : "memory");
    return ok != 0;
}
__device__ __forceinline__ void tma_row(void *dst, const void *src, uint32_t bytes, uint64_t *b) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(sa(dst)), "l"(src), "r"(bytes), "r"(sa(b)) : "memory");
}
__device__ __forceinline__ void sync_consumers() {
    asm volatile("bar.sync 1, %0;" ::"r"(kW * 32) : "memory");
}
__device__ __forceinline__ uint4 lds16(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}
// D += A * B, m16n8k16, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
                 "{%0, %1, %2, %3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float wsum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

__device__ float consumers_total(float v, float *red) {
    const int lane = threadIdx.x & 31, w = (threadIdx.x >> 5) - 1;
    v = wsum(v);
    sync_consumers();
    if (lane == 0) red[w] = v;
    sync_consumers();
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kW; ++i) s += red[i];
    return s;
}

__device__ __forceinline__ int nnew_of(const GemvArgs &a, int b) {
    int n = a.n_new[b];
    if (n < 1 || n > a.max_new) {
        set_err(a.err, kErrNNew);
        n = n < 1 ? 1 : a.max_new;
    }
    return n;
}

__device__ __forceinline__ int token_of(const GemvArgs &a, int tok) {
    if (tok < 0 || tok >= a.vocab) {
        set_err(a.err, kErrToken);
        return 0;
    }
    return tok;
}

// Activation rows [t0, t0 + tc) as bf16 in shared memory, row pitch xp
// elements; consumer threads only.
__device__ void stage_rows(const GemvArgs &a, int t0, int tc, uint16_t *X, int xp, float *red) {
    const int NT = kW * 32, tid = threadIdx.x - 32;
    const int kin = a.kin, d = a.d;
    const uint16_t *E = (const uint16_t *)a.embed;
    for (int t = 0; t < tc; ++t) {
        uint16_t *xr = X + (size_t)t * xp;
        const int row = t0 + t;
        if (a.pro == kProFusePrefill) {
            const int b = row / a.max_new, i = row % a.max_new;
            const int n = nnew_of(a, b);
            const bool valid = i < n;
            const int tok = valid ? token_of(a, a.tokens[b * a.max_new + i]) : 0;
            const uint16_t *hid = (const uint16_t *)a.hidden_in + ((size_t)b * a.max_new + i) * d;
            const uint16_t *er = E + (size_t)tok * d;
            for (int c = tid; c < d; c += NT) {
                xr[c] = valid ? er[c] : (uint16_t)0;
                xr[d + c] = valid ? hid[c] : (uint16_t)0;
            }
        } else if (a.pro == kProFuseDecode) {
            const int b = row;
            const int tok = token_of(a, a.draft[b * a.K + a.step - 2]);
            const uint16_t *er = E + (size_t)tok * d;
            const float *h = a.src + (size_t)b * d;
            for (int c = tid; c < d; c += NT) {
                xr[c] = er[c];
                xr[d + c] = f32_to_bf16(h[c]);
            }
        } else if (a.pro == kProNorm) {
            const int sr = a.src_prefill_rows ? (row * a.max_new + nnew_of(a, row) - 1) : row;
            const float *s = a.src + (size_t)sr * d;
            float inv = 1.f;
            if (a.gain) {
                float ss = 0.f;
                for (int c = tid; c < d; c += NT) ss = fmaf(s[c], s[c], ss);
                ss = consumers_total(ss, red);
                inv = 1.0f / sqrtf(ss / (float)d + a.eps);
            }
            const uint16_t *g = (const uint16_t *)a.gain;
            for (int c = tid; c < d; c += NT)
                xr[c] = f32_to_bf16(a.gain ? s[c] * inv * bf16_to_f32(g[c]) : s[c]);
        } else {
            const uint16_t *src = (const uint16_t *)a.act + (size_t)row * kin;
            for (int c = tid; c < kin; c += NT) xr[c] = src[c];
        }
    }
}

__device__ void merge_top8_warp(float (&v)[kTopK], int (&id)[kTopK]) {
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

struct MmaPlan {
    int kc;            // columns per row slice (a multiple of 256)
    int tc;            // activation rows per pass (<= 16)
    int xp;            // activation row pitch in elements
    int pitch;         // stage row pitch in bytes
    int stages;        // ring depth
    size_t stage_bytes;
};

// RPW: weight rows per unit (2 for gate/up pairs); HI: activation rows 8..15
// exist; TOPK: LM-head selection epilogue.
template <int RPW, bool HI, bool TOPK>
__global__ void __launch_bounds__(kThreadsM, 1) gemv_mma_kernel(const GemvArgs a, const MmaPlan pl) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t full[kStagesM], empty[kStagesM];
    __shared__ float red[kW];
    // per-tile partials of the 8 warps: [buffer][warp][r][activation row][weight row]
    __shared__ float s_red[2][kW][RPW][HI ? 16 : 8][8];
    __shared__ float s_val[TOPK ? (HI ? 16 : 8) : 1][8][kTopK];
    __shared__ int s_id[TOPK ? (HI ? 16 : 8) : 1][8][kTopK];
    __shared__ int s_last;

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int KC = pl.kc, S = pl.stages;
    const int u0 = (int)((long long)blockIdx.x * a.n_units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * a.n_units / gridDim.x);
    const int n_tiles = (u1 - u0 + 7) / 8;
    const int KS = (a.kin + KC - 1) / KC;
    const int n_pass = (a.T + pl.tc - 1) / pl.tc;
    const long total = (long)n_pass * n_tiles * KS;     // stages: pass, tile, K slice
    uint8_t *ring = smem;
    uint16_t *X = (uint16_t *)(smem + (size_t)S * pl.stage_bytes);

    pdl_trigger();
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            bar_init(&full[s], 1);
            bar_init(&empty[s], kW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        // stage i = (pass, tile, K slice) in order; slot s = i % S with
        // phase bit ph = (i / S) & 1, both kept incrementally (no divisions)
        long issued = 0;
        int s = 0, tile = 0, j = 0;
        uint32_t ph = 0;
        for (long i = 0; i < total; ++i) {
            int ok = 1;
            if (lane == 0) ok = bar_wait(&empty[s], ph ^ 1u, wait_bound(a.wait_polls, kWaitLimitM));
            ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
            if (!ok) {
                if (lane == 0) set_err(a.err, kErrTimeout);
                break;
            }
            const int first = u0 + tile * 8;
            const int rows = u1 - first < 8 ? u1 - first : 8;
            const int cols = a.kin - j * KC < KC ? a.kin - j * KC : KC;
            const uint32_t bytes = (uint32_t)cols * 2u;
            if (lane == 0) bar_arrive_tx(&full[s], bytes * (uint32_t)(rows * RPW));
            __syncwarp();
            if (lane < 8 * RPW) {
                const int r = lane / 8, rr = lane % 8;
                if (rr < rows)
                    tma_row(ring + (size_t)s * pl.stage_bytes + (size_t)lane * pl.pitch,
                            (const uint8_t *)a.W + (((size_t)first + rr + (size_t)r * a.pair_offset) * a.kin +
                                                    (size_t)j * KC) * 2,
                            bytes, &full[s]);
            }
            issued = i + 1;
            if (++j == KS) { j = 0; if (++tile == n_tiles) tile = 0; }
            if (++s == S) { s = 0; ph ^= 1u; }
        }
        // drain: the last S stages' copies land before this CTA may exit
        if (lane == 0) {
            const long first_i = issued > S ? issued - S : 0;
            int ds = (int)(first_i % S);
            uint32_t dph = (uint32_t)((first_i / S) & 1);
            for (long i = first_i; i < issued; ++i) {
                if (!bar_wait(&full[ds], dph)) set_err(a.err, kErrTimeout);
                if (++ds == S) { ds = 0; dph ^= 1u; }
            }
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    const int cw = warp - 1, g = lane >> 2, tq = lane & 3, ct = threadIdx.x - 32;
    const uint32_t ring_s = sa(ring), x_s = sa(X);
    constexpr int TR = HI ? 16 : 8;                          // activation rows in s_red
    bool dead = false;
    int s = 0;                                               // slot and phase of the next stage,
    uint32_t ph = 0;                                         // in the producer's order
    pdl_wait();

    for (int p = 0; p < n_pass; ++p) {
        const int t0 = p * pl.tc;
        const int tc = a.T - t0 < pl.tc ? a.T - t0 : pl.tc;
        stage_rows(a, t0, tc, X, pl.xp, red);
        sync_consumers();
        const bool row_lo = g < tc, row_hi = HI && (g + 8) < tc;
        // epilogue thread (activation row et, weight row en) and its top-8
        const int et = ct / 8, en = ct % 8;
        float lv[kTopK];
        int li[kTopK];
        if constexpr (TOPK) top8_init(lv, li);

        for (int tile = 0; tile < n_tiles; ++tile) {
            const int first = u0 + tile * 8;
            const int rows = u1 - first < 8 ? u1 - first : 8;
            // four independent accumulator sets (rotating over 32-column
            // groups) keep four MMA chains in flight; added in set order below
            float acc4[RPW][4][4];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int q = 0; q < 4; ++q) acc4[r][q][0] = acc4[r][q][1] = acc4[r][q][2] = acc4[r][q][3] = 0.f;
            for (int j = 0; j < KS; ++j) {
                if (!dead && !bar_wait(&full[s], ph, wait_bound(a.wait_polls, kWaitLimitM))) {
                    set_err(a.err, kErrTimeout);
                    dead = true;
                }
                const int cols = a.kin - j * KC < KC ? a.kin - j * KC : KC;
                const int cb = (int)((long)cw * cols / kW) / 32 * 32;       // this warp's column range
                const int ce = (int)((long)(cw + 1) * cols / kW) / 32 * 32;
                if (!dead) {
                    const uint32_t wrow = ring_s + (uint32_t)(s * pl.stage_bytes) + (uint32_t)(g * pl.pitch + tq * 16);
                    const uint32_t xlo = x_s + (uint32_t)((g * pl.xp + j * KC + tq * 8) * 2);
                    const uint32_t xhi = xlo + (uint32_t)(8 * pl.xp * 2);
                    for (int c0 = cb; c0 < ce; c0 += 128) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int c = c0 + 32 * q;
                            if (c < ce) {
                                const uint4 xa = row_lo ? lds16(xlo + (uint32_t)c * 2u) : make_uint4(0u, 0u, 0u, 0u);
                                const uint4 xb = row_hi ? lds16(xhi + (uint32_t)c * 2u) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                                for (int r = 0; r < RPW; ++r) {
                                    const uint4 wv = lds16(wrow + (uint32_t)(r * 8 * pl.pitch) + (uint32_t)c * 2u);
                                    mma16816(acc4[r][q], xa.x, xb.x, xa.y, xb.y, wv.x, wv.y);
                                    mma16816(acc4[r][q], xa.z, xb.z, xa.w, xb.w, wv.z, wv.w);
                                }
                            }
                        }
                    }
                }
                __syncwarp();
                // a warp that gave up on this stage does not release it (its copy
                // may still be in flight); the producer's wait then gives up
                if (lane == 0 && !dead) bar_arrive(&empty[s]);
                if (++s == S) { s = 0; ph ^= 1u; }
            }
            float acc[RPW][4];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[r][e] = ((acc4[r][0][e] + acc4[r][1][e]) + acc4[r][2][e]) + acc4[r][3][e];
            // add the 8 warps' partials: acc[r] = D[g][2tq], D[g][2tq+1], D[g+8][2tq], D[g+8][2tq+1]
            const int buf = tile & 1;
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                s_red[buf][cw][r][g][2 * tq] = acc[r][0];
                s_red[buf][cw][r][g][2 * tq + 1] = acc[r][1];
                if constexpr (HI) {
                    s_red[buf][cw][r][g + 8][2 * tq] = acc[r][2];
                    s_red[buf][cw][r][g + 8][2 * tq + 1] = acc[r][3];
                }
            }
            sync_consumers();
            if (!dead && et < tc && en < rows) {
                float z[RPW];
#pragma unroll
                for (int r = 0; r < RPW; ++r) {
                    float v = 0.f;
#pragma unroll
                    for (int w = 0; w < kW; ++w) v += s_red[buf][w][r][et][en];
                    z[r] = v;
                }
                const int row = t0 + et, u = first + en;
                if constexpr (TOPK) {
                    if (a.logits) a.logits[((size_t)row * a.K + a.step - 1) * a.vocab + u] = z[0];
                    top8_insert(lv, li, z[0], u);
                } else if constexpr (RPW == 2) {
                    Elem<uint16_t>::store((uint16_t *)a.out_act, (size_t)row * a.out_ld + u,
                                          z[0] / (1.0f + expf(-z[0])) * z[RPW - 1]);
                } else {
                    float val = z[0];
                    if (a.epi == kEpiResid) {
                        const int rrow = a.resid_prefill_rows ? (row * a.max_new + nnew_of(a, row) - 1) : row;
                        val += a.resid[(size_t)rrow * a.out_ld + u];
                        if (a.hidden_out) a.hidden_out[((size_t)row * a.K + a.step - 1) * a.d + u] = val;
                    }
                    a.out[(size_t)row * a.out_ld + u] = val;
                }
            }
        }

        if constexpr (TOPK) {
            // thread (et, en) holds the top-8 of row et over weight rows = en mod 8
            if (et < TR) {
#pragma unroll
                for (int i2 = 0; i2 < kTopK; ++i2) { s_val[et][en][i2] = lv[i2]; s_id[et][en][i2] = li[i2]; }
            }
            sync_consumers();
            for (int t = cw; t < tc; t += kW) {
                float v[kTopK];
                int id[kTopK];
                top8_init(v, id);
                for (int c2 = lane; c2 < 8 * kTopK; c2 += 32)
                    top8_insert(v, id, s_val[t][c2 / kTopK][c2 % kTopK], s_id[t][c2 / kTopK][c2 % kTopK]);
                merge_top8_warp(v, id);
                if (lane == 0) {
                    const size_t base = (((size_t)(t0 + t)) * gridDim.x + blockIdx.x) * kTopK;
#pragma unroll
                    for (int i2 = 0; i2 < kTopK; ++i2) { a.lm_part[base + i2] = v[i2]; a.lm_part_id[base + i2] = id[i2]; }
                }
            }
        }
        sync_consumers();
    }

    if constexpr (TOPK) {
        __threadfence();
        sync_consumers();
        if (threadIdx.x == 32) s_last = (atomicAdd(a.counter, 1) == (int)gridDim.x - 1);
        sync_consumers();
        if (!s_last) return;
        __threadfence();
        const int Gd = gridDim.x;
        for (int t = cw; t < a.T; t += kW) {
            float v[kTopK];
            int id[kTopK];
            top8_init(v, id);
            const size_t base = (size_t)t * Gd * kTopK;
            for (int c2 = lane; c2 < Gd * kTopK; c2 += 32)
                top8_insert(v, id, __ldcg(a.lm_part + base + c2), __ldcg(a.lm_part_id + base + c2));
            merge_top8_warp(v, id);
            if (lane == 0) {
                const size_t o = (size_t)t * a.K + a.step - 1;
                a.draft_out[o] = id[0];
#pragma unroll
                for (int i2 = 0; i2 < kTopK; ++i2) {
                    if (i2 < a.topk) {
                        if (a.topk_ids) a.topk_ids[o * a.topk + i2] = id[i2];
                        if (a.topk_logits) a.topk_logits[o * a.topk + i2] = v[i2];
                    }
                }
            }
        }
        if (threadIdx.x == 32) *a.counter = 0;
    }
}

// Stage: one 8-row tile (16 rows for gate/up) x KC columns, row copies of
// 4 KB (2 KB for gate/up); as many stages as fit next to the activation rows.
bool mma_plan(const GemvArgs &a, MmaPlan &pl, size_t &smem) {
    if (a.kin % 256 != 0) return false;          // 8 warps x 32-column groups
    const int RPW = a.epi == kEpiSwiGLU ? 2 : 1;
    pl.kc = RPW == 2 ? 1024 : 2048;
    while (pl.kc > a.kin) pl.kc /= 2;
    if (pl.kc < 256) return false;
    pl.pitch = pl.kc * 2 + 16;
    pl.stage_bytes = (size_t)RPW * 8 * pl.pitch;
    pl.xp = a.kin + 8;                            // +16 bytes per activation row
    for (int tc = a.T < 16 ? a.T : 16; tc >= 1; --tc) {
        const size_t x = (size_t)tc * pl.xp * 2;
        if (x + 3 * pl.stage_bytes > kSmemM) continue;
        size_t st = (kSmemM - x) / pl.stage_bytes;
        pl.stages = (int)(st > (size_t)kStagesM ? kStagesM : st);
        pl.tc = tc;
        smem = (size_t)pl.stages * pl.stage_bytes + x;
        return true;
    }
    return false;
}

template <int RPW, bool HI, bool TOPK>
cudaError_t launch_m(const GemvArgs &a, const MmaPlan &pl, int grid, size_t smem, cudaStream_t s, bool pdl) {
    return launch_k(gemv_mma_kernel<RPW, HI, TOPK>, dim3(grid), dim3(kThreadsM), smem, s, pdl, a, pl);
}

}  // namespace

bool gemv_mma_supported(const GemvArgs &a) {
    MmaPlan pl;
    size_t smem;
    return mma_plan(a, pl, smem);
}

cudaError_t prepare_gemv_mma_kernels() {
    cudaError_t e = cudaSuccess;
#define PRISM_SETM(R, H, T)                                                                          \
    if (e == cudaSuccess)                                                                            \
        e = cudaFuncSetAttribute(gemv_mma_kernel<R, H, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                 (int)kSmemM);
    PRISM_SETM(1, false, false) PRISM_SETM(1, true, false) PRISM_SETM(2, false, false)
    PRISM_SETM(2, true, false) PRISM_SETM(1, false, true) PRISM_SETM(1, true, true)
#undef PRISM_SETM
    return e;
}

cudaError_t launch_gemv_mma(const GemvArgs &a, int grid, cudaStream_t s, bool pdl) {
    MmaPlan pl;
    size_t smem;
    if (!mma_plan(a, pl, smem)) return cudaErrorInvalidValue;
    const bool hi = pl.tc > 8;
    if (a.epi == kEpiTopK)
        return hi ? launch_m<1, true, true>(a, pl, grid, smem, s, pdl) : launch_m<1, false, true>(a, pl, grid, smem, s, pdl);
    if (a.epi == kEpiSwiGLU)
        return hi ? launch_m<2, true, false>(a, pl, grid, smem, s, pdl) : launch_m<2, false, false>(a, pl, grid, smem, s, pdl);
    return hi ? launch_m<1, true, false>(a, pl, grid, smem, s, pdl) : launch_m<1, false, false>(a, pl, grid, smem, s, pdl);
}

}  // namespace prism
