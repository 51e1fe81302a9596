// Tensor-core (tcgen05) weight-streaming projections of the PRISM draft step.
//
// Each projection of a draft step (fusion F, QKV, O, gate/up, down, LM head;
// Sec. 3.2 and the Llama block) is D = W X^T with W [rows, kin] in bf16 and a
// handful of activation rows X [T, kin].  W is the A operand (M = 128 rows of
// W per tile, K-major), X the B operand (N = 16, K-major), D accumulates in
// fp32 in tensor memory.  Nothing on the SM touches individual weights:
//   * warp 0, one lane: TMA tensor loads of 128-row x 64-column boxes of W
//     (128-byte swizzle, the canonical K-major operand layout) into a ring of
//     shared-memory stages; it starts before griddepcontrol.wait, so the ring
//     fills while the previous kernel drains;
//   * warps 1-5 build X once per CTA in shared memory (embedding gather,
//     RMSNorm with its gain, bf16 rounding), already in the swizzled operand
//     layout; with T <= 8 only 8 rows are stored and the descriptor's 8-row
//     stride is 0, so the MMA's rows 8-15 re-read rows 0-7;
//   * warp 1, one lane: tcgen05.mma (kind::f16, M=128, N=16, K=16) per
//     32-byte K slice; tcgen05.commit releases a stage when its MMAs have
//     read it and signals a finished accumulator;
//   * warps 2-5: the epilogue reads the accumulator (tcgen05.ld, one TMEM
//     lane = one output row per thread) into registers while the MMA fills
//     the other of two accumulator buffers, and fuses the residual add,
//     SwiGLU, or the logits write and top-8 selection;
//   * split-K: with few 128-row tiles the contraction is split over CTAs
//     (CTA c takes K slice c % S); the partial sums go to a workspace and the
//     last CTA to finish a tile adds them in slice order, so results do not
//     depend on timing;
//   * every wait is bounded; on expiry the kernel sets the timeout bit of the
//     device error word, stops waiting, drains its copies and MMAs, frees its
//     tensor memory and returns.
#include <algorithm>
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"

namespace prism {

namespace {

constexpr int kTcThreads = 192;             // producer, MMA, 4 epilogue warps
constexpr int kStageThreads = kTcThreads - 32;
constexpr int kTileM = 128;
constexpr int kBoxK = 64;                   // bf16 elements per 128-byte swizzle row
constexpr uint32_t kBoxBytes = kTileM * 128;  // 16 KB
constexpr int kMmaN = 16;
constexpr int kTcMaxStages = 8;
constexpr int kMaxSplits = 8;
constexpr size_t kTcSmem = 212 * 1024;      // dynamic shared memory budget of the top-k list instances
// the other staged instances keep about 1 KB of static shared memory, so their
// rings can grow to what the 227 KB per-CTA limit leaves (more bytes in flight
// per SM: HBM reads scale with them up to tens of MB in flight device-wide)
constexpr size_t kTcSmemLarge = 225 * 1024;
constexpr size_t kXBudget = 128 * 1024;     // largest X slice
constexpr long kTcWaitLimit = 1L << 22;

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
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity, long limit = kTcWaitLimit) {
    for (long i = 0; i < limit; ++i)
        if (mbar_try(b, parity)) return true;
    return false;
}

// Whole-warp wait: lane 0 polls with a short back-off (a warp of spinning
// lanes would compete with the TMA and MMA traffic on shared memory), then
// every lane observes the completed phase.  Warp-uniform result.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t *b, uint32_t parity, long limit) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) {
        ok = false;
        for (long i = 0; i < limit; ++i) {
            if (mbar_try(b, parity)) { ok = true; break; }
            __nanosleep(64);
        }
    }
    ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
    if (ok) mbar_try(b, parity);
    return ok;
}

// 2-D TMA tensor load (box at column x, row y) into shared memory.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(dst), "l"((uint64_t)map), "r"(x), "r"(y), "r"(saddr(bar)) : "memory");
}
// The same with an L2 cache policy (pol != 0), else without.
__device__ __forceinline__ void tma_load_2d_pol(uint32_t dst, const CUtensorMap *map, int x, int y, uint64_t *bar,
                                                uint64_t pol) {
    if (pol == 0) {
        tma_load_2d(dst, map, x, y, bar);
        return;
    }
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
        "%3}], [%4], %5;" ::"r"(dst), "l"((uint64_t)map), "r"(x), "r"(y), "r"(saddr(bar)), "l"(pol) : "memory");
}

// tcgen05 shared-memory matrix descriptor: K-major operand in the 128-byte
// swizzle layout (8-row x 128-byte atoms, `sbo` bytes between 8-row groups).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFFu) >> 4);    // start address
    d |= (uint64_t)1 << 16;                     // leading-dimension offset (unused here)
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;  // stride-dimension offset
    d |= (uint64_t)1 << 46;                     // descriptor version
    d |= (uint64_t)2 << 61;                     // 128-byte swizzle
    return d;
}

// Instruction descriptor: bf16 A and B, fp32 D, both K-major, M = 128, N = 16.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kMmaN >> 3) << 17) |
                            ((uint32_t)(kTileM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a), "l"(b), "r"(kIdesc), "r"(accumulate));
}
// Arrive once on `bar` when every MMA this thread issued so far has completed.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(saddr(bar))
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 16 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void stage_sync() {   // warps 1-5
    asm volatile("bar.sync 1, %0;" ::"r"(kStageThreads) : "memory");
}
__device__ __forceinline__ void epi_sync() {     // warps 2-5
    asm volatile("bar.sync 2, 128;" ::: "memory");
}

__device__ __forceinline__ int clamp_n(const GemvArgs &a, int b) {
    int n = a.n_new[b];
    if (n < 1 || n > a.max_new) {
        set_err(a.err, kErrNNew);
        n = n < 1 ? 1 : a.max_new;
    }
    return n;
}
__device__ __forceinline__ int token_ok(const GemvArgs &a, int tok) {
    if (tok < 0 || tok >= a.vocab) {
        set_err(a.err, kErrToken);
        return 0;
    }
    return tok;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    return (uint32_t)f32_to_bf16(lo) | ((uint32_t)f32_to_bf16(hi) << 16);
}
struct TcPlan {
    int n_tiles;        // 128-row tiles of output units
    int nkb;            // 64-wide K blocks of the whole contraction
    int splits;         // K slices (CTA c works on slice c % splits)
    int stages;         // ring stages
    int kb_per_stage;   // K blocks per stage (each RPW boxes)
    uint32_t stage_bytes, x_bytes;
    float *part;        // split-K partial sums [splits][RPW][T][n_units]
    int *tile_ctr;      // per-tile arrival tickets (left at zero)
    int defer;          // split-K sums finished by splitk_finish_kernel, not the tile's last CTA
};

// X rows (bf16, swizzled K-major operand layout) for the K blocks [kb0, kb1).
// Threads of warps 1-5.  This runs once per CTA while the weight ring waits,
// so it is kept short in both senses: little code (it executes cold, one
// instruction-cache miss per line) and few dependent memory round trips
// (each costs microseconds behind a saturated HBM): a thread issues the loads
// of all its chunks of a row (up to kStageGroup) before using any.
constexpr int kStageGroup = 4;

__device__ __forceinline__ void ld32(const void *p, uint4 &lo, uint4 &hi) {
    lo = __ldcg((const uint4 *)p);
    hi = __ldcg((const uint4 *)p + 1);
}
__device__ __forceinline__ float sumsq8(const uint4 &lo, const uint4 &hi) {
    const float f[8] = {__uint_as_float(lo.x), __uint_as_float(lo.y), __uint_as_float(lo.z), __uint_as_float(lo.w),
                        __uint_as_float(hi.x), __uint_as_float(hi.y), __uint_as_float(hi.z), __uint_as_float(hi.w)};
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) s = fmaf(f[i], f[i], s);
    return s;
}
// 8 fp32 values (lo, hi), times scale and the bf16 gains g when use_g, rounded to bf16.
__device__ __forceinline__ uint4 round8r(const uint4 &lo, const uint4 &hi, float scale, bool use_g, const uint4 &g) {
    float v[8] = {__uint_as_float(lo.x), __uint_as_float(lo.y), __uint_as_float(lo.z), __uint_as_float(lo.w),
                  __uint_as_float(hi.x), __uint_as_float(hi.y), __uint_as_float(hi.z), __uint_as_float(hi.w)};
    if (use_g) {
        const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            v[2 * i] = v[2 * i] * scale * bf16lo(gw[i]);
            v[2 * i + 1] = v[2 * i + 1] * scale * bf16hi(gw[i]);
        }
    }
    return make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]), pack_bf16(v[6], v[7]));
}

// Deterministic sum over the staging threads (fixed shuffle tree, fixed warp order).
__device__ __forceinline__ float stage_sum(float v, float *red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    if ((threadIdx.x & 31) == 0) red[(threadIdx.x >> 5) - 1] = v;
    stage_sync();
    float tot = 0.f;
#pragma unroll
    for (int i = 0; i < kStageThreads / 32; ++i) tot += red[i];
    stage_sync();
    return tot;
}

template <int NB, int PRO>
__device__ void stage_x_tc(const GemvArgs &a, int kb0, int kb1, uint8_t *X, float *red) {
    const int tid = threadIdx.x - 32;
    const int d = a.d, kin = a.kin, T = a.T;
    // padding rows T..NB-1: zero (16-byte slot i of a K block holds row (i / 8) % NB)
    const int nslots = (kb1 - kb0) * NB * 8;
#pragma unroll 1
    for (int i = tid; i < nslots; i += kStageThreads)
        if (((i >> 3) & (NB - 1)) >= T) ((uint4 *)X)[i] = make_uint4(0, 0, 0, 0);

    const int c0 = kb0 * 8, c1 = kb1 * 8;     // 8-element chunks of this CTA's K range
#pragma unroll 1
    for (int t = 0; t < T; ++t) {
        // per-row sources
        const uint16_t *e_row = nullptr, *h_row = nullptr;
        const float *f_row = nullptr;
        bool valid = true;
        float inv = 1.f;
        if constexpr (PRO == kProFusePrefill) {
            const int b = t / a.max_new, r = t % a.max_new;
            valid = r < clamp_n(a, b);
            const int tok = valid ? token_ok(a, a.tokens[b * a.max_new + r]) : 0;
            e_row = (const uint16_t *)a.embed + (size_t)tok * d;
            h_row = (const uint16_t *)a.hidden_in + ((size_t)b * a.max_new + r) * d;
        } else if constexpr (PRO == kProFuseDecode) {
            e_row = (const uint16_t *)a.embed + (size_t)token_ok(a, a.draft[t * a.K + a.step - 2]) * d;
            f_row = a.src + (size_t)t * d;
        } else if constexpr (PRO == kProNorm) {
            const int sr = a.src_prefill_rows ? (t * a.max_new + clamp_n(a, t) - 1) : t;
            f_row = a.src + (size_t)sr * d;
            if (a.gain) {
                float ss = 0.f;
#pragma unroll 1
                for (int c = tid; c < d / 8; c += kStageGroup * kStageThreads) {
                    uint4 lo[kStageGroup], hi[kStageGroup];
#pragma unroll
                    for (int g = 0; g < kStageGroup; ++g)
                        if (c + g * kStageThreads < d / 8) ld32(f_row + (size_t)(c + g * kStageThreads) * 8, lo[g], hi[g]);
#pragma unroll
                    for (int g = 0; g < kStageGroup; ++g)
                        if (c + g * kStageThreads < d / 8) ss += sumsq8(lo[g], hi[g]);
                }
                inv = 1.0f / sqrtf(stage_sum(ss, red) / (float)d + a.eps);
            }
        } else {
            h_row = (const uint16_t *)a.act + (size_t)t * kin;
        }
        // this thread's chunks of the row: loads first, then convert and store
#pragma unroll 1
        for (int c = c0 + tid; c < c1; c += kStageGroup * kStageThreads) {
            uint4 lo[kStageGroup], hi[kStageGroup], gv[kStageGroup];
#pragma unroll
            for (int g = 0; g < kStageGroup; ++g) {
                const int k = (c + g * kStageThreads) * 8;
                lo[g] = hi[g] = gv[g] = make_uint4(0, 0, 0, 0);
                if (c + g * kStageThreads >= c1 || k >= kin || !valid) continue;
                if constexpr (PRO == kProFusePrefill) {
                    lo[g] = k < d ? __ldg((const uint4 *)(e_row + k)) : __ldcg((const uint4 *)(h_row + (k - d)));
                } else if constexpr (PRO == kProFuseDecode) {
                    if (k < d) lo[g] = __ldg((const uint4 *)(e_row + k));
                    else ld32(f_row + (k - d), lo[g], hi[g]);
                } else if constexpr (PRO == kProNorm) {
                    ld32(f_row + k, lo[g], hi[g]);
                    if (a.gain) gv[g] = __ldg((const uint4 *)((const uint16_t *)a.gain + k));
                } else {
                    lo[g] = __ldcg((const uint4 *)(h_row + k));
                }
            }
#pragma unroll
            for (int g = 0; g < kStageGroup; ++g) {
                const int cc = c + g * kStageThreads;
                if (cc >= c1) continue;
                uint4 v = lo[g];
                const int k = cc * 8;
                if (k < kin && valid) {
                    if constexpr (PRO == kProFuseDecode) {
                        if (k >= d) v = round8r(lo[g], hi[g], 1.f, false, gv[g]);
                    } else if constexpr (PRO == kProNorm) {
                        v = round8r(lo[g], hi[g], inv, a.gain != nullptr, gv[g]);
                    }
                }
                const int kb = cc >> 3, ci = cc & 7;
                *(uint4 *)(X + (size_t)(kb - kb0) * (NB * 128) + t * 128 + ((ci ^ (t & 7)) << 4)) = v;
            }
        }
    }
}

// Final epilogue of one output unit u for activation row t, given its
// accumulators (RPW = 2: gate, up).
template <int RPW>
__device__ __forceinline__ void finish_unit(const GemvArgs &a, int t, int u, float acc0, float acc1) {
    if constexpr (RPW == 2) {
        Elem<uint16_t>::store((uint16_t *)a.out_act, (size_t)t * a.out_ld + u, acc0 / (1.0f + expf(-acc0)) * acc1);
    } else {
        float val = acc0;
        if (a.epi == kEpiResid) {
            const int rrow = a.resid_prefill_rows ? (t * a.max_new + clamp_n(a, t) - 1) : t;
            val += a.resid[(size_t)rrow * a.out_ld + u];
            if (a.hidden_out) a.hidden_out[((size_t)t * a.K + a.step - 1) * a.d + u] = val;
        }
        a.out[(size_t)t * a.out_ld + u] = val;
    }
}

// Split-K: the last CTA of a tile adds the K slices of unit u for every
// activation row, in slice order, and finishes the unit.  The partial sums
// come from other SMs through L2, so the loads of several rows and all their
// slices (32 values; SB bounds the slice count) are issued before any is
// used: the round trips are T / C rather than T x splits.
template <int RPW, int SB>
__device__ __forceinline__ void reduce_slices_sb(const GemvArgs &a, const TcPlan &p, int T, int u) {
    constexpr int C = 32 / (SB * RPW);             // rows per batch of loads
    const int splits = p.splits;
#pragma unroll 1
    for (int t0 = 0; t0 < T; t0 += C) {
        float v[C][SB][RPW];
#pragma unroll
        for (int c = 0; c < C; ++c)
#pragma unroll
            for (int k = 0; k < SB; ++k)
#pragma unroll
                for (int r = 0; r < RPW; ++r)
                    v[c][k][r] = (t0 + c < T && k < splits)
                                     ? __ldcg(&p.part[(((size_t)k * RPW + r) * T + t0 + c) * a.n_units + u])
                                     : 0.f;
#pragma unroll
        for (int c = 0; c < C; ++c) {
            if (t0 + c >= T) break;
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int k = 0; k < SB; ++k)
                if (k < splits) {
                    s0 += v[c][k][0];
                    s1 += v[c][k][RPW - 1];
                }
            finish_unit<RPW>(a, t0 + c, u, s0, s1);
        }
    }
}
template <int RPW>
__device__ __forceinline__ void reduce_slices(const GemvArgs &a, const TcPlan &p, int T, int u) {
    if (T <= 4) {
        // few rows: the short loop (this code runs cold, once per tile)
        for (int t = 0; t < T; ++t) {
            float v0 = 0.f, v1 = 0.f;
            for (int k = 0; k < p.splits; ++k) {
                v0 += __ldcg(&p.part[(((size_t)k * RPW + 0) * T + t) * a.n_units + u]);
                if (RPW == 2) v1 += __ldcg(&p.part[(((size_t)k * RPW + 1) * T + t) * a.n_units + u]);
            }
            finish_unit<RPW>(a, t, u, v0, v1);
        }
    } else if (p.splits <= 2) reduce_slices_sb<RPW, 2>(a, p, T, u);
    else if (p.splits <= 4) reduce_slices_sb<RPW, 4>(a, p, T, u);
    else reduce_slices_sb<RPW, kMaxSplits>(a, p, T, u);
}

// ---------------------------------------------------------------- top-k lists
// A candidate list is kTopK packed keys (pack_best) in registers, best first;
// key 0 is the empty slot (below every real candidate).  Each epilogue thread
// keeps one list, for one activation row: with NB rows, P = 128 / NB threads
// share a row and each scans 128 / P of a tile's 128 logits.  The logits
// reach the scanning threads through a transposed shared-memory copy of one
// 16-column accumulator chunk at a time, so a scan is one compare per logit
// (a list changes only when a logit beats its last entry).  The P lists of a
// row are merged pairwise across lanes (bitonic merge), and the per-CTA lists
// of all CTAs once at the end.
constexpr int kTrMax = kTileM + 8;   // floats per transposed row, largest P

// One 16-column accumulator chunk (columns c0 .. c0 + 15) of a finished tile
// into the lists.  The four epilogue warps write their TMEM rows transposed
// (tr[j][row]: column j becomes a row of 128 logits), then the threads of
// those columns' rows scan them.  A transposed row is 128 + P floats long, so
// the 32 lanes of a scanning warp read 32 distinct banks.
// With P = 8 every epilogue thread scans: thread e takes row c0 + e / 8.
// With want_lse the scanning thread also adds each logit to its running
// log-sum-exp (lm, ls) of that row.
template <int P>
__device__ __forceinline__ void chunk_to_lists(const float (&acc)[16], int row, float *tr, int tile, int c0, int T,
                                               int n_units, bool dead, Key (&l)[kTopK], bool want_lse, float &lm,
                                               float &ls) {
    constexpr int S = kTileM + P;
#pragma unroll
    for (int j = 0; j < 16; ++j) tr[j * S + row] = acc[j];
    epi_sync();
    const int e = threadIdx.x - 64, t = (P == 8 ? c0 : 0) + e / P, q = e % P;
    if (!dead && t >= c0 && t < c0 + 16 && t < T) {
        const float *src = tr + (t - c0) * S;
#pragma unroll 4
        for (int i = 0; i < kTileM / P; ++i) {
            const int r = i * P + q, u = tile * kTileM + r;
            if (u < n_units) {
                key_insert(l, pack_best(src[r], u));
                if (want_lse) lse_add(lm, ls, src[r]);
            }
        }
    }
    epi_sync();
}

// The CTA's (max, sum exp) of each row: the 8 threads of a row combine
// theirs (fixed butterfly order), the first writes the CTA's partial.
__device__ __forceinline__ void lse_publish(const GemvArgs &a, float m, float s, int T, int t0) {
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o), s2 = __shfl_xor_sync(0xFFFFFFFFu, s, o);
        lse_combine(m, s, m2, s2);
    }
    const int e = threadIdx.x - 64, t = t0 + e / 8;
    if ((e & 7) == 0 && t < T) {
        float *pp = a.lse_part + ((size_t)t * gridDim.x + blockIdx.x) * 2;
        pp[0] = m;
        pp[1] = s;
    }
}

// The CTA's list of each row: the P threads of a row merge theirs and write
// it to the per-CTA partial lists ([row][CTA][kTopK] values and ids; id -1
// marks an empty slot), thread q the entries q, q + P, ...
template <int P>
__device__ __forceinline__ void lists_publish(const GemvArgs &a, Key (&l)[kTopK], int T, int t0 = 0) {
#pragma unroll 1
    for (int m = 1; m < P; m <<= 1) key_merge_xor(l, m);
    const int e = threadIdx.x - 64, t = t0 + e / P, q = e % P;
    if (t < T) {
#pragma unroll
        for (int r0 = 0; r0 < kTopK; r0 += P) {
            float v;
            int id;
            unpack_best(key_at(l, r0 + q), v, id);
            const size_t o = ((size_t)t * gridDim.x + blockIdx.x) * kTopK + r0 + q;
            a.lm_part[o] = v;
            a.lm_part_id[o] = id;
        }
    }
}

// This thread's share (candidates first, first + stride, ...) of row t's
// partial lists, as a sorted list.  Loads are issued 16 at a time; ROLLED
// inserts them through one copy of the insertion network (code that runs once
// per launch executes at instruction-cache-miss speed), otherwise unrolled.
template <bool ROLLED>
__device__ __forceinline__ void gather_keys(const GemvArgs &a, int t, int grid, int first, int stride, Key (&l)[kTopK]) {
    constexpr int kBatch = 16;
    const int ncand = grid * kTopK;
    const float *pv = a.lm_part + (size_t)t * ncand;
    const int *pi = a.lm_part_id + (size_t)t * ncand;
    key_clear(l);
#pragma unroll 1
    for (int c = first; c < ncand; c += kBatch * stride) {
        float v[kBatch];
        int id[kBatch];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int cc = c + b * stride;
            v[b] = cc < ncand ? __ldcg(pv + cc) : 0.f;
            id[b] = cc < ncand ? __ldcg(pi + cc) : -1;
        }
        if constexpr (ROLLED) {
#pragma unroll 1
            for (int b = 0; b < kBatch; ++b)
                if (id[b] >= 0) key_insert(l, pack_best(v[b], id[b]));
        } else {
#pragma unroll
            for (int b = 0; b < kBatch; ++b)
                if (id[b] >= 0) key_insert(l, pack_best(v[b], id[b]));
        }
    }
}

// Row t's final top-k from a list every lane of the warp holds: lane r < topk
// writes rank r.
__device__ __forceinline__ void write_row(const GemvArgs &a, int t, const Key (&l)[kTopK]) {
    const int lane = threadIdx.x & 31;
    if (lane < a.topk) {
        float v;
        int id;
        unpack_best(key_at(l, lane), v, id);
        const size_t o = (size_t)t * a.K + a.step - 1;
        if (lane == 0) a.draft_out[o] = id;
        if (a.topk_ids) a.topk_ids[o * a.topk + lane] = id;
        if (a.topk_logits) a.topk_logits[o * a.topk + lane] = v;
    }
}

// Packed top-1 (one row per accumulator column t < T): a warp's candidates
// of a tile, unit u of this lane with logit acc[t], join the warp's best of
// each row (thr_*, the same in every lane, mirrored in s_v / s_i for the CTA's
// join) in turn, lane by lane, where they beat it.
template <int N>
__device__ __forceinline__ void top1_scan(const float *acc, int T, bool valid, int u, float (&thr_v)[N],
                                          int (&thr_i)[N], float (&s_v)[N], int (&s_i)[N]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int t = 0; t < N; ++t) {
        if (t >= T) break;
        const float z = acc[t];
        unsigned m = __ballot_sync(0xFFFFFFFFu, valid && better(z, u, thr_v[t], thr_i[t]));
        while (m) {
            const int src = __ffs(m) - 1;
            m &= m - 1;
            const float zv = __shfl_sync(0xFFFFFFFFu, z, src);
            const int uv = __shfl_sync(0xFFFFFFFFu, u, src);
            if (!better(zv, uv, thr_v[t], thr_i[t])) continue;
            if (lane == 0) {
                s_v[t] = zv;
                s_i[t] = uv;
            }
            __syncwarp();
            thr_v[t] = s_v[t];
            thr_i[t] = s_i[t];
            __syncwarp();
        }
    }
}

// The CTA's best of each row (the four epilogue warps' s_v / s_i) joins a
// 64-bit atomic maximum; the last CTA to finish writes each row's top-1 and
// clears the maximum.  Epilogue warps only.
template <int N>
__device__ __forceinline__ void top1_join(const GemvArgs &a, int T, float (&s_v)[4][N], int (&s_i)[4][N],
                                          int &s_last) {
    const int ew = (threadIdx.x >> 5) - 2, lane = threadIdx.x & 31;
    epi_sync();
    if (ew == 0 && lane < T) {
        float bv = s_v[0][lane];
        int bi = s_i[0][lane];
#pragma unroll
        for (int w = 1; w < 4; ++w)
            if (better(s_v[w][lane], s_i[w][lane], bv, bi)) { bv = s_v[w][lane]; bi = s_i[w][lane]; }
        if (bi != 0x7FFFFFFF) atomicMax(a.best + lane, pack_best(bv, bi));
    }
    __threadfence();
    epi_sync();
    if (threadIdx.x == 64) s_last = atomicAdd(a.counter, 1) == (int)gridDim.x - 1;
    epi_sync();
    if (s_last) {
        __threadfence();
        if (ew == 0 && lane < T) {
            const Key key = atomicExch(a.best + lane, 0ull);
            float v;
            int id;
            unpack_best(key, v, id);
            const size_t o = (size_t)lane * a.K + a.step - 1;
            a.draft_out[o] = id;
            if (a.topk_ids) a.topk_ids[o] = id;
            if (a.topk_logits) a.topk_logits[o] = v;
        }
        if (threadIdx.x == 64) *a.counter = 0;
    }
}

// TK: 0 no selection; 1 top-1 through the packed 64-bit atomic maximum; 2 top-k
// through the register lists (separate instances, so neither carries the
// other's code).
template <int NB, int RPW, int TK, int PRO>
__global__ void __launch_bounds__(kTcThreads, 1)
    gemv_tc_kernel(const GemvArgs a, const TcPlan p, const __grid_constant__ CUtensorMap tmW) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kTcMaxStages], empty[kTcMaxStages], acc_full[2], acc_empty[2], mma_done;
    __shared__ uint32_t s_tmem;
    __shared__ float red[kStageThreads / 32];
    constexpr bool TOPK = TK != 0;
    __shared__ float s_val[TK == 1 ? 4 : 1][TK == 1 ? NB : 1];   // top-1: each epilogue warp's best per row
    __shared__ int s_id[TK == 1 ? 4 : 1][TK == 1 ? NB : 1];
    __shared__ float s_tr[TK == 2 ? 16 : 1][TK == 2 ? kTrMax : 1];
    __shared__ int s_last;
    constexpr uint32_t kCols = RPW == 1 ? 32 : 64;   // two accumulator buffers x RPW x 16 columns

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long lim = wait_bound(a.wait_polls, kTcWaitLimit);
    uint8_t *base = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *ring = base;
    uint8_t *X = base + (size_t)p.stages * p.stage_bytes;
    const int S = p.stages;
    const int ks = blockIdx.x % p.splits;
    const int tiles_step = gridDim.x / p.splits;
    const int kb0 = (int)((long)ks * p.nkb / p.splits), kb1 = (int)((long)(ks + 1) * p.nkb / p.splits);
    const int n_kst = (kb1 - kb0 + p.kb_per_stage - 1) / p.kb_per_stage;
    int my_tiles = 0;
    for (int tile = blockIdx.x / p.splits; tile < p.n_tiles; tile += tiles_step) ++my_tiles;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);
        }
        mbar_init(&mma_done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmW) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&s_tmem)),
                     "r"(kCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    pdl_trigger();

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            const uint64_t wpol = a.w_evict_first ? l2_evict_first_policy() : 0ull;
            int s = 0, issued = 0;
            uint32_t ph = 0;
            bool dead = false;
            for (int i = 0; i < my_tiles && !dead; ++i) {
                const int tile = blockIdx.x / p.splits + i * tiles_step;
                for (int q = 0; q < n_kst; ++q) {
                    if (!mbar_wait(&empty[s], ph ^ 1, lim)) {
                        set_err(a.err, kErrTimeout);
                        dead = true;
                        break;
                    }
                    const int kbs = kb0 + q * p.kb_per_stage;
                    const int nkb = kb1 - kbs < p.kb_per_stage ? kb1 - kbs : p.kb_per_stage;
                    mbar_arrive_tx(&full[s], (uint32_t)nkb * RPW * kBoxBytes);
                    const uint32_t st = saddr(ring) + (uint32_t)s * p.stage_bytes;
                    for (int j = 0; j < nkb; ++j)
#pragma unroll
                        for (int r = 0; r < RPW; ++r)
                            tma_load_2d_pol(st + (uint32_t)(j * RPW + r) * kBoxBytes, &tmW, (kbs + j) * kBoxK,
                                        tile * kTileM + r * a.pair_offset, &full[s], wpol);
                    ++issued;
                    if (++s == S) { s = 0; ph ^= 1; }
                }
            }
            if (!dead) prefetch_l2_share(a.pf_next, a.pf_next_bytes, blockIdx.x, gridDim.x);
            // drain: the copies in flight land before this CTA may exit
            const int first = issued > S ? issued - S : 0;
            for (int i = first; i < issued; ++i)
                if (!mbar_wait(&full[i % S], (uint32_t)((i / S) & 1))) set_err(a.err, kErrTimeout);
        }
    } else {
        pdl_wait();
        stage_x_tc<NB, PRO>(a, kb0, kb1, X, red);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        stage_sync();

        if (warp == 1) {
            // ------------------------------------------------------------ MMA
            if (lane == 0) {
                int s = 0;
                uint32_t ph = 0;
                bool dead = false;
                const uint32_t xb = saddr(X);
                const uint32_t sbo_b = NB == 16 ? 1024u : 0u;
                for (int i = 0; i < my_tiles && !dead; ++i) {
                    const int ab = i & 1;
                    if (!mbar_wait(&acc_empty[ab], ((i >> 1) & 1) ^ 1, lim)) {
                        set_err(a.err, kErrTimeout);
                        dead = true;
                        break;
                    }
                    tc_fence_after();
                    for (int q = 0; q < n_kst; ++q) {
                        if (!mbar_wait(&full[s], ph, lim)) {
                            set_err(a.err, kErrTimeout);
                            dead = true;
                            break;
                        }
                        tc_fence_after();
                        const int kbs = kb0 + q * p.kb_per_stage;
                        const int nkb = kb1 - kbs < p.kb_per_stage ? kb1 - kbs : p.kb_per_stage;
                        const uint32_t st = saddr(ring) + (uint32_t)s * p.stage_bytes;
                        for (int j = 0; j < nkb; ++j) {
                            const uint32_t xa = xb + (uint32_t)(kbs + j - kb0) * (NB * 128);
#pragma unroll
                            for (int kk = 0; kk < kBoxK / 16; ++kk) {
                                const uint64_t bd = sw128_desc(xa + kk * 32, sbo_b);
#pragma unroll
                                for (int r = 0; r < RPW; ++r) {
                                    const uint64_t ad =
                                        sw128_desc(st + (uint32_t)(j * RPW + r) * kBoxBytes + kk * 32, 1024);
                                    mma_bf16(tmem + (uint32_t)((ab * RPW + r) * kMmaN), ad, bd,
                                             (q | j | kk) != 0 ? 1u : 0u);
                                }
                            }
                        }
                        mma_commit(&empty[s]);
                        if (++s == S) { s = 0; ph ^= 1; }
                    }
                    if (!dead) mma_commit(&acc_full[ab]);
                }
                mma_commit(&mma_done);
                if (!mbar_wait(&mma_done, 0)) set_err(a.err, kErrTimeout);
            }
            __syncwarp();
        } else {
            // ------------------------------------------------------------ epilogue
            const int ew = warp - 2;                   // 0..3
            const int quarter = warp & 3;              // TMEM lanes 32*quarter .. +31
            const int row = quarter * 32 + lane;
            const int T = a.T;
            // top-1 with the 64-bit atomic maximum: per warp and row the best so
            // far (thr, cached in registers); otherwise the register lists
            constexpr bool top1 = TK == 1;
            float thr_v[NB];
            int thr_i[NB];
            Key lst[kTopK];
            if constexpr (TOPK) {
#pragma unroll
                for (int t = 0; t < NB; ++t) { thr_v[t] = -INFINITY; thr_i[t] = 0x7FFFFFFF; }
                if constexpr (TK == 1) {
                    if (lane < NB) { s_val[ew][lane] = -INFINITY; s_id[ew][lane] = 0x7FFFFFFF; }
                }
                key_clear(lst);
                __syncwarp();
            }
            float lse_m = -INFINITY, lse_s = 0.f;     // this thread's row, with a.lse_part
            bool dead = false;
            for (int i = 0; i < my_tiles; ++i) {
                const int tile = blockIdx.x / p.splits + i * tiles_step;
                const int ab = i & 1;
                if (!dead && !mbar_wait_warp(&acc_full[ab], (i >> 1) & 1, lim)) {
                    if (lane == 0) set_err(a.err, kErrTimeout);
                    dead = true;
                }
                float acc[RPW][16];
                if (!dead) {
                    tc_fence_after();
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
                        tmem_ld16(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((ab * RPW + r) * kMmaN),
                                  acc[r]);
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acc_empty[ab]);
                } else {
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
#pragma unroll
                        for (int t = 0; t < 16; ++t) acc[r][t] = 0.f;
                }

                const int u = tile * kTileM + row;
                const bool valid = !dead && u < a.n_units;
                if constexpr (TOPK) {
                    if (valid && a.logits) {
#pragma unroll
                        for (int t = 0; t < NB; ++t)
                            if (t < T) a.logits[((size_t)t * a.K + a.step - 1) * a.vocab + u] = acc[0][t];
                    }
                    if constexpr (top1) {
                        top1_scan<NB>(acc[0], T, valid, u, thr_v, thr_i, s_val[ew], s_id[ew]);
                    } else {
                        chunk_to_lists<8>(acc[0], row, &s_tr[0][0], tile, 0, T, a.n_units, dead, lst,
                                          a.lse_part != nullptr, lse_m, lse_s);
                    }
                } else if (p.splits == 1) {
                    if (valid) {
#pragma unroll
                        for (int t = 0; t < NB; ++t) {
                            if (t >= T) break;
                            finish_unit<RPW>(a, t, u, acc[0][t], acc[RPW - 1][t]);
                        }
                    }
                } else {
                    // split-K: publish this slice, the tile's last CTA adds all slices in order
                    if (valid) {
#pragma unroll
                        for (int r = 0; r < RPW; ++r)
#pragma unroll
                            for (int t = 0; t < NB; ++t) {
                                if (t >= T) break;
                                p.part[(((size_t)ks * RPW + r) * T + t) * a.n_units + u] = acc[r][t];
                            }
                    }
                    __threadfence();
                    epi_sync();
                    if (threadIdx.x == 64) s_last = atomicAdd(&p.tile_ctr[tile], 1) == p.splits - 1;
                    epi_sync();
                    if (s_last) {
                        __threadfence();
                        if (valid) reduce_slices<RPW>(a, p, T, u);
                        if (threadIdx.x == 64) p.tile_ctr[tile] = 0;
                    }
                    epi_sync();
                }
            }
            if constexpr (top1) {
                top1_join<NB>(a, T, s_val, s_id, s_last);
            } else if constexpr (TOPK) {
                lists_publish<8>(a, lst, T);
                if (a.lse_part) lse_publish(a, lse_m, lse_s, T, 0);
                __threadfence();
                epi_sync();
                if (threadIdx.x == 64) s_last = !a.defer_merge && atomicAdd(a.counter, 1) == (int)gridDim.x - 1;
                epi_sync();
                if (s_last) {
                    __threadfence();
                    // one warp per row over every CTA's list
                    for (int t = ew; t < T; t += 4) {
                        gather_keys<true>(a, t, gridDim.x, lane, 32, lst);
#pragma unroll 1
                        for (int m = 1; m < 32; m <<= 1) key_merge_xor(lst, m);
                        write_row(a, t, lst);
                    }
                    if (threadIdx.x == 64) *a.counter = 0;
                }
            }
        }
    }

    if (warp == 0) return;   // the producer takes no part in tensor memory
    // teardown: every tcgen05 operation of this CTA is complete before the free
    tc_fence_before();
    stage_sync();
    tc_fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols));
}

// ------------------------------------------------------------------ streamed
// Variant for many activation rows (T > 16): the B operand is not staged
// whole but streams through the ring next to W.  Each stage holds, per K
// block, the RPW boxes of W and one box of the activation rows X (NB rows x
// 64 columns, the same 128-byte swizzle), fetched by TMA from a bf16 X
// buffer that a prep kernel (or the previous projection, for the copy
// prologue) has written.  MMA N = NB (16 .. 256); rows of X past T arrive as
// zeros.  The epilogue reads the NB accumulator columns 16 at a time.  With
// top-k, the per-row merge across CTAs is left to topk_merge_kernel.
template <int NB, int RPW, int TK>
__global__ void __launch_bounds__(kTcThreads, 1)
    gemv_tcs_kernel(const GemvArgs a, const TcPlan p, const __grid_constant__ CUtensorMap tmW,
                    const __grid_constant__ CUtensorMap tmX) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kTcMaxStages], empty[kTcMaxStages], acc_full[2], acc_empty[2], mma_done;
    __shared__ uint32_t s_tmem;
    constexpr bool TOPK = TK != 0, LISTS = TK == 2;   // TK: 0 none, 1 packed top-1, 2 top-k lists
    __shared__ float s_tr[LISTS ? 16 : 1][LISTS ? kTrMax : 1];
    __shared__ float s_val[TK == 1 ? 4 : 1][TK == 1 ? NB : 1];   // top-1: each epilogue warp's best per row
    __shared__ int s_id[TK == 1 ? 4 : 1][TK == 1 ? NB : 1];
    __shared__ int s_last;
    constexpr uint32_t kXBox = NB * 128;                              // one X box
    constexpr uint32_t kColsNeed = 2 * RPW * NB;
    constexpr uint32_t kCols = kColsNeed <= 32 ? 32 : kColsNeed <= 64 ? 64 : kColsNeed <= 128 ? 128
                               : kColsNeed <= 256 ? 256 : 512;
    static_assert(kColsNeed <= 512, "accumulators exceed tensor memory");
    constexpr uint32_t kIdescN = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(NB >> 3) << 17) |
                                 ((uint32_t)(kTileM >> 4) << 24);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long lim = wait_bound(a.wait_polls, kTcWaitLimit);
    uint8_t *ring = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int S = p.stages;
    const uint32_t kb_bytes = RPW * kBoxBytes + kXBox;                // one K block in a stage
    const int ks = blockIdx.x % p.splits;
    const int tiles_step = gridDim.x / p.splits;
    const int kb0 = (int)((long)ks * p.nkb / p.splits), kb1 = (int)((long)(ks + 1) * p.nkb / p.splits);
    const int n_kst = (kb1 - kb0 + p.kb_per_stage - 1) / p.kb_per_stage;
    int my_tiles = 0;
    for (int tile = blockIdx.x / p.splits; tile < p.n_tiles; tile += tiles_step) ++my_tiles;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);
        }
        mbar_init(&mma_done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmW) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmX) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&s_tmem)),
                     "r"(kCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    pdl_trigger();

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            const uint64_t wpol = a.w_evict_first ? l2_evict_first_policy() : 0ull;
            int s = 0, issued = 0;
            uint32_t ph = 0;
            bool dead = false;
            const int total = my_tiles * n_kst;
            // item f of this CTA: tile, first K block and K blocks of its stage
            auto item = [&](int f, int &tile, int &kbs, int &nkb) {
                tile = blockIdx.x / p.splits + (f / n_kst) * tiles_step;
                kbs = kb0 + (f % n_kst) * p.kb_per_stage;
                nkb = kb1 - kbs < p.kb_per_stage ? kb1 - kbs : p.kb_per_stage;
            };
            auto load_w = [&](int f, int stage) {
                int tile, kbs, nkb;
                item(f, tile, kbs, nkb);
                const uint32_t st = saddr(ring) + (uint32_t)stage * p.stage_bytes;
                for (int j = 0; j < nkb; ++j)
#pragma unroll
                    for (int r = 0; r < RPW; ++r)
                        tma_load_2d_pol(st + (uint32_t)j * kb_bytes + (uint32_t)r * kBoxBytes, &tmW, (kbs + j) * kBoxK,
                                        tile * kTileM + r * a.pair_offset, &full[stage], wpol);
            };
            auto load_x = [&](int f, int stage) {
                int tile, kbs, nkb;
                item(f, tile, kbs, nkb);
                const uint32_t st = saddr(ring) + (uint32_t)stage * p.stage_bytes;
                for (int j = 0; j < nkb; ++j)
                    tma_load_2d(st + (uint32_t)j * kb_bytes + RPW * kBoxBytes, &tmX, (kbs + j) * kBoxK, 0, &full[stage]);
            };
            auto arm = [&](int f, int stage) {
                int tile, kbs, nkb;
                item(f, tile, kbs, nkb);
                mbar_arrive_tx(&full[stage], (uint32_t)nkb * kb_bytes);
            };
            // The first ring pass: the stages are free (fresh barriers), and the
            // weight boxes do not depend on the previous kernel, so they are
            // requested before the dependency wait; X is the previous kernel's
            // output, so its boxes of those stages follow the wait.  Each stage's
            // barrier expects both from the start, so it completes only when both
            // have landed.
            const int pre = total < S ? total : S;
            for (int f = 0; f < pre; ++f) {
                arm(f, f);
                load_w(f, f);
            }
            pdl_wait();
            for (int f = 0; f < pre; ++f) load_x(f, f);
            issued = pre;
            s = pre % S;
            ph = pre == S ? 1u : 0u;
            for (int f = pre; f < total; ++f) {
                if (!mbar_wait(&empty[s], ph ^ 1, lim)) {
                    set_err(a.err, kErrTimeout);
                    dead = true;
                    break;
                }
                arm(f, s);
                load_w(f, s);
                load_x(f, s);
                ++issued;
                if (++s == S) { s = 0; ph ^= 1; }
            }
            if (!dead) prefetch_l2_share(a.pf_next, a.pf_next_bytes, blockIdx.x, gridDim.x);
            const int first = issued > S ? issued - S : 0;
            for (int i = first; i < issued; ++i)
                if (!mbar_wait(&full[i % S], (uint32_t)((i / S) & 1))) set_err(a.err, kErrTimeout);
        }
    } else {
        pdl_wait();
        if (warp == 1) {
            // ------------------------------------------------------------ MMA
            if (lane == 0) {
                int s = 0;
                uint32_t ph = 0;
                bool dead = false;
                for (int i = 0; i < my_tiles && !dead; ++i) {
                    const int ab = i & 1;
                    if (!mbar_wait(&acc_empty[ab], ((i >> 1) & 1) ^ 1, lim)) {
                        set_err(a.err, kErrTimeout);
                        dead = true;
                        break;
                    }
                    tc_fence_after();
                    for (int q = 0; q < n_kst; ++q) {
                        if (!mbar_wait(&full[s], ph, lim)) {
                            set_err(a.err, kErrTimeout);
                            dead = true;
                            break;
                        }
                        tc_fence_after();
                        const int kbs = kb0 + q * p.kb_per_stage;
                        const int nkb = kb1 - kbs < p.kb_per_stage ? kb1 - kbs : p.kb_per_stage;
                        const uint32_t st = saddr(ring) + (uint32_t)s * p.stage_bytes;
                        for (int j = 0; j < nkb; ++j) {
                            const uint32_t xa = st + (uint32_t)j * kb_bytes + RPW * kBoxBytes;
#pragma unroll
                            for (int kk = 0; kk < kBoxK / 16; ++kk) {
                                const uint64_t bd = sw128_desc(xa + kk * 32, 1024);
#pragma unroll
                                for (int r = 0; r < RPW; ++r) {
                                    const uint64_t ad =
                                        sw128_desc(st + (uint32_t)j * kb_bytes + (uint32_t)r * kBoxBytes + kk * 32, 1024);
                                    const uint32_t acc = (q | j | kk) != 0 ? 1u : 0u;
                                    asm volatile(
                                        "{\n\t.reg .pred pp;\n\tsetp.ne.b32 pp, %4, 0;\n\t"
                                        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, pp;\n\t}"
                                        ::"r"(tmem + (uint32_t)((ab * RPW + r) * NB)), "l"(ad), "l"(bd),
                                        "r"(kIdescN), "r"(acc));
                                }
                            }
                        }
                        mma_commit(&empty[s]);
                        if (++s == S) { s = 0; ph ^= 1; }
                    }
                    if (!dead) mma_commit(&acc_full[ab]);
                }
                mma_commit(&mma_done);
                if (!mbar_wait(&mma_done, 0)) set_err(a.err, kErrTimeout);
            }
            __syncwarp();
        } else {
            // ------------------------------------------------------------ epilogue
            const int ew = warp - 2;
            const int quarter = warp & 3;
            const int row = quarter * 32 + lane;
            const int T = a.T;
            // top-k: every 16-row chunk of a tile is scanned by all 128 epilogue
            // threads, 8 per row (each thread keeps one list per chunk position)
            constexpr int kNL = LISTS ? NB / 16 : 1;
            Key lst[kNL][kTopK];
            float lse_m[kNL], lse_s[kNL];         // per chunk position, with a.lse_part
            if constexpr (LISTS) {
#pragma unroll
                for (int cc = 0; cc < kNL; ++cc) {
                    key_clear(lst[cc]);
                    lse_m[cc] = -INFINITY;
                    lse_s[cc] = 0.f;
                }
            }
            // top-1: per warp and row the best so far (the same in every lane)
            constexpr int kN1 = TK == 1 ? NB : 1;
            float thr_v[kN1];
            int thr_i[kN1];
            if constexpr (TK == 1) {
#pragma unroll
                for (int t = 0; t < NB; ++t) { thr_v[t] = -INFINITY; thr_i[t] = 0x7FFFFFFF; }
                if (lane < NB) { s_val[ew][lane] = -INFINITY; s_id[ew][lane] = 0x7FFFFFFF; }
                __syncwarp();
            }
            bool dead = false;
            for (int i = 0; i < my_tiles; ++i) {
                const int tile = blockIdx.x / p.splits + i * tiles_step;
                const int ab = i & 1;
                if (!dead && !mbar_wait_warp(&acc_full[ab], (i >> 1) & 1, lim)) {
                    if (lane == 0) set_err(a.err, kErrTimeout);
                    dead = true;
                }
                const int u = tile * kTileM + row;
                const bool valid = !dead && u < a.n_units;
                if constexpr (TOPK) {
#pragma unroll
                    for (int cc = 0; cc < kNL; ++cc) {
                        const int c0 = 16 * cc;
                        if (c0 >= T) break;
                        float acc[16];
                        if (!dead) {
                            tc_fence_after();
                            tmem_ld16(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(ab * NB + c0), acc);
                        } else {
#pragma unroll
                            for (int tt = 0; tt < 16; ++tt) acc[tt] = 0.f;
                        }
                        if (valid && a.logits) {
#pragma unroll
                            for (int tt = 0; tt < 16; ++tt)
                                if (c0 + tt < T) a.logits[((size_t)(c0 + tt) * a.K + a.step - 1) * a.vocab + u] = acc[tt];
                        }
                        if constexpr (LISTS)
                            chunk_to_lists<8>(acc, row, &s_tr[0][0], tile, c0, T, a.n_units, dead, lst[cc],
                                              a.lse_part != nullptr, lse_m[cc], lse_s[cc]);
                        else
                            top1_scan<kN1>(acc, T, valid, u, thr_v, thr_i, s_val[ew], s_id[ew]);
                    }
                }
                // accumulator columns 16 at a time (all RPW sets of one chunk together)
                for (int c0 = 0; c0 < (TOPK ? 0 : NB); c0 += 16) {
                    float acc[RPW][16];
                    if (!dead) {
                        tc_fence_after();
#pragma unroll
                        for (int r = 0; r < RPW; ++r)
                            tmem_ld16(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((ab * RPW + r) * NB + c0),
                                      acc[r]);
                    }
                    if (c0 >= T) continue;
                    if (p.splits == 1) {
                        if (valid) {
#pragma unroll
                            for (int tt = 0; tt < 16; ++tt) {
                                if (c0 + tt >= T) break;
                                finish_unit<RPW>(a, c0 + tt, u, acc[0][tt], acc[RPW - 1][tt]);
                            }
                        }
                    } else if (valid) {
#pragma unroll
                        for (int r = 0; r < RPW; ++r)
#pragma unroll
                            for (int tt = 0; tt < 16; ++tt) {
                                if (c0 + tt >= T) break;
                                p.part[(((size_t)ks * RPW + r) * T + c0 + tt) * a.n_units + u] = acc[r][tt];
                            }
                    }
                }
                if (!dead) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acc_empty[ab]);
                }
                if constexpr (!TOPK) {
                    if (p.splits > 1 && !p.defer) {
                        __threadfence();
                        epi_sync();
                        if (threadIdx.x == 64) s_last = atomicAdd(&p.tile_ctr[tile], 1) == p.splits - 1;
                        epi_sync();
                        if (s_last) {
                            __threadfence();
                            if (valid) reduce_slices<RPW>(a, p, T, u);
                            if (threadIdx.x == 64) p.tile_ctr[tile] = 0;
                        }
                        epi_sync();
                    }
                }
            }
            if constexpr (LISTS) {
                // this CTA's list of every row; the cross-CTA merge is a separate kernel
#pragma unroll
                for (int cc = 0; cc < kNL; ++cc) {
                    lists_publish<8>(a, lst[cc], T, 16 * cc);
                    if (a.lse_part) lse_publish(a, lse_m[cc], lse_s[cc], T, 16 * cc);
                }
            } else if constexpr (TK == 1) {
                top1_join<kN1>(a, T, s_val, s_id, s_last);
            }
        }
    }

    if (warp == 0) return;
    tc_fence_before();
    stage_sync();
    tc_fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols));
}

// Split-K sums of a streamed projection with many activation rows: the
// projection kernel only publishes its slices, and this kernel adds them, one
// thread per (row t, unit u) with all slices loaded at once, in slice order
// (the same sums as the last-CTA path), and finishes the unit.  Inline in the
// projection, the last CTA of a tile would read T x 128 x splits partial sums
// through L2 while the tile's other work waits behind it.
// The grid is at most a few CTAs per SM, all resident at once (a grid of
// one CTA per output element came to many waves, which the next projection's
// early-started CTAs delayed further): each thread strides over the outputs.
constexpr int kFinishCtasPerSm = 4;
template <int RPW>
__global__ void __launch_bounds__(256) splitk_finish_kernel(const GemvArgs a, const float *part, int splits) {
    pdl_trigger();
    pdl_wait();
    const long total = (long)a.T * a.n_units;
    for (long e = (long)blockIdx.x * 256 + threadIdx.x; e < total; e += (long)gridDim.x * 256) {
        const int t = (int)(e / a.n_units), u = (int)(e % a.n_units);
        float v[kMaxSplits][RPW];
#pragma unroll
        for (int k = 0; k < kMaxSplits; ++k)
#pragma unroll
            for (int r = 0; r < RPW; ++r)
                v[k][r] = k < splits ? __ldcg(&part[(((size_t)k * RPW + r) * a.T + t) * a.n_units + u]) : 0.f;
        float s0 = 0.f, s1 = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxSplits; ++k)
            if (k < splits) {
                s0 += v[k][0];
                s1 += v[k][RPW - 1];
            }
        finish_unit<RPW>(a, t, u, s0, s1);
    }
}

// Cross-CTA top-k merge of the streamed LM head: one CTA (4 warps) per row;
// each warp merges a quarter of the row's candidates, warp 0 the four lists.
// This kernel runs once per row and step, right after the LM head, with
// HBM busy streaming the next step's weights: its instructions arrive at
// cache-miss speed, so it is written with rolled loops (one copy of the
// insertion and merge networks).
__global__ void __launch_bounds__(128) topk_merge_kernel(const GemvArgs a, int grid) {
    // It runs once per row while HBM streams the next weights, so each load
    // round trip waits behind full queues: the candidates and the h^ half of
    // the next fusion row are all requested before any is used, and the
    // E(token) half in one more batch once the token is known.
    constexpr int kB = 16;                          // candidates per thread in the first batch
    constexpr int kG = 4;                           // 8-element groups of a row per thread and batch
    __shared__ Key s_k[4][kTopK];
    __shared__ int s_tok;
    pdl_trigger();
    pdl_wait();
    const int t = blockIdx.x, w = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
    const int ncand = grid * kTopK, d = a.d, ng = d / 8;
    const float *pv = a.lm_part + (size_t)t * ncand;
    const int *pi = a.lm_part_id + (size_t)t * ncand;
    float cv[kB];
    int ci[kB];
#pragma unroll
    for (int b = 0; b < kB; ++b) {
        const int cc = tid + b * 128;
        cv[b] = cc < ncand ? __ldcg(pv + cc) : 0.f;
        ci[b] = cc < ncand ? __ldcg(pi + cc) : -1;
    }
    uint4 *x = a.next_fuse ? (uint4 *)(a.next_x + (size_t)t * 2 * d) : nullptr;
    if (x) {
        // the h^ half of the next decode step's fusion row does not depend on the token
        const float4 *h = (const float4 *)(a.src + (size_t)t * d);
#pragma unroll 1
        for (int c0 = 0; c0 < ng; c0 += 128 * kG) {
            float4 v0[kG], v1[kG];
#pragma unroll
            for (int q = 0; q < kG; ++q) {
                const int c = c0 + tid + q * 128;
                v0[q] = c < ng ? __ldcg(h + 2 * c) : make_float4(0.f, 0.f, 0.f, 0.f);
                v1[q] = c < ng ? __ldcg(h + 2 * c + 1) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int q = 0; q < kG; ++q) {
                const int c = c0 + tid + q * 128;
                if (c < ng)
                    x[ng + c] = make_uint4(pack_bf16x2(v0[q].x, v0[q].y), pack_bf16x2(v0[q].z, v0[q].w),
                                           pack_bf16x2(v1[q].x, v1[q].y), pack_bf16x2(v1[q].z, v1[q].w));
            }
        }
    }
    Key l[kTopK];
    key_clear(l);
#pragma unroll 1
    for (int b = 0; b < kB; ++b)
        if (ci[b] >= 0) key_insert(l, pack_best(cv[b], ci[b]));
#pragma unroll 1
    for (int cc = tid + kB * 128; cc < ncand; cc += 128) key_insert(l, pack_best(__ldcg(pv + cc), __ldcg(pi + cc)));
#pragma unroll 1
    for (int m = 1; m < 32; m <<= 1) key_merge_xor(l, m);
    if (lane == 0) {
#pragma unroll
        for (int i = 0; i < kTopK; ++i) s_k[w][i] = l[i];
    }
    __syncthreads();
    if (w == 0) {
#pragma unroll
        for (int i = 0; i < kTopK; ++i) l[i] = lane < 4 ? s_k[lane][i] : 0ull;
        // every lane ends with the merged list (write_row reads rank r from lane r)
#pragma unroll 1
        for (int m = 1; m < 32; m <<= 1) key_merge_xor(l, m);
        write_row(a, t, l);
        if (lane == 0) {
            float v;
            int id;
            unpack_best(l[0], v, id);
            s_tok = id;
        }
    }
    if (x) {
        // the token's half of the next decode step's fusion row: E(token)
        __syncthreads();
        const uint4 *e = (const uint4 *)((const uint16_t *)a.embed + (size_t)token_ok(a, s_tok) * d);
#pragma unroll 1
        for (int c0 = 0; c0 < ng; c0 += 128 * kG) {
            uint4 r[kG];
#pragma unroll
            for (int q = 0; q < kG; ++q) {
                const int c = c0 + tid + q * 128;
                r[q] = c < ng ? __ldg(e + c) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int q = 0; q < kG; ++q) {
                const int c = c0 + tid + q * 128;
                if (c < ng) x[c] = r[q];
            }
        }
    }
}

// Split-K sums of one activation row per CTA (Store and Resid epilogues of a
// streamed projection), in slice order like splitk_finish_kernel, and the
// next projection's activation row: RMSNorm of the finished row with
// next_gain (or the row as it is when next_gain is null), rounded to bf16,
// into next_x.  One kernel instead of the finish and the next row
// preparation.  It sits on the critical path between two projections, so a
// thread holds its values in registers and issues all its loads at once (the
// gain, a weight, before the dependency wait).  n_units <= kRowMaxUnits.
// VEC float4 groups per thread, at most SPL slices (instances keep the
// loads in flight within the register budget of 1024 threads).
constexpr int kRowThreads = 1024;
constexpr int kRowMaxUnits = kRowThreads * 4 * 2;           // 8192
template <int kRowVec, int SPL>
__global__ void __launch_bounds__(kRowThreads) splitk_finish_row_kernel(const GemvArgs a, const float *part,
                                                                      int splits) {
    __shared__ float red[kRowThreads / 32];
    pdl_trigger();
    const int t = blockIdx.x, n = a.n_units, tid = threadIdx.x;
    const uint16_t *g = a.next_norm ? (const uint16_t *)a.next_gain : nullptr;
    uint2 gw[kRowVec];
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
        const int u = (tid + i * kRowThreads) * 4;
        gw[i] = g && u < n ? __ldg((const uint2 *)(g + u)) : make_uint2(0u, 0u);
    }
    pdl_wait();
    const int rrow = a.epi == kEpiResid && a.resid_prefill_rows ? t * a.max_new + clamp_n(a, t) - 1 : t;
    float4 v[kRowVec][SPL], q[kRowVec];
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
        const int u = (tid + i * kRowThreads) * 4;
        if (u >= n) continue;
#pragma unroll
        for (int k = 0; k < SPL; ++k)
            if (k < splits) v[i][k] = __ldcg((const float4 *)&part[((size_t)k * a.T + t) * n + u]);
        if (a.epi == kEpiResid) q[i] = __ldcg((const float4 *)&a.resid[(size_t)rrow * a.out_ld + u]);
    }
    float4 r[kRowVec];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
        const int u = (tid + i * kRowThreads) * 4;
        r[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (u >= n) continue;
#pragma unroll
        for (int k = 0; k < SPL; ++k)
            if (k < splits) {
                r[i].x += v[i][k].x;
                r[i].y += v[i][k].y;
                r[i].z += v[i][k].z;
                r[i].w += v[i][k].w;
            }
        if (a.epi == kEpiResid) {
            r[i].x += q[i].x;
            r[i].y += q[i].y;
            r[i].z += q[i].z;
            r[i].w += q[i].w;
            if (a.hidden_out) {
                float *ho = a.hidden_out + ((size_t)t * a.K + a.step - 1) * a.d + u;
                ho[0] = r[i].x;
                ho[1] = r[i].y;
                ho[2] = r[i].z;
                ho[3] = r[i].w;
            }
        }
        *(float4 *)&a.out[(size_t)t * a.out_ld + u] = r[i];
        ss = fmaf(r[i].x, r[i].x, ss);
        ss = fmaf(r[i].y, r[i].y, ss);
        ss = fmaf(r[i].z, r[i].z, ss);
        ss = fmaf(r[i].w, r[i].w, ss);
    }
    if (!a.next_norm) return;
    float inv = 1.f;
    if (g) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
        if ((tid & 31) == 0) red[tid >> 5] = ss;
    }
    __syncthreads();
    if (g) {
        float tot = 0.f;
#pragma unroll
        for (int i = 0; i < kRowThreads / 32; ++i) tot += red[i];
        inv = 1.0f / sqrtf(tot / (float)n + a.eps);
    }
    uint2 *x = (uint2 *)(a.next_x + (size_t)t * n);
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
        const int u = (tid + i * kRowThreads) * 4;
        if (u >= n) continue;
        float y[4] = {r[i].x, r[i].y, r[i].z, r[i].w};
        if (g) {
            y[0] = y[0] * inv * bf16lo(gw[i].x);
            y[1] = y[1] * inv * bf16hi(gw[i].x);
            y[2] = y[2] * inv * bf16lo(gw[i].y);
            y[3] = y[3] * inv * bf16hi(gw[i].y);
        }
        x[u / 4] = make_uint2(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]));
    }
}

// Activation rows of a projection as a bf16 buffer X [T][kin] (the streamed
// kernel's B operand): embedding gather and concatenation, or RMSNorm with
// its gain, rounded to bf16.  One CTA of 256 threads per row.
__global__ void __launch_bounds__(256) prep_x_kernel(const GemvArgs a, uint16_t *X) {
    __shared__ float red[8];
    pdl_trigger();
    pdl_wait();
    // 16-byte vectors (d is a multiple of 8): a thread issues its loads of a
    // row before using any
    const int t = blockIdx.x, tid = threadIdx.x;
    const int d = a.d, kin = a.kin;
    uint4 *xr = (uint4 *)(X + (size_t)t * kin);
    if (a.pro == kProNorm) {
        const int sr = a.src_prefill_rows ? (t * a.max_new + clamp_n(a, t) - 1) : t;
        const float4 *src = (const float4 *)(a.src + (size_t)sr * d);
        float inv = 1.f;
        if (a.gain) {
            float ss = 0.f;
            for (int c = tid; c < d / 4; c += 256) {
                const float4 v = __ldcg(src + c);
                ss = fmaf(v.x, v.x, ss);
                ss = fmaf(v.y, v.y, ss);
                ss = fmaf(v.z, v.z, ss);
                ss = fmaf(v.w, v.w, ss);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
            if ((tid & 31) == 0) red[tid >> 5] = ss;
            __syncthreads();
            float tot = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) tot += red[i];
            inv = 1.0f / sqrtf(tot / (float)d + a.eps);
        }
        const uint4 *g = (const uint4 *)a.gain;
        for (int c = tid; c < d / 8; c += 256) {
            const float4 v0 = __ldcg(src + 2 * c), v1 = __ldcg(src + 2 * c + 1);
            float y[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            if (g) {
                const uint4 gw = __ldg(g + c);
                const uint32_t gg[4] = {gw.x, gw.y, gw.z, gw.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    y[2 * i] = y[2 * i] * inv * bf16lo(gg[i]);
                    y[2 * i + 1] = y[2 * i + 1] * inv * bf16hi(gg[i]);
                }
            }
            xr[c] = make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]), pack_bf16x2(y[4], y[5]),
                               pack_bf16x2(y[6], y[7]));
        }
    } else if (a.pro == kProFuseDecode) {
        const int tok = token_ok(a, a.draft[t * a.K + a.step - 2]);
        const uint4 *e = (const uint4 *)((const uint16_t *)a.embed + (size_t)tok * d);
        const float4 *h = (const float4 *)(a.src + (size_t)t * d);
        for (int c = tid; c < d / 8; c += 256) {
            const uint4 ev = __ldg(e + c);
            const float4 h0 = __ldcg(h + 2 * c), h1 = __ldcg(h + 2 * c + 1);
            xr[c] = ev;
            xr[d / 8 + c] = make_uint4(pack_bf16x2(h0.x, h0.y), pack_bf16x2(h0.z, h0.w), pack_bf16x2(h1.x, h1.y),
                                       pack_bf16x2(h1.z, h1.w));
        }
    } else if (a.pro == kProFusePrefill) {
        const int b = t / a.max_new, r = t % a.max_new;
        const bool valid = r < clamp_n(a, b);
        const int tok = valid ? token_ok(a, a.tokens[b * a.max_new + r]) : 0;
        const uint4 *e = (const uint4 *)((const uint16_t *)a.embed + (size_t)tok * d);
        const uint4 *h = (const uint4 *)((const uint16_t *)a.hidden_in + ((size_t)b * a.max_new + r) * d);
        const uint4 z = make_uint4(0u, 0u, 0u, 0u);
        for (int c = tid; c < d / 8; c += 256) {
            xr[c] = valid ? __ldg(e + c) : z;
            xr[d / 8 + c] = valid ? __ldg(h + c) : z;
        }
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

template <int NB>
cudaError_t dispatch_tc(const GemvArgs &a, const TcPlan &p, const CUtensorMap &m, int grid, size_t smem,
                        cudaStream_t s, bool pdl) {
    const dim3 g(grid), b(kTcThreads);
    if (a.epi == kEpiTopK && a.pro == kProNorm) {
        if (a.topk == 1 && a.best != nullptr)
            return launch_k(gemv_tc_kernel<NB, 1, 1, kProNorm>, g, b, smem, s, pdl, a, p, m);
        return launch_k(gemv_tc_kernel<NB, 1, 2, kProNorm>, g, b, smem, s, pdl, a, p, m);
    }
    if (a.epi == kEpiSwiGLU && a.pro == kProNorm)
        return launch_k(gemv_tc_kernel<NB, 2, 0, kProNorm>, g, b, smem, s, pdl, a, p, m);
    if (a.epi == kEpiStore || a.epi == kEpiResid) {
        switch (a.pro) {
            case kProFusePrefill: return launch_k(gemv_tc_kernel<NB, 1, 0, kProFusePrefill>, g, b, smem, s, pdl, a, p, m);
            case kProFuseDecode: return launch_k(gemv_tc_kernel<NB, 1, 0, kProFuseDecode>, g, b, smem, s, pdl, a, p, m);
            case kProNorm: return launch_k(gemv_tc_kernel<NB, 1, 0, kProNorm>, g, b, smem, s, pdl, a, p, m);
            case kProCopy: return launch_k(gemv_tc_kernel<NB, 1, 0, kProCopy>, g, b, smem, s, pdl, a, p, m);
        }
    }
    return cudaErrorInvalidValue;
}

template <int NB>
cudaError_t set_tc_attrs(int bytes) {
    cudaError_t e = cudaSuccess;
#define PRISM_TC_ATTR(RPW, TK, PRO)                                                                      \
    if (e == cudaSuccess)                                                                                \
        e = cudaFuncSetAttribute(gemv_tc_kernel<NB, RPW, TK, PRO>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    PRISM_TC_ATTR(1, 2, kProNorm)
    bytes = (int)kTcSmemLarge;
    PRISM_TC_ATTR(1, 1, kProNorm)
    PRISM_TC_ATTR(2, 0, kProNorm)
    PRISM_TC_ATTR(1, 0, kProFusePrefill)
    PRISM_TC_ATTR(1, 0, kProFuseDecode)
    PRISM_TC_ATTR(1, 0, kProNorm)
    PRISM_TC_ATTR(1, 0, kProCopy)
#undef PRISM_TC_ATTR
    return e;
}

// Split count and ring for one projection: the fewest K blocks on the
// busiest CTA, then the fewest splits.
bool tc_plan(const GemvArgs &a, int sms, TcPlan &p, int &grid, size_t &smem) {
    if (a.T < 1 || a.T > kMmaN || a.kin % 8 || a.n_units < 1) return false;
    if ((a.epi == kEpiTopK || a.epi == kEpiSwiGLU) && a.pro != kProNorm) return false;
    const int RPW = a.epi == kEpiSwiGLU ? 2 : 1;
    const int NB = a.T <= 8 ? 8 : 16;
    const int nkb = (a.kin + kBoxK - 1) / kBoxK;
    const int n_tiles = (a.n_units + kTileM - 1) / kTileM;
    const int max_s = a.epi == kEpiTopK ? 1 : kMaxSplits;
    long best = -1;
    int best_s = 0, best_ctas = 0;
    for (int sp = 1; sp <= max_s && sp <= nkb; ++sp) {
        const int per = (nkb + sp - 1) / sp;
        if ((size_t)NB * 128 * per > kXBudget) continue;
        int ctas = sms / sp;
        if (ctas > n_tiles) ctas = n_tiles;
        if (ctas < 1) break;
        const long cost = (long)((n_tiles + ctas - 1) / ctas) * per;
        if (best < 0 || cost < best) { best = cost; best_s = sp; best_ctas = ctas; }
    }
    if (best < 0) return false;
    p.n_tiles = n_tiles;
    p.nkb = nkb;
    p.splits = best_s;
    p.x_bytes = (uint32_t)(NB * 128 * ((nkb + best_s - 1) / best_s));
    const bool lists = a.epi == kEpiTopK && !(a.topk == 1 && a.best != nullptr);
    const size_t room = (lists ? kTcSmem : kTcSmemLarge) - 1024 - p.x_bytes;
    // 48 KB stages when three fit, 32 KB ones when four fit, else 16 KB
    p.kb_per_stage = RPW != 1 ? 1 : room >= 3 * 3 * (size_t)kBoxBytes ? 3 : room >= 4 * 2 * (size_t)kBoxBytes ? 2 : 1;
    p.stage_bytes = (uint32_t)p.kb_per_stage * RPW * kBoxBytes;
    p.stages = (int)(room / p.stage_bytes);
    if (p.stages > kTcMaxStages) p.stages = kTcMaxStages;
    if (p.stages < 2) return false;
    if (a.even_waves && a.epi == kEpiTopK && best_s == 1) {
        const int waves = (n_tiles + best_ctas - 1) / best_ctas;
        best_ctas = (n_tiles + waves - 1) / waves;
    }
    grid = best_ctas * best_s;
    smem = 1024 + (size_t)p.stages * p.stage_bytes + p.x_bytes;
    return true;
}

}  // namespace

template <int NB, int RPW, int TK>
cudaError_t set_tcs_attr(int bytes) {
    return cudaFuncSetAttribute(gemv_tcs_kernel<NB, RPW, TK>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

int tcs_nb(int T, int RPW, bool topk) {
    int nb = 16;
    while (nb < T) nb *= 2;
    const int cap = topk ? 64 : (RPW == 2 ? 128 : 256);
    return nb <= cap ? nb : 0;
}

// The selection a streamed launch makes: 0 none, 1 the packed top-1 (one
// 16-row tile of activation rows), 2 top-k lists.
int tcs_tk(const GemvArgs &a, int NB) {
    if (a.epi != kEpiTopK) return 0;
    return a.stream_top1 && a.topk == 1 && a.best && NB == 16 ? 1 : 2;
}

// static shared memory of a streamed kernel (barriers, top-1 bests, top-k lists)
size_t tcs_static(int NB, int tk) {
    return 512 + (tk == 2 ? (size_t)16 * kTrMax * 4 : tk == 1 ? (size_t)4 * NB * 8 : 64);
}

bool tcs_plan(const GemvArgs &a, int sms, TcPlan &p, int &grid, size_t &smem, int &NB) {
    const bool topk = a.epi == kEpiTopK;
    const int RPW = a.epi == kEpiSwiGLU ? 2 : 1;
    if (a.T < 1 || a.kin % 8 || a.n_units < 1) return false;
    NB = tcs_nb(a.T, RPW, topk);
    if (!NB) return false;
    const int nkb = (a.kin + kBoxK - 1) / kBoxK;
    const int n_tiles = (a.n_units + kTileM - 1) / kTileM;
    // No split when the tiles alone already occupy most SMs in one wave: a
    // split then buys little streaming time and costs a finish pass over
    // every partial sum (gate/up at 112 tiles: 2440 -> 2197 us per round at
    // batch 64, 1663 -> 1615 us at batch 16)
    const bool one_wave = n_tiles <= sms && 10 * n_tiles >= 7 * sms;
    const int max_s = topk || one_wave ? 1 : kMaxSplits;
    long best = -1;
    int best_s = 0, best_ctas = 0;
    for (int sp = 1; sp <= max_s && sp <= nkb; ++sp) {
        const int per = (nkb + sp - 1) / sp;
        int ctas = sms / sp;
        if (ctas > n_tiles) ctas = n_tiles;
        if (ctas < 1) break;
        const long cost = (long)((n_tiles + ctas - 1) / ctas) * per;
        if (best < 0 || cost < best) { best = cost; best_s = sp; best_ctas = ctas; }
    }
    if (best < 0) return false;
    const size_t kb_bytes = (size_t)RPW * kBoxBytes + (size_t)NB * 128;
    // the packed top-1 instance takes the larger budget (its ring is what an
    // LM head at batch 1 gains by streaming its row); the others 212 KB at most
    const int tk = tcs_tk(a, NB);
    const size_t dyn = tk == 1 ? kTcSmemLarge
                               : std::min((size_t)220 * 1024 - tcs_static(NB, tk), kTcSmem);
    const size_t room = dyn - 1024;
    p.n_tiles = n_tiles;
    p.nkb = nkb;
    p.splits = best_s;
    // the largest stage of up to 64 KB of which four still fit (larger
    // stages stream faster than more, smaller ones)
    p.kb_per_stage = 1;
    for (int k = 3; k >= 2; --k)
        if (k * kb_bytes <= 64 * 1024 && room >= 4 * (size_t)k * kb_bytes) { p.kb_per_stage = k; break; }
    p.stage_bytes = (uint32_t)(p.kb_per_stage * kb_bytes);
    p.x_bytes = 0;
    p.stages = (int)(room / p.stage_bytes);
    if (p.stages > kTcMaxStages) p.stages = kTcMaxStages;
    if (p.stages < 2) return false;
    if (a.even_waves && topk && best_s == 1) {
        const int waves = (n_tiles + best_ctas - 1) / best_ctas;
        best_ctas = (n_tiles + waves - 1) / waves;
    }
    grid = best_ctas * best_s;
    smem = 1024 + (size_t)p.stages * p.stage_bytes;
    return true;
}

template <int NB>
cudaError_t dispatch_tcs(const GemvArgs &a, const TcPlan &p, const CUtensorMap &mw, const CUtensorMap &mx, int grid,
                         size_t smem, cudaStream_t s, bool pdl) {
    const dim3 g(grid), b(kTcThreads);
    if (a.epi == kEpiTopK) {
        if constexpr (NB == 16)
            if (tcs_tk(a, NB) == 1) return launch_k(gemv_tcs_kernel<NB, 1, 1>, g, b, smem, s, pdl, a, p, mw, mx);
        if constexpr (NB <= 64) return launch_k(gemv_tcs_kernel<NB, 1, 2>, g, b, smem, s, pdl, a, p, mw, mx);
        return cudaErrorInvalidValue;
    }
    if (a.epi == kEpiSwiGLU) {
        if constexpr (NB <= 128) return launch_k(gemv_tcs_kernel<NB, 2, 0>, g, b, smem, s, pdl, a, p, mw, mx);
        return cudaErrorInvalidValue;
    }
    return launch_k(gemv_tcs_kernel<NB, 1, 0>, g, b, smem, s, pdl, a, p, mw, mx);
}

cudaError_t prepare_gemv_tc_kernels() {
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess) return e;
        if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
        g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    }
    cudaError_t e = set_tc_attrs<8>((int)kTcSmem);
    if (e == cudaSuccess) e = set_tc_attrs<16>((int)kTcSmem);
    const int b = (int)kTcSmem;
    // per instance: what the 220 KB budget leaves after its static shared memory
#define PRISM_TCS(NB, RPW, TK)                                                                          \
    if (e == cudaSuccess)                                                                               \
        e = set_tcs_attr<NB, RPW, TK>((int)std::min((size_t)b, (size_t)220 * 1024 - tcs_static(NB, TK)));
    PRISM_TCS(16, 1, 0) PRISM_TCS(32, 1, 0) PRISM_TCS(64, 1, 0) PRISM_TCS(128, 1, 0)
    PRISM_TCS(256, 1, 0) PRISM_TCS(16, 2, 0) PRISM_TCS(32, 2, 0) PRISM_TCS(64, 2, 0)
    PRISM_TCS(128, 2, 0) PRISM_TCS(16, 1, 2) PRISM_TCS(32, 1, 2) PRISM_TCS(64, 1, 2)
#undef PRISM_TCS
    if (e == cudaSuccess) e = set_tcs_attr<16, 1, 1>((int)kTcSmemLarge);
    return e;
}

cudaError_t make_weight_map(CUtensorMap *m, const void *W, int rows, int kin) {
    if (!g_encode) return cudaErrorNotSupported;
    if (((uintptr_t)W & 15) || (kin % 8) || rows < 1) return cudaErrorInvalidValue;
    cuuint64_t dims[2] = {(cuuint64_t)kin, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)kin * 2};
    cuuint32_t box[2] = {(cuuint32_t)kBoxK, (cuuint32_t)kTileM};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(W), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_cache_map(CUtensorMap *m, const void *cache, int heads, int max_ctx, int D, int rows_per_box) {
    if (!g_encode) return cudaErrorNotSupported;
    if (((uintptr_t)cache & 15) || (D % 64) || heads < 1 || max_ctx < 1 || rows_per_box < 1 || rows_per_box > 256)
        return cudaErrorInvalidValue;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)max_ctx, (cuuint64_t)heads};
    cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)max_ctx * D * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)rows_per_box, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(cache), dims, strides, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

bool gemv_tc_supported(const GemvArgs &a, int sms) {
    TcPlan p{};
    int grid;
    size_t smem;
    return tc_plan(a, sms, p, grid, smem);
}

int gemv_tc_tiles(const GemvArgs &a) { return (a.n_units + kTileM - 1) / kTileM; }

bool gemv_tcs_supported(const GemvArgs &a, int sms) {
    TcPlan p{};
    int grid, NB;
    size_t smem;
    return tcs_plan(a, sms, p, grid, smem, NB);
}

size_t gemv_tcs_workspace_floats(const GemvArgs &a, int sms) {
    TcPlan p{};
    int grid, NB;
    size_t smem;
    if (!tcs_plan(a, sms, p, grid, smem, NB) || p.splits == 1) return 0;
    return (size_t)p.splits * (a.epi == kEpiSwiGLU ? 2 : 1) * a.T * a.n_units;
}

cudaError_t launch_gemv_tcs(const GemvArgs &a, const CUtensorMap &mw, int sms, float *part, int *tile_ctr,
                            uint16_t *xbuf, cudaStream_t s, bool pdl, bool *next_done) {
    if (next_done) *next_done = false;
    TcPlan p{};
    int grid, NB;
    size_t smem;
    if (!tcs_plan(a, sms, p, grid, smem, NB)) return cudaErrorInvalidValue;
    p.part = part;
    p.tile_ctr = tile_ctr;
    p.defer = p.splits > 1;
    if (p.splits > 1 && (!part || !tile_ctr)) return cudaErrorInvalidValue;
    // the activation rows as a bf16 [T][kin] buffer: the copy prologue's
    // source as it is, otherwise written by prep_x_kernel
    const void *x = a.act;
    cudaError_t e = cudaSuccess;
    if (a.pro != kProCopy) {
        if (!xbuf) return cudaErrorInvalidValue;
        e = launch_k(prep_x_kernel, dim3(a.T), dim3(256), 0, s, pdl, a, xbuf);
        if (e != cudaSuccess) return e;
        x = xbuf;
        pdl = true;
    }
    CUtensorMap mx;
    if (!g_encode) return cudaErrorNotSupported;
    {
        cuuint64_t dims[2] = {(cuuint64_t)a.kin, (cuuint64_t)a.T};
        cuuint64_t strides[1] = {(cuuint64_t)a.kin * 2};
        cuuint32_t box[2] = {(cuuint32_t)kBoxK, (cuuint32_t)NB};
        cuuint32_t estr[2] = {1, 1};
        if (((uintptr_t)x & 15) ||
            g_encode(&mx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(x), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    switch (NB) {
        case 16: e = dispatch_tcs<16>(a, p, mw, mx, grid, smem, s, pdl); break;
        case 32: e = dispatch_tcs<32>(a, p, mw, mx, grid, smem, s, pdl); break;
        case 64: e = dispatch_tcs<64>(a, p, mw, mx, grid, smem, s, pdl); break;
        case 128: e = dispatch_tcs<128>(a, p, mw, mx, grid, smem, s, pdl); break;
        default: e = dispatch_tcs<256>(a, p, mw, mx, grid, smem, s, pdl); break;
    }
    if (e == cudaSuccess && a.epi == kEpiTopK && tcs_tk(a, NB) == 2) {
        GemvArgs m = a;
        m.next_fuse = a.next_fuse && a.next_x && a.d % 8 == 0;
        if (!a.defer_merge) e = launch_k(topk_merge_kernel, dim3(a.T), dim3(128), 0, s, true, m, grid);
        if (e == cudaSuccess && next_done) *next_done = !a.defer_merge && m.next_fuse != 0;
    }
    if (e == cudaSuccess && p.defer) {
        if (a.epi != kEpiSwiGLU && a.next_norm && a.next_x && a.n_units % 4 == 0 && a.n_units <= kRowMaxUnits) {
            // one CTA per row: the sums, then the next projection's normalised row
            const float *pp = (const float *)part;
            const dim3 rg(a.T), rb(kRowThreads);
            if (a.n_units <= kRowThreads * 4)
                e = p.splits <= 2   ? launch_k(splitk_finish_row_kernel<1, 2>, rg, rb, 0, s, true, a, pp, p.splits)
                    : p.splits <= 4 ? launch_k(splitk_finish_row_kernel<1, 4>, rg, rb, 0, s, true, a, pp, p.splits)
                                    : launch_k(splitk_finish_row_kernel<1, 8>, rg, rb, 0, s, true, a, pp, p.splits);
            else
                e = p.splits <= 2   ? launch_k(splitk_finish_row_kernel<2, 2>, rg, rb, 0, s, true, a, pp, p.splits)
                    : p.splits <= 4 ? launch_k(splitk_finish_row_kernel<2, 4>, rg, rb, 0, s, true, a, pp, p.splits)
                                    : launch_k(splitk_finish_row_kernel<2, 8>, rg, rb, 0, s, true, a, pp, p.splits);
            if (e == cudaSuccess && next_done) *next_done = true;
        } else {
            long nb = ((long)a.T * a.n_units + 255) / 256;
            if (nb > (long)kFinishCtasPerSm * sms) nb = (long)kFinishCtasPerSm * sms;
            const dim3 fg((unsigned)nb);
            e = a.epi == kEpiSwiGLU
                    ? launch_k(splitk_finish_kernel<2>, fg, dim3(256), 0, s, true, a, (const float *)part, p.splits)
                    : launch_k(splitk_finish_kernel<1>, fg, dim3(256), 0, s, true, a, (const float *)part, p.splits);
        }
    }
    return e;
}

size_t gemv_tc_workspace_floats(const GemvArgs &a, int sms) {
    TcPlan p{};
    int grid;
    size_t smem;
    if (!tc_plan(a, sms, p, grid, smem) || p.splits == 1) return 0;
    return (size_t)p.splits * (a.epi == kEpiSwiGLU ? 2 : 1) * a.T * a.n_units;
}

cudaError_t launch_gemv_tc(const GemvArgs &a, const CUtensorMap &m, int sms, float *part, int *tile_ctr,
                           cudaStream_t s, bool pdl) {
    TcPlan p{};
    int grid;
    size_t smem;
    if (!tc_plan(a, sms, p, grid, smem)) return cudaErrorInvalidValue;
    p.part = part;
    p.tile_ctr = tile_ctr;
    if (p.splits > 1 && (!part || !tile_ctr)) return cudaErrorInvalidValue;
    return a.T <= 8 ? dispatch_tc<8>(a, p, m, grid, smem, s, pdl) : dispatch_tc<16>(a, p, m, grid, smem, s, pdl);
}

}  // namespace prism
