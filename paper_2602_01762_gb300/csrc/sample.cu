// Sampled drafting and speculative-sampling acceptance (Sec. 2 at a
// temperature T > 0), sm_103a.
//
// Drafting: after the LM head of step k has written its logits z, each draft
// token is drawn from p_draft = softmax(z / T) by the Gumbel-max rule: the
// argmax of z_i / T + G_i with G_i = -log(-log U_i) is distributed as
// softmax(z / T).  The logits of one row are split over many CTAs; each keeps
// a running (max, sum of exp) of z / T and its best perturbed score, and the
// last CTA of the row merges them in CTA order and writes the token and
// lse = log sum_i exp(z_i / T), so that p_draft(x) = exp(z_x / T - lse).
//
// Acceptance: one CTA per sequence walks the K drafted positions; x is
// accepted when r * p_draft(x) < p_target(x) (r < min(1, p_target /
// p_draft)); the first rejected position draws its replacement from
// max(0, p_target - p_draft) by an inverse-CDF search over the vocabulary (a
// residual that is zero everywhere falls back to p_target); after a full
// accept the extra token is drawn from p_target at position K.
//
// Random numbers: the n-th output of SplitMix64 (Steele, Lea and Flood,
// OOPSLA 2014) started from state `seed`, with the counter
// n = (stream << 60) | (b << 40) | (k << 32) | i, mapped to (0, 1) as
// ((x >> 41) + 1/2) / 2^23 (exact in float32).  Streams: 1 draft sampling
// (i = token id), 2 the acceptance test of position k, 3 the token drawn at
// position k (k = K: the extra token after a full accept).
#include "common.cuh"

namespace prism {

namespace {

constexpr int kSampleThreads = 256;
constexpr int kAcceptThreads = 1024;

__device__ __forceinline__ uint64_t splitmix_at(uint64_t seed, uint64_t n) {
    uint64_t z = seed + (n + 1) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ float uniform01(uint64_t seed, uint32_t stream, uint32_t b, uint32_t k, uint32_t i) {
    const uint64_t n = ((uint64_t)stream << 60) | ((uint64_t)b << 40) | ((uint64_t)k << 32) | (uint64_t)i;
    return ((float)(splitmix_at(seed, n) >> 41) + 0.5f) * (1.0f / 8388608.0f);
}

// (max, sum of exp(v - max)) of two parts, combined.
__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2) {
    if (m2 == -INFINITY) return;
    if (m == -INFINITY) { m = m2; s = s2; return; }
    if (m2 > m) { s = s * expf(m - m2) + s2; m = m2; }
    else s += s2 * expf(m2 - m);
}
// better perturbed score: larger, ties to the lower id
__device__ __forceinline__ bool score_better(float v, int i, float bv, int bi) { return v > bv || (v == bv && i < bi); }

// grid (blocks per row, B); a CTA takes `chunk` consecutive logits of row b.
__global__ void __launch_bounds__(kSampleThreads) sample_kernel(const SampleArgs a) {
    __shared__ float s_m[kSampleThreads / 32], s_s[kSampleThreads / 32], s_v[kSampleThreads / 32];
    __shared__ int s_i[kSampleThreads / 32];
    __shared__ int s_last;
    pdl_trigger();
    pdl_wait();
    const int b = blockIdx.y, blk = blockIdx.x, nblk = gridDim.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint64_t seed = *a.seed;
    const float inv_t = 1.0f / a.temperature;
    const float *z = a.logits + ((size_t)b * a.K + a.step - 1) * a.V;
    const int lo = blk * a.chunk, hi = min(a.V, lo + a.chunk);
    float m = -INFINITY, s = 0.f, bv = -INFINITY;
    int bi = 0x7FFFFFFF;
    for (int i = lo + tid; i < hi; i += kSampleThreads) {
        const float v = z[i] * inv_t;
        lse_merge(m, s, v, 1.f);
        const float u = uniform01(seed, 1, (uint32_t)b, (uint32_t)(a.step - 1), (uint32_t)i);
        const float g = v - logf(-logf(u));
        if (score_better(g, i, bv, bi)) { bv = g; bi = i; }
    }
    // block: warps in a fixed tree, then warp 0 over the warps in order
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o), s2 = __shfl_xor_sync(0xFFFFFFFFu, s, o);
        const float v2 = __shfl_xor_sync(0xFFFFFFFFu, bv, o);
        const int i2 = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
        lse_merge(m, s, m2, s2);
        if (score_better(v2, i2, bv, bi)) { bv = v2; bi = i2; }
    }
    if (lane == 0) { s_m[warp] = m; s_s[warp] = s; s_v[warp] = bv; s_i[warp] = bi; }
    __syncthreads();
    if (tid == 0) {
        for (int w = 1; w < kSampleThreads / 32; ++w) {
            lse_merge(m, s, s_m[w], s_s[w]);
            if (score_better(s_v[w], s_i[w], bv, bi)) { bv = s_v[w]; bi = s_i[w]; }
        }
        float *part = a.part + ((size_t)b * a.max_blocks + blk) * 4;
        part[0] = m;
        part[1] = s;
        part[2] = bv;
        part[3] = __int_as_float(bi);
        __threadfence();
        s_last = atomicAdd(a.counter + b, 1) == nblk - 1;
    }
    __syncthreads();
    if (!s_last || warp != 0) return;
    // the row's last CTA: lane l merges partials l, l + 32, ... (loads first),
    // then the lanes merge in a fixed butterfly order
    __threadfence();
    constexpr int kPer = kSampleMaxBlocks / 32;
    float pm[kPer], ps[kPer], pv[kPer];
    int pi[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int q = lane + 32 * i;
        const float4 v = q < nblk ? __ldcg((const float4 *)(a.part + ((size_t)b * a.max_blocks + q) * 4))
                                  : make_float4(-INFINITY, 0.f, -INFINITY, __int_as_float(0x7FFFFFFF));
        pm[i] = v.x;
        ps[i] = v.y;
        pv[i] = v.z;
        pi[i] = __float_as_int(v.w);
    }
    float M = -INFINITY, S = 0.f, BV = -INFINITY;
    int BI = 0x7FFFFFFF;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        lse_merge(M, S, pm[i], ps[i]);
        if (score_better(pv[i], pi[i], BV, BI)) { BV = pv[i]; BI = pi[i]; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, M, o), s2 = __shfl_xor_sync(0xFFFFFFFFu, S, o);
        const float v2 = __shfl_xor_sync(0xFFFFFFFFu, BV, o);
        const int i2 = __shfl_xor_sync(0xFFFFFFFFu, BI, o);
        lse_merge(M, S, m2, s2);
        if (score_better(v2, i2, BV, BI)) { BV = v2; BI = i2; }
    }
    if (lane == 0) {
        const size_t o = (size_t)b * a.K + a.step - 1;
        a.draft[o] = BI;
        a.lse[o] = M + logf(S);
        a.counter[b] = 0;
    }
}

// Inverse-CDF draw over w(0 .. V) (non-negative, not normalised), by the whole
// CTA: thread t sums the contiguous chunk t, an inclusive scan gives the
// chunk bounds, and the thread whose bounds hold u * total searches its
// chunk.  Returns the token in every thread, or -1 when every weight is 0.
template <typename W>
__device__ int draw_block(W w, int V, float u, float *s_scan, int *s_tok) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int C = (V + kAcceptThreads - 1) / kAcceptThreads;
    const int lo = min(V, tid * C), hi = min(V, lo + C);
    float sum = 0.f;
    int last = -1;
    for (int i = lo; i < hi; ++i) {
        const float wi = w(i);
        if (wi > 0.f) last = i;
        sum += wi;
    }
    // inclusive scan: within the warp, then over the warp totals
    float incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float x = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += x;
    }
    if (lane == 31) s_scan[warp] = incl;
    if (tid == 0) *s_tok = -1;
    __syncthreads();
    if (warp == 0) {
        float t = s_scan[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float x = __shfl_up_sync(0xFFFFFFFFu, t, o);
            if (lane >= o) t += x;
        }
        s_scan[lane] = t;
    }
    __syncthreads();
    // chunk t covers [excl, incl); neighbours share each bound bit for bit
    // (a warp's last bound is the warp-level sum the next warp starts from)
    const float base = warp > 0 ? s_scan[warp - 1] : 0.f;
    const float total = s_scan[kAcceptThreads / 32 - 1];
    float excl = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
    if (lane == 0) excl = 0.f;
    excl += base;
    incl = lane == 31 ? s_scan[warp] : incl + base;
    const float target = u * total;
    if (total > 0.f && sum > 0.f && excl <= target && target < incl) {
        float c = excl;
        int tok = last;
        for (int i = lo; i < hi; ++i) {
            c += w(i);
            if (c > target) { tok = i; break; }
        }
        *s_tok = tok;
    }
    __syncthreads();
    int tok = *s_tok;
    if (tok < 0 && total > 0.f) {
        // u * total rounded onto the top of the range: the last positive weight
        __syncthreads();
        if (tid == 0) *s_tok = -1;
        __syncthreads();
        atomicMax(s_tok, last);
        __syncthreads();
        tok = *s_tok;
    }
    __syncthreads();
    return tok;
}

__global__ void __launch_bounds__(kAcceptThreads) accept_sampled_kernel(const AcceptSampledArgs a) {
    __shared__ float s_scan[kAcceptThreads / 32];
    __shared__ int s_tok, s_dec;
    const int b = blockIdx.x, tid = threadIdx.x, K = a.K, V = a.V;
    const uint64_t seed = *a.seed;
    const float inv_t = 1.0f / a.temperature;
    int acc = 0, extra = -1;
    for (; acc < K; ++acc) {
        const size_t row = (size_t)b * K + acc;
        const float *z = a.logits + row * V;
        const float *pt = a.target + ((size_t)b * (K + 1) + acc) * V;
        const float lse = a.lse[row];
        if (tid == 0) {
            int x = a.draft[row];
            if (x < 0 || x >= V) {
                set_err(a.err, kErrToken);
                x = 0;
            }
            const float pd = expf(z[x] * inv_t - lse);
            const float r = uniform01(seed, 2, (uint32_t)b, (uint32_t)acc, 0);
            s_dec = r * pd < pt[x];
        }
        __syncthreads();
        const bool accepted = s_dec;
        __syncthreads();
        if (accepted) continue;
        const float u = uniform01(seed, 3, (uint32_t)b, (uint32_t)acc, 0);
        extra = draw_block([&](int i) { return fmaxf(0.f, pt[i] - expf(z[i] * inv_t - lse)); }, V, u, s_scan, &s_tok);
        if (extra < 0) extra = draw_block([&](int i) { return pt[i]; }, V, u, s_scan, &s_tok);
        break;
    }
    if (acc == K) {
        const float *pt = a.target + ((size_t)b * (K + 1) + K) * V;
        extra = draw_block([&](int i) { return pt[i]; }, V, uniform01(seed, 3, (uint32_t)b, (uint32_t)K, 0), s_scan,
                           &s_tok);
    }
    if (tid == 0) {
        a.accept_len[b] = acc;
        for (int j = 0; j <= K; ++j) {
            int v = -1;
            if (j < acc) v = a.draft[(size_t)b * K + j];
            else if (j == acc) v = extra;
            a.out_tokens[(size_t)b * (K + 1) + j] = v;
        }
        a.kv_len[b] += a.n_new[b];
    }
}

}  // namespace

int sample_blocks(int V, int *chunk) {
    int c = 2048;
    while ((V + c - 1) / c > kSampleMaxBlocks) c *= 2;
    if (chunk) *chunk = c;
    return (V + c - 1) / c;
}

cudaError_t launch_sample(const SampleArgs &args, int B, cudaStream_t s, bool pdl) {
    SampleArgs a = args;
    const int nblk = sample_blocks(a.V, &a.chunk);
    a.max_blocks = kSampleMaxBlocks;
    return launch_k(sample_kernel, dim3(nblk, B), dim3(kSampleThreads), 0, s, pdl, a);
}

cudaError_t launch_accept_sampled(const AcceptSampledArgs &a, cudaStream_t s) {
    return launch_k(accept_sampled_kernel, dim3(a.B), dim3(kAcceptThreads), 0, s, false, a);
}

}  // namespace prism
