/*
 * CPU oracle of one PRISM draft round.
 *
 * TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the benchmark's
 * CPU-baseline leg may call it; the CUDA path never does, and the two share
 * no code.  Arithmetic is IEEE double throughout (fp64), with no blocking,
 * fusion or reordering: every dot product is one left-to-right loop.
 *
 * What it computes (PRISM, Sec. 3.2 "Draft with PRISM", notation of Table 2):
 *   step 1 (prefill): for each accepted token x_i with its target hidden
 *     state, the fused input F_{f_map(1)}(E(x_i), h) passes through the
 *     transformer layer L_{f_map(1)} with causal attention over the draft KV
 *     cache; the last output row is h^_0 and x^_1 = argmax LM_head(h^_0).
 *   steps k = 2..K (decode): H_in = F_{f_map(k)}(E(x^_{k-1}), h^_{k-2});
 *     h^_{k-1} = L_{f_map(k)}(H_in) with the shared KV cache;
 *     x^_k = argmax LM_head(h^_{k-1}).
 *   greedy acceptance (Sec. 2 "Speculative Decoding", the rejection rule at
 *     temperature 0): the longest prefix on which draft and target agree,
 *     followed by the target's token at the first disagreement.
 *   sampled drafting and acceptance (Sec. 2, at a temperature tau > 0): each
 *     step draws x^_k from p_draft = softmax(z / tau) instead of taking the
 *     argmax; a draft token x is accepted when r < min(1, p_target(x) /
 *     p_draft(x)), and the first rejected position draws its replacement from
 *     max(0, p_target - p_draft) normalised.
 *   tree drafting (the tree of Sec. 3.2 and Sec. 4, read as a dynamic top-w
 *     expansion; see orc_draft_tree): each step expands the w best frontier
 *     rows by their w best tokens, scores candidates by summed draft
 *     log-probabilities, and the verified tree is the best n_nodes of the
 *     pool; its greedy acceptance follows the target's tokens from the root.
 *
 * Readings where the paper is silent (each is a reading, not a quote):
 *   fusion F = one bias-free linear map W_fuse [d, 2d] applied to the
 *     concatenation [E(x); h] in that order;
 *   transformer layer = Llama pre-norm block (RMSNorm, grouped-query attention
 *     with rotate-half RoPE, SwiGLU MLP, no biases), matching the Llama targets
 *     of Sec. 4;
 *   an RMSNorm with gain g_final precedes the frozen LM head (switchable);
 *     the un-normed h^ is what feeds the next step;
 *   argmax ties go to the lowest token id; top-k lists are sorted by logit
 *     descending, then id ascending;
 *   bf16 numeric contract (round_acts = 1): each projection's activation
 *     operand is rounded to bf16 (nearest even) right before the product, and
 *     K/V are rounded to the cache's storage type when stored; the residual
 *     stream, q, scores, softmax and logits are not rounded.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int32_t hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab, n_steps;
    int32_t bf16;        /* 1: weights, E, LM head, hidden inputs and KV cache hold bf16
                            bit patterns (uint16); 0: they hold float32 */
    int32_t round_acts;  /* 1: apply the bf16 rounding of projection operands */
    int32_t final_norm;  /* 1: RMSNorm(h^) * g_final before the LM head */
    int32_t topk;        /* candidates reported per step (>= 1) */
    int32_t max_ctx;     /* cache capacity in positions */
    double rope_theta, rms_eps;
} orc_config;

typedef struct {
    const void *w_fuse;    /* [d, 2d] */
    const void *g_attn;    /* [d] */
    const void *w_qkv;     /* [(Hq + 2 Hkv) D, d]: q rows, then k rows, then v rows */
    const void *w_o;       /* [d, Hq D] */
    const void *g_mlp;     /* [d] */
    const void *w_gate_up; /* [2F, d]: gate rows [0, F), up rows [F, 2F) */
    const void *w_down;    /* [d, F] */
    const void *g_final;   /* [d] */
} orc_module;

/* ---------------------------------------------------------------- scalars */

static double bf16_bits_to_double(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* Round a double to the nearest bf16 value (ties to even), for values in the
 * normal float range.  bf16 keeps 7 explicit mantissa bits of the 52. */
double orc_round_bf16(double x) {
    uint64_t u;
    memcpy(&u, &x, 8);
    uint64_t keep_lsb = (u >> 45) & 1u;
    u += 0x00000FFFFFFFFFFFULL + keep_lsb;
    u &= ~0x00001FFFFFFFFFFFULL;
    memcpy(&x, &u, 8);
    return x;
}

static uint16_t double_to_bf16_bits(double x) {
    float f = (float)orc_round_bf16(x); /* exact: the value already has 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, 4);
    return (uint16_t)(u >> 16);
}

/* Threads the oracle's parallel loops use. */
int orc_num_threads(void) { return omp_get_max_threads(); }

/* Round an array of doubles to bf16 bit patterns (nearest even). */
void orc_round_bf16_bits(const double *x, int64_t n, uint16_t *out) {
    for (int64_t i = 0; i < n; ++i) out[i] = double_to_bf16_bits(x[i]);
}

static double load_el(const void *p, int64_t i, int bf16) {
    return bf16 ? bf16_bits_to_double(((const uint16_t *)p)[i]) : (double)((const float *)p)[i];
}

static void store_el(void *p, int64_t i, int bf16, double v) {
    if (bf16)
        ((uint16_t *)p)[i] = double_to_bf16_bits(v);
    else
        ((float *)p)[i] = (float)v;
}

static void round_vec(double *v, int64_t n, int on) {
    if (!on) return;
    for (int64_t i = 0; i < n; ++i) v[i] = orc_round_bf16(v[i]);
}

/* ---------------------------------------------------------------- ops */

/* y[r] = sum_c W[r, c] x[c], W row-major [rows, cols]. */
void orc_matvec(const void *W, int bf16, int64_t rows, int64_t cols, const double *x, double *y) {
#pragma omp parallel for schedule(static) if (rows * cols > (1 << 16))
    for (int64_t r = 0; r < rows; ++r) {
        double acc = 0.0;
        const int64_t base = r * cols;
        for (int64_t c = 0; c < cols; ++c) acc += load_el(W, base + c, bf16) * x[c];
        y[r] = acc;
    }
}

/* RMSNorm: out = x / sqrt(mean(x^2) + eps) * g. */
void orc_rmsnorm(const double *x, const double *g, int64_t n, double eps, double *out) {
    double ss = 0.0;
    for (int64_t i = 0; i < n; ++i) ss += x[i] * x[i];
    double inv = 1.0 / sqrt(ss / (double)n + eps);
    for (int64_t i = 0; i < n; ++i) out[i] = x[i] * inv * g[i];
}

/* Rotary position embedding of one head vector at position pos, rotate-half
 * pairing (j, j + D/2) with angle pos * theta^(-2j/D). */
void orc_rope(double *v, int32_t D, int64_t pos, double theta) {
    int32_t half = D / 2;
    for (int32_t j = 0; j < half; ++j) {
        double ang = (double)pos * pow(theta, -2.0 * (double)j / (double)D);
        double c = cos(ang), s = sin(ang);
        double a = v[j], b = v[j + half];
        v[j] = a * c - b * s;
        v[j + half] = b * c + a * s;
    }
}

/* Softmax attention of one query head over positions [0, n_pos) of one KV
 * head: scores (q . k_j) / sqrt(D), softmax over j, weighted sum of v_j.
 * kv rows are row_stride elements apart in storage of the given type. */
void orc_attend(const double *q, const void *kc, const void *vc, int bf16, int64_t row_stride,
                int64_t n_pos, int32_t D, double *o) {
    double *s = (double *)malloc(sizeof(double) * (size_t)(n_pos > 0 ? n_pos : 1));
    double scale = 1.0 / sqrt((double)D);
    double mx = -INFINITY;
    for (int64_t j = 0; j < n_pos; ++j) {
        double dot = 0.0;
        for (int32_t t = 0; t < D; ++t) dot += q[t] * load_el(kc, j * row_stride + t, bf16);
        s[j] = dot * scale;
        if (s[j] > mx) mx = s[j];
    }
    double den = 0.0;
    for (int64_t j = 0; j < n_pos; ++j) {
        s[j] = exp(s[j] - mx);
        den += s[j];
    }
    for (int32_t t = 0; t < D; ++t) o[t] = 0.0;
    for (int64_t j = 0; j < n_pos; ++j)
        for (int32_t t = 0; t < D; ++t) o[t] += s[j] * load_el(vc, j * row_stride + t, bf16);
    for (int32_t t = 0; t < D; ++t) o[t] /= den;
    free(s);
}

static double silu(double t) { return t / (1.0 + exp(-t)); }

/* ---------------------------------------------------------------- layer */

typedef struct {
    double *x0, *n1, *qkv, *o, *a, *n2, *gu, *mm, *y;
    double *g_attn, *g_mlp, *g_final;
} scratch;

static void widen(const void *p, int bf16, int64_t n, double *out) {
    for (int64_t i = 0; i < n; ++i) out[i] = load_el(p, i, bf16);
}

/* One row through fusion + transformer layer of module m.  u = [E(x); h]
 * (already rounded per the contract).  The row's q and k are rotated at
 * position pos and its K/V are stored at cache slot `slot` of sequence b's
 * cache.  Attention runs over the cache slots vis[0..n_vis) in that order, or
 * over [0, pos] when vis is NULL (the chain, where slot == pos).  Writes the
 * layer output to y. */
static void layer_row_at(const orc_config *c, const orc_module *m, const double *u, int64_t pos,
                         int64_t slot, const int64_t *vis, int64_t n_vis, void *kc_b, void *vc_b,
                         scratch *w) {
    const int64_t d = c->hidden, Hq = c->n_q_heads, Hkv = c->n_kv_heads, D = c->head_dim, F = c->ffn;
    const int bf = c->bf16, ra = c->round_acts;
    const int64_t group = Hq / Hkv;

    /* fusion F_i(E(x), h) */
    orc_matvec(m->w_fuse, bf, d, 2 * d, u, w->x0);

    /* attention sub-block */
    widen(m->g_attn, bf, d, w->g_attn);
    orc_rmsnorm(w->x0, w->g_attn, d, c->rms_eps, w->n1);
    round_vec(w->n1, d, ra);
    orc_matvec(m->w_qkv, bf, (Hq + 2 * Hkv) * D, d, w->n1, w->qkv);
    double *q = w->qkv, *k = w->qkv + Hq * D, *v = w->qkv + (Hq + Hkv) * D;
    for (int64_t h = 0; h < Hq; ++h) orc_rope(q + h * D, (int32_t)D, pos, c->rope_theta);
    for (int64_t g = 0; g < Hkv; ++g) orc_rope(k + g * D, (int32_t)D, pos, c->rope_theta);
    for (int64_t g = 0; g < Hkv; ++g)
        for (int64_t t = 0; t < D; ++t) {
            int64_t idx = (g * c->max_ctx + slot) * D + t;
            store_el(kc_b, idx, bf, k[g * D + t]);
            store_el(vc_b, idx, bf, v[g * D + t]);
        }
    const size_t el = bf ? 2 : 4;
    if (!vis) {
#pragma omp parallel for schedule(static) if (pos > 256)
        for (int64_t h = 0; h < Hq; ++h) {
            int64_t g = h / group;
            const char *kb = (const char *)kc_b + (size_t)(g * c->max_ctx * D) * el;
            const char *vb = (const char *)vc_b + (size_t)(g * c->max_ctx * D) * el;
            orc_attend(q + h * D, kb, vb, bf, D, pos + 1, (int32_t)D, w->o + h * D);
        }
    } else {
        /* gather the visible rows of each KV head, then plain softmax attention */
        char *kt = malloc((size_t)(n_vis * D) * el), *vt = malloc((size_t)(n_vis * D) * el);
        for (int64_t g = 0; g < Hkv; ++g) {
            for (int64_t i = 0; i < n_vis; ++i) {
                const size_t src = (size_t)((g * c->max_ctx + vis[i]) * D) * el;
                memcpy(kt + (size_t)(i * D) * el, (const char *)kc_b + src, (size_t)D * el);
                memcpy(vt + (size_t)(i * D) * el, (const char *)vc_b + src, (size_t)D * el);
            }
            for (int64_t h = g * group; h < (g + 1) * group; ++h)
                orc_attend(q + h * D, kt, vt, bf, D, n_vis, (int32_t)D, w->o + h * D);
        }
        free(kt);
        free(vt);
    }
    round_vec(w->o, Hq * D, ra);
    orc_matvec(m->w_o, bf, d, Hq * D, w->o, w->a);
    for (int64_t i = 0; i < d; ++i) w->a[i] += w->x0[i];

    /* MLP sub-block */
    widen(m->g_mlp, bf, d, w->g_mlp);
    orc_rmsnorm(w->a, w->g_mlp, d, c->rms_eps, w->n2);
    round_vec(w->n2, d, ra);
    orc_matvec(m->w_gate_up, bf, 2 * F, d, w->n2, w->gu);
    for (int64_t j = 0; j < F; ++j) w->mm[j] = silu(w->gu[j]) * w->gu[F + j];
    round_vec(w->mm, F, ra);
    orc_matvec(m->w_down, bf, d, F, w->mm, w->y);
    for (int64_t i = 0; i < d; ++i) w->y[i] += w->a[i];
}

/* The chain's row: rotary position = cache slot = pos, causal window [0, pos]. */
static void layer_row(const orc_config *c, const orc_module *m, const double *u, int64_t pos,
                      void *kc_b, void *vc_b, scratch *w) {
    layer_row_at(c, m, u, pos, pos, NULL, 0, kc_b, vc_b, w);
}

/* ---------------------------------------------------------------- selection */

static const double *g_sort_keys;
static int cmp_desc(const void *pa, const void *pb) {
    int32_t a = *(const int32_t *)pa, b = *(const int32_t *)pb;
    double va = g_sort_keys[a], vb = g_sort_keys[b];
    if (va > vb) return -1;
    if (va < vb) return 1;
    return (a > b) - (a < b);
}

/* LM head on h^ (after the optional final RMSNorm) and top-k selection. */
static void select_tokens(const orc_config *c, const void *lm_head, const orc_module *m,
                          const double *h, double *z, int32_t *order, scratch *w,
                          int32_t *top_ids, double *top_vals) {
    const int64_t d = c->hidden, V = c->vocab;
    double *nf = w->n1; /* reuse */
    if (c->final_norm) {
        widen(m->g_final, c->bf16, d, w->g_final);
        orc_rmsnorm(h, w->g_final, d, c->rms_eps, nf);
    } else {
        memcpy(nf, h, sizeof(double) * (size_t)d);
    }
    round_vec(nf, d, c->round_acts);
    orc_matvec(lm_head, c->bf16, V, d, nf, z);
    for (int32_t i = 0; i < V; ++i) order[i] = i;
    g_sort_keys = z;
    qsort(order, (size_t)V, sizeof(int32_t), cmp_desc);
    for (int32_t r = 0; r < c->topk; ++r) {
        top_ids[r] = order[r];
        top_vals[r] = z[order[r]];
    }
}

/* ---------------------------------------------------------------- sampling */

/* Random numbers of sampled drafting and acceptance: the n-th output of
 * SplitMix64 (Steele, Lea and Flood, OOPSLA 2014) started from state `seed`,
 * i.e. the finaliser applied to seed + (n + 1) * gamma, with the counter
 * n = (stream << 60) | (b << 40) | (k << 32) | i (b < 2^20, k < 2^8,
 * i < 2^32).  Mapped to the open interval (0, 1) as ((x >> 41) + 1/2) / 2^23:
 * 24 significant bits, so float32 holds the value exactly and a float32
 * implementation draws the very same numbers.  Streams: 1 = draft sampling (i = token
 * id), 2 = the acceptance test of position k, 3 = the replacement or extra
 * token drawn at position k. */
uint64_t orc_splitmix_at(uint64_t seed, uint64_t n) {
    uint64_t z = seed + (n + 1) * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

double orc_uniform(uint64_t seed, int32_t stream, int64_t b, int64_t k, int64_t i) {
    const uint64_t n = ((uint64_t)stream << 60) | ((uint64_t)b << 40) | ((uint64_t)k << 32) | (uint64_t)i;
    return ((double)(orc_splitmix_at(seed, n) >> 41) + 0.5) / 8388608.0;
}

/* One draw from p_draft = softmax(z / tau) over V logits by the Gumbel-max
 * rule (the argmax of z_i / tau + G_i, G_i = -log(-log U_i) independent
 * standard Gumbel variables, is distributed as softmax(z / tau)); ties go to
 * the lower id.  lse = log sum_i exp(z_i / tau), so p_draft(x) =
 * exp(z_x / tau - lse).  margin = best minus second-best perturbed score. */
void orc_sample_gumbel(const double *z, int64_t V, double tau, uint64_t seed, int64_t b, int64_t k,
                       int32_t *token, double *lse, double *margin) {
    double m = -INFINITY;
    for (int64_t i = 0; i < V; ++i) m = fmax(m, z[i] / tau);
    double s = 0.0;
    for (int64_t i = 0; i < V; ++i) s += exp(z[i] / tau - m);
    *lse = m + log(s);
    double best = -INFINITY, second = -INFINITY;
    int32_t arg = 0;
    for (int64_t i = 0; i < V; ++i) {
        const double v = z[i] / tau - log(-log(orc_uniform(seed, 1, b, k, i)));
        if (v > best) {
            second = best;
            best = v;
            arg = (int32_t)i;
        } else if (v > second) {
            second = v;
        }
    }
    *token = arg;
    *margin = best - second;
}

/* Inverse-CDF draw from the non-negative weights w[0..V) (not necessarily
 * normalised): the first i whose running sum exceeds u * total. */
static int32_t draw_cdf(const double *w, int64_t V, double u) {
    double total = 0.0;
    for (int64_t i = 0; i < V; ++i) total += w[i];
    const double t = u * total;
    double c = 0.0;
    int32_t last = 0;
    for (int64_t i = 0; i < V; ++i) {
        if (w[i] > 0.0) last = (int32_t)i;
        c += w[i];
        if (c > t) return (int32_t)i;
    }
    return last;
}

/* Speculative-sampling acceptance (Sec. 2) of B sequences with K drafted
 * tokens each.  z: the draft logits [B, K, V]; lse: log sum exp(z / tau) per
 * (b, k); pt: the target's distributions [B, K + 1, V] (rows sum to 1);
 * seq_index[b]: the sequence's index in the random streams.  For k = 0..K-1
 * in turn, x = draft[b, k] is accepted when r * p_draft(x) < p_target(x)
 * (r < min(1, p_target / p_draft) without the division), r = uniform(2, b,
 * k).  At the first rejected position k the replacement is drawn from
 * max(0, p_target - p_draft) (uniform(3, b, k)); if that residual is zero
 * everywhere, from p_target.  When all K are accepted, the extra token is
 * drawn from p_target at position K (uniform(3, b, K)).  accept_len[b] = the
 * accepted count a; out_tokens[b] = the a accepted drafts followed by the
 * drawn token, the rest -1; kv_len[b] += n_new[b]. */
void orc_accept_sampled(int32_t B, int32_t K, int64_t V, const int32_t *seq_index, const int32_t *draft,
                        const double *z, const double *lse, double tau, const double *pt, uint64_t seed,
                        const int32_t *n_new, int32_t *kv_len, int32_t *accept_len, int32_t *out_tokens) {
    double *w = malloc(sizeof(double) * (size_t)V);
    for (int32_t b = 0; b < B; ++b) {
        const int64_t sb = seq_index ? seq_index[b] : b;
        int32_t a = 0, extra = -1;
        for (; a < K; ++a) {
            const int32_t x = draft[b * K + a];
            const double *zk = z + ((int64_t)b * K + a) * V, *pk = pt + ((int64_t)b * (K + 1) + a) * V;
            const double pd = exp(zk[x] / tau - lse[b * K + a]);
            const double r = orc_uniform(seed, 2, sb, a, 0);
            if (r * pd < pk[x]) continue;
            double tot = 0.0;
            for (int64_t i = 0; i < V; ++i) {
                w[i] = fmax(0.0, pk[i] - exp(zk[i] / tau - lse[b * K + a]));
                tot += w[i];
            }
            const double u = orc_uniform(seed, 3, sb, a, 0);
            extra = tot > 0.0 ? draw_cdf(w, V, u) : draw_cdf(pk, V, u);
            break;
        }
        if (a == K) extra = draw_cdf(pt + ((int64_t)b * (K + 1) + K) * V, V, orc_uniform(seed, 3, sb, K, 0));
        accept_len[b] = a;
        for (int32_t j = 0; j <= K; ++j) {
            int32_t v = -1;
            if (j < a) v = draft[b * K + j];
            else if (j == a) v = extra;
            out_tokens[b * (K + 1) + j] = v;
        }
        kv_len[b] = kv_len[b] + n_new[b];
    }
    free(w);
}

/* ---------------------------------------------------------------- round */

/* Returns 0 on success; 1 bad argument; 2 token id out of range; 3 cache
 * capacity exceeded (kv_len + n_new + K - 1 > max_ctx).
 * steps[k] is the module of draft step k+1 (the surjection f_map applied).
 * Outputs: draft_ids [B, K]; topk_ids/topk_logits [B, K, topk];
 * logits [B, K, V] and hidden_out [B, K, d] when non-NULL. */
/* The round with sampled drafting when tau > 0 (see orc_sample_gumbel):
 * seq_index[b] names sequence b in the random streams (NULL: b itself);
 * draft_lse / draft_margin [B, K] receive lse and the Gumbel margin of each
 * draw when non-NULL.  With tau <= 0 this is the greedy round. */
int orc_draft_round_sampled(const orc_config *c, const void *embed, const void *lm_head,
                            const orc_module *steps, int32_t B, int32_t max_new,
                            const int32_t *tokens, const void *hidden, const int32_t *n_new,
                            const int32_t *kv_len, void *k_cache, void *v_cache,
                            int32_t *draft_ids, int32_t *topk_ids, double *topk_logits,
                            double *logits, double *hidden_out, double tau, uint64_t seed,
                            const int32_t *seq_index, double *draft_lse, double *draft_margin) {
    const int64_t d = c->hidden, V = c->vocab, K = c->n_steps, F = c->ffn;
    const int64_t Hq = c->n_q_heads, Hkv = c->n_kv_heads, D = c->head_dim;
    const int bf = c->bf16;
    if (K < 1 || c->topk < 1 || c->topk > V || Hq % Hkv != 0 || D % 2 != 0) return 1;
    for (int32_t b = 0; b < B; ++b) {
        if (n_new[b] < 1 || n_new[b] > max_new || kv_len[b] < 0) return 1;
        if ((int64_t)kv_len[b] + n_new[b] + K - 1 > c->max_ctx) return 3;
        for (int32_t i = 0; i < n_new[b]; ++i)
            if (tokens[b * max_new + i] < 0 || tokens[b * max_new + i] >= V) return 2;
    }
    scratch w;
    w.x0 = calloc((size_t)d, 8); w.n1 = calloc((size_t)d, 8);
    w.qkv = calloc((size_t)((Hq + 2 * Hkv) * D), 8); w.o = calloc((size_t)(Hq * D), 8);
    w.a = calloc((size_t)d, 8); w.n2 = calloc((size_t)d, 8);
    w.gu = calloc((size_t)(2 * F), 8); w.mm = calloc((size_t)F, 8); w.y = calloc((size_t)d, 8);
    w.g_attn = calloc((size_t)d, 8); w.g_mlp = calloc((size_t)d, 8); w.g_final = calloc((size_t)d, 8);
    double *u = calloc((size_t)(2 * d), 8), *hhat = calloc((size_t)d, 8);
    double *z = calloc((size_t)V, 8);
    int32_t *order = calloc((size_t)V, 4);
    int32_t *tid = calloc((size_t)c->topk, 4);
    double *tval = calloc((size_t)c->topk, 8);
    const size_t el = bf ? 2 : 4;
    const int64_t cache_seq = Hkv * (int64_t)c->max_ctx * D;

    for (int32_t b = 0; b < B; ++b) {
        void *kc_b = (char *)k_cache + (size_t)(b * cache_seq) * el;
        void *vc_b = (char *)v_cache + (size_t)(b * cache_seq) * el;
        const int64_t L = kv_len[b], n = n_new[b];
        int32_t prev = -1;
        for (int64_t k = 1; k <= K; ++k) {
            const orc_module *m = &steps[k - 1];
            if (k == 1) {
                /* prefill: rows x_1..x_n with their hidden states, positions L..L+n-1 */
                for (int64_t i = 0; i < n; ++i) {
                    int32_t x = tokens[b * max_new + i];
                    for (int64_t t = 0; t < d; ++t) {
                        u[t] = load_el(embed, (int64_t)x * d + t, bf);
                        u[d + t] = load_el(hidden, ((int64_t)b * max_new + i) * d + t, bf);
                    }
                    round_vec(u, 2 * d, c->round_acts);
                    layer_row(c, m, u, L + i, kc_b, vc_b, &w);
                }
            } else {
                for (int64_t t = 0; t < d; ++t) {
                    u[t] = load_el(embed, (int64_t)prev * d + t, bf);
                    u[d + t] = hhat[t];
                }
                round_vec(u, 2 * d, c->round_acts);
                layer_row(c, m, u, L + n + k - 2, kc_b, vc_b, &w);
            }
            memcpy(hhat, w.y, sizeof(double) * (size_t)d);
            select_tokens(c, lm_head, m, hhat, z, order, &w, tid, tval);
            prev = tid[0];
            if (tau > 0.0) {
                double lse, margin;
                orc_sample_gumbel(z, V, tau, seed, seq_index ? seq_index[b] : b, k - 1, &prev, &lse, &margin);
                if (draft_lse) draft_lse[b * K + (k - 1)] = lse;
                if (draft_margin) draft_margin[b * K + (k - 1)] = margin;
            }
            draft_ids[b * K + (k - 1)] = prev;
            for (int32_t r = 0; r < c->topk; ++r) {
                if (topk_ids) topk_ids[(b * K + (k - 1)) * c->topk + r] = tid[r];
                if (topk_logits) topk_logits[(b * K + (k - 1)) * c->topk + r] = tval[r];
            }
            if (logits) memcpy(logits + (b * K + (k - 1)) * V, z, sizeof(double) * (size_t)V);
            if (hidden_out) memcpy(hidden_out + (b * K + (k - 1)) * d, hhat, sizeof(double) * (size_t)d);
        }
    }
    free(w.x0); free(w.n1); free(w.qkv); free(w.o); free(w.a); free(w.n2); free(w.gu);
    free(w.mm); free(w.y); free(w.g_attn); free(w.g_mlp); free(w.g_final);
    free(u); free(hhat); free(z); free(order); free(tid); free(tval);
    return 0;
}

int orc_draft_round(const orc_config *c, const void *embed, const void *lm_head,
                    const orc_module *steps, int32_t B, int32_t max_new,
                    const int32_t *tokens, const void *hidden, const int32_t *n_new,
                    const int32_t *kv_len, void *k_cache, void *v_cache,
                    int32_t *draft_ids, int32_t *topk_ids, double *topk_logits,
                    double *logits, double *hidden_out) {
    return orc_draft_round_sampled(c, embed, lm_head, steps, B, max_new, tokens, hidden, n_new, kv_len,
                                   k_cache, v_cache, draft_ids, topk_ids, topk_logits, logits, hidden_out,
                                   0.0, 0, NULL, NULL, NULL);
}

/* Greedy acceptance (temperature 0).  accept_len[b] = largest a in [0, K]
 * with draft[b, j] == target[b, j] for all j < a; out_tokens[b] =
 * draft[b, 0:a] followed by target[b, a], the rest -1; kv_len[b] += n_new[b]
 * (only the step-1 rows are committed; draft-step rows are scratch). */
void orc_accept_greedy(int32_t B, int32_t K, const int32_t *draft, const int32_t *target,
                       const int32_t *n_new, int32_t *kv_len, int32_t *accept_len,
                       int32_t *out_tokens) {
    for (int32_t b = 0; b < B; ++b) {
        int32_t a = 0;
        while (a < K && draft[b * K + a] == target[b * (K + 1) + a]) ++a;
        accept_len[b] = a;
        for (int32_t j = 0; j <= K; ++j) {
            int32_t v = -1;
            if (j < a) v = draft[b * K + j];
            else if (j == a) v = target[b * (K + 1) + a];
            out_tokens[b * (K + 1) + j] = v;
        }
        kv_len[b] += n_new[b];
    }
}

/* ---------------------------------------------------------------- tree drafting */

/* Tree-structured drafting.  PRISM states that its step-wise modules work
 * unchanged with tree-shaped drafts (Sec. 3.2, after the recurrence), and
 * evaluates a 6-step, 4-branch tree with at most 16 verified tokens (Sec. 4).
 * The paper does not spell the tree out; this oracle reads it as the dynamic
 * top-w expansion of EAGLE-2, where a candidate's score is the sum of the
 * draft log-probabilities along its path:
 *   step 1: the prefill as in the chain gives h^_0 and logits z; the w best
 *     tokens of z are the depth-1 candidates, score = z_x - lse(z).  All w
 *     form the first frontier.
 *   step k = 2..K: frontier node j (token t, emitted by a row with output
 *     h^) is processed by step k's module as its own row: input
 *     [E(t); h^], rotary position L + n + k - 2 (its depth), K/V stored at
 *     cache slot L + n + (k - 2) w + j, attention over the committed rows
 *     [0, L + n) plus the slots of the rows that processed its ancestors and
 *     its own slot.  The row's w best tokens become candidates with score =
 *     parent score + z_x - lse(z).  The next frontier is the w best of these
 *     w^2 candidates (score descending, then pool index ascending).
 *   end: the verified tree is the n_nodes best candidates of the whole pool
 *     (score descending, then pool index ascending), listed in pool order.
 *     The pool lists shallower entries first and log-probabilities are <= 0,
 *     so a parent always ranks before its children: every chosen node's
 *     parent is chosen too, and parents precede children in the list.
 * Pool layout per sequence: P = w + (K - 1) w^2 entries; depth-1 candidate r
 * at index r; candidate r of row j at step k at w + (k - 2) w^2 + j w + r.
 *
 * follow_tokens [B, P] / follow_frontier [B, K, w] (both or neither): use
 * these candidate tokens and frontier choices instead of the oracle's own
 * (scores are still the oracle's), so that another implementation's tree can
 * be recomputed node by node.
 * Outputs: pool_tokens / pool_parent (pool index, -1 = root) / pool_score
 * [B, P]; frontier [B, K, w] (pool indices chosen after each step);
 * row_logits [B, K, w, V], row_lse [B, K, w] and row_hidden [B, K, w, d]
 * when non-NULL (step 1 fills only row 0); tree_* [B, n_nodes] (tree_parent
 * is the parent's position in the tree, -1 = root; tree_pool the pool index).
 * Returns 0; 1 bad argument; 2 token id out of range; 3 cache capacity
 * (kv_len + n_new + (K - 1) w > max_ctx); 4 invalid follow input. */
static const double *g_tree_score;
static int cmp_tree(const void *pa, const void *pb) {
    int32_t a = *(const int32_t *)pa, b = *(const int32_t *)pb;
    if (g_tree_score[a] > g_tree_score[b]) return -1;
    if (g_tree_score[a] < g_tree_score[b]) return 1;
    return a < b ? -1 : (a > b);   /* equal scores: lower pool index first */
}

static double log_sum_exp(const double *z, int64_t V) {
    double m = -INFINITY;
    for (int64_t i = 0; i < V; ++i) m = fmax(m, z[i]);
    double s = 0.0;
    for (int64_t i = 0; i < V; ++i) s += exp(z[i] - m);
    return m + log(s);
}

int orc_draft_tree(const orc_config *c, const void *embed, const void *lm_head, const orc_module *steps,
                   int32_t B, int32_t max_new, const int32_t *tokens, const void *hidden,
                   const int32_t *n_new, const int32_t *kv_len, void *k_cache, void *v_cache,
                   int32_t width, int32_t n_nodes, const int32_t *follow_tokens,
                   const int32_t *follow_frontier, int32_t *pool_tokens, int32_t *pool_parent,
                   double *pool_score, int32_t *frontier, double *row_logits, double *row_lse,
                   double *row_hidden, int32_t *tree_tokens, int32_t *tree_parent, int32_t *tree_depth,
                   double *tree_score, int32_t *tree_pool) {
    const int64_t d = c->hidden, V = c->vocab, K = c->n_steps, F = c->ffn;
    const int64_t Hq = c->n_q_heads, Hkv = c->n_kv_heads, D = c->head_dim;
    const int64_t w_ = width, P = width + (K - 1) * (int64_t)width * width;
    const int bf = c->bf16;
    if (K < 1 || width < 1 || width > V || n_nodes < 1 || n_nodes > P || Hq % Hkv != 0 || D % 2 != 0) return 1;
    if ((follow_tokens == NULL) != (follow_frontier == NULL)) return 1;
    for (int32_t b = 0; b < B; ++b) {
        if (n_new[b] < 1 || n_new[b] > max_new || kv_len[b] < 0) return 1;
        if ((int64_t)kv_len[b] + n_new[b] + (K - 1) * w_ > c->max_ctx) return 3;
        for (int32_t i = 0; i < n_new[b]; ++i)
            if (tokens[b * max_new + i] < 0 || tokens[b * max_new + i] >= V) return 2;
    }
    scratch w;
    w.x0 = calloc((size_t)d, 8); w.n1 = calloc((size_t)d, 8);
    w.qkv = calloc((size_t)((Hq + 2 * Hkv) * D), 8); w.o = calloc((size_t)(Hq * D), 8);
    w.a = calloc((size_t)d, 8); w.n2 = calloc((size_t)d, 8);
    w.gu = calloc((size_t)(2 * F), 8); w.mm = calloc((size_t)F, 8); w.y = calloc((size_t)d, 8);
    w.g_attn = calloc((size_t)d, 8); w.g_mlp = calloc((size_t)d, 8); w.g_final = calloc((size_t)d, 8);
    double *u = calloc((size_t)(2 * d), 8);
    double *z = calloc((size_t)V, 8);
    int32_t *order = calloc((size_t)V, 4);
    int32_t *tid = calloc((size_t)width, 4);
    double *tval = calloc((size_t)width, 8);
    /* h^ of every row of the round: row 0 = the prefill's last row, then
     * (k - 2) w + j + 1 for row j of step k */
    double *H = calloc((size_t)((1 + (K - 1) * w_) * d), 8);
    /* cache-slot offsets (from L + n) of each row's own and ancestors' rows */
    int64_t *anc = calloc((size_t)((1 + (K - 1) * w_) * K), 8);
    int32_t *n_anc = calloc((size_t)(1 + (K - 1) * w_), 4);
    int64_t *vis = calloc((size_t)(c->max_ctx), 8);
    int32_t *idx = calloc((size_t)P, 4), *depth = calloc((size_t)P, 4), *pos_in_tree = calloc((size_t)P, 4);
    orc_config ct = *c;
    ct.topk = width;
    const size_t el = bf ? 2 : 4;
    const int64_t cache_seq = Hkv * (int64_t)c->max_ctx * D;
    int rc = 0;

    for (int64_t e = 0; e < P; ++e) depth[e] = e < w_ ? 1 : (int32_t)(2 + (e - w_) / (w_ * w_));
    for (int32_t b = 0; b < B && rc == 0; ++b) {
        void *kc_b = (char *)k_cache + (size_t)(b * cache_seq) * el;
        void *vc_b = (char *)v_cache + (size_t)(b * cache_seq) * el;
        const int64_t L = kv_len[b], n = n_new[b];
        int32_t *ptok = pool_tokens + (int64_t)b * P, *ppar = pool_parent + (int64_t)b * P;
        double *psc = pool_score + (int64_t)b * P;
        int32_t *front = frontier + (int64_t)b * K * w_;
        if (row_logits) memset(row_logits + (int64_t)b * K * w_ * V, 0, sizeof(double) * (size_t)(K * w_ * V));
        if (row_lse) memset(row_lse + (int64_t)b * K * w_, 0, sizeof(double) * (size_t)(K * w_));
        if (row_hidden) memset(row_hidden + (int64_t)b * K * w_ * d, 0, sizeof(double) * (size_t)(K * w_ * d));
        for (int64_t k = 1; k <= K && rc == 0; ++k) {
            const orc_module *m = &steps[k - 1];
            const int64_t rows = k == 1 ? 1 : w_;
            const int64_t base = k == 1 ? 0 : w_ + (k - 2) * w_ * w_;
            for (int64_t j = 0; j < rows && rc == 0; ++j) {
                const int64_t row = k == 1 ? 0 : 1 + (k - 2) * w_ + j;
                int64_t parent = -1;
                if (k == 1) {
                    for (int64_t i = 0; i < n; ++i) {
                        int32_t x = tokens[b * max_new + i];
                        for (int64_t t = 0; t < d; ++t) {
                            u[t] = load_el(embed, (int64_t)x * d + t, bf);
                            u[d + t] = load_el(hidden, ((int64_t)b * max_new + i) * d + t, bf);
                        }
                        round_vec(u, 2 * d, c->round_acts);
                        layer_row(c, m, u, L + i, kc_b, vc_b, &w);
                    }
                    n_anc[row] = 0;
                } else {
                    parent = front[(k - 2) * w_ + j];
                    /* the row that emitted the parent candidate */
                    const int64_t erow = parent < w_ ? 0 : 1 + (k - 3) * w_ + (parent - (w_ + (k - 3) * w_ * w_)) / w_;
                    const int64_t slot_off = (k - 2) * w_ + j;
                    n_anc[row] = n_anc[erow] + 1;
                    for (int32_t i = 0; i < n_anc[erow]; ++i) anc[row * K + i] = anc[erow * K + i];
                    anc[row * K + n_anc[erow]] = slot_off;
                    const int32_t x = ptok[parent];
                    for (int64_t t = 0; t < d; ++t) {
                        u[t] = load_el(embed, (int64_t)x * d + t, bf);
                        u[d + t] = H[erow * d + t];
                    }
                    round_vec(u, 2 * d, c->round_acts);
                    int64_t nv = 0;
                    for (int64_t p = 0; p < L + n; ++p) vis[nv++] = p;
                    for (int32_t i = 0; i < n_anc[row]; ++i) vis[nv++] = L + n + anc[row * K + i];
                    layer_row_at(c, m, u, L + n + k - 2, L + n + slot_off, vis, nv, kc_b, vc_b, &w);
                }
                memcpy(H + row * d, w.y, sizeof(double) * (size_t)d);
                select_tokens(&ct, lm_head, m, w.y, z, order, &w, tid, tval);
                const double lse = log_sum_exp(z, V);
                const int64_t ri = ((int64_t)b * K + (k - 1)) * w_ + j;
                if (row_logits) memcpy(row_logits + ri * V, z, sizeof(double) * (size_t)V);
                if (row_lse) row_lse[ri] = lse;
                if (row_hidden) memcpy(row_hidden + ri * d, w.y, sizeof(double) * (size_t)d);
                for (int64_t r = 0; r < w_; ++r) {
                    const int64_t e = base + j * w_ + r;
                    int32_t x = tid[r];
                    if (follow_tokens) {
                        x = follow_tokens[(int64_t)b * P + e];
                        if (x < 0 || x >= V) { rc = 4; break; }
                        for (int64_t r2 = 0; r2 < r; ++r2)
                            if (ptok[base + j * w_ + r2] == x) rc = 4;
                    }
                    ptok[e] = x;
                    ppar[e] = (int32_t)parent;
                    psc[e] = (parent < 0 ? 0.0 : psc[parent]) + (z[x] - lse);
                }
            }
            if (rc) break;
            /* the next frontier: the w best of this step's candidates */
            const int64_t ncand = rows * w_;
            for (int64_t e = 0; e < ncand; ++e) idx[e] = (int32_t)(base + e);
            g_tree_score = psc;
            qsort(idx, (size_t)ncand, sizeof(int32_t), cmp_tree);
            for (int64_t j = 0; j < w_; ++j) {
                int32_t e = idx[j];
                if (follow_frontier) {
                    e = follow_frontier[((int64_t)b * K + (k - 1)) * w_ + j];
                    if (e < base || e >= base + ncand) rc = 4;
                    for (int64_t j2 = 0; j2 < j; ++j2)
                        if (front[(k - 1) * w_ + j2] == e) rc = 4;
                }
                front[(k - 1) * w_ + j] = e;
            }
        }
        if (rc) break;
        /* the verified tree: the n_nodes best of the pool, listed in pool order */
        for (int64_t e = 0; e < P; ++e) idx[e] = (int32_t)e;
        g_tree_score = psc;
        qsort(idx, (size_t)P, sizeof(int32_t), cmp_tree);
        for (int64_t e = 0; e < P; ++e) pos_in_tree[e] = -1;
        for (int64_t i = 0; i < n_nodes; ++i) pos_in_tree[idx[i]] = 0;
        int32_t np = 0;
        for (int64_t e = 0; e < P; ++e)
            if (pos_in_tree[e] == 0) pos_in_tree[e] = np++;
        for (int64_t e = 0; e < P; ++e) {
            if (pos_in_tree[e] < 0) continue;
            const int64_t o = (int64_t)b * n_nodes + pos_in_tree[e];
            tree_pool[o] = (int32_t)e;
            tree_tokens[o] = ptok[e];
            tree_depth[o] = depth[e];
            tree_score[o] = psc[e];
            tree_parent[o] = ppar[e] < 0 ? -1 : pos_in_tree[ppar[e]];
            if (ppar[e] >= 0 && pos_in_tree[ppar[e]] < 0) rc = 4;   /* cannot happen: see above */
        }
    }
    free(w.x0); free(w.n1); free(w.qkv); free(w.o); free(w.a); free(w.n2); free(w.gu);
    free(w.mm); free(w.y); free(w.g_attn); free(w.g_mlp); free(w.g_final);
    free(u); free(z); free(order); free(tid); free(tval); free(H); free(anc); free(n_anc); free(vis);
    free(idx); free(depth); free(pos_in_tree);
    return rc;
}

/* Greedy acceptance of a draft tree (Sec. 2's temperature-0 rule applied
 * along the tree, as in tree-based verification): target_next[b, 0] is the
 * target's token after the last accepted token (the root) and
 * target_next[b, 1 + i] its token after tree node i.  From the root, repeatedly
 * accept the child whose token equals the target's token at the current node;
 * stop when no child matches.  accept_len[b] = accepted nodes a (0..K);
 * accept_nodes[b, 0:a] their tree positions (rest -1); out_tokens[b] = their
 * tokens followed by the target's token at the last accepted node (rest -1);
 * kv_len[b] += n_new[b]. */
void orc_accept_tree(int32_t B, int32_t n_nodes, int32_t K, const int32_t *tree_tokens,
                     const int32_t *tree_parent, const int32_t *target_next, const int32_t *n_new,
                     int32_t *kv_len, int32_t *accept_len, int32_t *accept_nodes, int32_t *out_tokens) {
    for (int32_t b = 0; b < B; ++b) {
        const int32_t *tok = tree_tokens + (int64_t)b * n_nodes, *par = tree_parent + (int64_t)b * n_nodes;
        const int32_t *tn = target_next + (int64_t)b * (n_nodes + 1);
        int32_t cur = -1, a = 0;
        for (int32_t j = 0; j < K; ++j) accept_nodes[b * K + j] = -1;
        for (int32_t j = 0; j <= K; ++j) out_tokens[b * (K + 1) + j] = -1;
        while (a < K) {
            const int32_t want = tn[cur + 1];
            int32_t next = -1;
            for (int32_t i = 0; i < n_nodes && next < 0; ++i)
                if (par[i] == cur && tok[i] == want) next = i;
            if (next < 0) break;
            accept_nodes[b * K + a] = next;
            out_tokens[b * (K + 1) + a] = tok[next];
            ++a;
            cur = next;
        }
        out_tokens[b * (K + 1) + a] = tn[cur + 1];
        accept_len[b] = a;
        kv_len[b] = kv_len[b] + n_new[b];   /* only the step-1 rows are committed */
    }
}
