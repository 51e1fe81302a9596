"""Pins of the oracle's sampled drafting and acceptance (Sec. 2, temperature > 0).

What fixes these functions, other than the oracle itself:
  * the random numbers are the published SplitMix64 sequence (golden file);
  * the Gumbel-max draw follows softmax(z / T) (a chi-square test against the
    closed form), its log-sum-exp equals scipy's, and at a tiny temperature it
    is the argmax;
  * speculative sampling is lossless: with drafts drawn from p_draft, the first
    output token is distributed as p_target (chi-square), whatever p_draft is;
  * the same at a later position (its own draft and target distributions),
    and the extra token after K accepted drafts follows p_target at K;
  * special cases: p_target = p_draft accepts everything; a draft token the
    target gives probability 0 is always rejected and replaced by a token where
    p_target > p_draft;
  * inside a round, every sampled token is the Gumbel draw of that step's own
    logits with the sequence's index in the full batch.
The last test plants mistakes in copies of the sampling code and checks that
these pins catch each one.
"""
from __future__ import annotations

import os

import numpy as np
import pytest
from scipy import special, stats

import oracle
import synth
from tests import test_oracle_pins as pins

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")
P_MIN = 1e-4          # chi-square p-value below which a distribution test fails


def test_random_numbers_are_the_published_splitmix64_sequence():
    vals = [int(x) for x in open(os.path.join(GOLDEN, "splitmix64_reference.txt"))
            if x.strip() and not x.startswith("#")]
    seed, outs = vals[0], vals[1:]
    assert [oracle.splitmix_at(seed, n) for n in range(len(outs))] == outs
    # counter 0..4 of stream 0, sequence 0, position 0: the top 23 bits, centred in their cell
    for n, x in enumerate(outs):
        u = oracle.uniform(seed, 0, 0, 0, n)
        assert 0.0 < u < 1.0 and u * 2 ** 23 - 0.5 == x >> 41
        assert float(np.float32(u)) == u          # exact in float32


def test_uniforms_are_uniform_and_streams_differ():
    u = np.array([oracle.uniform(99, 1, b, 3, 7) for b in range(20000)])
    assert stats.kstest(u, "uniform").pvalue > P_MIN
    v = np.array([oracle.uniform(99, 2, b, 3, 7) for b in range(20000)])
    assert abs(np.corrcoef(u, v)[0, 1]) < 0.03


def test_gumbel_draws_follow_softmax():
    z = np.array([0.3, -1.2, 2.0, 0.0, 1.1, -0.4])
    tau = 0.8
    n = 30000
    toks = np.empty(n, dtype=np.int64)
    for b in range(n):
        toks[b], lse, _ = oracle.sample_gumbel(z, tau, 2024, b, 1)
    assert abs(lse - special.logsumexp(z / tau)) < 1e-12
    p = special.softmax(z / tau)
    counts = np.bincount(toks, minlength=z.size)
    assert stats.chisquare(counts, p * n).pvalue > P_MIN


def test_gumbel_draw_at_tiny_temperature_is_the_argmax():
    rng = np.random.default_rng(5)
    for b in range(200):
        z = rng.normal(size=50)
        assert oracle.sample_gumbel(z, 1e-4, 77, b, 0)[0] == int(np.argmax(z))


def _draws(z, tau, seed, n, k=0):
    return np.array([oracle.sample_gumbel(z, tau, seed, b, k)[0] for b in range(n)], dtype=np.int32)


def test_speculative_sampling_is_lossless():
    """Drafts from p_draft, acceptance against p_target: the first output token
    is distributed as p_target (the property Sec. 2 states for the rule)."""
    V, n, tau, seed = 6, 40000, 1.0, 31337
    zd = np.array([1.5, 0.2, -0.3, 0.9, -2.0, 0.4])          # p_draft = softmax(zd)
    pt = np.array([0.05, 0.30, 0.10, 0.15, 0.25, 0.15])        # p_target, far from p_draft
    draft = _draws(zd, tau, seed, n)[:, None]
    z = np.broadcast_to(zd, (n, 1, V))
    lse = np.full((n, 1), special.logsumexp(zd / tau))
    target = np.broadcast_to(np.stack([pt, pt]), (n, 2, V))
    r = oracle.accept_sampled(draft, z, lse, tau, target, seed, np.ones(n, np.int32), np.zeros(n, np.int32))
    first = r["out_tokens"][:, 0]
    assert stats.chisquare(np.bincount(first, minlength=V), pt * n).pvalue > P_MIN
    # and some drafts were rejected, some accepted (the test exercises both branches)
    assert 0.2 < r["accept_len"].mean() < 0.9


def test_lossless_at_every_position():
    """Two draft positions with their own draft and target distributions: the
    first output token follows p_target[0]; where the first draft is accepted,
    the second output token follows p_target[1] (the rule applied at that
    position, with its own random numbers)."""
    V, K, n, tau, seed = 5, 2, 40000, 1.0, 777
    zd = np.array([[1.2, -0.5, 0.3, 0.0, -1.0],
                   [-0.8, 0.9, 0.1, 1.4, -0.2]])
    pt = np.array([[0.10, 0.35, 0.25, 0.20, 0.10],
                   [0.40, 0.05, 0.30, 0.05, 0.20],
                   [0.20, 0.20, 0.20, 0.20, 0.20]])
    draft = np.stack([_draws(zd[k], tau, seed, n, k) for k in range(K)], axis=1)
    z = np.broadcast_to(zd, (n, K, V))
    lse = np.broadcast_to(special.logsumexp(zd / tau, axis=-1), (n, K))
    target = np.broadcast_to(pt, (n, K + 1, V))
    r = oracle.accept_sampled(draft, z, lse, tau, target, seed, np.ones(n, np.int32), np.zeros(n, np.int32))
    out, a = r["out_tokens"], r["accept_len"]
    assert stats.chisquare(np.bincount(out[:, 0], minlength=V), pt[0] * n).pvalue > P_MIN
    sel = a >= 1
    m = int(sel.sum())
    assert m > n // 4
    assert stats.chisquare(np.bincount(out[sel, 1], minlength=V), pt[1] * m).pvalue > P_MIN


def test_bonus_token_follows_the_targets_last_distribution():
    """When every draft is accepted, the extra token is drawn from p_target at
    position K."""
    V, K, n, tau = 5, 2, 20000, 1.0
    zd = np.array([0.5, -0.2, 0.1, 0.8, -1.0])
    pd = special.softmax(zd / tau)
    last = np.array([0.70, 0.05, 0.05, 0.15, 0.05])
    target = np.broadcast_to(np.stack([pd, pd, last]), (n, K + 1, V))
    draft = np.stack([_draws(zd, tau, 9, n, k) for k in range(K)], axis=1)
    z = np.broadcast_to(zd, (n, K, V))
    lse = np.full((n, K), special.logsumexp(zd / tau))
    r = oracle.accept_sampled(draft, z, lse, tau, target, 9, np.ones(n, np.int32), np.zeros(n, np.int32))
    assert (r["accept_len"] == K).all()
    assert stats.chisquare(np.bincount(r["out_tokens"][:, K], minlength=V), last * n).pvalue > P_MIN


def test_equal_distributions_accept_everything():
    V, K, n, tau = 5, 3, 500, 0.7
    rng = np.random.default_rng(8)
    z = rng.normal(size=(n, K, V))
    lse = special.logsumexp(z / tau, axis=-1)
    pd = np.exp(z / tau - lse[..., None])
    extra = rng.dirichlet(np.ones(V), size=n)
    target = np.concatenate([pd, extra[:, None]], axis=1)
    draft = np.array([[oracle.sample_gumbel(z[b, k], tau, 3, b, k)[0] for k in range(K)] for b in range(n)])
    r = oracle.accept_sampled(draft, z, lse, tau, target, 3, np.full(n, 2, np.int32), np.full(n, 10, np.int32))
    assert (r["accept_len"] == K).all()
    assert (r["out_tokens"][:, :K] == draft).all()
    assert (r["kv_len"] == 12).all()
    # the extra token follows the target's last distribution
    counts = np.zeros(V)
    for b in range(n):
        counts[r["out_tokens"][b, K]] += 1
    assert (counts > 0).sum() >= 3


def test_a_token_the_target_excludes_is_replaced_where_target_exceeds_draft():
    V, n, tau = 8, 2000, 1.0
    rng = np.random.default_rng(12)
    z = rng.normal(size=(n, 1, V))
    lse = special.logsumexp(z / tau, axis=-1)
    pd = np.exp(z / tau - lse[..., None])
    draft = np.array([[int(np.argmax(z[b, 0]))] for b in range(n)])
    pt = rng.dirichlet(np.ones(V), size=(n, 2))
    for b in range(n):
        pt[b, 0, draft[b, 0]] = 0.0
        pt[b, 0] /= pt[b, 0].sum()
    r = oracle.accept_sampled(draft, z, lse, tau, pt, 5, np.ones(n, np.int32), np.zeros(n, np.int32))
    assert (r["accept_len"] == 0).all()
    rep = r["out_tokens"][:, 0]
    assert (r["out_tokens"][:, 1] == -1).all()
    assert all(pt[b, 0, rep[b]] > pd[b, 0, rep[b]] for b in range(n))


def test_sampled_round_draws_from_its_own_logits():
    w = pins.PIN.with_(batch=3, topk=2)
    W, I = pins.pin_case(w)
    tau, seed = 0.9, 4242
    full = oracle.draft_round(w.shape, W, I, topk=2, want_logits=True, temperature=tau, seed=seed)
    K = w.shape.n_steps
    for b in range(w.batch):
        for k in range(K):
            tok, lse, margin = oracle.sample_gumbel(full["logits"][b, k], tau, seed, b, k)
            assert tok == full["draft_ids"][b, k]
            assert abs(lse - full["draft_lse"][b, k]) < 1e-12 and margin == full["draft_margin"][b, k]
            assert lse == pytest.approx(special.logsumexp(full["logits"][b, k] / tau), abs=1e-10)
    # a subset of sequences keeps each sequence's random stream
    sub = oracle.draft_round(w.shape, W, I, topk=2, want_logits=True, temperature=tau, seed=seed, seqs=[2, 0])
    assert (sub["draft_ids"] == full["draft_ids"][[2, 0]]).all()
    # the step chain follows the sampled token: the round differs from the greedy one
    greedy = oracle.draft_round(w.shape, W, I, topk=2, want_logits=True)
    assert (greedy["draft_ids"][:, 0] == greedy["topk_ids"][:, 0, 0]).all()
    assert (full["draft_ids"] != greedy["draft_ids"]).any()


def test_sampled_round_at_tiny_temperature_is_the_greedy_round():
    W, I = pins.pin_case()
    s = oracle.draft_round(pins.PIN_SHAPE, W, I, topk=3, temperature=1e-6, seed=1)
    g = oracle.draft_round(pins.PIN_SHAPE, W, I, topk=3)
    assert (s["draft_ids"] == g["draft_ids"]).all()


SAMPLING_PINS = [
    test_gumbel_draws_follow_softmax,
    test_gumbel_draw_at_tiny_temperature_is_the_argmax,
    test_speculative_sampling_is_lossless,
    test_lossless_at_every_position,
    test_bonus_token_follows_the_targets_last_distribution,
    test_equal_distributions_accept_everything,
    test_a_token_the_target_excludes_is_replaced_where_target_exceeds_draft,
    test_sampled_round_draws_from_its_own_logits,
]

# (name, original text, planted mistake)
MUTANTS = [
    ("gumbel-sign", "const double v = z[i] / tau - log(-log(", "const double v = z[i] / tau + log(-log("),
    ("gumbel-temperature", "const double v = z[i] / tau", "const double v = z[i]"),
    ("accept-inequality", "if (r * pd < pk[x]) continue;", "if (r * pk[x] < pd) continue;"),
    ("residual-direction", "w[i] = fmax(0.0, pk[i] - exp(", "w[i] = fmax(0.0, -pk[i] + 2.0 * exp("),
    ("replacement-stream", "const double u = orc_uniform(seed, 3, sb, a, 0);", "const double u = orc_uniform(seed, 2, sb, a, 0);"),
    ("round-stream-index", "seq_index ? seq_index[b] : b, k - 1, &prev", "b, k - 1, &prev"),
    ("bonus-position", "+ K) * V, V, orc_uniform(seed, 3, sb, K, 0)", "+ K - 1) * V, V, orc_uniform(seed, 3, sb, K, 0)"),
    ("target-position", "*pk = pt + ((int64_t)b * (K + 1) + a) * V;", "*pk = pt + ((int64_t)b * (K + 1)) * V;"),
    ("draft-lse-position", "const double pd = exp(zk[x] / tau - lse[b * K + a]);",
     "const double pd = exp(zk[x] / tau - lse[b * K]);"),
    ("replacement-not-residual", "extra = tot > 0.0 ? draw_cdf(w, V, u) : draw_cdf(pk, V, u);", "extra = draw_cdf(pk, V, u);"),
    ("accept-stream-position", "const double r = orc_uniform(seed, 2, sb, a, 0);", "const double r = orc_uniform(seed, 2, sb, 0, 0);"),
]


def _caught() -> bool:
    for pin in SAMPLING_PINS:
        try:
            pin()
        except (AssertionError, ValueError, FloatingPointError):
            return True
    return False


@pytest.mark.parametrize("name,orig,mut", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_sampling_mistake_is_caught(tmp_path, name, orig, mut):
    src = open(SRC).read()
    assert src.count(orig) == 1, f"mutation anchor for {name} not found exactly once"
    p = tmp_path / "mutant.c"
    p.write_text(src.replace(orig, mut))
    lib = oracle.compile_source(str(p), str(tmp_path / f"libmutant_{name}.so"))
    with oracle.variant(lib):
        assert _caught(), f"planted mistake '{name}' was not caught by any pin"
