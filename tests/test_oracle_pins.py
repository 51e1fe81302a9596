"""Pins of the CPU oracle against things other than itself.

Each check is chosen so that a plausible mistake in the oracle (a dropped
term, a wrong sign or index, a transposed operand) fails at least one of
them; ``test_oracle_mutants.py`` plants such mistakes in copies of the
oracle and confirms that they are caught.
"""
from __future__ import annotations

import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

import oracle
import synth
from synth.workloads import Shape, Workload
from tests.libref import reference_round

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")

# A tiny grouped-query shape (4 query heads share 2 KV heads) so that the
# head grouping is exercised; f32 storage and no bf16 rounding, so the oracle
# and the library reference differ only by fp64 summation order.
PIN_SHAPE = Shape("pin-gqa", 64, 4, 2, 16, 96, 300, 3, "f32", 10000.0)
PIN = Workload("pin", PIN_SHAPE, batch=3, ctx_lo=0, ctx_hi=9, n_new=4, topk=3, seed=11,
               gain_sigma=0.2)


def pin_case(w: Workload = PIN, ragged=True):
    W = synth.make_weights(w)
    I = synth.make_round_inputs(w)
    if ragged and w.batch > 1:
        I["n_new"][1] = 2               # ragged prefill lengths
        I["tokens"][1, 2:] = 0
        I["hidden"][1, 2:] = 0
    return W, I


def max_rel(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return float(np.max(np.abs(a - b)) / max(1e-300, float(np.max(np.abs(b)))))


# ------------------------------------------------------------------ generator

def test_splitmix64_matches_published_outputs():
    vals = [int(x) for x in open(os.path.join(GOLDEN, "splitmix64_reference.txt"))
            if x.strip() and not x.startswith("#")]
    assert synth.splitmix64_sequence(vals[0], 5) == vals[1:]


def test_generator_moments_and_slices():
    a = synth.bf16_to_f32(synth.normal(3, "moments", (1 << 20,), 0.02, "bf16")).astype(np.float64)
    assert abs(a.mean()) < 1e-4 and abs(a.std() / 0.02 - 1) < 5e-3
    b = synth.normal(3, "moments", (1 << 20,), 1.0, "f32")
    # the stream depends on (seed, tag, index) only: scaling sigma scales every draw
    assert np.allclose(b.astype(np.float64) * 0.02, synth.bf16_to_f32(
        synth.normal(3, "moments", (1 << 20,), 0.02, "bf16")), atol=0.02 * 2 ** -7 * 5)
    u = synth.uniform_int(5, "ids", (200000,), 0, 9)
    assert u.min() == 0 and u.max() == 9 and abs(np.bincount(u).min() / 20000 - 1) < 0.05


# ------------------------------------------------------------------ single ops

def test_round_bf16_matches_library_conversion():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(20000) * np.exp(rng.uniform(-20, 20, 20000))).astype(np.float32)
    ours = np.array([oracle.round_bf16(float(v)) for v in x])
    lib = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(ours, lib)
    # ties go to even: 1 + 2^-8 is halfway between 1 and 1 + 2^-7
    assert oracle.round_bf16(1.0 + 2 ** -8) == 1.0
    assert oracle.round_bf16(1.0 + 3 * 2 ** -8) == 1.0 + 2 ** -6
    assert oracle.round_bf16(-(1.0 + 2 ** -8)) == -1.0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_matvec_matches_library_matmul(dtype):
    W = synth.normal(1, "mv", (37, 129), 1.0, dtype)
    x = np.random.default_rng(1).standard_normal(129)
    Wd = synth.bf16_to_f32(W) if dtype == "bf16" else W
    ref = np.asarray(Wd, np.float64) @ x
    assert max_rel(oracle.matvec(W, x), ref) < 1e-13


def test_rmsnorm_matches_library_and_invariants():
    rng = np.random.default_rng(2)
    x, g = rng.standard_normal(257), rng.uniform(0.5, 1.5, 257)
    out = oracle.rmsnorm(x, g, 1e-5)
    lib = Fn.rms_norm(torch.from_numpy(x), (257,), weight=torch.from_numpy(g), eps=1e-5).numpy()
    assert max_rel(out, lib) < 1e-14
    # scale invariance (eps = 0) and unit mean square of out / g
    assert max_rel(oracle.rmsnorm(7.5 * x, g, 0.0), oracle.rmsnorm(x, g, 0.0)) < 1e-14
    assert abs(np.mean((oracle.rmsnorm(x, np.ones(257), 0.0)) ** 2) - 1) < 1e-13


def test_rope_closed_forms():
    rng = np.random.default_rng(3)
    D, theta = 16, 10000.0
    q, k = rng.standard_normal(D), rng.standard_normal(D)
    assert np.array_equal(oracle.rope(q, 0, theta), q)                        # position 0 = identity
    assert abs(np.linalg.norm(oracle.rope(q, 37, theta)) - np.linalg.norm(q)) < 1e-12
    # relative position: <R_p q, R_p' k> depends only on p - p'
    d1 = oracle.rope(q, 40, theta) @ oracle.rope(k, 33, theta)
    d2 = oracle.rope(q, 107, theta) @ oracle.rope(k, 100, theta)
    assert abs(d1 - d2) < 1e-11
    # complex form: (x_j + i x_{j+D/2}) * exp(i p theta^(-2j/D))
    p = 12
    z = (q[:D // 2] + 1j * q[D // 2:]) * np.exp(1j * p * theta ** (-2.0 * np.arange(D // 2) / D))
    assert max_rel(oracle.rope(q, p, theta), np.concatenate([z.real, z.imag])) < 1e-13
    # pair 0 (frequency theta^0 = 1) turns by exactly `pos` radians
    r = oracle.rope(np.eye(D)[0], 1, theta)
    assert abs(r[0] - np.cos(1.0)) < 1e-15 and abs(r[D // 2] - np.sin(1.0)) < 1e-15


def test_attention_brute_force_and_special_cases():
    rng = np.random.default_rng(4)
    for n in (1, 2, 7):
        q = rng.standard_normal(8)
        k = rng.standard_normal((n, 8)).astype(np.float32)
        v = rng.standard_normal((n, 8)).astype(np.float32)
        s = k.astype(np.float64) @ q / np.sqrt(8)
        p = np.exp(s) / np.exp(s).sum()                                      # no max shift
        assert max_rel(oracle.attend(q, k, v), p @ v.astype(np.float64)) < 1e-12
    v = rng.standard_normal((5, 8)).astype(np.float32)
    same = np.tile(rng.standard_normal(8).astype(np.float32), (5, 1))
    assert max_rel(oracle.attend(rng.standard_normal(8), same, v), v.astype(np.float64).mean(0)) < 1e-13
    assert max_rel(oracle.attend(rng.standard_normal(8), v[:1], v[:1]), v[0]) < 1e-15


# ------------------------------------------------------------------ the round

def _compare_with_reference(W, I, w, round_acts=False, final_norm=True):
    got = oracle.draft_round(w.shape, W, I, topk=w.topk, round_acts=round_acts,
                             final_norm=final_norm, want_logits=True)
    ref = reference_round(w.shape, W, I, topk=w.topk, round_acts=round_acts, final_norm=final_norm)
    return got, ref


def reference_agrees(w: Workload = PIN, tol=1e-10) -> bool:
    W, I = pin_case(w)
    got, ref = _compare_with_reference(W, I, w)
    ok = np.array_equal(got["draft_ids"], ref["draft_ids"])
    ok &= np.array_equal(got["topk_ids"], ref["topk_ids"])
    ok &= max_rel(got["logits"], ref["logits"]) < tol
    ok &= max_rel(got["hidden_out"], ref["hidden_out"]) < tol
    ok &= max_rel(got["k_cache"], ref["k_cache"]) < 1e-6
    ok &= max_rel(got["v_cache"], ref["v_cache"]) < 1e-6
    return bool(ok)


@pytest.mark.parametrize("f_map", [(0, 1, 2), (0, 0, 0), (0, 1, 1)])
def test_round_matches_library_reference(f_map):
    """Per-step modules, the shared-weights special case (one block reused
    for every step: a single-block EAGLE/HASS-style drafter) and the two-module
    layout of the paper's experiments (module 1 prefill, module 2 decode)."""
    assert reference_agrees(PIN.with_(f_map=f_map))


def test_round_without_final_norm_matches_reference():
    W, I = pin_case()
    got, ref = _compare_with_reference(W, I, PIN, final_norm=False)
    assert np.array_equal(got["draft_ids"], ref["draft_ids"])
    assert max_rel(got["logits"], ref["logits"]) < 1e-10


def test_bf16_contract_matches_reference():
    w = PIN.with_(shape=Shape("pin-gqa-bf16", 64, 4, 2, 16, 96, 300, 3, "bf16", 10000.0))
    W, I = pin_case(w)
    got, ref = _compare_with_reference(W, I, w, round_acts=True)
    # both round fp64 to bf16 directly (the oracle by bit manipulation, the
    # reference through frexp / rint), so every rounding point agrees exactly
    assert max_rel(got["logits"], ref["logits"]) < 1e-9
    assert max_rel(got["hidden_out"], ref["hidden_out"]) < 1e-9
    assert np.array_equal(got["draft_ids"], ref["draft_ids"])
    for key in ("k_cache", "v_cache"):      # bf16 bit patterns against the reference's rounded doubles
        assert np.array_equal(synth.bf16_to_f32(got[key]).astype(np.float64), ref[key])


def test_prefill_equals_sequential_decode():
    """Step 1 over n rows equals n single-row rounds that carry the cache."""
    w = PIN.with_(batch=1, ctx_lo=0, ctx_hi=0, n_new=6, topk=1)
    W, I = pin_case(w, ragged=False)
    full = oracle.draft_round(w.shape, W, I)
    cache_k, cache_v = I["k_cache"].copy(), I["v_cache"].copy()
    for i in range(6):
        one = dict(I, tokens=I["tokens"][:, i:i + 1], hidden=I["hidden"][:, i:i + 1],
                   n_new=np.array([1], np.int32), kv_len=np.array([i], np.int32),
                   k_cache=cache_k, v_cache=cache_v)
        r = oracle.draft_round(w.shape, W, one)
        cache_k, cache_v = r["k_cache"], r["v_cache"]
    assert np.array_equal(r["draft_ids"], full["draft_ids"])
    assert np.array_equal(r["hidden_out"], full["hidden_out"])
    assert np.array_equal(cache_k[:, :, :6], full["k_cache"][:, :, :6])
    assert np.array_equal(cache_v[:, :, :6], full["v_cache"][:, :, :6])


def test_step_parameter_sets_are_independent():
    W, I = pin_case()
    base = oracle.draft_round(PIN.shape, W, I, want_logits=True)
    for j in (1, 2):
        W2 = {**W, "modules": {m: dict(mod) for m, mod in W["modules"].items()}}
        W2["modules"][j]["w_down"] = W2["modules"][j]["w_down"] * np.float32(1.5)
        pert = oracle.draft_round(PIN.shape, W2, I, want_logits=True)
        assert np.array_equal(pert["logits"][:, :j], base["logits"][:, :j])
        assert np.array_equal(pert["hidden_out"][:, :j], base["hidden_out"][:, :j])
        assert not np.array_equal(pert["logits"][:, j], base["logits"][:, j])


def test_argmax_ties_go_to_lowest_id():
    """With an all-zero LM head every logit ties at 0: the chained token must
    be id 0 and the top-k list must run 0, 1, 2, ..."""
    shape = Shape("tie", 16, 2, 2, 8, 24, 20, 2, "f32", 10000.0)
    w = Workload("tie", shape, 1, 2, 2, 1, 3, 3)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    W["lm_head"][:] = 0.0
    r = oracle.draft_round(shape, W, I, topk=3)
    assert (r["draft_ids"] == 0).all()
    assert (r["topk_ids"] == np.arange(3)).all()


def test_topk_lists_are_the_sorted_logits():
    """The top-k list of every step is numpy's stable sort of that step's
    logits (descending value, ascending id), and the greedy chain takes its
    first entry."""
    W, I = pin_case()
    k = 7
    r = oracle.draft_round(PIN_SHAPE, W, I, topk=k, want_logits=True)
    z = r["logits"]
    order = np.argsort(-z, axis=-1, kind="stable")[..., :k]
    assert np.array_equal(r["topk_ids"], order)
    assert np.array_equal(r["topk_logits"], np.take_along_axis(z, order, axis=-1))
    assert np.array_equal(r["draft_ids"], order[..., 0])


# ------------------------------------------------------------------ closed forms

def _structured(shape, fuse_half, n_new=3, seed=5):
    """Weights where the block reduces to a closed form: W_o = W_down = 0 so
    h^ equals the fusion output; W_fuse selects one half of [E(x); h]."""
    w = Workload("cf", shape, 2, 3, 3, n_new, 2, seed)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    d = shape.hidden
    for mod in W["modules"].values():
        sel = np.zeros((d, 2 * d), np.float32)
        sel[:, (0 if fuse_half == "embed" else d):][:, :d] = np.eye(d)
        mod["w_fuse"] = sel
        mod["w_o"] = np.zeros_like(mod["w_o"])
        mod["w_down"] = np.zeros_like(mod["w_down"])
    return w, W, I


def test_closed_form_draft_repeats_last_token():
    """E = c * identity rows and LM head = E: h^ = E(x), so every draft step
    re-predicts the last accepted token (checks the [E(x); h] order, that step 1
    uses the last prefill row and that decode steps embed x^_{k-1})."""
    shape = Shape("cf", 32, 2, 2, 16, 40, 32, 4, "f32", 10000.0)
    w, W, I = _structured(shape, "embed")
    W["embed"] = (np.eye(32) * 0.5).astype(np.float32)
    W["lm_head"] = W["embed"].copy()
    out = oracle.draft_round(shape, W, I)
    last = I["tokens"][np.arange(2), I["n_new"] - 1]
    assert np.array_equal(out["draft_ids"], np.repeat(last[:, None], 4, axis=1))


def test_closed_form_hidden_passthrough():
    """W_fuse picks the hidden-state half: h^_0 is the last accepted row's
    target hidden state exactly, every later step feeds h^_{k-2} back
    unchanged, and with LM head = identity the draft token is argmax(h)."""
    shape = Shape("cf", 32, 2, 2, 16, 40, 32, 4, "f32", 10000.0)
    w, W, I = _structured(shape, "hidden")
    W["lm_head"] = np.eye(32, dtype=np.float32)
    out = oracle.draft_round(shape, W, I)
    last_h = I["hidden"][np.arange(2), I["n_new"] - 1].astype(np.float64)
    assert np.array_equal(out["hidden_out"], np.repeat(last_h[:, None], 4, axis=1))
    assert np.array_equal(out["draft_ids"], np.repeat(np.argmax(last_h, 1)[:, None], 4, axis=1))


def test_closed_form_uniform_attention():
    """W_q = 0 makes every score zero, so each query head returns the plain
    mean of its KV head's values over positions [0, p]; with W_v = 0 the new
    rows add zeros.  With W_o = identity, W_down = 0 and W_fuse picking E(x),
    h^ = E(x) + mean(V) head by head."""
    shape = Shape("cf", 32, 4, 2, 8, 40, 50, 2, "f32", 10000.0)
    w = Workload("cf", shape, 1, 6, 6, 1, 1, 9)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    d, D, Hkv = 32, 8, 2
    for mod in W["modules"].values():
        sel = np.zeros((d, 2 * d), np.float32)
        sel[:, :d] = np.eye(d)
        mod["w_fuse"] = sel
        mod["w_qkv"][: 4 * D] = 0            # q rows
        mod["w_qkv"][6 * D:] = 0             # v rows
        mod["w_o"] = np.eye(d, dtype=np.float32)
        mod["w_down"] = np.zeros_like(mod["w_down"])
    out = oracle.draft_round(shape, W, I)
    L = 6
    V = I["v_cache"][0].astype(np.float64)  # [Hkv, max_ctx, D]
    for k in range(2):
        p = L + k                            # step 1 row at L, step 2 row at L + 1
        tok = I["tokens"][0, 0] if k == 0 else out["draft_ids"][0, 0]
        mean = np.concatenate([V[h // 2, :L].sum(0) / (p + 1) for h in range(4)])
        exp = W["embed"][tok].astype(np.float64) + mean
        assert max_rel(out["hidden_out"][0, k], exp) < 1e-12


# ------------------------------------------------------------------ acceptance

def test_accept_exhaustive_patterns():
    for K in range(1, 8):
        pats = np.array([[(m >> j) & 1 for j in range(K)] for m in range(2 ** K)], np.int32)
        draft = np.arange(K, dtype=np.int32)[None].repeat(len(pats), 0) + 10
        target = np.concatenate([np.where(pats == 1, draft, 99), np.full((len(pats), 1), 7)], 1)
        n_new = np.ones(len(pats), np.int32)
        r = oracle.accept_greedy(draft, target.astype(np.int32), n_new, np.full(len(pats), 5, np.int32))
        a = r["accept_len"]
        exp_a = np.array([next((j for j in range(K) if p[j] == 0), K) for p in pats])
        assert np.array_equal(a, exp_a) and a.min() >= 0 and a.max() <= K
        assert np.array_equal(a == K, pats.all(1))
        for i in range(len(pats)):
            out = r["out_tokens"][i]
            assert np.array_equal(out[:a[i]], draft[i, :a[i]]) and out[a[i]] == target[i, a[i]]
            assert (out[a[i] + 1:] == -1).all()
        assert (r["kv_len"] == 6).all()


def _rejection_sampling(p_target, p_draft, draft, rng):
    """The speculative-sampling rule of Sec. 2 for one sequence: accept token i
    when r < min(1, p_t/p_d); on the first rejection draw from the normalised
    max(0, p_t - p_d); if all pass, draw the extra token from p_t."""
    out = []
    for i, x in enumerate(draft):
        r = rng.uniform()
        if r < min(1.0, p_target[i][x] / p_draft[i][x]):
            out.append(int(x))
            continue
        resid = np.maximum(0.0, p_target[i] - p_draft[i])
        out.append(int(rng.choice(len(resid), p=resid / resid.sum())))
        return len(out) - 1, out
    out.append(int(rng.choice(len(p_target[-1]), p=p_target[-1])))
    return len(draft), out


def test_greedy_acceptance_is_the_zero_temperature_rule():
    rng = np.random.default_rng(6)
    V, K = 11, 5
    for _ in range(300):
        draft = rng.integers(0, V, K)
        target = np.where(rng.uniform(size=K + 1) < 0.6, np.append(draft, 0), rng.integers(0, V, K + 1))
        one_hot = lambda t: np.eye(V)[t]
        a_ref, out_ref = _rejection_sampling([one_hot(t) for t in target],
                                             [one_hot(t) for t in draft], draft, rng)
        r = oracle.accept_greedy(draft[None].astype(np.int32), target[None].astype(np.int32),
                                 np.ones(1, np.int32), np.zeros(1, np.int32))
        assert r["accept_len"][0] == a_ref
        assert list(r["out_tokens"][0, :a_ref + 1]) == out_ref


# ------------------------------------------------------------------ input checks

def test_oracle_rejects_bad_inputs():
    W, I = pin_case()
    bad = dict(I, kv_len=np.array([I["max_ctx"] - 3, 0, 0], np.int32))
    with pytest.raises(ValueError):
        oracle.draft_round(PIN.shape, W, bad)
    bad = dict(I, tokens=I["tokens"].copy())
    bad["tokens"][0, 0] = PIN.shape.vocab
    with pytest.raises(ValueError):
        oracle.draft_round(PIN.shape, W, bad)


def test_golden_tiny_round():
    """Regression against stored oracle outputs written by
    tests/golden/make_golden.py (oracle + generator only)."""
    import json
    g = json.load(open(os.path.join(GOLDEN, "tiny_rounds.json")))
    for name, exp in g.items():
        w = synth.WORKLOADS[name]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
        got = oracle.draft_round(w.shape, W, I, topk=4, want_logits=True)
        assert got["draft_ids"].tolist() == exp["draft_ids"]
        assert got["topk_ids"].tolist() == exp["topk_ids"]
        assert max_rel(got["topk_logits"], np.array(exp["topk_logits"])) < 1e-12
        assert max_rel(got["hidden_out"][:, :, :8], np.array(exp["hidden_head"])) < 1e-12
