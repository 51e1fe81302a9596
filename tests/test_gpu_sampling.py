"""Sampled drafting and speculative-sampling acceptance (Sec. 2 at T > 0) on
the GPU, through the C ABI, against the oracle on the same inputs and the
same random streams.

The draws are compared where they are decided with room to spare: a draft
token where the oracle's Gumbel margin (best minus second-best perturbed
score) exceeds twice the step's logit deviation over T plus 1e-3, an
acceptance decision where r * p_draft and p_target differ by more than 1e-4
relative, and a drawn token by the inverse-CDF bracket it must fall in.
"""
from __future__ import annotations

import numpy as np
import pytest
from scipy import special, stats

import oracle
import synth
from synth.workloads import Shape
from tests.gpu_harness import GpuModel, sample_seqs
from tests.parity import ATOL, REL_L2, rel_l2
from tests.test_gpu_round import MID_W, mid_case

TAU = 0.8
SEED = 0x1234_5678_9ABC_DEF0


def _seed_tensor(seed):
    import torch
    return torch.tensor([np.int64(np.uint64(seed).view(np.int64))], dtype=torch.int64, device="cuda")


def sampled_gpu_round(w, W, I, *, tau, seed, topk, model=None, repeat=1):
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    own = model is None
    model = model or GpuModel(W)
    dr = model.drafter(w.shape, list(W["f_map"]), max_batch=w.batch, max_ctx=int(I["max_ctx"]),
                       max_new=I["tokens"].shape[1], topk=topk)
    B, K, V = I["tokens"].shape[0], w.shape.n_steps, w.shape.vocab
    i32, f32 = torch.int32, torch.float32
    runs = []
    try:
        for _ in range(repeat):
            t = {n: to_device(I[n]) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
            out = {"draft_ids": torch.full((B, K), -7, dtype=i32, device="cuda"),
                   "logits": torch.zeros((B, K, V), dtype=f32, device="cuda"),
                   "lse": torch.zeros((B, K), dtype=f32, device="cuda"),
                   "topk_ids": torch.zeros((B, K, topk), dtype=i32, device="cuda"),
                   "topk_logits": torch.zeros((B, K, topk), dtype=f32, device="cuda")}
            s = _seed_tensor(seed)
            dr.draft_round_sampled(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"],
                                   tau, s, out["draft_ids"], out["logits"], out["lse"], out["topk_ids"],
                                   out["topk_logits"])
            flags = dr.sync_status()
            res = {k: to_numpy(v) for k, v in out.items()}
            res["flags"] = flags
            runs.append(res)
    finally:
        dr.close()
        if own:
            model.close()
        torch.cuda.empty_cache()
    return runs if repeat > 1 else runs[0]


def compare_sampled(g, o, seqs, K, tau):
    """Free-running chain: step 1 strict, later steps by rel-L2 (chain reading);
    ids where the Gumbel margin clears the deviation; stop a sequence after an
    exempt divergence."""
    compared = exempt = 0
    for j, b in enumerate(seqs):
        for k in range(K):
            zg, zo = g["logits"][b, k], o["logits"][j, k]
            ma = float(np.max(np.abs(zg - zo)))
            if k == 0:
                assert ma <= ATOL, f"seq {b} step 1: logit max-abs {ma:.3e}"
            assert rel_l2(zg, zo) <= REL_L2
            assert abs(g["lse"][b, k] - o["draft_lse"][j, k]) <= ma / tau + 1e-4 + 1e-6 * abs(o["draft_lse"][j, k])
            thr = 2 * ma / tau + 1e-3
            if o["draft_margin"][j, k] > thr:
                assert g["draft_ids"][b, k] == o["draft_ids"][j, k], (
                    f"seq {b} step {k + 1}: drawn {g['draft_ids'][b, k]} != oracle {o['draft_ids'][j, k]} "
                    f"(margin {o['draft_margin'][j, k]:.3e})")
                compared += 1
            else:
                exempt += 1
            if g["draft_ids"][b, k] != o["draft_ids"][j, k]:
                break
    return compared, exempt


def _case(name):
    if name == "mid":
        return MID_W, *mid_case()
    w = synth.WORKLOADS[name]
    return w, synth.make_weights(w), synth.make_round_inputs(w)


@pytest.mark.gpu
@pytest.mark.parametrize("name,n_sample", [("tiny-bf16", 1), ("mid", 3), ("l3-8b-b1", 1), ("l3-8b-b16", 3)])
def test_sampled_round_matches_oracle(name, n_sample):
    w, W, I = _case(name)
    g = sampled_gpu_round(w, W, I, tau=TAU, seed=SEED, topk=w.topk)
    assert g["flags"] == 0
    seqs = sample_seqs(w.batch, n_sample)
    o = oracle.draft_round(w.shape, W, I, topk=w.topk, want_logits=True, want_hidden=False, seqs=seqs,
                           temperature=TAU, seed=SEED)
    compared, exempt = compare_sampled(g, o, seqs, w.shape.n_steps, TAU)
    assert compared >= len(seqs)


@pytest.mark.gpu
def test_sampled_round_replays_with_the_seed_it_reads():
    """A captured round reads the seed when it runs: the same seed gives the
    same draws bit for bit, another seed other draws."""
    w, W, I = _case("tiny-bf16")
    model = GpuModel(W)
    try:
        a, b = sampled_gpu_round(w, W, I, tau=TAU, seed=SEED, topk=1, model=model, repeat=2)
        c = sampled_gpu_round(w, W, I, tau=TAU, seed=SEED + 1, topk=1, model=model)
    finally:
        model.close()
    for key in ("draft_ids", "logits", "lse"):
        assert np.array_equal(a[key], b[key]), key
    assert not np.array_equal(a["draft_ids"], c["draft_ids"])


def _accept_drafter(V, K, B):
    from paper_2602_01762_gb300 import Drafter
    sh = Shape("accept-only", 64, 1, 1, 64, 64, V, K, "f32", 10000.0)
    return Drafter.from_shape(sh, max_batch=B, max_ctx=4, max_new=1, topk=1)


def _gpu_accept(V, K, draft, z, lse, tau, pt, seed, n_new, kv_len):
    import torch
    from paper_2602_01762_gb300.host import to_numpy
    B = draft.shape[0]
    dr = _accept_drafter(V, K, B)
    try:
        dev = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), dtype=dt, device="cuda")
        kv = dev(kv_len, torch.int32)
        acc = torch.full((B,), -7, dtype=torch.int32, device="cuda")
        out = torch.full((B, K + 1), -7, dtype=torch.int32, device="cuda")
        dr.accept_sampled(dev(draft, torch.int32), dev(z, torch.float32), dev(lse, torch.float32), tau,
                          dev(pt, torch.float32), _seed_tensor(seed), dev(n_new, torch.int32), kv, acc, out)
        flags = dr.sync_status()
        return {"accept_len": to_numpy(acc), "out_tokens": to_numpy(out), "kv_len": to_numpy(kv), "flags": flags}
    finally:
        dr.close()


def _accept_inputs(B, K, V, tau, seed, spread, rng):
    z = (rng.normal(size=(B, K, V)) * 2.0).astype(np.float32)
    lse = special.logsumexp(z.astype(np.float64) / tau, axis=-1).astype(np.float32)
    draft = np.array([[oracle.sample_gumbel(z[b, k].astype(np.float64), tau, seed, b, k)[0] for k in range(K)]
                      for b in range(B)], dtype=np.int32)
    zt = np.concatenate([z.astype(np.float64) / tau + spread * rng.normal(size=(B, K, V)),
                         rng.normal(size=(B, 1, V))], axis=1)
    pt = special.softmax(zt, axis=-1).astype(np.float32)
    return draft, z, lse, pt


@pytest.mark.gpu
@pytest.mark.parametrize("V", [4096, 128256])
def test_sampled_acceptance_matches_oracle(V):
    B, K, tau, seed = 32 if V > 10000 else 256, 5, TAU, SEED ^ V
    rng = np.random.default_rng(V)
    draft, z, lse, pt = _accept_inputs(B, K, V, tau, seed, 0.6, rng)
    n_new = rng.integers(1, 4, size=B).astype(np.int32)
    kv_len = rng.integers(0, 100, size=B).astype(np.int32)
    g = _gpu_accept(V, K, draft, z, lse, tau, pt, seed, n_new, kv_len)
    assert g["flags"] == 0
    o = oracle.accept_sampled(draft, z.astype(np.float64), lse.astype(np.float64), tau, pt.astype(np.float64),
                              seed, n_new, kv_len)
    assert np.array_equal(g["kv_len"], kv_len + n_new)
    z64, lse64, pt64 = z.astype(np.float64), lse.astype(np.float64), pt.astype(np.float64)
    same_len = exact = 0
    for b in range(B):
        # the decisions up to the oracle's stopping point, with their margins
        marginal = False
        for k in range(min(o["accept_len"][b] + 1, K)):
            x = draft[b, k]
            pd = np.exp(z64[b, k, x] / tau - lse64[b, k])
            r = oracle.uniform(seed, 2, b, k, 0)
            if abs(r * pd - pt64[b, k, x]) <= 1e-4 * max(r * pd, pt64[b, k, x]):
                marginal = True
        if marginal:
            continue
        a = o["accept_len"][b]
        assert g["accept_len"][b] == a, f"seq {b}: accepted {g['accept_len'][b]} != oracle {a}"
        assert np.array_equal(g["out_tokens"][b, :a], draft[b, :a])
        assert (g["out_tokens"][b, a + 1:] == -1).all()
        same_len += 1
        # the drawn token lies in the inverse-CDF bracket of its uniform
        if a < K:
            w = np.maximum(0.0, pt64[b, a] - np.exp(z64[b, a] / tau - lse64[b, a]))
            if w.sum() == 0.0:
                w = pt64[b, a]
        else:
            w = pt64[b, K]
        u = oracle.uniform(seed, 3, b, a, 0)
        c = np.cumsum(w)
        target = u * c[-1]
        t = g["out_tokens"][b, a]
        assert 0 <= t < V and w[t] > 0.0
        lo = c[t - 1] if t > 0 else 0.0
        slack = 1e-5 * c[-1]
        assert lo - slack <= target <= c[t] + slack, f"seq {b}: token {t} outside its bracket"
        exact += int(t == o["out_tokens"][b, a])
    assert same_len >= int(0.9 * B)
    assert exact >= int(0.9 * same_len)
    assert 0 < o["accept_len"].mean() < K                 # both branches exercised


@pytest.mark.gpu
def test_sampled_acceptance_is_lossless_on_the_gpu():
    """Drafts drawn from p_draft, accepted on the GPU: the first output token is
    distributed as p_target (chi-square)."""
    V, K, B, tau, seed = 8, 1, 40000, 1.0, 777
    zd = np.array([1.5, 0.2, -0.3, 0.9, -2.0, 0.4, 0.0, -1.0])
    pt = np.array([0.05, 0.25, 0.10, 0.15, 0.20, 0.10, 0.10, 0.05])
    draft = np.array([[oracle.sample_gumbel(zd, tau, seed, b, 0)[0]] for b in range(B)], dtype=np.int32)
    z = np.broadcast_to(zd.astype(np.float32), (B, K, V))
    lse = np.full((B, K), special.logsumexp(zd / tau), dtype=np.float32)
    target = np.broadcast_to(np.stack([pt, pt]).astype(np.float32), (B, K + 1, V))
    g = _gpu_accept(V, K, draft, z, lse, tau, target, seed, np.ones(B, np.int32), np.zeros(B, np.int32))
    first = g["out_tokens"][:, 0]
    assert stats.chisquare(np.bincount(first, minlength=V), pt * B).pvalue > 1e-4
    o = oracle.accept_sampled(draft, z.astype(np.float64), lse.astype(np.float64), tau, target.astype(np.float64),
                              seed, np.ones(B, np.int32), np.zeros(B, np.int32))
    assert np.mean(o["out_tokens"][:, 0] == first) > 0.999
