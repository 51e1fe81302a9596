"""GPU tests of the steady-state draft loop (``prism_draft_loop``): rounds
back to back on the device, each acceptance writing the next round's tokens,
n_new and kv_len.

  * against the oracle run as the same loop on the host (its own drafts,
    acceptances and next-round inputs); targets come from the oracle's drafts
    (per position the draft token with probability 1/2, else uniform).  Draft
    ids are compared where the oracle's top-1 margin exceeds the chain's
    tolerance: MARGIN at step 1; at later steps, where h^ is re-rounded step
    after step and the loop returns no logits, twice the largest logit
    deviation the chain comparison allows there (max(ATOL, ENVELOPE_FACTOR
    times the oracle's one-ulp envelope of that round)).  Acceptance lengths,
    output tokens, n_new and kv_len exactly.  A sequence whose drafts
    legitimately differ (a margin-exempt id) is not compared in later rounds;
  * every round once more from the oracle's state at its start (teacher
    forcing per round): a single GPU round on the oracle loop's inputs of
    that round, through the chain comparison with logits (step 1 strictly,
    the envelope along the chain, every later step forced from the oracle's
    state);
  * against the library's own single-round calls (prism_draft_round then
    prism_accept_greedy, next-round inputs prepared on the host): bit-identical.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from synth.workloads import Shape, Workload
from tests.gpu_harness import GpuModel
from tests.parity import ATOL, ENVELOPE_FACTOR, MARGIN, one_ulp_envelope
from tests.test_gpu_round import _check

pytestmark = pytest.mark.gpu

MID = Shape("mid-gqa", 1024, 8, 2, 128, 2816, 32000, 4, "bf16", 500000.0)
CASES = {
    "tiny-bf16": Workload("tiny-loop", synth.workloads.TINY_BF16, 3, 16, 40, 1, 1, 0),
    "mid": Workload("mid-loop", MID, 3, 100, 700, 1, 1, 21, gain_sigma=0.1, f_map=(0, 1, 1, 2)),
}
ROUNDS = 4


def loop_inputs(w):
    K = w.shape.n_steps
    I = synth.make_round_inputs(w, max_new=K + 1)
    # room for every round's prefill (up to K + 1 rows) and draft rows
    mc = (w.ctx_hi + (ROUNDS + 1) * (K + 1) + K + 15) // 16 * 16
    for key in ("k_cache", "v_cache"):
        a = I[key]
        pad = np.zeros(a.shape[:2] + (mc,) + a.shape[3:], a.dtype)
        pad[:, :, :a.shape[2]] = a
        I[key] = pad
    I["max_ctx"] = mc
    hid = np.stack([synth.normal(w.seed, f"loop_hidden_{r}", I["hidden"].shape, 1.0, w.shape.dtype)
                    for r in range(ROUNDS)])
    return I, hid


def oracle_loop(w, W, I0, hid):
    K, B = w.shape.n_steps, w.batch
    I = dict(I0)
    rounds = []
    for r in range(ROUNDS):
        I["hidden"] = hid[r]
        o = oracle.draft_round(w.shape, W, I, topk=2, want_logits=True)
        env = one_ulp_envelope(w.shape, W, I, list(range(B)), o)
        tgt = synth.make_targets(w.with_(seed=w.seed + 100 + r), o["draft_ids"])
        a = oracle.accept_greedy(o["draft_ids"], tgt, I["n_new"], I["kv_len"])
        rounds.append({"draft": o["draft_ids"], "top": o["topk_logits"], "target": tgt, "envelope": env,
                       "inputs": dict(I), "accept_len": a["accept_len"], "out_tokens": a["out_tokens"],
                       "kv_len": a["kv_len"]})
        tokens = np.zeros_like(I["tokens"])
        for b in range(B):
            n = int(a["accept_len"][b]) + 1
            tokens[b, :n] = a["out_tokens"][b, :n]
        I = dict(I, tokens=tokens, n_new=(a["accept_len"] + 1).astype(np.int32), kv_len=a["kv_len"],
                 k_cache=o["k_cache"], v_cache=o["v_cache"])
    return rounds


def gpu_loop(w, W, I, hid, target, model):
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    K, B = w.shape.n_steps, w.batch
    dr = model.drafter(w.shape, list(W["f_map"]), max_batch=B, max_ctx=int(I["max_ctx"]), max_new=K + 1, topk=1)
    t = {n: to_device(I[n]) for n in ("tokens", "n_new", "kv_len", "k_cache", "v_cache")}
    hd = to_device(hid)
    i32 = torch.int32
    draft = torch.full((ROUNDS, B, K), -7, dtype=i32, device="cuda")
    acc = torch.full((ROUNDS, B), -7, dtype=i32, device="cuda")
    out = torch.full((ROUNDS, B, K + 1), -7, dtype=i32, device="cuda")
    dr.draft_loop(t["tokens"], hd, t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], to_device(target), draft,
                  acc, out)
    flags = dr.sync_status()
    res = {"draft": to_numpy(draft), "accept_len": to_numpy(acc), "out_tokens": to_numpy(out),
           "tokens": to_numpy(t["tokens"]), "n_new": to_numpy(t["n_new"]), "kv_len": to_numpy(t["kv_len"]),
           "k_cache": to_numpy(t["k_cache"]), "flags": flags}
    dr.close()
    return res


def stepwise(w, W, I, hid, target, model):
    """The same rounds through prism_draft_round + prism_accept_greedy, next
    round's inputs prepared on the host from the device's outputs."""
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    K, B = w.shape.n_steps, w.batch
    dr = model.drafter(w.shape, list(W["f_map"]), max_batch=B, max_ctx=int(I["max_ctx"]), max_new=K + 1, topk=1)
    t = {n: to_device(I[n]) for n in ("tokens", "n_new", "kv_len", "k_cache", "v_cache")}
    i32 = torch.int32
    drafts, accs, outs = [], [], []
    for r in range(ROUNDS):
        ids = torch.empty((B, K), dtype=i32, device="cuda")
        dr.draft_round(t["tokens"], to_device(hid[r]), t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], ids)
        acc = torch.empty(B, dtype=i32, device="cuda")
        out = torch.empty((B, K + 1), dtype=i32, device="cuda")
        dr.accept_greedy(ids, to_device(target[r]), t["n_new"], t["kv_len"], acc, out)
        assert dr.sync_status() == 0
        a, o = to_numpy(acc), to_numpy(out)
        tok = to_numpy(t["tokens"])
        for b in range(B):
            tok[b, :a[b] + 1] = o[b, :a[b] + 1]
        t["tokens"] = to_device(tok)
        t["n_new"] = to_device((a + 1).astype(np.int32))
        drafts.append(to_numpy(ids))
        accs.append(a)
        outs.append(o)
    res = {"draft": np.stack(drafts), "accept_len": np.stack(accs), "out_tokens": np.stack(outs),
           "kv_len": to_numpy(t["kv_len"]), "k_cache": to_numpy(t["k_cache"])}
    dr.close()
    return res


@pytest.mark.parametrize("case", sorted(CASES))
def test_loop_matches_oracle_loop_and_single_rounds(case):
    w = CASES[case]
    K, B = w.shape.n_steps, w.batch
    W = synth.make_weights(w)
    I, hid = loop_inputs(w)
    orc = oracle_loop(w, W, I, hid)
    target = np.stack([r["target"] for r in orc])
    model = GpuModel(W)
    try:
        g = gpu_loop(w, W, I, hid, target, model)
        s = stepwise(w, W, I, hid, target, model)
    finally:
        model.close()
    assert g["flags"] == 0
    # the loop on the device equals the same rounds called one by one
    for key in ("draft", "accept_len", "out_tokens", "kv_len", "k_cache"):
        assert np.array_equal(g[key], s[key]), key
    # against the oracle, per sequence while the two stay in step
    compared = accepted = 0
    for b in range(B):
        for r, o in enumerate(orc):
            same = True
            for k in range(K):
                margin = o["top"][b, k, 0] - o["top"][b, k, 1]
                thr = MARGIN if k == 0 else 2 * max(ATOL, ENVELOPE_FACTOR * o["envelope"][b, k])
                if g["draft"][r, b, k] != o["draft"][b, k]:
                    assert margin <= thr, f"round {r} seq {b} step {k + 1}: id differs at margin {margin:.3e}"
                    same = False
                    break
            if not same:
                break
            compared += 1
            accepted += int(o["accept_len"][b])
            assert g["accept_len"][r, b] == o["accept_len"][b]
            assert np.array_equal(g["out_tokens"][r, b], o["out_tokens"][b])
            if r == ROUNDS - 1:
                assert g["kv_len"][b] == o["kv_len"][b]
                assert g["n_new"][b] == o["accept_len"][b] + 1
                n = int(g["n_new"][b])
                assert np.array_equal(g["tokens"][b, :n], o["out_tokens"][b, :n])
    print(case, "rounds compared", compared, "accepted drafts", accepted)
    assert compared >= B * 2 and accepted >= 1
    # every round from the oracle's own state at its start
    for r, o in enumerate(orc):
        _, _, rep = _check(w, W, o["inputs"], list(range(B)), topk=2)
        print(case, "round", r, "forced", rep)


def test_loop_rejects_short_max_new():
    import torch
    from paper_2602_01762_gb300 import PrismError
    w = CASES["tiny-bf16"]
    W = synth.make_weights(w)
    model = GpuModel(W)
    K, B = w.shape.n_steps, w.batch
    dr = model.drafter(w.shape, list(W["f_map"]), max_batch=B, max_ctx=64, max_new=K, topk=1)
    z = lambda *s: torch.zeros(s, dtype=torch.int32, device="cuda")
    kc = torch.zeros((B, w.shape.n_kv_heads, 64, w.shape.head_dim), dtype=torch.bfloat16, device="cuda")
    hid = torch.zeros((1, B, K, w.shape.hidden), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(PrismError, match="CAPACITY"):
        dr.draft_loop(z(B, K), hid, z(B), z(B), kc, kc.clone(), z(1, B, K + 1), z(1, B, K), z(1, B), z(1, B, K + 1))
    dr.close()
    model.close()
