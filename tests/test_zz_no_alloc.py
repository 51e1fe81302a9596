"""The LM-head entry point that allocates no device memory.

``prism_lm_head_topk_static`` is for callers that cannot call cudaMalloc (a
server whose caching allocator already holds the memory it may use, a plugin
limited to its host's pool, a process that fixes its whole device-memory
budget at start-up): it keeps its scratch in a static device array inside the library
instead of a context workspace.  Here it must reproduce what the draft round
itself selects at each step: fed a step's hidden rows (the round's
``hidden_out``) and that step's final-norm gain, its logits and its top-k must
match the round's within the parity tolerances, over two calls in a row (the
second reuses the scratch the first left behind).  Its logits are also held
to the oracle's final norm and LM head applied to the same rows, at the
Llama-3-8B vocabulary with the largest batch the static scratch takes.

This file is collected last (``zz``) so that a run stopping at the first
failure has run every other test before it.
"""
from __future__ import annotations

import ctypes

import numpy as np
import pytest

import oracle
import synth
from tests.parity import ATOL, MARGIN, REL_L2, _as_f64, rel_l2
from tests.test_gpu_round import MID_W, mid_case


def _oracle_lm_head(h, g_final, lm_head, eps, bf16):
    """The oracle's selection stage on given hidden rows: RMSNorm with the gain,
    the normed row rounded to bf16 under the bf16 contract, then the LM head,
    all in fp64.  h fp32 [B, d]; g_final and lm_head as stored (bf16 bits or
    fp32).  Returns logits [B, V]."""
    g = _as_f64(g_final)
    rows = []
    for b in range(h.shape[0]):
        nf = oracle.rmsnorm(h[b].astype(np.float64), g, eps)
        if bf16:
            nf = _as_f64(oracle.to_bf16_bits(nf))
        rows.append(oracle.matvec(lm_head, nf))
    return np.stack(rows)


def _check_against_oracle(st, z, topk):
    """Static-call outputs against oracle logits z [B, V]: max-abs and relative
    L2 per row, top-1 and ranked top-k ids wherever the oracle's gaps exceed
    the margin.  Returns the number of ids compared."""
    compared = 0
    for b in range(z.shape[0]):
        assert np.abs(st["logits"][b] - z[b]).max() <= ATOL, f"row {b}: logit max-abs"
        assert rel_l2(st["logits"][b], z[b]) <= REL_L2, f"row {b}: logit rel-L2"
        order = np.lexsort((np.arange(z.shape[1]), -z[b]))[:topk + 1]
        top = z[b][order]
        for r in range(topk):
            lo = top[r - 1] - top[r] if r > 0 else np.inf
            if min(lo, top[r] - top[r + 1]) > MARGIN:
                assert st["topk_ids"][b, r] == order[r], f"row {b}: top-{r + 1} id"
                if r == 0:
                    assert st["draft"][b] == order[0], f"row {b}: draft id"
                compared += 1
        assert np.abs(st["topk_logits"][b] - z[b][st["topk_ids"][b]]).max() <= ATOL
    return compared


def _static_call(h, g_final, lm_head, topk):
    import torch
    from paper_2602_01762_gb300 import lm_head_topk_static
    B, V = h.shape[0], lm_head.shape[0]
    out = {
        "draft": torch.full((B,), -7, dtype=torch.int32, device="cuda"),
        "topk_ids": torch.full((B, topk), -7, dtype=torch.int32, device="cuda"),
        "topk_logits": torch.zeros((B, topk), dtype=torch.float32, device="cuda"),
        "logits": torch.zeros((B, V), dtype=torch.float32, device="cuda"),
        "flags": torch.full((1,), -1, dtype=torch.int32, device="cuda"),
    }
    lm_head_topk_static(h, g_final, lm_head, out["draft"], out["topk_ids"], out["topk_logits"],
                        out["logits"], out["flags"], rms_eps=1e-5)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _compare(st, rnd, k):
    """Static-call outputs against the round's step-k outputs."""
    logits = rnd["logits"][:, k - 1]
    assert np.abs(st["logits"] - logits).max() <= ATOL
    assert np.abs(st["topk_logits"] - rnd["topk_logits"][:, k - 1]).max() <= ATOL
    compared = 0
    for b in range(logits.shape[0]):
        top2 = np.sort(logits[b])[-2:]
        if top2[1] - top2[0] < MARGIN:      # near-tie: either id is a correct top-1
            continue
        assert st["draft"][b] == rnd["draft_ids"][b, k - 1]
        assert st["topk_ids"][b, 0] == rnd["topk_ids"][b, k - 1, 0]
        compared += 1
    return compared


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["mid-bf16", "tiny-f32"])
def test_static_lm_head_matches_round_on_two_calls(case):
    import torch
    from tests.gpu_harness import gpu_round

    if case == "mid-bf16":
        w = MID_W
        W, I = mid_case()
    else:
        w = synth.WORKLOADS["tiny-f32"]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
    topk = 8
    rnd = gpu_round(w, W, I, topk=topk, keep=True)
    try:
        assert rnd["flags"] == 0
        model = rnd["_model"]
        hidden_dev = rnd["_out"]["hidden_out"]                  # [B, K, d] fp32 on the device
        compared = 0
        for k in (1, 2):                                         # two calls in a row
            h = hidden_dev[:, k - 1].contiguous()
            g_final = model.modules[W["f_map"][k - 1]]["g_final"]
            st = _static_call(h, g_final, model.lm_head, topk)
            assert st["flags"][0] == 0, f"device error word {st['flags'][0]}"
            compared += _compare(st, rnd, k)
            z = _oracle_lm_head(h.cpu().numpy(), W["modules"][W["f_map"][k - 1]]["g_final"], W["lm_head"],
                                w.shape.rms_eps, w.shape.dtype == "bf16")
            compared += _check_against_oracle(st, z, topk)
        assert compared >= 4
    finally:
        rnd["_drafter"].close()
        rnd["_model"].close()
        torch.cuda.empty_cache()


@pytest.mark.gpu
def test_static_lm_head_full_scratch_at_llama3_vocabulary():
    """64 rows (the partial lists fill the static array exactly) over the
    Llama-3-8B LM head (128256 x 4096, bf16), then 37 other rows on the
    scratch the first call left: both against the oracle."""
    import torch
    from paper_2602_01762_gb300.host import to_device
    V, d, seed = 128256, 4096, 41
    lm_host = synth.normal(seed, "lm_head", (V, d), 0.02, "bf16")
    g_host = synth.normal(seed, "g_final", (d,), 0.1, "bf16", mean=1.0)
    lm, g = to_device(lm_host), to_device(g_host)
    try:
        compared = 0
        for B, tag in ((64, "h_a"), (37, "h_b")):               # two calls in a row
            h_host = synth.normal(seed, tag, (B, d), 1.0, "f32")
            st = _static_call(to_device(h_host), g, lm, 8)
            assert st["flags"][0] == 0, f"device error word {st['flags'][0]}"
            z = _oracle_lm_head(h_host, g_host, lm_host, 1e-5, True)
            compared += _check_against_oracle(st, z, 8)
        assert compared >= 101
    finally:
        del lm, g
        torch.cuda.empty_cache()


def test_static_lm_head_rejects_sizes_beyond_its_scratch():
    """Host-side checks that run before any device work (no GPU needed)."""
    from paper_2602_01762_gb300 import library
    lib = library()
    fake = ctypes.c_void_p(1 << 20)                  # 16-byte aligned, never dereferenced
    args = dict(dtype=1, hidden=1024, vocab=32000, batch=65, topk=8)
    st = lib.prism_lm_head_topk_static(*args.values(), 1e-5, fake, None, fake, fake, None, None, None, None, None)
    assert st == 3                                   # PRISM_ERR_CAPACITY
    assert b"64" in lib.prism_get_error(None)
    st = lib.prism_lm_head_topk_static(1, 1024, 32000, 0, 8, 1e-5, fake, None, fake, fake, None, None, None, None, None)
    assert st == 2                                   # PRISM_ERR_SHAPE
    st = lib.prism_lm_head_topk_static(1, 1024, 32000, 4, 8, 1e-5, None, None, fake, fake, None, None, None, None, None)
    assert st == 1                                   # PRISM_ERR_INVALID_ARG
