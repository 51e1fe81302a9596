"""The LM-head entry point that allocates no device memory.

``prism_lm_head_topk_static`` is for callers that cannot call cudaMalloc (a
server whose caching allocator already holds the memory it may use, a plugin
limited to its host's pool, code enqueued under a capture mode that forbids
allocation): it keeps its scratch in a static device array inside the library
instead of a context workspace.  Here it must reproduce what the draft round
itself selects at each step: fed a step's hidden rows (the round's
``hidden_out``) and that step's final-norm gain, its logits and its top-k must
match the round's within the parity tolerances, over two calls in a row (the
second reuses the scratch the first left behind).

This file is collected last (``zz``) so that a run stopping at the first
failure has run every other test before it.
"""
from __future__ import annotations

import ctypes

import numpy as np
import pytest

import synth
from tests.parity import ATOL, MARGIN
from tests.test_gpu_round import MID_W, mid_case


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
        assert compared >= 2
    finally:
        rnd["_drafter"].close()
        rnd["_model"].close()
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
