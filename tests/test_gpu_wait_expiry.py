"""A bounded device wait that gives up, on the GPU.

Every wait between two roles of a ring kernel is bounded; when it gives up
the kernel sets the timeout bit of the device error word and winds down,
still waiting for the copies and MMAs it has in flight (the wind-down paths
are model-checked in tests/test_wait_expiry_cpu.py).  The option
``wait_polls`` bounds those waits per call: < 0 makes every one of them give
up at once, a small count makes them give up part-way through.  Here the
tiny drafter's round (streamed tcgen05 projections for the 64-row prefill,
staged ones and the CUDA-core ring for the single rows, the fused attention
cluster, with 8 or 4 compute warps) runs with both settings: the error word carries the timeout bit,
prism_sync_status returns PRISM_ERR_TIMEOUT, nothing faults, and the next
round on the same context, with the bound back to its default, matches the
oracle.
"""
from __future__ import annotations

import pytest

import oracle
import synth
from tests.gpu_harness import GpuModel, run_round
from tests.parity import compare_cache, compare_round, one_ulp_envelope

pytestmark = pytest.mark.gpu

PRISM_ERR_TIMEOUT = 8
TIMEOUT_BIT = 8


@pytest.mark.parametrize("attn", [{}, {"attn_warps": 4}], ids=["8-warp-attention", "4-warp-attention"])
def test_waits_that_give_up_report_timeout_and_the_context_recovers(attn):
    w = synth.WORKLOADS["tiny-bf16"]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    K = w.shape.n_steps
    model = GpuModel(W)
    try:
        dr = model.drafter(w.shape, list(W["f_map"]), max_batch=w.batch, max_ctx=int(I["max_ctx"]),
                           max_new=I["tokens"].shape[1], topk=4)
        # every role-to-role wait gives up at once: no copy or MMA is issued
        # past the first one, and every kernel reports it
        g = run_round(dr, I, n_steps=K, topk=4, options={"wait_polls": -1, **attn})
        assert g["flags"] & TIMEOUT_BIT
        assert dr.last_status == PRISM_ERR_TIMEOUT
        # one poll per wait: the waits give up part-way, with copies in flight
        g = run_round(dr, I, n_steps=K, topk=4, options={"wait_polls": 1, **attn})
        assert dr.last_status in (0, PRISM_ERR_TIMEOUT)
        # the built-in bound again: the same context drafts correctly
        g = run_round(dr, I, n_steps=K, topk=4, options={"wait_polls": 0, **attn})
        assert g["flags"] == 0 and dr.last_status == 0
        dr.close()
    finally:
        model.close()
    o = oracle.draft_round(w.shape, W, I, topk=5, want_logits=True, seqs=[0])
    compare_round(g, o, I, [0], K, 4, chain=True, envelope=one_ulp_envelope(w.shape, W, I, [0], o))
    compare_cache(g["k_cache"], g["v_cache"], o["k_cache"], o["v_cache"], I, [0], K)
