"""The oracle's own sensitivity along the draft chain (CPU).

Under the bf16 numeric contract every activation operand is rounded to bf16
before its projection, and the chain feeds each step's h^ into the next
step's fusion (Sec. 3.2, the decode recurrence).  A change of one ulp in one
input element therefore flips later bf16 roundings, and each flip moves the
next step's input by a full bf16 ulp.  These tests measure that on the oracle
itself (no GPU): how far its own logits move, step by step, when one element
of the last input hidden row moves by one ulp.  They pin the reading the GPU
parity tests rest on: along a free-running chain no fp32 implementation can
stay within the max-abs bar the oracle is compared at, because the oracle
does not stay within it of itself; the deviation a GPU is allowed there is
measured, not assumed (``tests.parity.one_ulp_envelope``).
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from tests.parity import ATOL, one_ulp_envelope
from tests.test_gpu_round import MID_W, mid_case


def _fp32_activation_move(w, W, I, seqs):
    """The same one-ulp changes with the bf16 rounding points switched off
    (fp32 activations): the move of a smooth function of the input."""
    base = oracle.draft_round(w.shape, W, I, topk=1, want_logits=True, seqs=seqs, round_acts=False)
    return one_ulp_envelope(w.shape, W, I, seqs, base, round_acts=False)


def _check(w, W, I, seqs):
    base = oracle.draft_round(w.shape, W, I, topk=1, want_logits=True, seqs=seqs)
    again = oracle.draft_round(w.shape, W, I, topk=1, want_logits=True, seqs=seqs)
    assert np.array_equal(base["logits"], again["logits"])         # the oracle is deterministic
    env = one_ulp_envelope(w.shape, W, I, seqs, base)
    smooth = _fp32_activation_move(w, W, I, seqs)
    assert np.all(env[:, 0] > 0)
    # the rounding cascade, not the model's conditioning, makes the move:
    # without the bf16 rounding points the same changes move the logits at
    # least three times less at every step
    assert np.all(3 * smooth < env), (smooth, env)
    # and it grows along the chain
    assert np.all(env[:, -1] > 2 * env[:, 0])
    return env


def test_one_ulp_sensitivity_mid_size():
    W, I = mid_case()
    env = _check(MID_W, W, I, [0, 1, 2])
    print(np.round(env, 4))
    assert np.all(env[:, -1] > 0.015)


@pytest.mark.slow
def test_one_ulp_moves_the_llama3_8b_chain_beyond_the_max_abs_bar():
    """Llama-3-8B shape, batch 1, context 2048, K = 5 (the benchmark's round):
    one ulp of one input element moves the oracle's own logits by more than
    ATOL within the round."""
    w = synth.WORKLOADS["l3-8b-b1"]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    env = _check(w, W, I, [0])
    print(np.round(env, 4))
    assert env[0, 0] > 0.01
    assert env[0, -1] > ATOL
