"""GPU parity with a vocabulary that is not a multiple of the LM head's
128-row tile, so that the last tile of the LM head is partial.

The argmax and top-k of a draft step run over the whole vocabulary (Sec. 3.2,
the selection of each draft token).  A partial last tile exercises the
selection epilogues' bounds: rows past V must never enter a list, and the
last real rows must.  Covered: top-1 and top-8, the staged LM-head kernel
(fewer than 8 activation rows) and the streamed one (8 rows or more), the
sampled draw and the tree's top-w lists with its log-sum-exp pass.
"""
from __future__ import annotations

from dataclasses import replace

import pytest

import oracle
import synth
from synth.workloads import Workload
from tests.gpu_harness import sample_seqs
from tests.test_gpu_round import MID_W, _check
from tests.test_gpu_sampling import TAU, SEED, compare_sampled, sampled_gpu_round
from tests.test_gpu_tree import ragged, run_case

pytestmark = pytest.mark.gpu

# 4000 = 31 * 128 + 32: the last LM-head tile holds 32 real rows
TINY_V4000 = replace(synth.workloads.TINY_BF16, name="tiny-bf16-v4000", vocab=4000)


def _tiny(batch, n_new, ctx, topk):
    return Workload("tiny-bf16-v4000", TINY_V4000, batch, ctx, ctx, n_new, topk, 7)


@pytest.mark.parametrize("topk", [1, 8])
@pytest.mark.parametrize("batch,n_new,ctx", [(1, 64, 0), (1, 1, 63), (9, 1, 40)],
                         ids=["staged-prefill", "staged-decode", "streamed-b9"])
def test_ragged_vocabulary_round(topk, batch, n_new, ctx):
    w = _tiny(batch, n_new, ctx, topk)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    _, _, rep = _check(w, W, I, sample_seqs(batch, 3), topk=topk)
    assert rep["ids_compared"] >= 1


def test_ragged_vocabulary_mid_size():
    """Mid-size drafter with V = 32064 (250 full tiles and one of 64 rows), top-8."""
    w = MID_W.with_(shape=replace(MID_W.shape, name="mid-gqa-v32064", vocab=32064))
    W, I = mid_case_for(w)
    _, _, rep = _check(w, W, I, [0, 1, 2], topk=8)
    assert rep["ids_compared"] >= 6


def mid_case_for(w):
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    I["n_new"][:] = [4, 1, 3]                 # the ragged prefill lengths of the mid-size case
    for b, n in enumerate(I["n_new"]):
        I["tokens"][b, n:] = 0
        I["hidden"][b, n:] = 0
    return W, I


def test_ragged_vocabulary_sampled_round():
    w = _tiny(3, 4, 20, 1)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    g = sampled_gpu_round(w, W, I, tau=TAU, seed=SEED, topk=1)
    assert g["flags"] == 0
    seqs = [0, 1, 2]
    o = oracle.draft_round(w.shape, W, I, topk=1, want_logits=True, want_hidden=False, seqs=seqs,
                           temperature=TAU, seed=SEED)
    compared, _ = compare_sampled(g, o, seqs, w.shape.n_steps, TAU)
    assert compared >= len(seqs)


def test_ragged_vocabulary_tree():
    base = synth.WORKLOADS["tiny-bf16-tree"]
    w = base.with_(shape=replace(base.shape, name="tiny-bf16-k4-v4000", vocab=4000))
    W = synth.make_weights(w)
    I = ragged(w, synth.make_round_inputs(w))
    _, _, rep = run_case(w, W, I, list(range(w.batch)))
    assert rep["ids_compared"] >= 10
