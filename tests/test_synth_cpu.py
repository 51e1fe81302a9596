"""The input recipe (synth/): seeded, synthetic inputs with the shapes and
distributions the workloads state, shared by both sides and free of the
method's arithmetic.  These tests check the recipe's stated properties."""
from __future__ import annotations

import numpy as np
import pytest

import synth
from synth.workloads import WORKLOADS, max_ctx_of


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_cache_capacity_covers_every_round(name):
    """kv_len + n_new + the round's draft rows (K for the chain, (K - 1) w for
    a tree) fit the cache for the longest committed context the recipe draws."""
    w = WORKLOADS[name]
    K = w.shape.n_steps
    need = w.ctx_hi + w.n_new + max(K, (K - 1) * w.tree_width)
    mc = max_ctx_of(w)
    assert need <= mc and mc % 16 == 0 and mc - need < 16


def test_round_inputs_follow_the_recipe():
    w = WORKLOADS["tiny-bf16"].with_(batch=6, ctx_lo=5, ctx_hi=40, n_new=3)
    I = synth.make_round_inputs(w, max_new=5)
    B, V = w.batch, w.shape.vocab
    assert I["tokens"].shape == (B, 5) and (I["tokens"][:, 3:] == 0).all()
    assert (I["tokens"] >= 0).all() and (I["tokens"] < V).all()
    assert (I["n_new"] == 3).all()
    assert ((I["kv_len"] >= 5) & (I["kv_len"] <= 40)).all() and len(set(I["kv_len"].tolist())) > 1
    hid = synth.bf16_to_f32(I["hidden"])
    assert (hid[:, 3:] == 0).all() and abs(hid[:, :3].std() - 1.0) < 0.05
    k = synth.bf16_to_f32(I["k_cache"])
    for b in range(B):
        L = int(I["kv_len"][b])
        assert (k[b, :, L:] == 0).all()                     # rows past the committed length are empty
        assert abs(k[b, :, :L].std() - 1.0) < 0.1
    # the same seed gives the same inputs; another seed other ones
    J = synth.make_round_inputs(w, max_new=5)
    assert all(np.array_equal(I[n], J[n]) for n in ("tokens", "hidden", "kv_len", "k_cache"))
    K2 = synth.make_round_inputs(w.with_(seed=w.seed + 1), max_new=5)
    assert not np.array_equal(I["k_cache"], K2["k_cache"])


def test_weights_follow_the_recipe():
    w = WORKLOADS["tiny-bf16"].with_(f_map=(0, 1, 1))
    W = synth.make_weights(w)
    assert set(W["modules"]) == {0, 1} and tuple(W["f_map"]) == (0, 1, 1)
    m = W["modules"][1]
    wq = synth.bf16_to_f32(m["w_qkv"])
    assert abs(wq.std() / 0.02 - 1) < 0.02 and abs(wq.mean()) < 1e-3
    assert (synth.bf16_to_f32(m["g_attn"]) == 1.0).all()          # gains are ones
    g = synth.make_weights(w.with_(gain_sigma=0.1))["modules"][0]["g_mlp"]
    g = synth.bf16_to_f32(g)
    assert abs(g.mean() - 1.0) < 0.02 and abs(g.std() - 0.1) < 0.02
    # modules differ from each other
    assert not np.array_equal(W["modules"][0]["w_o"], W["modules"][1]["w_o"])


def test_chain_targets_copy_the_draft_half_the_time():
    w = WORKLOADS["tiny-bf16"].with_(batch=4000)
    K, V = w.shape.n_steps, w.shape.vocab
    draft = synth.uniform_int(77, "drafts", (w.batch, K), 0, V - 1).astype(np.int32)
    t = synth.make_targets(w, draft)
    assert t.shape == (w.batch, K + 1) and (t >= 0).all() and (t < V).all()
    agree = (t[:, :K] == draft).mean()
    assert abs(agree - (0.5 + 0.5 / V)) < 0.02


def test_tree_targets_pick_a_child_half_the_time():
    w = WORKLOADS["tiny-bf16-tree"].with_(batch=3000)
    V = w.shape.vocab
    # a fixed tree: root -> nodes 0, 1; node 0 -> node 2; nodes 1 and 2 are leaves
    B, n = w.batch, 3
    tok = np.tile(np.array([[10, 20, 30]], np.int32), (B, 1))
    par = np.tile(np.array([[-1, -1, 0]], np.int32), (B, 1))
    t = synth.make_tree_targets(w, tok, par)
    assert t.shape == (B, n + 1) and (t >= 0).all() and (t < V).all()
    root = t[:, 0]
    assert abs(np.isin(root, [10, 20]).mean() - 0.5) < 0.03
    assert abs((root == 10).mean() - 0.25) < 0.03            # the child is chosen uniformly
    assert abs((t[:, 1] == 30).mean() - 0.5) < 0.03           # node 0's only child
    assert (t[:, 2] == 10).mean() < 0.01 and (t[:, 3] == 30).mean() < 0.01   # leaves: uniform
