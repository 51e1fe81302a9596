"""Pins of the oracle's tree drafting and tree acceptance.

What fixes these functions, other than the oracle itself:
  * every processed row equals the library reference (``tests/libref.py``,
    written with torch routines) run as a CHAIN forced down that row's path:
    same module per step, same rotary position (the depth), attention over the
    committed rows plus exactly the path's earlier rows.  This pins the tree
    mask, the cache-slot / position split and the pairing of each token with
    the hidden state of the row that emitted it;
  * the KV rows a tree row stores equal the chain's rows at that depth;
  * scores are sums of log-softmax values taken with scipy along each path;
  * candidates, frontiers and the verified tree equal brute-force sorts;
  * with one branch and n_nodes = K the tree is the greedy chain;
  * acceptance equals a brute-force search over all root paths, and on a
    chain-shaped tree equals the chain's greedy acceptance.
The last test plants mistakes in copies of the tree code and checks that
these pins catch each one.
"""
from __future__ import annotations

import os
from dataclasses import replace

import numpy as np
import pytest
from scipy import special

import oracle
import synth
from tests import test_oracle_pins as pins
from tests.libref import reference_round

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

TREE_SHAPE = replace(pins.PIN_SHAPE, name="pin-tree", n_steps=4)
TREE = pins.PIN.with_(shape=TREE_SHAPE, batch=2, tree_width=3, tree_nodes=10)


def tree_case():
    return pins.pin_case(TREE)


def _path(o, b, e):
    """Tokens from the root to pool entry e of sequence b."""
    toks = []
    while e >= 0:
        toks.append(int(o["pool_tokens"][b, e]))
        e = int(o["pool_parent"][b, e])
    return toks[::-1]


def _rows(K, w):
    """(step k, row j) of every processed row."""
    return [(1, 0)] + [(k, j) for k in range(2, K + 1) for j in range(w)]


def test_tree_rows_equal_the_reference_chain_forced_down_their_path():
    W, I = tree_case()
    K, w = TREE_SHAPE.n_steps, TREE.tree_width
    o = oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=TREE.tree_nodes, want_hidden=True)
    B = I["tokens"].shape[0]
    for b in range(B):
        L, n = int(I["kv_len"][b]), int(I["n_new"][b])
        for k, j in _rows(K, w):
            path = [] if k == 1 else _path(o, b, int(o["frontier"][b, k - 2, j]))
            assert len(path) == k - 1
            forced = np.zeros((B, K - 1), np.int32)
            forced[b, :k - 1] = path
            ref = reference_round(TREE_SHAPE, W, I, forced=forced)
            assert pins.max_rel(o["row_logits"][b, k - 1, j], ref["logits"][b, k - 1]) < 1e-9, (b, k, j)
            assert pins.max_rel(o["row_hidden"][b, k - 1, j], ref["hidden_out"][b, k - 1]) < 1e-9, (b, k, j)
            if k >= 2:
                # the row's K/V sit at slot L + n + (k - 2) w + j, the chain's at L + n + k - 2
                slot, pos = L + n + (k - 2) * w + j, L + n + k - 2
                assert pins.max_rel(o["k_cache"][b, :, slot], ref["k_cache"][b, :, pos]) < 1e-6
                assert pins.max_rel(o["v_cache"][b, :, slot], ref["v_cache"][b, :, pos]) < 1e-6


def test_tree_rows_under_the_bf16_contract_equal_the_reference_chain():
    """The same, with bf16 weights, caches and operand rounding: the reference
    rounds fp64 to bf16 by another route, so every rounding point must agree."""
    shape = replace(TREE_SHAPE, name="pin-tree-bf16", dtype="bf16")
    w = TREE.with_(shape=shape)
    W, I = pins.pin_case(w)
    K, wd = shape.n_steps, w.tree_width
    o = oracle.draft_tree(shape, W, I, width=wd, n_nodes=w.tree_nodes, want_hidden=True)
    B = I["tokens"].shape[0]
    for b in range(B):
        for k, j in _rows(K, wd):
            path = [] if k == 1 else _path(o, b, int(o["frontier"][b, k - 2, j]))
            forced = np.zeros((B, K - 1), np.int32)
            forced[b, :k - 1] = path
            ref = reference_round(shape, W, I, forced=forced, round_acts=True)
            assert pins.max_rel(o["row_logits"][b, k - 1, j], ref["logits"][b, k - 1]) < 1e-9, (b, k, j)
            assert pins.max_rel(o["row_hidden"][b, k - 1, j], ref["hidden_out"][b, k - 1]) < 1e-9, (b, k, j)


def test_committed_rows_untouched_and_step1_rows_as_chain():
    W, I = tree_case()
    o = oracle.draft_tree(TREE_SHAPE, W, I, width=TREE.tree_width, n_nodes=TREE.tree_nodes)
    ref = reference_round(TREE_SHAPE, W, I)
    for b in range(I["tokens"].shape[0]):
        L, n = int(I["kv_len"][b]), int(I["n_new"][b])
        assert np.array_equal(o["k_cache"][b, :, :L], I["k_cache"][b, :, :L])
        assert pins.max_rel(o["k_cache"][b, :, L:L + n], ref["k_cache"][b, :, L:L + n]) < 1e-6


def test_scores_candidates_frontiers_and_tree_by_brute_force():
    W, I = tree_case()
    K, w, m = TREE_SHAPE.n_steps, TREE.tree_width, TREE.tree_nodes
    o = oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=m)
    P = oracle.pool_size(K, w)
    for b in range(I["tokens"].shape[0]):
        # candidates: each row's w best tokens (logit descending, id ascending)
        for k, j in _rows(K, w):
            z = o["row_logits"][b, k - 1, j]
            best = np.lexsort((np.arange(z.size), -z))[:w]
            base = 0 if k == 1 else w + (k - 2) * w * w
            assert list(o["pool_tokens"][b, base + j * w: base + (j + 1) * w]) == list(best)
            assert abs(o["row_lse"][b, k - 1, j] - special.logsumexp(z)) < 1e-9 * abs(special.logsumexp(z))
        # scores: log-softmax summed along each path
        depth = np.array([1 if e < w else 2 + (e - w) // (w * w) for e in range(P)])
        for e in range(P):
            s, node = 0.0, e
            while node >= 0:
                d = depth[node]
                if d == 1:
                    k, j = 1, 0
                else:
                    k, j = d, (node - (w + (d - 2) * w * w)) // w
                lp = special.log_softmax(o["row_logits"][b, k - 1, j])
                s += lp[o["pool_tokens"][b, node]]
                node = o["pool_parent"][b, node]
            assert abs(o["pool_score"][b, e] - s) < 1e-9 * max(1.0, abs(s))
        # frontiers: the w best of each step's candidates; parents are the previous frontier
        sc = o["pool_score"][b]
        for k in range(1, K + 1):
            base = 0 if k == 1 else w + (k - 2) * w * w
            cand = np.arange(base, base + (w if k == 1 else w * w))
            want = cand[np.lexsort((cand, -sc[cand]))][:w]
            assert list(o["frontier"][b, k - 1]) == list(want)
            if k >= 2:
                for j in range(w):
                    assert set(o["pool_parent"][b, base + j * w: base + (j + 1) * w]) == {o["frontier"][b, k - 2, j]}
        # the verified tree: the m best of the pool, in pool order, parents inside and first
        allidx = np.arange(P)
        best = np.sort(allidx[np.lexsort((allidx, -sc))][:m])
        assert list(o["tree_pool"][b]) == list(best)
        for i, e in enumerate(best):
            assert o["tree_tokens"][b, i] == o["pool_tokens"][b, e]
            assert o["tree_depth"][b, i] == depth[e]
            p = o["tree_parent"][b, i]
            if depth[e] == 1:
                assert p == -1
            else:
                assert 0 <= p < i and best[p] == o["pool_parent"][b, e]


def test_one_branch_tree_is_the_greedy_chain():
    W, I = tree_case()
    K = TREE_SHAPE.n_steps
    o = oracle.draft_tree(TREE_SHAPE, W, I, width=1, n_nodes=K)
    c = oracle.draft_round(TREE_SHAPE, W, I, topk=1, want_logits=True)
    assert np.array_equal(o["tree_tokens"], c["draft_ids"])
    assert np.array_equal(o["tree_depth"], np.tile(np.arange(1, K + 1), (I["tokens"].shape[0], 1)))
    assert np.array_equal(o["tree_parent"], np.tile(np.arange(-1, K - 1), (I["tokens"].shape[0], 1)))
    assert pins.max_rel(o["row_logits"][:, :, 0], c["logits"]) < 1e-12
    assert np.array_equal(o["k_cache"], c["k_cache"]) and np.array_equal(o["v_cache"], c["v_cache"])


def test_following_a_tree_recomputes_it():
    W, I = tree_case()
    K, w, m = TREE_SHAPE.n_steps, TREE.tree_width, TREE.tree_nodes
    o = oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=m)
    f = oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=m,
                          follow={"pool_tokens": o["pool_tokens"], "frontier": o["frontier"]})
    for key in ("pool_tokens", "pool_parent", "pool_score", "frontier", "tree_tokens", "tree_parent", "row_logits"):
        assert np.array_equal(o[key], f[key]), key
    # another valid frontier (reversed choice order, one swapped candidate)
    # still gives rows that equal the chain forced down their paths
    fr = o["frontier"].copy()
    fr[:, 1] = fr[:, 1, ::-1]
    base = w
    fr[0, 1, 0] = next(e for e in range(base, base + w * w) if e not in fr[0, 1])
    g = oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=m, want_hidden=True,
                          follow={"pool_tokens": o["pool_tokens"], "frontier": fr})
    b, k, j = 0, 3, 0
    path = _path(g, b, int(g["frontier"][b, k - 2, j]))
    forced = np.zeros((I["tokens"].shape[0], K - 1), np.int32)
    forced[b, :k - 1] = path
    ref = reference_round(TREE_SHAPE, W, I, forced=forced)
    assert pins.max_rel(g["row_logits"][b, k - 1, j], ref["logits"][b, k - 1]) < 1e-9
    with pytest.raises(ValueError):
        bad = fr.copy()
        bad[0, 2, 0] = 0                      # not a candidate of step 3
        oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=m,
                          follow={"pool_tokens": o["pool_tokens"], "frontier": bad})


def test_tree_rejects_bad_arguments():
    W, I = tree_case()
    K, w = TREE_SHAPE.n_steps, TREE.tree_width
    with pytest.raises(ValueError):
        oracle.draft_tree(TREE_SHAPE, W, I, width=w, n_nodes=oracle.pool_size(K, w) + 1)
    J = dict(I)
    J["kv_len"] = I["kv_len"].copy()
    J["kv_len"][0] = int(I["max_ctx"]) - int(I["n_new"][0]) - (K - 1) * w + 1
    with pytest.raises(ValueError):
        oracle.draft_tree(TREE_SHAPE, W, J, width=w, n_nodes=5)


# ------------------------------------------------------------------ acceptance

def _brute_accept(tokens, parent, target, K):
    """Deepest node whose whole root path matches the target's tokens."""
    n = len(tokens)
    best, best_path = 0, []
    for i in range(n):
        path, node = [], i
        while node >= 0:
            path.append(node)
            node = parent[node]
        path = path[::-1]
        ok = all(tokens[p] == target[(parent[p] + 1)] for p in path)
        if ok and len(path) > best:
            best, best_path = len(path), path
    return best, best_path


def _random_tree(rng, n, K, V):
    depth = [0] * n
    parent, tokens = [], []
    for i in range(n):
        cands = [-1] + [p for p in range(i) if depth[p] < K]
        p = int(rng.choice(cands))
        parent.append(p)
        depth[i] = 1 if p < 0 else depth[p] + 1
        sib = {tokens[q] for q in range(i) if parent[q] == p}
        t = int(rng.integers(0, V))
        while t in sib:
            t = int(rng.integers(0, V))
        tokens.append(t)
    return np.array(tokens, np.int32), np.array(parent, np.int32)


def test_tree_acceptance_matches_brute_force():
    rng = np.random.default_rng(7)
    K, V, n = 5, 20, 12
    for _ in range(400):
        tok, par = _random_tree(rng, n, K, V)
        tgt = rng.integers(0, V, n + 1).astype(np.int32)
        # make a matching child likely
        for node in range(-1, n):
            kids = np.flatnonzero(par == node)
            if kids.size and rng.random() < 0.6:
                tgt[node + 1] = tok[rng.choice(kids)]
        r = oracle.accept_tree(tok[None], par[None], tgt[None], np.array([2]), np.array([10]), K)
        a, path = _brute_accept(tok, par, tgt, K)
        assert r["accept_len"][0] == a
        assert list(r["accept_nodes"][0, :a]) == path and all(r["accept_nodes"][0, a:] == -1)
        last = path[-1] if path else -1
        assert list(r["out_tokens"][0, :a + 1]) == [int(tok[p]) for p in path] + [int(tgt[last + 1])]
        assert all(r["out_tokens"][0, a + 1:] == -1)
        assert r["kv_len"][0] == 12


def test_chain_shaped_tree_acceptance_is_greedy_acceptance():
    rng = np.random.default_rng(3)
    K, V = 6, 5
    for _ in range(200):
        draft = rng.integers(0, V, (1, K)).astype(np.int32)
        target = rng.integers(0, V, (1, K + 1)).astype(np.int32)
        target[0, :K] = np.where(rng.random(K) < 0.7, draft[0], target[0, :K])
        g = oracle.accept_greedy(draft, target, np.array([1]), np.array([0]))
        t = oracle.accept_tree(draft, np.arange(-1, K - 1, dtype=np.int32)[None], target, np.array([1]),
                               np.array([0]), K)
        assert g["accept_len"][0] == t["accept_len"][0]
        assert np.array_equal(g["out_tokens"], t["out_tokens"])


# ------------------------------------------------------------------ pin strength

TREE_MUTANTS = [
    ("tree-rope-at-slot", "layer_row_at(c, m, u, L + n + k - 2, L + n + slot_off,",
     "layer_row_at(c, m, u, L + n + slot_off, L + n + slot_off,"),
    ("tree-no-ancestors", "for (int32_t i = 0; i < n_anc[erow]; ++i) anc[row * K + i] = anc[erow * K + i];",
     "n_anc[row] = 1;"),
    ("tree-hidden-of-root", "u[d + t] = H[erow * d + t];", "u[d + t] = H[t];"),
    ("tree-score-no-parent", "psc[e] = (parent < 0 ? 0.0 : psc[parent]) + (z[x] - lse);", "psc[e] = z[x] - lse;"),
    ("tree-score-logit", "psc[e] = (parent < 0 ? 0.0 : psc[parent]) + (z[x] - lse);",
     "psc[e] = (parent < 0 ? 0.0 : psc[parent]) + z[x];"),
    ("tree-emitting-row", "const int64_t erow = parent < w_ ? 0 : 1 + (k - 3) * w_ + (parent - (w_ + (k - 3) * w_ * w_)) / w_;",
     "const int64_t erow = parent < w_ ? 0 : 1 + (k - 3) * w_ + (parent - (w_ + (k - 3) * w_ * w_)) % w_;"),
    ("tree-frontier-skips-best", "int32_t e = idx[j];", "int32_t e = idx[j + 1 < ncand ? j + 1 : j];"),
    ("tree-final-size", "for (int64_t i = 0; i < n_nodes; ++i) pos_in_tree[idx[i]] = 0;",
     "for (int64_t i = 0; i < n_nodes; ++i) pos_in_tree[idx[i + (i + 1 < n_nodes ? 0 : 1)]] = 0;"),
    ("accept-tree-wrong-target", "const int32_t want = tn[cur + 1];", "const int32_t want = tn[a];"),
    ("tree-prefill-hidden-shift", "\n                            u[d + t] = load_el(hidden, ((int64_t)b * max_new + i) * d + t, bf);",
     "\n                            u[d + t] = i > 0 ? load_el(hidden, ((int64_t)b * max_new + i - 1) * d + t, bf) : 0.0;"),
    ("tree-round-input", "round_vec(u, 2 * d, c->round_acts);\n                    int64_t nv = 0;", "int64_t nv = 0;"),
    ("accept-tree-commit", "kv_len[b] = kv_len[b] + n_new[b];   /* only", "kv_len[b] = kv_len[b] + n_new[b] + a;   /* only"),
    ("accept-tree-bonus", "out_tokens[b * (K + 1) + a] = tn[cur + 1];", "out_tokens[b * (K + 1) + a] = tn[a];"),
]

TREE_PINS = [
    test_tree_rows_equal_the_reference_chain_forced_down_their_path,
    test_tree_rows_under_the_bf16_contract_equal_the_reference_chain,
    test_scores_candidates_frontiers_and_tree_by_brute_force,
    test_tree_acceptance_matches_brute_force,
]


def _caught() -> bool:
    for pin in TREE_PINS:
        try:
            pin()
        except (AssertionError, ValueError, FloatingPointError):
            return True
    return False


@pytest.mark.parametrize("name,orig,mut", TREE_MUTANTS, ids=[m[0] for m in TREE_MUTANTS])
def test_planted_tree_mistake_is_caught(tmp_path, name, orig, mut):
    src = open(SRC).read()
    assert src.count(orig) == 1, f"mutation anchor for {name} not found exactly once"
    p = tmp_path / "mutant.c"
    p.write_text(src.replace(orig, mut))
    lib = oracle.compile_source(str(p), str(tmp_path / f"libmutant_{name}.so"))
    with oracle.variant(lib):
        assert _caught(), f"planted mistake '{name}' was not caught by any pin"
