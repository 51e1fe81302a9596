"""GPU parity of tree drafting and tree acceptance against the CPU oracle,
through the C ABI.

The oracle recomputes the GPU's own tree (``follow``: the GPU's candidate
tokens and frontier choices), so every processed row can be compared.  Along
the tree the hidden state is re-rounded to bf16 at every step, exactly as in
the chain, so the bar is the chain's:
  * step 1 strictly (max-abs and relative L2);
  * later steps of the free-running tree by relative L2, and max-abs within
    ENVELOPE_FACTOR times the oracle's own one-ulp envelope of the same tree
    (``tree_envelope``); id and order decisions compared where the oracle's
    gaps exceed max(MARGIN, twice the measured max-abs deviation);
  * every row of steps 2..K once more from the oracle's own state (teacher
    forcing, ``forced_tree_rows``): the row's token, its emitting row's h^ and
    a cache holding the oracle's committed rows and the row's ancestors, run
    on the GPU as a one-step round, strictly: max-abs, relative L2 and the
    row's candidates wherever the oracle's gaps exceed MARGIN.
Decisions the GPU takes from its own numbers (frontiers, the verified tree,
its structure) are checked exactly against a re-sort of those numbers.
"""
from __future__ import annotations

from dataclasses import replace

import numpy as np
import pytest

import oracle
import synth
from synth.workloads import Shape, Workload
from tests.gpu_harness import GpuModel
from tests.parity import ATOL, ENVELOPE_FACTOR, MARGIN, REL_L2, _as_f64, rel_l2

pytestmark = pytest.mark.gpu

MID = Shape("mid-gqa-k4", 1024, 8, 2, 128, 2816, 32000, 4, "bf16", 500000.0)
MID_TREE = Workload("mid-tree", MID, batch=4, ctx_lo=100, ctx_hi=700, n_new=3, topk=1, seed=23,
                    gain_sigma=0.1, f_map=(0, 1, 1, 2), tree_width=4, tree_nodes=16)


def ragged(w, I):
    I = dict(I)
    I["n_new"] = I["n_new"].copy()
    if w.batch > 1 and w.n_new > 1:
        I["n_new"][1] = 1
        I["tokens"] = I["tokens"].copy()
        I["hidden"] = I["hidden"].copy()
        I["tokens"][1, 1:] = 0
        I["hidden"][1, 1:] = 0
    return I


def gpu_tree(w, W, I, *, width, n_nodes, model=None, options=None, repeat=1):
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    own = model is None
    model = model or GpuModel(W)
    B, K, V = w.batch, w.shape.n_steps, w.shape.vocab
    from paper_2602_01762_gb300 import Drafter
    dr = Drafter.from_shape(w.shape, max_batch=B, max_ctx=int(I["max_ctx"]), max_new=I["tokens"].shape[1],
                            topk=1, max_tree_width=width)
    dr.load_shared_weights(model.embed, model.lm_head)
    for k, m in enumerate(W["f_map"]):
        dr.load_step_weights(k, model.modules[m])
    for k, v in (options or {}).items():
        dr.set_option(k, v)
    P = oracle.pool_size(K, width)
    i32, f32 = torch.int32, torch.float32
    res = []
    for _ in range(repeat):
        t = {n: to_device(I[n]) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
        out = {
            "tree_tokens": torch.full((B, n_nodes), -7, dtype=i32, device="cuda"),
            "tree_parents": torch.full((B, n_nodes), -7, dtype=i32, device="cuda"),
            "tree_depths": torch.full((B, n_nodes), -7, dtype=i32, device="cuda"),
            "tree_scores": torch.zeros((B, n_nodes), dtype=f32, device="cuda"),
            "pool_tokens": torch.full((B, P), -7, dtype=i32, device="cuda"),
            "pool_parents": torch.full((B, P), -7, dtype=i32, device="cuda"),
            "pool_scores": torch.zeros((B, P), dtype=f32, device="cuda"),
            "frontier": torch.full((B, K, width), -7, dtype=i32, device="cuda"),
            "row_logits": torch.zeros((K, B, width, V), dtype=f32, device="cuda"),
        }
        dr.draft_tree(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], width,
                      out["tree_tokens"], out["tree_parents"], out["tree_depths"], out["tree_scores"],
                      out["pool_tokens"], out["pool_parents"], out["pool_scores"], out["frontier"],
                      out["row_logits"])
        flags = dr.sync_status()
        r = {k: to_numpy(v) for k, v in out.items()}
        r["row_logits"] = r["row_logits"].transpose(1, 0, 2, 3)     # [B, K, w, V] like the oracle
        r["k_cache"], r["v_cache"], r["flags"] = to_numpy(t["k_cache"]), to_numpy(t["v_cache"]), flags
        res.append(r)
    dr.close()
    if own:
        model.close()
    torch.cuda.empty_cache()
    return res if repeat > 1 else res[0]


def _order(scores, idx):
    """Indices sorted by score descending, then index ascending (float32 keys)."""
    return idx[np.lexsort((idx, -scores[idx]))]


def check_self_consistent(g, K, w, m):
    """Decisions the GPU took from its own numbers, re-sorted here: exact."""
    B, P = g["pool_scores"].shape
    for b in range(B):
        sc = g["pool_scores"][b].astype(np.float32)
        for k in range(1, K + 1):
            base = 0 if k == 1 else w + (k - 2) * w * w
            cand = np.arange(base, base + (w if k == 1 else w * w))
            assert list(g["frontier"][b, k - 1]) == list(_order(sc, cand)[:w]), f"seq {b} step {k}: frontier"
            if k >= 2:
                for j in range(w):
                    par = g["pool_parents"][b, base + j * w: base + (j + 1) * w]
                    assert set(par) == {g["frontier"][b, k - 2, j]}
        best = np.sort(_order(sc, np.arange(P))[:m])
        pos = {int(e): i for i, e in enumerate(best)}
        for i, e in enumerate(best):
            assert g["tree_tokens"][b, i] == g["pool_tokens"][b, e]
            d = 1 if e < w else 2 + (e - w) // (w * w)
            assert g["tree_depths"][b, i] == d
            par = g["pool_parents"][b, e]
            assert g["tree_parents"][b, i] == (-1 if par < 0 else pos[int(par)])
            assert g["tree_scores"][b, i] == g["pool_scores"][b, e]


def tree_envelope(shape, W, I, seqs, follow, base, *, width, n_nodes, trials: int = 3):
    """The oracle's own sensitivity along the tree: ``trials`` oracle tree
    rounds following the same tree (``follow``), each with ONE element of the
    last input hidden row of every sequence moved by one ulp of its storage
    type, against the unperturbed oracle tree ``base``.  Returns [len(seqs),
    K]: per step the largest max-abs move of any row's logits over the
    trials, made non-decreasing along the steps."""
    K, d = shape.n_steps, shape.hidden
    env = np.zeros((len(seqs), K))
    for t in range(trials):
        hid = I["hidden"].copy()
        e = (t + 1) * d // (trials + 1)
        for b in seqs:
            i = int(I["n_new"][b]) - 1
            if hid.dtype == np.uint16:
                hid[b, i, e] = np.uint16(hid[b, i, e] + 1)
            else:
                hid[b, i, e] = np.nextafter(hid[b, i, e], np.float32(np.inf))
        o = oracle.draft_tree(shape, W, dict(I, hidden=hid), width=width, n_nodes=n_nodes, follow=follow,
                              seqs=seqs)
        move = np.abs(o["row_logits"] - base["row_logits"]).max(axis=(2, 3))      # [seqs, K]
        env = np.maximum(env, move)
    return np.maximum.accumulate(env, axis=1)


def _tree_row_path(g, b, k, j, w):
    """(emitting step, emitting row) of row j of step k >= 2 of sequence b in
    the GPU's tree, and the rows (step, row) of its ancestors at steps
    2..k-1, nearest first."""
    def emitter(kk, jj):
        parent = int(g["frontier"][b, kk - 2, jj])
        if parent < w:
            return 1, 0
        return kk - 1, (parent - (w + (kk - 3) * w * w)) // w
    em = emitter(k, j)
    anc = []
    cur = em
    while cur[0] >= 2:
        anc.append(cur)
        cur = emitter(*cur)
    return em, anc


def forced_tree_rows(w, W, I, g, o, seqs, width, model, report):
    """Every row of steps 2..K recomputed on the GPU from the oracle's state.

    A tree row at step k is the chain's row at position L + n + k - 2 whose
    visible keys are the committed and prefill rows plus its ancestors'
    rows (Sec. 3.2's recurrence along one path of the tree; the oracle pins
    show the two equal).  So each row runs as a one-step round of step k's
    module: token = the row's candidate token, hidden = the oracle's h^ of
    the emitting row (rounded to the storage type, as the fusion input is),
    cache = the oracle's rows [0, L + n) followed by the oracle's ancestor
    rows at the positions L + n + i - 2 of their steps i, and kv_len =
    L + n + k - 2.  ``o`` must hold ``row_hidden`` and the oracle's caches.
    Returns the number of rows compared."""
    from tests.gpu_harness import run_round
    K, V = w.shape.n_steps, w.shape.vocab
    bf16 = I["hidden"].dtype == np.uint16
    rows = 0
    for k in range(2, K + 1):
        items = [(jj, b, j) for jj, b in enumerate(seqs) for j in range(width)]
        Bf = len(items)
        hsh = I["k_cache"].shape
        kc = np.zeros((Bf,) + hsh[1:], I["k_cache"].dtype)
        vc = np.zeros_like(kc)
        tokens = np.zeros((Bf, 1), np.int32)
        hidden = np.zeros((Bf, 1, w.shape.hidden), I["hidden"].dtype)
        kv = np.zeros(Bf, np.int32)
        for f, (jj, b, j) in enumerate(items):
            L, n = int(I["kv_len"][b]), int(I["n_new"][b])
            (ek, ej), anc = _tree_row_path(g, b, k, j, width)
            parent = int(g["frontier"][b, k - 2, j])
            tokens[f, 0] = g["pool_tokens"][b, parent]
            h = o["row_hidden"][jj, ek - 1, ej]
            hidden[f, 0] = oracle.to_bf16_bits(h) if bf16 else h.astype(np.float32)
            kc[f, :, :L + n] = o["k_cache"][jj, :, :L + n]
            vc[f, :, :L + n] = o["v_cache"][jj, :, :L + n]
            for (ak, aj) in anc:
                slot, pos = L + n + (ak - 2) * width + aj, L + n + ak - 2
                kc[f, :, pos] = o["k_cache"][jj, :, slot]
                vc[f, :, pos] = o["v_cache"][jj, :, slot]
            kv[f] = L + n + k - 2
        Ik = {"tokens": tokens, "hidden": hidden, "n_new": np.ones(Bf, np.int32), "kv_len": kv,
              "k_cache": kc, "v_cache": vc, "max_ctx": I["max_ctx"]}
        dr = model.drafter(w.shape, [W["f_map"][k - 1]], max_batch=Bf, max_ctx=int(I["max_ctx"]), max_new=1,
                           topk=width)
        gk = run_round(dr, Ik, n_steps=1, topk=width)
        dr.close()
        assert gk["flags"] == 0, f"device error word {gk['flags']}"
        for f, (jj, b, j) in enumerate(items):
            zg, zo = gk["logits"][f, 0].astype(np.float64), o["row_logits"][jj, k - 1, j]
            ma, rl = float(np.max(np.abs(zg - zo))), rel_l2(zg, zo)
            report["forced_max_abs_logit"] = max(report.get("forced_max_abs_logit", 0.0), ma)
            assert ma <= ATOL, f"seq {b} step {k} row {j} (forced): logit max-abs {ma:.3e}"
            assert rl <= REL_L2, f"seq {b} step {k} row {j} (forced): logit rel-L2 {rl:.3e}"
            order = np.lexsort((np.arange(V), -zo))
            top = zo[order[:width + 1]]
            for r in range(width):
                lo = top[r - 1] - top[r] if r > 0 else np.inf
                if min(lo, top[r] - top[r + 1]) > MARGIN:
                    report["forced_ids_compared"] = report.get("forced_ids_compared", 0) + 1
                    assert gk["topk_ids"][f, 0, r] == order[r], f"seq {b} step {k} row {j} (forced): candidate {r}"
            # the row's own key and value, at its chain position and at its tree slot
            L, n = int(I["kv_len"][b]), int(I["n_new"][b])
            pos, slot = L + n + k - 2, L + n + (k - 2) * width + j
            for gc, oc in ((gk["k_cache"], o["k_cache"]), (gk["v_cache"], o["v_cache"])):
                assert rel_l2(_as_f64(gc[f, :, pos]), _as_f64(oc[jj, :, slot])) <= REL_L2
            rows += 1
    return rows


def compare_tree(g, o, I, seqs, K, w, m, report, envelope):
    """g: GPU outputs over the full batch; o: the oracle following g's tree on
    `seqs`; envelope: ``tree_envelope`` of the same tree."""
    rep = report
    for key in ("rows", "ids_compared", "frontier_compared", "tree_compared"):
        rep.setdefault(key, 0)
    rep.setdefault("max_abs_logit", 0.0)
    rep.setdefault("max_rel_l2_logit", 0.0)
    rep.setdefault("max_score_err", 0.0)
    rep.setdefault("max_abs_over_envelope", 0.0)
    for jj, b in enumerate(seqs):
        ma_row = {}
        for k in range(1, K + 1):
            rows = 1 if k == 1 else w
            base = 0 if k == 1 else w + (k - 2) * w * w
            ma_step = 0.0
            for j in range(rows):
                zg, zo = g["row_logits"][b, k - 1, j].astype(np.float64), o["row_logits"][jj, k - 1, j]
                ma = float(np.max(np.abs(zg - zo)))
                rl = rel_l2(zg, zo)
                rep["rows"] += 1
                rep["max_abs_logit"] = max(rep["max_abs_logit"], ma)
                rep["max_rel_l2_logit"] = max(rep["max_rel_l2_logit"], rl)
                ma_step = max(ma_step, ma)
                ma_row[(k, j)] = ma
                if k == 1:
                    assert ma <= ATOL, f"seq {b} step 1: logit max-abs {ma:.3e}"
                else:
                    env = float(envelope[jj, k - 1])
                    rep["max_abs_over_envelope"] = max(rep["max_abs_over_envelope"], ma / max(env, 1e-30))
                    bar = max(ATOL, ENVELOPE_FACTOR * env)
                    assert ma <= bar, (f"seq {b} step {k} row {j}: logit max-abs {ma:.3e} > {bar:.3e} "
                                       f"({ENVELOPE_FACTOR} x the oracle's one-ulp envelope {env:.3e})")
                assert rl <= REL_L2, f"seq {b} step {k} row {j}: logit rel-L2 {rl:.3e}"
                thr = max(MARGIN, 2 * ma) if k > 1 else MARGIN
                # the row's w candidates: the oracle's best w where its gaps allow
                cand = g["pool_tokens"][b, base + j * w: base + (j + 1) * w]
                assert len(set(cand.tolist())) == w
                order = np.lexsort((np.arange(zo.size), -zo))
                top = zo[order[:w + 1]]
                for r in range(w):
                    lo = top[r - 1] - top[r] if r > 0 else np.inf
                    hi = top[r] - top[r + 1]
                    if min(lo, hi) > thr:
                        rep["ids_compared"] += 1
                        assert cand[r] == order[r], f"seq {b} step {k} row {j}: candidate {r}"
                # every GPU candidate is within thr of the oracle's w-th best logit
                assert np.all(zo[cand] >= top[w - 1] - thr), f"seq {b} step {k} row {j}: candidate outside top-w"
        # pool scores: oracle's log-probabilities along the same paths
        # (log-sum-exp is 1-Lipschitz in the max norm, so one level of a path
        # moves by at most twice its row's max-abs logit deviation)
        P = o["pool_score"].shape[1]
        depth = np.array([1 if e < w else 2 + (e - w) // (w * w) for e in range(P)])
        tol = np.zeros(P)
        for e in range(P):
            row = (1, 0) if depth[e] == 1 else (depth[e], (e - (w + (depth[e] - 2) * w * w)) // w)
            par = int(g["pool_parents"][b, e])
            tol[e] = (tol[par] if par >= 0 else 0.0) + 2 * ma_row[row] + 1e-5 * (1 + abs(o["pool_score"][jj, e]))
        err = np.abs(g["pool_scores"][b].astype(np.float64) - o["pool_score"][jj])
        rep["max_score_err"] = max(rep["max_score_err"], float(err.max()))
        assert np.all(err <= tol), f"seq {b}: pool score error {err.max():.3e}"
        # frontier and tree: equal to the oracle's choice wherever its boundary gap exceeds the tolerance
        so = o["pool_score"][jj]
        for k in range(2, K + 1):
            base = w + (k - 2) * w * w
            cand = np.arange(base, base + w * w)
            srt = _order(so, cand)
            gap = so[srt[w - 1]] - so[srt[w]] if cand.size > w else np.inf
            tk = 2 * tol[cand].max()
            if gap > tk:
                rep["frontier_compared"] += 1
                assert set(g["frontier"][b, k - 1]) == set(srt[:w]), f"seq {b} step {k}: frontier set"
            assert np.all(so[g["frontier"][b, k - 1]] >= so[srt[w - 1]] - tk)
        srt = _order(so, np.arange(P))
        if m < P:
            e_in, e_out = srt[m - 1], srt[m]
            if so[e_in] - so[e_out] > tol[e_in] + tol[e_out]:
                rep["tree_compared"] += 1
                assert list(o["tree_pool"][jj]) == sorted(srt[:m])
                assert np.array_equal(g["tree_tokens"][b], o["tree_tokens"][jj])
                assert np.array_equal(g["tree_parents"][b], o["tree_parent"][jj])
                assert np.array_equal(g["tree_depths"][b], o["tree_depth"][jj])
    return rep


def compare_tree_cache(g, o, I, seqs, K, w):
    for jj, b in enumerate(seqs):
        L, n = int(I["kv_len"][b]), int(I["n_new"][b])
        for gc, ic, oc in ((g["k_cache"], I["k_cache"], o["k_cache"]), (g["v_cache"], I["v_cache"], o["v_cache"])):
            assert np.array_equal(gc[b, :, :L], ic[b, :, :L]), f"seq {b}: committed rows modified"
            assert rel_l2(_as_f64(gc[b, :, L:L + n]), _as_f64(oc[jj, :, L:L + n])) <= REL_L2
            # draft slots of the first tree step (depth-1 nodes): inputs differ only by rounding
            got = _as_f64(gc[b, :, L + n:L + n + w])
            exp = _as_f64(oc[jj, :, L + n:L + n + w])
            assert rel_l2(got, exp) <= REL_L2, f"seq {b}: tree KV rows rel-L2 {rel_l2(got, exp):.3e}"


def run_case(w, W, I, seqs, *, width=None, n_nodes=None, options=None, forced=True):
    width = width or w.tree_width
    n_nodes = n_nodes or w.tree_nodes
    K = w.shape.n_steps
    model = GpuModel(W)
    try:
        g = gpu_tree(w, W, I, width=width, n_nodes=n_nodes, options=options, model=model)
        assert g["flags"] == 0, f"device error word {g['flags']}"
        check_self_consistent(g, K, width, n_nodes)
        follow = {"pool_tokens": g["pool_tokens"][seqs], "frontier": g["frontier"][seqs]}
        o = oracle.draft_tree(w.shape, W, I, width=width, n_nodes=n_nodes, follow=follow, seqs=seqs,
                              want_hidden=forced)
        env = tree_envelope(w.shape, W, I, seqs, follow, o, width=width, n_nodes=n_nodes)
        rep = compare_tree(g, o, I, seqs, K, width, n_nodes, {}, env)
        compare_tree_cache(g, o, I, seqs, K, width)
        if forced and K > 1:
            rep["forced_rows"] = forced_tree_rows(w, W, I, g, o, seqs, width, model, rep)
            assert rep["forced_rows"] == len(seqs) * (K - 1) * width
    finally:
        model.close()
    return g, o, rep


@pytest.mark.parametrize("name", ["tiny-bf16-tree", "tiny-f32-tree", "tiny-bf16-tree-peaked"])
def test_tiny_tree(name):
    w = synth.WORKLOADS["tiny-bf16-tree"]
    if name == "tiny-f32-tree":
        w = w.with_(shape=replace(w.shape, name="tiny-f32-k4", dtype="f32"))
    if name == "tiny-bf16-tree-peaked":
        # larger weights spread the logits, so that frontier and tree choices
        # clear the tolerance and are compared set for set
        w = w.with_(weight_sigma=0.2, seed=5, batch=6)
    W = synth.make_weights(w)
    I = ragged(w, synth.make_round_inputs(w))
    _, _, rep = run_case(w, W, I, list(range(w.batch)))
    print(name, rep)
    assert rep["ids_compared"] >= 10
    if name == "tiny-bf16-tree-peaked":
        assert rep["frontier_compared"] >= 4 and rep["tree_compared"] >= 1


def test_mid_tree_streamed_rows():
    """B * w = 16 rows: the projections stream their activation rows."""
    W = synth.make_weights(MID_TREE)
    I = ragged(MID_TREE, synth.make_round_inputs(MID_TREE))
    _, _, rep = run_case(MID_TREE, W, I, [0, 1, 3])
    print(rep)
    assert rep["ids_compared"] >= 10


def test_tiny_tree_staged_rows():
    """The tree's 12 rows per step (3 sequences x 4 branches) staged in
    shared memory (tc_stream_rows = 16) instead of streamed: the staged
    tcgen05 projections and LM head with 16-row operands."""
    w = synth.WORKLOADS["tiny-bf16-tree"]
    W = synth.make_weights(w)
    I = ragged(w, synth.make_round_inputs(w))
    _, _, rep = run_case(w, W, I, list(range(w.batch)), options={"tc_stream_rows": 16})
    assert rep["ids_compared"] >= 10


@pytest.mark.parametrize("width,n_nodes", [(1, 4), (2, 5), (8, 40)])
def test_tree_widths(width, n_nodes):
    W = synth.make_weights(MID_TREE)
    I = ragged(MID_TREE, synth.make_round_inputs(MID_TREE))
    _, _, rep = run_case(MID_TREE, W, I, [0, 2], width=width, n_nodes=n_nodes)
    assert rep["rows"] >= 2


@pytest.mark.parametrize("name", ["l3-8b-b1-tree", "l3-8b-b1-tree-m2"])
def test_full_size_tree_l3_8b_b1(name):
    """The paper's tree (6 steps, 4 branches, 16 verified) on the Llama-3-8B
    shape at batch 1, in the launch configuration the benchmark times; with a
    module per step and with the paper's two modules."""
    w = synth.WORKLOADS[name]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    _, _, rep = run_case(w, W, I, [0])
    print(rep)
    assert rep["ids_compared"] >= 10


def test_one_branch_tree_follows_the_chain():
    """Width 1 and n_nodes = K: the tree is the greedy chain of prism_draft_round."""
    from tests.gpu_harness import gpu_round
    W = synth.make_weights(MID_TREE)
    I = ragged(MID_TREE, synth.make_round_inputs(MID_TREE))
    K = MID.n_steps
    g = gpu_tree(MID_TREE, W, I, width=1, n_nodes=K)
    c = gpu_round(MID_TREE, W, I, topk=2)
    o = oracle.draft_round(MID, W, I, topk=2)
    for b in range(MID_TREE.batch):
        for k in range(K):
            assert np.all(g["tree_parents"][b] == np.arange(-1, K - 1))
            margin = o["topk_logits"][b, k, 0] - o["topk_logits"][b, k, 1]
            if g["tree_tokens"][b, k] != c["draft_ids"][b, k]:
                assert margin <= 5 * MARGIN, f"seq {b} step {k + 1}: tree and chain differ at margin {margin:.3e}"
                break
            assert rel_l2(g["row_logits"][b, k, 0], c["logits"][b, k]) <= REL_L2


def test_tree_replays_and_eager_are_bit_identical():
    W = synth.make_weights(MID_TREE)
    I = ragged(MID_TREE, synth.make_round_inputs(MID_TREE))
    a, b2 = gpu_tree(MID_TREE, W, I, width=4, n_nodes=16, repeat=2)
    e = gpu_tree(MID_TREE, W, I, width=4, n_nodes=16, options={"use_graph": 0})
    for key in ("tree_tokens", "tree_parents", "tree_scores", "pool_scores", "frontier", "row_logits",
                "k_cache", "v_cache"):
        assert np.array_equal(a[key], b2[key]), key
        assert np.array_equal(a[key], e[key]), key


def test_tree_acceptance_matches_oracle():
    import torch
    from paper_2602_01762_gb300 import Drafter
    from paper_2602_01762_gb300.host import to_device, to_numpy
    w = MID_TREE
    W = synth.make_weights(w)
    I = ragged(w, synth.make_round_inputs(w))
    g = gpu_tree(w, W, I, width=4, n_nodes=16)
    K, B = w.shape.n_steps, w.batch
    dr = Drafter.from_shape(w.shape, max_batch=B, max_ctx=int(I["max_ctx"]), max_new=I["tokens"].shape[1],
                            max_tree_width=4)
    for trial in range(3):
        tgt = synth.make_tree_targets(w.with_(seed=w.seed + trial), g["tree_tokens"], g["tree_parents"])
        o = oracle.accept_tree(g["tree_tokens"], g["tree_parents"], tgt, I["n_new"], I["kv_len"], K)
        d = {n: to_device(a) for n, a in (("tt", g["tree_tokens"]), ("tp", g["tree_parents"]), ("tn", tgt),
                                          ("n_new", I["n_new"]), ("kv", I["kv_len"]))}
        acc = torch.empty(B, dtype=torch.int32, device="cuda")
        nodes = torch.empty((B, K), dtype=torch.int32, device="cuda")
        out = torch.empty((B, K + 1), dtype=torch.int32, device="cuda")
        dr.accept_tree(d["tt"], d["tp"], d["tn"], d["n_new"], d["kv"], acc, nodes, out)
        assert dr.sync_status() == 0
        assert np.array_equal(to_numpy(acc), o["accept_len"])
        assert np.array_equal(to_numpy(nodes), o["accept_nodes"])
        assert np.array_equal(to_numpy(out), o["out_tokens"])
        assert np.array_equal(to_numpy(d["kv"]), o["kv_len"])
    dr.close()


def test_tree_rejects_bad_arguments():
    import torch
    from paper_2602_01762_gb300 import Drafter, PrismError
    from paper_2602_01762_gb300.host import to_device
    w = MID_TREE
    W = synth.make_weights(w)
    I = synth.make_round_inputs(w)
    model = GpuModel(W)
    dr = Drafter.from_shape(w.shape, max_batch=w.batch, max_ctx=int(I["max_ctx"]), max_new=I["tokens"].shape[1],
                            max_tree_width=2)
    dr.load_shared_weights(model.embed, model.lm_head)
    for k, m in enumerate(W["f_map"]):
        dr.load_step_weights(k, model.modules[m])
    t = {n: to_device(I[n]) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
    B = w.batch
    o = [torch.zeros((B, 4), dtype=torch.int32, device="cuda") for _ in range(3)]
    sc = torch.zeros((B, 4), dtype=torch.float32, device="cuda")
    with pytest.raises(PrismError, match="CAPACITY"):          # width above max_tree_width
        dr.draft_tree(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], 3,
                      o[0], o[1], o[2], sc)
    big = [torch.zeros((B, 1000), dtype=torch.int32, device="cuda") for _ in range(3)]
    with pytest.raises(PrismError, match="INVALID_ARG"):       # n_nodes above the pool size
        dr.draft_tree(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], 2,
                      big[0], big[1], big[2], torch.zeros((B, 1000), dtype=torch.float32, device="cuda"))
    dr.close()
    model.close()


@pytest.mark.parametrize("K,width,n_nodes", [(1, 4, 3), (9, 8, 40)])
def test_tree_step_count_edges(K, width, n_nodes):
    """One step (the tree is the best candidates of the prefill row alone) and
    (K - 1) * width = 64, every bit of the ancestor mask in use."""
    base = synth.WORKLOADS["tiny-bf16-tree"]
    w = base.with_(shape=replace(base.shape, name=f"tiny-bf16-k{K}", n_steps=K), tree_width=width, tree_nodes=n_nodes)
    W = synth.make_weights(w)
    I = ragged(w, synth.make_round_inputs(w))
    _, _, rep = run_case(w, W, I, list(range(w.batch)))
    assert rep["rows"] == w.batch * (1 + (K - 1) * width)
