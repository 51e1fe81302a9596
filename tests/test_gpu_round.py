"""GPU parity of the draft round against the CPU oracle, through the C ABI.

Sizes: the tiny drafter (several CTAs per projection, a ragged prefill of 64
rows), a mid-size grouped-query drafter with a ragged batch, and every
full-size Llama-shaped workload in the launch configuration the benchmark
times (full batch on the GPU; the oracle computes an evenly spread sample of
the independent sequences).
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from synth.workloads import Shape, Workload
from tests.gpu_harness import (GpuModel, forced_step_inputs, gpu_round, oracle_step, run_round,
                               sample_seqs)
from tests.parity import compare_cache, compare_round, one_ulp_envelope

pytestmark = pytest.mark.gpu

MID = Shape("mid-gqa", 1024, 8, 2, 128, 2816, 32000, 4, "bf16", 500000.0)
MID_W = Workload("mid", MID, batch=3, ctx_lo=100, ctx_hi=700, n_new=4, topk=8, seed=21,
                 gain_sigma=0.1, f_map=(0, 1, 1, 2))


def mid_case():
    W, I = synth.make_weights(MID_W), synth.make_round_inputs(MID_W)
    I["n_new"][:] = [4, 1, 3]                 # ragged prefill lengths
    for b, n in enumerate(I["n_new"]):
        I["tokens"][b, n:] = 0
        I["hidden"][b, n:] = 0
    return W, I


def _check(w, W, I, seqs, *, topk, options=None):
    """Free-running round on the full batch, then every later step recomputed
    from the oracle's state (teacher forcing) in the same batch shape."""
    K = w.shape.n_steps
    model = GpuModel(W)
    try:
        g = gpu_round(w, W, I, topk=topk, model=model, options=options)
        assert g["flags"] == 0, f"device error word {g['flags']}"
        # one candidate more than is compared: the margin of the last compared
        # rank is its gap to the next one
        o = oracle.draft_round(w.shape, W, I, topk=topk + 1, want_logits=True, seqs=seqs)
        env = one_ulp_envelope(w.shape, W, I, seqs, o)
        rep = compare_round(g, o, I, seqs, K, topk, chain=True, envelope=env)
        compare_cache(g["k_cache"], g["v_cache"], o["k_cache"], o["v_cache"], I, seqs, K)
        forced = {}
        for k in range(2, K + 1):
            Ik = forced_step_inputs(I, o, seqs, k)
            dr = model.drafter(w.shape, [W["f_map"][k - 1]], max_batch=w.batch, max_ctx=int(I["max_ctx"]),
                               max_new=1, topk=topk)
            gk = run_round(dr, Ik, n_steps=1, topk=topk, options=options)
            dr.close()
            assert gk["flags"] == 0
            compare_round(gk, oracle_step(o, k), Ik, seqs, 1, topk, report=forced)
            compare_cache(gk["k_cache"], gk["v_cache"], o["k_cache"], o["v_cache"], Ik, seqs, 1)
        rep["forced"] = forced
    finally:
        model.close()
    return g, o, rep


@pytest.mark.parametrize("name", ["tiny-f32", "tiny-bf16", "tiny-f32-decode"])
def test_tiny_round(name):
    w = synth.WORKLOADS[name]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    _, _, rep = _check(w, W, I, [0], topk=4)
    assert rep["ids_compared"] >= 1


def test_mid_ragged_batch_round():
    W, I = mid_case()
    _, _, rep = _check(MID_W, W, I, [0, 1, 2], topk=8)
    print(rep)
    assert rep["ids_compared"] >= 6


@pytest.mark.slow
@pytest.mark.parametrize("name,n_sample", [("l3-8b-b1", 1), ("l3-8b-b1-m2", 1), ("l3-8b-b16", 3), ("l3-8b-b64", 3),
                                           ("l2-7b-b8", 3), ("l3-70b-b32", 2)])
def test_full_size_round(name, n_sample):
    w = synth.WORKLOADS[name]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    seqs = sample_seqs(w.batch, n_sample)
    _, _, rep = _check(w, W, I, seqs, topk=w.topk)
    print(name, rep)
    assert rep["ids_compared"] >= 1


def test_modes_are_bit_identical():
    """Graph replay vs eager launches, with and without programmatic
    dependent launch, and a second replay: identical bits."""
    W, I = mid_case()
    runs = [gpu_round(MID_W, W, I, topk=8, options={"use_graph": g, "use_pdl": p})
            for g, p in ((1, 1), (0, 0), (0, 1), (1, 0))]
    for r in runs[1:]:
        for key in ("draft_ids", "topk_ids", "topk_logits", "logits", "hidden_out", "k_cache", "v_cache"):
            assert np.array_equal(r[key], runs[0][key]), key


@pytest.mark.parametrize("options", [{"gemv_tcgen05": 0}, {"gemv_tcgen05": 0, "gemv_cuda_core": 0}],
                         ids=["cuda-core-ring", "mma-sync"])
def test_fallback_projection_kernels_match_oracle(options):
    """The kernels that carry projections the tcgen05 kernel does not take
    (more than 16 activation rows, fp32 weights): the CUDA-core TMA-ring
    kernel and the warp-level mma.sync kernel, forced for every projection."""
    W, I = mid_case()
    g = gpu_round(MID_W, W, I, topk=8, options=options)
    assert g["flags"] == 0
    o = oracle.draft_round(MID_W.shape, W, I, topk=8, want_logits=True, seqs=[0, 1, 2])
    env = one_ulp_envelope(MID_W.shape, W, I, [0, 1, 2], o)
    compare_round(g, o, I, [0, 1, 2], MID_W.shape.n_steps, 8, chain=True, envelope=env)
    compare_cache(g["k_cache"], g["v_cache"], o["k_cache"], o["v_cache"], I, [0, 1, 2], MID_W.shape.n_steps)


TCGEN05 = {"gemv_tcgen05": 2}      # every projection, gate/up included, on the tcgen05 kernel


@pytest.mark.parametrize("case", ["tiny-bf16", "mid"])
def test_tcgen05_projection_path_matches_oracle(case):
    """Projections on the tcgen05 kernel (TMA tensor loads, MMA into tensor
    memory, split-K for short outputs); prefill rows beyond 16 stay on the
    CUDA-core kernel, so the tiny case mixes both."""
    if case == "mid":
        w = MID_W
        W, I = mid_case()
        seqs = [0, 1, 2]
    else:
        w = synth.WORKLOADS[case]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
        seqs = [0]
    _, _, rep = _check(w, W, I, seqs, topk=8, options=TCGEN05)
    print(case, rep)
    assert rep["ids_compared"] >= 1


@pytest.mark.parametrize("case", ["tiny-bf16", "tiny-f32", "mid"])
def test_split_attention_path_matches_oracle(case):
    """Attention as two kernels (RoPE/append, then split-KV attention with a
    last-CTA combine) instead of the fused cluster kernel."""
    if case == "mid":
        w = MID_W
        W, I = mid_case()
        seqs = [0, 1, 2]
    else:
        w = synth.WORKLOADS[case]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
        seqs = [0]
    _, _, rep = _check(w, W, I, seqs, topk=4, options={"attn_fused": 0})
    assert rep["ids_compared"] >= 1


def test_fused_attention_on_cuda_cores_matches_oracle():
    """The fused RoPE/append/attention kernel with QK^T and PV on CUDA cores
    instead of tensor-core MMAs, at a size whose context spans several chunks."""
    W, I = mid_case()
    _, _, rep = _check(MID_W, W, I, [0, 1, 2], topk=4, options={"attn_tc": 0})
    assert rep["ids_compared"] >= 1


def test_four_warp_cluster_attention_matches_oracle():
    """The cluster attention kernel with 4 compute warps (64-key stages, two
    CTAs per SM) and a cluster of CTAs per (sequence, KV head) merging
    through distributed shared memory."""
    W, I = mid_case()
    _, _, rep = _check(MID_W, W, I, [0, 1, 2], topk=4, options={"attn_warps": 4})
    assert rep["ids_compared"] >= 1


def test_tcgen05_modes_bit_identical():
    """Graph replay, eager launches, with and without programmatic dependent
    launch: identical outputs on the tcgen05 path (split-K sums in fixed order)."""
    W, I = mid_case()
    model = GpuModel(W)
    try:
        runs = []
        for graph, pdl in ((1, 1), (0, 1), (0, 0), (1, 0)):
            dr = model.drafter(MID_W.shape, list(W["f_map"]), max_batch=MID_W.batch, max_ctx=int(I["max_ctx"]),
                               max_new=I["tokens"].shape[1], topk=8)
            r = run_round(dr, I, n_steps=MID_W.shape.n_steps, topk=8,
                          options=dict(TCGEN05, use_graph=graph, use_pdl=pdl))
            dr.close()
            assert r["flags"] == 0
            runs.append(r)
        for r in runs[1:]:
            for key in ("draft_ids", "topk_ids", "topk_logits", "logits", "hidden_out", "k_cache", "v_cache"):
                assert np.array_equal(r[key], runs[0][key]), key
    finally:
        model.close()


STAGED = {"tc_stream_rows": 8}      # fewer than 8 activation rows staged in shared memory


@pytest.mark.parametrize("case,topk", [("tiny-bf16", 4), ("mid", 8), ("mid", 1)])
def test_staged_projection_path_matches_oracle(case, topk):
    """The tcgen05 projections with their activation rows staged whole in
    shared memory (built per CTA: embedding gather, RMSNorm, bf16 rounding)
    and split-K sums added by each tile's last CTA, which the rounds of fewer
    than tc_stream_rows rows take; by default every row streams."""
    if case == "mid":
        w = MID_W
        W, I = mid_case()
        seqs = [0, 1, 2]
    else:
        w = synth.WORKLOADS[case]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
        seqs = [0]
    _, _, rep = _check(w, W, I, seqs, topk=topk, options=STAGED)
    assert rep["ids_compared"] >= 1


@pytest.mark.parametrize("lm_stream", [1, 0], ids=["streamed", "staged"])
def test_mid_top1_round(lm_stream):
    """The greedy top-1 round at mid size (3 rows, a vocabulary of 32000 in
    250 tiles of 128 rows, hidden size 1024): the LM head with its rows
    streamed beside the weights and the packed top-1 joined in the kernel,
    and with its rows staged in shared memory, both against the oracle,
    free-running and teacher-forced."""
    W, I = mid_case()
    _, _, rep = _check(MID_W, W, I, [0, 1, 2], topk=1, options={"lm_stream": lm_stream})
    assert rep["ids_compared"] >= 1


@pytest.mark.slow
@pytest.mark.parametrize("name,n_sample", [("l3-8b-b1", 1), ("l3-8b-b16", 3)])
def test_cuda_core_full_size_round(name, n_sample):
    """Full-size rounds with every projection on the CUDA-core ring kernel."""
    w = synth.WORKLOADS[name]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    _, _, rep = _check(w, W, I, sample_seqs(w.batch, n_sample), topk=w.topk, options={"gemv_tcgen05": 0})
    print(name, rep)
    assert rep["ids_compared"] >= 1


def test_graph_replay_is_repeatable():
    import torch
    W, I = mid_case()
    g = gpu_round(MID_W, W, I, topk=8, keep=True)
    dr, t, out = g["_drafter"], g["_t"], g["_out"]
    first = out["logits"].clone()
    for _ in range(3):
        dr.draft_round(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"],
                       out["draft_ids"], out["topk_ids"], out["topk_logits"], out["logits"], out["hidden_out"])
    assert dr.sync_status() == 0
    assert torch.equal(first, out["logits"])
    dr.close()


def test_accept_greedy_matches_oracle():
    import torch
    from paper_2602_01762_gb300 import Drafter
    from paper_2602_01762_gb300.host import to_device, to_numpy
    K, B = 5, 700
    rng = np.random.default_rng(9)
    draft = rng.integers(0, 50, (B, K)).astype(np.int32)
    target = np.concatenate([draft, rng.integers(0, 50, (B, 1))], 1).astype(np.int32)
    flip = rng.uniform(size=(B, K)) < 0.3
    target[:, :K][flip] = (target[:, :K][flip] + 1) % 50
    n_new = rng.integers(1, 7, B).astype(np.int32)
    kv = rng.integers(0, 1000, B).astype(np.int32)
    exp = oracle.accept_greedy(draft, target, n_new, kv)
    dr = Drafter(hidden=64, n_q_heads=2, n_kv_heads=2, head_dim=64, ffn=64, vocab=64, n_steps=K,
                 max_batch=B, max_ctx=64, max_new=1)
    t = [to_device(x) for x in (draft, target, n_new, kv)]
    acc = torch.empty(B, dtype=torch.int32, device="cuda")
    out = torch.empty((B, K + 1), dtype=torch.int32, device="cuda")
    dr.accept_greedy(t[0], t[1], t[2], t[3], acc, out)
    assert dr.sync_status() == 0
    assert np.array_equal(to_numpy(acc), exp["accept_len"])
    assert np.array_equal(to_numpy(out), exp["out_tokens"])
    assert np.array_equal(to_numpy(t[3]), exp["kv_len"])
    dr.close()


def test_round_then_accept_then_next_round():
    """The steady-state loop: draft, accept against targets built from the
    oracle's drafts (half forced agreement), commit, and draft again from the
    accepted tokens.  The GPU chain and the oracle chain each carry their own
    cache and acceptance results; both rounds match."""
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    w = synth.WORKLOADS["tiny-bf16"].with_(batch=2, ctx_lo=5, ctx_hi=9, n_new=2)
    K = w.shape.n_steps
    W, I = synth.make_weights(w), synth.make_round_inputs(w, max_new=K + 1)
    g = gpu_round(w, W, I, topk=2, keep=True)
    o = oracle.draft_round(w.shape, W, I, topk=2, want_logits=True)
    compare_round(g, o, I, [0, 1], K, 2, chain=True, envelope=one_ulp_envelope(w.shape, W, I, [0, 1], o))
    assert np.array_equal(g["draft_ids"], o["draft_ids"])
    target = synth.make_targets(w, o["draft_ids"])
    exp = oracle.accept_greedy(o["draft_ids"], target, I["n_new"], I["kv_len"])
    dr, t, out = g["_drafter"], g["_t"], g["_out"]
    acc = torch.empty(2, dtype=torch.int32, device="cuda")
    toks = torch.empty((2, K + 1), dtype=torch.int32, device="cuda")
    dr.accept_greedy(out["draft_ids"], to_device(target), t["n_new"], t["kv_len"], acc, toks)
    assert dr.sync_status() == 0
    g_acc, g_toks, g_kv = to_numpy(acc), to_numpy(toks), to_numpy(t["kv_len"])
    assert np.array_equal(g_acc, exp["accept_len"])
    assert np.array_equal(g_toks, exp["out_tokens"])
    assert np.array_equal(g_kv, exp["kv_len"])
    dr.close()

    def next_inputs(acc_len, out_tokens, kv_len, k_cache, v_cache):
        keep = np.arange(K + 1)[None, :] <= acc_len[:, None]
        hid = synth.normal(w.seed, "hidden2", I["hidden"].shape, 1.0, w.shape.dtype)
        hid[~keep] = 0
        return dict(I, n_new=(acc_len + 1).astype(np.int32),
                    tokens=np.where(keep, out_tokens, 0).astype(np.int32), hidden=hid,
                    kv_len=kv_len.astype(np.int32), k_cache=k_cache, v_cache=v_cache)

    I2_gpu = next_inputs(g_acc, g_toks, g_kv, g["k_cache"], g["v_cache"])
    I2_orc = next_inputs(exp["accept_len"], exp["out_tokens"], exp["kv_len"], o["k_cache"], o["v_cache"])
    g2 = gpu_round(w, W, I2_gpu, topk=2)
    o2 = oracle.draft_round(w.shape, W, I2_orc, topk=2, want_logits=True)
    compare_round(g2, o2, I2_gpu, [0, 1], K, 2, chain=True,
                  envelope=one_ulp_envelope(w.shape, W, I2_orc, [0, 1], o2))
    compare_cache(g2["k_cache"], g2["v_cache"], o2["k_cache"], o2["v_cache"], I2_gpu, [0, 1], K)


def test_device_error_word():
    """Out-of-range token ids, cache positions and n_new set the device error
    word (the kernels clamp or skip; nothing traps) and the context stays usable."""
    w = synth.WORKLOADS["tiny-bf16"].with_(batch=2, ctx_lo=3, ctx_hi=3, n_new=1)
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    bad = dict(I, tokens=I["tokens"].copy())
    bad["tokens"][1, 0] = w.shape.vocab + 5
    assert gpu_round(w, W, bad, topk=1)["flags"] & 1
    bad = dict(I, kv_len=np.array([3, I["max_ctx"] - 1], np.int32))
    assert gpu_round(w, W, bad, topk=1)["flags"] & 2
    bad = dict(I, n_new=np.array([1, 0], np.int32))
    assert gpu_round(w, W, bad, topk=1)["flags"] & 4
    assert gpu_round(w, W, I, topk=1)["flags"] == 0


def test_abi_rejects_bad_arguments():
    import torch
    from paper_2602_01762_gb300 import Drafter, PrismError
    from paper_2602_01762_gb300.host import to_device
    w = synth.WORKLOADS["tiny-bf16"]
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    dr = Drafter.from_shape(w.shape, max_batch=1, max_ctx=int(I["max_ctx"]), max_new=64)
    t = {n: to_device(I[n]) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
    ids = torch.empty((1, 3), dtype=torch.int32, device="cuda")
    with pytest.raises(PrismError, match="NOT_LOADED"):
        dr.draft_round(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], ids)
    lib = dr.lib
    assert lib.prism_draft_round(dr.h, 1, *([None] * 12)) == 1          # null tensors
    assert lib.prism_draft_round(dr.h, 2, *([None] * 12)) == 3          # batch > max_batch
    assert lib.prism_accept_greedy(dr.h, 5, *([None] * 7)) == 1
    x = torch.zeros(8, dtype=torch.int32, device="cuda")
    p = x.data_ptr()
    assert lib.prism_accept_greedy(dr.h, 5, p, p, p, p, p, p, None) == 3  # batch > max_batch
    assert lib.prism_set_option(dr.h, b"no_such_option", 1) == 1
    dr.close()
