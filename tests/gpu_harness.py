"""Run draft rounds through the C ABI (via the Python binding) on synthetic
inputs and bring every output back as numpy.

Two kinds of runs:
  * the free-running round (all K steps chained on the device);
  * a teacher-forced single step k: a one-step drafter bound to step k's
    module, started from the ORACLE's state after step k-1 (its draft token
    x^_{k-1}, its h^_{k-2} rounded to bf16 as the fusion input, and its KV
    cache).  Oracle outputs feed the GPU here, never the reverse.
"""
from __future__ import annotations

from dataclasses import replace

import numpy as np


class GpuModel:
    """Embedding, LM head and every module uploaded once."""

    def __init__(self, W):
        from paper_2602_01762_gb300 import STEP_TENSORS
        from paper_2602_01762_gb300.host import to_device
        self.W = W
        self.embed = to_device(W["embed"])
        self.lm_head = to_device(W["lm_head"])
        self.modules = {m: {n: to_device(mod[n]) for n in STEP_TENSORS} for m, mod in W["modules"].items()}

    def drafter(self, shape, step_modules, *, max_batch, max_ctx, max_new, topk):
        from paper_2602_01762_gb300 import Drafter
        sh = replace(shape, n_steps=len(step_modules))
        dr = Drafter.from_shape(sh, max_batch=max_batch, max_ctx=max_ctx, max_new=max_new, topk=topk)
        dr.load_shared_weights(self.embed, self.lm_head)
        for k, m in enumerate(step_modules):
            dr.load_step_weights(k, self.modules[m])
        return dr

    def close(self):
        import torch
        self.embed = self.lm_head = None
        self.modules = {}
        torch.cuda.empty_cache()


def run_round(dr, I, *, n_steps, topk, logits=True, hidden=True, keep=False, options=None):
    import torch
    from paper_2602_01762_gb300.host import to_device, to_numpy
    B = I["tokens"].shape[0]
    for k, v in (options or {}).items():
        dr.set_option(k, v)
    t = {n: to_device(I[n]) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
    i32, f32 = torch.int32, torch.float32
    out = {
        "draft_ids": torch.full((B, n_steps), -7, dtype=i32, device="cuda"),
        "topk_ids": torch.full((B, n_steps, topk), -7, dtype=i32, device="cuda"),
        "topk_logits": torch.zeros((B, n_steps, topk), dtype=f32, device="cuda"),
        "logits": torch.zeros((B, n_steps, dr.vocab), dtype=f32, device="cuda") if logits else None,
        "hidden_out": torch.zeros((B, n_steps, dr.hidden), dtype=f32, device="cuda") if hidden else None,
    }
    dr.draft_round(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"],
                   out["draft_ids"], out["topk_ids"], out["topk_logits"], out["logits"], out["hidden_out"])
    flags = dr.sync_status()
    res = {k: (None if v is None else to_numpy(v)) for k, v in out.items()}
    res["k_cache"] = to_numpy(t["k_cache"])
    res["v_cache"] = to_numpy(t["v_cache"])
    res["flags"] = flags
    if keep:
        res["_t"], res["_out"] = t, out
    return res


def gpu_round(w, W, I, *, topk, logits=True, hidden=True, options=None, keep=False, model=None):
    """Free-running round of workload w (all K steps) on inputs I."""
    import torch
    own = model is None
    model = model or GpuModel(W)
    dr = model.drafter(w.shape, list(W["f_map"]), max_batch=w.batch, max_ctx=int(I["max_ctx"]),
                       max_new=I["tokens"].shape[1], topk=topk)
    res = run_round(dr, I, n_steps=w.shape.n_steps, topk=topk, logits=logits, hidden=hidden,
                    keep=keep, options=options)
    if keep:
        res["_drafter"], res["_model"] = dr, model
    else:
        dr.close()
        if own:
            model.close()
        torch.cuda.empty_cache()
    return res


def forced_step_inputs(I, orc, seqs, k: int) -> dict:
    """Inputs of a one-step round that recomputes draft step k (k >= 2) from
    the oracle's state, for the sampled sequences `seqs` (the others get
    valid filler rows whose outputs are ignored)."""
    import oracle
    B = I["tokens"].shape[0]
    tokens = I["tokens"][:, :1].copy()
    hidden = I["hidden"][:, :1].copy()
    kv = (I["kv_len"] + I["n_new"] + (k - 2)).astype(np.int32)
    kc, vc = I["k_cache"].copy(), I["v_cache"].copy()
    bf16 = I["hidden"].dtype == np.uint16
    for j, b in enumerate(seqs):
        tokens[b, 0] = orc["draft_ids"][j, k - 2]
        h = orc["hidden_out"][j, k - 2]
        hidden[b, 0] = oracle.to_bf16_bits(h) if bf16 else h.astype(np.float32)
        kc[b] = orc["k_cache"][j]
        vc[b] = orc["v_cache"][j]
    return {"tokens": tokens, "hidden": hidden, "n_new": np.ones(B, np.int32), "kv_len": kv,
            "k_cache": kc, "v_cache": vc, "max_ctx": I["max_ctx"]}


def oracle_step(orc, k: int) -> dict:
    """Oracle outputs of draft step k alone (as a one-step round)."""
    sl = slice(k - 1, k)
    return {n: (None if orc.get(n) is None else orc[n][:, sl])
            for n in ("draft_ids", "topk_ids", "topk_logits", "logits", "hidden_out")} | {
        "k_cache": orc["k_cache"], "v_cache": orc["v_cache"]}


def sample_seqs(B: int, n: int) -> list:
    """Evenly spread sample of sequence indices, always including the first and last."""
    if B <= n:
        return list(range(B))
    return sorted(set(np.linspace(0, B - 1, n).round().astype(int).tolist()))
