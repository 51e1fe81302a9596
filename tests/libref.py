"""Independent reference of a PRISM draft round built from PyTorch library
routines (fp64 on the CPU), used only to pin the oracle.

It is written differently from the oracle on purpose: the step-1 prefill is
one batched pass with a causal mask handed to
``torch.nn.functional.scaled_dot_product_attention`` (not a row-by-row
loop), grouped-query attention repeats KV heads with ``repeat_interleave``,
RMSNorm is ``torch.nn.functional.rms_norm`` and the rotary embedding is a
complex multiplication z * exp(i * pos * theta_j) on the pairs
(x_j, x_{j+D/2}) rather than the real 2x2 rotation.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as Fn

from synth import bf16_to_f32

f64 = torch.float64


def _t(a) -> torch.Tensor:
    a = np.asarray(a)
    if a.dtype == np.uint16:
        a = bf16_to_f32(a)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))


def _bf16(t: torch.Tensor) -> torch.Tensor:
    """Round to the nearest bf16 value, ties to even, directly from fp64:
    x = m * 2^e with 0.5 <= |m| < 1, and bf16 keeps 8 significant bits, so the
    result is rint(m * 2^8) / 2^8 * 2^e (numpy's rint rounds half to even).
    (torch's own conversion goes through float32 and can round twice.)"""
    x = t.detach().numpy()
    m, e = np.frexp(x)
    return torch.from_numpy(np.ldexp(np.rint(m * 256.0) / 256.0, e))


def _rope(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """x [rows, heads, D]; pos [rows]."""
    D = x.shape[-1]
    half = D // 2
    inv = theta ** (-2.0 * torch.arange(half, dtype=f64) / D)
    ang = pos.to(f64)[:, None, None] * inv[None, None, :]
    rot = torch.polar(torch.ones_like(ang), ang)
    z = torch.complex(x[..., :half], x[..., half:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def reference_round(shape, weights, inputs, *, topk=1, round_acts=False, final_norm=True, forced=None):
    """``forced`` [B, K-1]: tokens fed to steps 2..K in place of the previous
    step's argmax (a chain that follows a given path)."""
    d, Hq, Hkv, D, F = shape.hidden, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    K, eps = shape.n_steps, shape.rms_eps
    grp = Hq // Hkv
    bf_store = shape.dtype == "bf16"
    R = _bf16 if round_acts else (lambda t: t)
    store = _bf16 if bf_store else (lambda t: t.to(torch.float32).to(f64))
    E, LM = _t(weights["embed"]), _t(weights["lm_head"])
    mods = {m: {k: _t(v) for k, v in mod.items()} for m, mod in weights["modules"].items()}
    B = inputs["tokens"].shape[0]
    out_ids = np.zeros((B, K), np.int32)
    out_top = np.zeros((B, K, topk), np.int32)
    out_logits = np.zeros((B, K, shape.vocab))
    out_hidden = np.zeros((B, K, d))
    kc_all = _t(inputs["k_cache"]).clone()
    vc_all = _t(inputs["v_cache"]).clone()
    for b in range(B):
        L, n = int(inputs["kv_len"][b]), int(inputs["n_new"][b])
        kc, vc = kc_all[b], vc_all[b]          # [Hkv, max_ctx, D]
        H = _t(inputs["hidden"][b])
        prev, hhat = None, None
        for k in range(1, K + 1):
            m = mods[weights["f_map"][k - 1]]
            if k == 1:
                toks = torch.from_numpy(np.asarray(inputs["tokens"][b, :n], dtype=np.int64))
                U = torch.cat([E[toks], H[:n]], dim=1)
                pos = L + torch.arange(n)
            else:
                U = torch.cat([E[prev], hhat])[None, :]
                pos = torch.tensor([L + n + k - 2])
            U = R(U)
            X0 = U @ m["w_fuse"].T
            N1 = R(Fn.rms_norm(X0, (d,), weight=m["g_attn"], eps=eps))
            QKV = N1 @ m["w_qkv"].T
            rows = QKV.shape[0]
            q = _rope(QKV[:, :Hq * D].reshape(rows, Hq, D), pos, shape.rope_theta)
            kk = _rope(QKV[:, Hq * D:(Hq + Hkv) * D].reshape(rows, Hkv, D), pos, shape.rope_theta)
            vv = QKV[:, (Hq + Hkv) * D:].reshape(rows, Hkv, D)
            kc[:, pos, :] = store(kk.transpose(0, 1))
            vc[:, pos, :] = store(vv.transpose(0, 1))
            T = int(pos[-1]) + 1
            keys = kc[:, :T].repeat_interleave(grp, dim=0)
            vals = vc[:, :T].repeat_interleave(grp, dim=0)
            mask = torch.arange(T)[None, :] <= pos[:, None]
            O = Fn.scaled_dot_product_attention(q.transpose(0, 1), keys, vals, attn_mask=mask)
            O = R(O.transpose(0, 1).reshape(rows, Hq * D))
            A = X0 + O @ m["w_o"].T
            N2 = R(Fn.rms_norm(A, (d,), weight=m["g_mlp"], eps=eps))
            GU = N2 @ m["w_gate_up"].T
            M = R(Fn.silu(GU[:, :F]) * GU[:, F:])
            Y = A + M @ m["w_down"].T
            hhat = Y[-1]
            nf = Fn.rms_norm(hhat, (d,), weight=m["g_final"], eps=eps) if final_norm else hhat
            z = LM @ R(nf)
            zs = z.numpy()
            order = np.lexsort((np.arange(zs.size), -zs))
            prev = int(order[0])
            out_ids[b, k - 1] = prev
            if forced is not None and k < K:
                prev = int(forced[b, k - 1])
            out_top[b, k - 1] = order[:topk]
            out_logits[b, k - 1] = zs
            out_hidden[b, k - 1] = hhat.numpy()
    return {"draft_ids": out_ids, "topk_ids": out_top, "logits": out_logits,
            "hidden_out": out_hidden, "k_cache": kc_all.numpy(), "v_cache": vc_all.numpy()}
