"""Synthetic workloads: the model shapes and the input recipe of each.

Shapes follow the Llama targets the paper drafts for (Llama-2-7B and
Llama-3-8B, Sec. 4 "Target LLMs"), plus a tiny drafter and a Llama-3-70B
shape.  No trained weights or datasets are used: every tensor is drawn from
the counter-based generator of this package.

Recipe (per workload seed, one stream tag per tensor):
  * matrices, token embedding E and LM head: normal, sigma 0.02;
  * RMSNorm gains: ones (``gain_sigma`` > 0 gives 1 + normal(gain_sigma));
  * target hidden states: normal, sigma 1;
  * accepted token ids: uniform in [0, vocab);
  * committed draft-KV rows [0, L_b): normal, sigma 1, stored as the cache
    dtype and taken as already rotary-encoded;
  * per-sequence committed length L_b: uniform in [ctx_lo, ctx_hi];
  * acceptance targets: per position, with probability 1/2 the draft token,
    otherwise uniform in [0, vocab); the bonus position is uniform.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

from . import normal, uniform_int, uniform01


@dataclass(frozen=True)
class Shape:
    name: str
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    n_steps: int
    dtype: str              # "f32" or "bf16": weights, embeddings, hidden states, KV cache
    rope_theta: float
    rms_eps: float = 1e-5

    @property
    def qkv_rows(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    def module_params(self) -> int:
        d, F = self.hidden, self.ffn
        return (d * 2 * d + self.qkv_rows * d + d * self.n_q_heads * self.head_dim
                + 2 * F * d + d * F + 3 * d)


@dataclass(frozen=True)
class Workload:
    name: str
    shape: Shape
    batch: int
    ctx_lo: int             # committed draft-KV length per sequence: uniform in [ctx_lo, ctx_hi]
    ctx_hi: int
    n_new: int              # accepted tokens fed to the step-1 prefill of each sequence
    topk: int
    seed: int
    weight_sigma: float = 0.02
    gain_sigma: float = 0.0
    f_map: tuple = field(default=())   # module index of each step; () = one module per step
    tree_width: int = 0     # > 0: tree drafting with this many branches per node
    tree_nodes: int = 0     # verified tree size of a tree round

    def modules(self) -> tuple:
        return self.f_map if self.f_map else tuple(range(self.shape.n_steps))

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


TINY_F32 = Shape("tiny-f32", 256, 4, 4, 64, 688, 4096, 3, "f32", 10000.0)
TINY_BF16 = replace(TINY_F32, name="tiny-bf16", dtype="bf16")
L3_8B = Shape("llama3-8b", 4096, 32, 8, 128, 14336, 128256, 5, "bf16", 500000.0)
L2_7B = Shape("llama2-7b", 4096, 32, 32, 128, 11008, 32000, 7, "bf16", 10000.0)
L3_70B = Shape("llama3-70b", 8192, 64, 8, 128, 28672, 128256, 5, "bf16", 500000.0)

WORKLOADS = {
    # tiny drafter: the 64 target hidden states are the step-1 prefill of an empty draft cache
    "tiny-f32": Workload("tiny-f32", TINY_F32, 1, 0, 0, 64, 1, 0),
    "tiny-bf16": Workload("tiny-bf16", TINY_BF16, 1, 0, 0, 64, 1, 0),
    "tiny-f32-decode": Workload("tiny-f32-decode", TINY_F32, 1, 63, 63, 1, 1, 0),
    "l3-8b-b1": Workload("l3-8b-b1", L3_8B, 1, 2048, 2048, 1, 1, 1),
    "l3-8b-b16": Workload("l3-8b-b16", L3_8B, 16, 512, 4096, 1, 8, 2),
    "l3-8b-b64": Workload("l3-8b-b64", L3_8B, 64, 512, 4096, 1, 8, 2),
    "l2-7b-b8": Workload("l2-7b-b8", L2_7B, 8, 1024, 1024, 1, 1, 3),
    "l3-70b-b32": Workload("l3-70b-b32", L3_70B, 32, 4096, 4096, 1, 1, 4),
    # tree drafting: w branches per node, the n best candidates verified
    "tiny-bf16-tree": Workload("tiny-bf16-tree", replace(TINY_BF16, name="tiny-bf16-k4", n_steps=4), 3, 16, 40, 3,
                               1, 0, gain_sigma=0.1, tree_width=4, tree_nodes=16),
    # the tree the paper evaluates (Sec. 4): 6 steps, 4 branches, 16 verified tokens, batch 1
    "l3-8b-b1-tree": Workload("l3-8b-b1-tree", replace(L3_8B, name="llama3-8b-k6", n_steps=6), 1, 2048, 2048, 1,
                              1, 1, tree_width=4, tree_nodes=16),
    # the module layout of the paper's experiments (Sec. 4): two modules, the first for the prefill
    # step and the second for every decoding step
    "l3-8b-b1-m2": Workload("l3-8b-b1-m2", L3_8B, 1, 2048, 2048, 1, 1, 1, f_map=(0, 1, 1, 1, 1)),
    "l3-8b-b1-tree-m2": Workload("l3-8b-b1-tree-m2", replace(L3_8B, name="llama3-8b-k6", n_steps=6), 1, 2048, 2048,
                                 1, 1, 1, f_map=(0, 1, 1, 1, 1, 1), tree_width=4, tree_nodes=16),
}


def max_ctx_of(w: Workload) -> int:
    """Cache capacity: longest committed context + new rows + draft rows (K for
    the chain, (K - 1) * width for a tree), rounded up to 16."""
    need = w.ctx_hi + w.n_new + max(w.shape.n_steps, (w.shape.n_steps - 1) * w.tree_width)
    return (need + 15) // 16 * 16


def _module_tensor_shapes(s: Shape) -> dict:
    d, F = s.hidden, s.ffn
    return {
        "w_fuse": (d, 2 * d),
        "g_attn": (d,),
        "w_qkv": (s.qkv_rows, d),
        "w_o": (d, s.n_q_heads * s.head_dim),
        "g_mlp": (d,),
        "w_gate_up": (2 * F, d),      # rows [0, F) gate, rows [F, 2F) up
        "w_down": (d, F),
        "g_final": (d,),
    }


STEP_TENSORS = ("w_fuse", "g_attn", "w_qkv", "w_o", "g_mlp", "w_gate_up", "w_down", "g_final")


def make_weights(w: Workload) -> dict:
    """Embedding, LM head and one parameter set per distinct module.

    Returns {"embed", "lm_head", "modules": {m: {name: array}}, "f_map": tuple}.
    bf16 tensors are uint16 bit patterns; f32 tensors are float32."""
    s, seed, dt = w.shape, w.seed, w.shape.dtype
    out = {
        "embed": normal(seed, "embed", (s.vocab, s.hidden), w.weight_sigma, dt),
        "lm_head": normal(seed, "lm_head", (s.vocab, s.hidden), w.weight_sigma, dt),
        "modules": {},
        "f_map": w.modules(),
    }
    for m in sorted(set(w.modules())):
        mod = {}
        for name, shp in _module_tensor_shapes(s).items():
            if name.startswith("g_"):
                if w.gain_sigma > 0:
                    mod[name] = normal(seed, f"m{m}.{name}", shp, w.gain_sigma, dt, mean=1.0)
                else:
                    mod[name] = _ones(shp, dt)
            else:
                mod[name] = normal(seed, f"m{m}.{name}", shp, w.weight_sigma, dt)
        out["modules"][m] = mod
    return out


def _ones(shape, dt):
    if dt == "bf16":
        return np.full(shape, 0x3F80, dtype=np.uint16)
    return np.ones(shape, dtype=np.float32)


def make_round_inputs(w: Workload, max_new: int | None = None) -> dict:
    """Inputs of one draft round: accepted tokens, their target hidden states,
    per-sequence counts, committed KV lengths and the pre-filled KV cache."""
    s, seed, dt = w.shape, w.seed, w.shape.dtype
    B, n = w.batch, w.n_new
    max_new = max_new or n
    mc = max_ctx_of(w)
    tokens = np.zeros((B, max_new), dtype=np.int32)
    tokens[:, :n] = uniform_int(seed, "tokens", (B, max_new), 0, s.vocab - 1)[:, :n]
    hid = normal(seed, "hidden", (B, max_new, s.hidden), 1.0, dt)
    hid[:, n:] = 0
    kv_len = uniform_int(seed, "ctx_len", (B,), w.ctx_lo, w.ctx_hi)
    kshape = (B, s.n_kv_heads, mc, s.head_dim)
    k_cache = normal(seed, "k_prior", kshape, 1.0, dt)
    v_cache = normal(seed, "v_prior", kshape, 1.0, dt)
    for b in range(B):
        k_cache[b, :, kv_len[b]:, :] = 0
        v_cache[b, :, kv_len[b]:, :] = 0
    return {
        "tokens": tokens,
        "hidden": hid,
        "n_new": np.full((B,), n, dtype=np.int32),
        "kv_len": kv_len.astype(np.int32),
        "k_cache": k_cache,
        "v_cache": v_cache,
        "max_ctx": mc,
    }


def make_targets(w: Workload, draft_ids: np.ndarray) -> np.ndarray:
    """Target tokens [B, K+1] for greedy acceptance: each position copies the
    draft token with probability 1/2, else a uniform id; the bonus slot is uniform."""
    B, K, V = w.batch, w.shape.n_steps, w.shape.vocab
    u = uniform01(w.seed, "target_u", (B, K))
    rnd = uniform_int(w.seed, "target_tok", (B, K + 1), 0, V - 1)
    tgt = rnd.copy()
    tgt[:, :K] = np.where(u < 0.5, draft_ids, rnd[:, :K])
    return tgt.astype(np.int32)


def make_tree_targets(w: Workload, tree_tokens: np.ndarray, tree_parent: np.ndarray) -> np.ndarray:
    """Target tokens [B, n + 1] for greedy tree acceptance: entry 0 is the
    target's token after the root, entry 1 + i its token after tree node i.
    Each entry is, with probability 1/2, the token of a uniformly chosen child
    of that node (when it has one), else a uniform id."""
    B, n = tree_tokens.shape
    V = w.shape.vocab
    u = uniform01(w.seed, "tree_target_u", (B, n + 1))
    pick = uniform01(w.seed, "tree_target_pick", (B, n + 1))
    rnd = uniform_int(w.seed, "tree_target_tok", (B, n + 1), 0, V - 1)
    out = rnd.copy()
    for b in range(B):
        for node in range(-1, n):
            kids = [i for i in range(n) if tree_parent[b, i] == node]
            if kids and u[b, node + 1] < 0.5:
                out[b, node + 1] = tree_tokens[b, kids[int(pick[b, node + 1] * len(kids))]]
    return out.astype(np.int32)
