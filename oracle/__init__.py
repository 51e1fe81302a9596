"""CPU oracle of one PRISM draft round (fp64 C, see ``oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use it.  The CUDA path never imports it and
shares no code with it.

Pins: every function here is checked against something other than itself in
``tests/test_oracle_pins.py`` (library routines, closed forms, invariants,
brute force on tiny inputs and an independent library-based reference block).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

STEP_TENSORS = ("w_fuse", "g_attn", "w_qkv", "w_o", "g_mlp", "w_gate_up", "w_down", "g_final")


class _Config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "hidden", "n_q_heads", "n_kv_heads", "head_dim", "ffn", "vocab", "n_steps",
        "bf16", "round_acts", "final_norm", "topk", "max_ctx")] + [
        ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double)]


class _Module(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in STEP_TENSORS]


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        compile_source(_SRC, _LIB)
    return _LIB


def compile_source(src: str, out: str) -> str:
    """Compile an oracle source file into a shared library at ``out``."""
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                           src, "-o", tmp, "-lm"])
    os.replace(tmp, out)
    return out


def _bind(path: str):
    lib = ctypes.CDLL(path)
    vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    lib.orc_round_bf16.argtypes = [dbl]
    lib.orc_round_bf16.restype = dbl
    lib.orc_matvec.argtypes = [vp, ctypes.c_int, i64, i64, vp, vp]
    lib.orc_rmsnorm.argtypes = [vp, vp, i64, dbl, vp]
    lib.orc_rope.argtypes = [vp, i32, i64, dbl]
    lib.orc_attend.argtypes = [vp, vp, vp, ctypes.c_int, i64, i64, i32, vp]
    lib.orc_draft_round.argtypes = [ctypes.POINTER(_Config), vp, vp, ctypes.POINTER(_Module),
                                    i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.orc_draft_round.restype = ctypes.c_int
    u64 = ctypes.c_uint64
    lib.orc_draft_round_sampled.argtypes = [ctypes.POINTER(_Config), vp, vp, ctypes.POINTER(_Module),
                                            i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                            dbl, u64, vp, vp, vp]
    lib.orc_draft_round_sampled.restype = ctypes.c_int
    lib.orc_splitmix_at.argtypes = [u64, u64]
    lib.orc_splitmix_at.restype = u64
    lib.orc_uniform.argtypes = [u64, i32, i64, i64, i64]
    lib.orc_uniform.restype = dbl
    lib.orc_sample_gumbel.argtypes = [vp, i64, dbl, u64, i64, i64, vp, vp, vp]
    lib.orc_sample_gumbel.restype = None
    lib.orc_accept_sampled.argtypes = [i32, i32, i64, vp, vp, vp, vp, dbl, vp, u64, vp, vp, vp, vp]
    lib.orc_accept_sampled.restype = None
    lib.orc_accept_greedy.argtypes = [i32, i32, vp, vp, vp, vp, vp, vp]
    lib.orc_draft_tree.argtypes = [ctypes.POINTER(_Config), vp, vp, ctypes.POINTER(_Module), i32, i32,
                                   vp, vp, vp, vp, vp, vp, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                   vp, vp, vp, vp, vp]
    lib.orc_draft_tree.restype = ctypes.c_int
    lib.orc_accept_tree.argtypes = [i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.orc_accept_tree.restype = None
    lib.orc_num_threads.restype = ctypes.c_int
    lib.orc_round_bf16_bits.argtypes = [vp, i64, vp]
    lib.orc_round_bf16_bits.restype = None
    for f in (lib.orc_matvec, lib.orc_rmsnorm, lib.orc_rope, lib.orc_attend, lib.orc_accept_greedy):
        f.restype = None
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(build())
    return _lib


class variant:
    """Use another compiled copy of the oracle (e.g. one with a planted
    mistake, built by a pin-strength test) inside a ``with`` block."""

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib
        _load()
        with _lock:
            self._saved, _lib = _lib, _bind(self.path)
        return self

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self._saved
        return False


def _ptr(a):
    return None if a is None else a.ctypes.data


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ------------------------------------------------------------------ single ops

def round_bf16(x: float) -> float:
    return float(_load().orc_round_bf16(float(x)))


def num_threads() -> int:
    """Threads used by the oracle's parallel loops (OpenMP)."""
    return int(_load().orc_num_threads())


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to bf16 bit patterns (uint16) with the oracle's rule."""
    x = _c(x, np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().orc_round_bf16_bits(x.ctypes.data, x.size, out.ctypes.data)
    return out


def matvec(W: np.ndarray, x: np.ndarray) -> np.ndarray:
    """y = W x in fp64; W float32 [rows, cols] or bf16 bit patterns (uint16)."""
    bf = W.dtype == np.uint16
    W = _c(W, np.uint16 if bf else np.float32)
    x = _c(x, np.float64)
    y = np.empty(W.shape[0], dtype=np.float64)
    _load().orc_matvec(W.ctypes.data, int(bf), W.shape[0], W.shape[1], x.ctypes.data, y.ctypes.data)
    return y


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    x = _c(x, np.float64)
    g = _c(g, np.float64)
    out = np.empty_like(x)
    _load().orc_rmsnorm(x.ctypes.data, g.ctypes.data, x.size, eps, out.ctypes.data)
    return out


def rope(v: np.ndarray, pos: int, theta: float) -> np.ndarray:
    v = _c(v, np.float64).copy()
    _load().orc_rope(v.ctypes.data, v.size, pos, theta)
    return v


def attend(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Softmax attention of one query over rows of k, v ([n, D], float32)."""
    q = _c(q, np.float64)
    k = _c(k, np.float32)
    v = _c(v, np.float32)
    o = np.empty(q.size, dtype=np.float64)
    _load().orc_attend(q.ctypes.data, k.ctypes.data, v.ctypes.data, 0, k.shape[1], k.shape[0],
                       q.size, o.ctypes.data)
    return o


# ------------------------------------------------------------------ round

def config_of(shape, *, topk: int, max_ctx: int, round_acts: bool | None = None,
              final_norm: bool = True) -> _Config:
    bf = shape.dtype == "bf16"
    return _Config(shape.hidden, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                   shape.vocab, shape.n_steps, int(bf), int(bf if round_acts is None else round_acts),
                   int(final_norm), topk, max_ctx, float(shape.rope_theta), float(shape.rms_eps))


def draft_round(shape, weights: dict, inputs: dict, *, topk: int = 1, round_acts: bool | None = None,
                final_norm: bool = True, want_logits: bool = False, want_hidden: bool = True,
                seqs=None, temperature: float = 0.0, seed: int = 0) -> dict:
    """Run one draft round on the host.

    ``weights``: {"embed", "lm_head", "modules": {m: {...}}, "f_map"} as made
    by the synthetic generator (bf16 arrays are uint16 bit patterns).
    ``inputs``: {"tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache", "max_ctx"}.
    ``seqs``: optional list of sequence indices to compute (sequences are
    independent); outputs then cover only those sequences, in that order.
    The caches in ``inputs`` are not modified; updated copies are returned.
    ``temperature`` > 0: each draft token is drawn from softmax(z / T) with
    the random streams of ``seed`` (sequence numbers are the indices in the
    full batch); the result then also holds ``draft_lse`` and ``draft_margin``."""
    lib = _load()
    bf = shape.dtype == "bf16"
    wdt = np.uint16 if bf else np.float32
    K = shape.n_steps
    sel = list(range(inputs["tokens"].shape[0])) if seqs is None else list(seqs)
    B = len(sel)
    tokens = _c(inputs["tokens"][sel], np.int32)
    max_new = tokens.shape[1]
    hidden = _c(inputs["hidden"][sel], wdt)
    n_new = _c(inputs["n_new"][sel], np.int32)
    kv_len = _c(inputs["kv_len"][sel], np.int32)
    k_cache = _c(inputs["k_cache"][sel], wdt).copy()
    v_cache = _c(inputs["v_cache"][sel], wdt).copy()
    cfg = config_of(shape, topk=topk, max_ctx=int(inputs["max_ctx"]), round_acts=round_acts,
                    final_norm=final_norm)
    keep = []
    mods = (_Module * K)()
    for k in range(K):
        mod = weights["modules"][weights["f_map"][k]]
        arrs = [_c(mod[n], wdt) for n in STEP_TENSORS]
        keep.extend(arrs)
        mods[k] = _Module(*[a.ctypes.data for a in arrs])
    embed = _c(weights["embed"], wdt)
    lm = _c(weights["lm_head"], wdt)
    draft = np.empty((B, K), dtype=np.int32)
    tids = np.empty((B, K, topk), dtype=np.int32)
    tvals = np.empty((B, K, topk), dtype=np.float64)
    logits = np.empty((B, K, shape.vocab), dtype=np.float64) if want_logits else None
    hout = np.empty((B, K, shape.hidden), dtype=np.float64) if want_hidden else None
    seq_index = _c(np.asarray(sel), np.int32)
    lse = np.empty((B, K), dtype=np.float64)
    margin = np.empty((B, K), dtype=np.float64)
    rc = lib.orc_draft_round_sampled(ctypes.byref(cfg), embed.ctypes.data, lm.ctypes.data, mods, B, max_new,
                                     tokens.ctypes.data, hidden.ctypes.data, n_new.ctypes.data,
                                     kv_len.ctypes.data, k_cache.ctypes.data, v_cache.ctypes.data,
                                     draft.ctypes.data, tids.ctypes.data, tvals.ctypes.data,
                                     _ptr(logits), _ptr(hout), float(temperature), int(seed),
                                     seq_index.ctypes.data, lse.ctypes.data, margin.ctypes.data)
    if rc != 0:
        raise ValueError(f"oracle draft round rejected its input (code {rc})")
    out = {"draft_ids": draft, "topk_ids": tids, "topk_logits": tvals, "logits": logits,
           "hidden_out": hout, "k_cache": k_cache, "v_cache": v_cache}
    if temperature > 0:
        out["draft_lse"] = lse
        out["draft_margin"] = margin
    return out


def accept_greedy(draft: np.ndarray, target: np.ndarray, n_new: np.ndarray, kv_len: np.ndarray) -> dict:
    draft = _c(draft, np.int32)
    target = _c(target, np.int32)
    B, K = draft.shape
    kv = _c(kv_len, np.int32).copy()
    acc = np.empty(B, dtype=np.int32)
    out = np.empty((B, K + 1), dtype=np.int32)
    _load().orc_accept_greedy(B, K, draft.ctypes.data, target.ctypes.data, _c(n_new, np.int32).ctypes.data,
                              kv.ctypes.data, acc.ctypes.data, out.ctypes.data)
    return {"accept_len": acc, "out_tokens": out, "kv_len": kv}


# ------------------------------------------------------------------ sampling (temperature > 0)

def splitmix_at(seed: int, n: int) -> int:
    """The n-th output of SplitMix64 started from state ``seed``."""
    return int(_load().orc_splitmix_at(int(seed) & (2 ** 64 - 1), int(n)))


def uniform(seed: int, stream: int, b: int, k: int, i: int) -> float:
    """The random number of (stream, sequence b, position k, index i), in (0, 1)."""
    return float(_load().orc_uniform(int(seed) & (2 ** 64 - 1), stream, b, k, i))


def sample_gumbel(z: np.ndarray, tau: float, seed: int, b: int, k: int):
    """One draw from softmax(z / tau): (token, log-sum-exp of z / tau, Gumbel margin)."""
    z = _c(z, np.float64)
    tok = ctypes.c_int32(0)
    lse = ctypes.c_double(0.0)
    margin = ctypes.c_double(0.0)
    _load().orc_sample_gumbel(z.ctypes.data, z.size, float(tau), int(seed) & (2 ** 64 - 1), b, k,
                              ctypes.byref(tok), ctypes.byref(lse), ctypes.byref(margin))
    return int(tok.value), float(lse.value), float(margin.value)


def accept_sampled(draft: np.ndarray, logits: np.ndarray, lse: np.ndarray, tau: float, target_probs: np.ndarray,
                   seed: int, n_new: np.ndarray, kv_len: np.ndarray, seq_index=None) -> dict:
    """Speculative-sampling acceptance: draft [B, K], logits [B, K, V], lse [B, K],
    target_probs [B, K + 1, V]."""
    draft = _c(draft, np.int32)
    B, K = draft.shape
    z = _c(logits, np.float64)
    lse = _c(lse, np.float64)
    pt = _c(target_probs, np.float64)
    V = z.shape[-1]
    assert z.shape == (B, K, V) and pt.shape == (B, K + 1, V) and lse.shape == (B, K)
    idx = _c(np.arange(B) if seq_index is None else seq_index, np.int32)
    kv = _c(kv_len, np.int32).copy()
    acc = np.empty(B, dtype=np.int32)
    out = np.empty((B, K + 1), dtype=np.int32)
    _load().orc_accept_sampled(B, K, V, idx.ctypes.data, draft.ctypes.data, z.ctypes.data, lse.ctypes.data,
                               float(tau), pt.ctypes.data, int(seed) & (2 ** 64 - 1),
                               _c(n_new, np.int32).ctypes.data, kv.ctypes.data, acc.ctypes.data,
                               out.ctypes.data)
    return {"accept_len": acc, "out_tokens": out, "kv_len": kv}


# ------------------------------------------------------------------ tree drafting

def pool_size(n_steps: int, width: int) -> int:
    """Candidates of one tree round: w at depth 1, then w * w per later step."""
    return width + (n_steps - 1) * width * width


def draft_tree(shape, weights: dict, inputs: dict, *, width: int, n_nodes: int, follow: dict | None = None,
               round_acts: bool | None = None, final_norm: bool = True, want_logits: bool = True,
               want_hidden: bool = False, seqs=None) -> dict:
    """One tree-drafting round on the host (``orc_draft_tree``).

    ``follow``: {"pool_tokens" [B, P], "frontier" [B, K, w]} over the same
    sequences as ``seqs`` (or the full batch): recompute that tree instead of
    choosing candidates and frontiers.  Returns the pool (tokens, parents,
    scores), the frontier chosen after each step, per-row logits / lse
    ([B, K, w, ...]; step 1 fills row 0 only), the verified tree and the
    updated caches."""
    lib = _load()
    bf = shape.dtype == "bf16"
    wdt = np.uint16 if bf else np.float32
    K, V, d = shape.n_steps, shape.vocab, shape.hidden
    sel = list(range(inputs["tokens"].shape[0])) if seqs is None else list(seqs)
    B = len(sel)
    P = pool_size(K, width)
    tokens = _c(inputs["tokens"][sel], np.int32)
    max_new = tokens.shape[1]
    hidden = _c(inputs["hidden"][sel], wdt)
    n_new = _c(inputs["n_new"][sel], np.int32)
    kv_len = _c(inputs["kv_len"][sel], np.int32)
    k_cache = _c(inputs["k_cache"][sel], wdt).copy()
    v_cache = _c(inputs["v_cache"][sel], wdt).copy()
    cfg = config_of(shape, topk=width, max_ctx=int(inputs["max_ctx"]), round_acts=round_acts,
                    final_norm=final_norm)
    keep = []
    mods = (_Module * K)()
    for k in range(K):
        mod = weights["modules"][weights["f_map"][k]]
        arrs = [_c(mod[n], wdt) for n in STEP_TENSORS]
        keep.extend(arrs)
        mods[k] = _Module(*[a.ctypes.data for a in arrs])
    embed = _c(weights["embed"], wdt)
    lm = _c(weights["lm_head"], wdt)
    ft = ff = None
    if follow is not None:
        ft = _c(follow["pool_tokens"], np.int32)
        ff = _c(follow["frontier"], np.int32)
        assert ft.shape == (B, P) and ff.shape == (B, K, width)
    out = {
        "pool_tokens": np.empty((B, P), np.int32), "pool_parent": np.empty((B, P), np.int32),
        "pool_score": np.empty((B, P), np.float64), "frontier": np.empty((B, K, width), np.int32),
        "row_logits": np.empty((B, K, width, V), np.float64) if want_logits else None,
        "row_lse": np.empty((B, K, width), np.float64),
        "row_hidden": np.empty((B, K, width, d), np.float64) if want_hidden else None,
        "tree_tokens": np.empty((B, n_nodes), np.int32), "tree_parent": np.empty((B, n_nodes), np.int32),
        "tree_depth": np.empty((B, n_nodes), np.int32), "tree_score": np.empty((B, n_nodes), np.float64),
        "tree_pool": np.empty((B, n_nodes), np.int32),
    }
    rc = lib.orc_draft_tree(ctypes.byref(cfg), embed.ctypes.data, lm.ctypes.data, mods, B, max_new,
                            tokens.ctypes.data, hidden.ctypes.data, n_new.ctypes.data, kv_len.ctypes.data,
                            k_cache.ctypes.data, v_cache.ctypes.data, int(width), int(n_nodes), _ptr(ft), _ptr(ff),
                            out["pool_tokens"].ctypes.data, out["pool_parent"].ctypes.data,
                            out["pool_score"].ctypes.data, out["frontier"].ctypes.data, _ptr(out["row_logits"]),
                            out["row_lse"].ctypes.data, _ptr(out["row_hidden"]), out["tree_tokens"].ctypes.data,
                            out["tree_parent"].ctypes.data, out["tree_depth"].ctypes.data,
                            out["tree_score"].ctypes.data, out["tree_pool"].ctypes.data)
    if rc != 0:
        raise ValueError(f"oracle tree round rejected its input (code {rc})")
    out["k_cache"], out["v_cache"] = k_cache, v_cache
    return out


def accept_tree(tree_tokens: np.ndarray, tree_parent: np.ndarray, target_next: np.ndarray, n_new: np.ndarray,
                kv_len: np.ndarray, n_steps: int) -> dict:
    """Greedy acceptance of a draft tree (``orc_accept_tree``)."""
    tt = _c(tree_tokens, np.int32)
    tp = _c(tree_parent, np.int32)
    tn = _c(target_next, np.int32)
    B, m = tt.shape
    assert tn.shape == (B, m + 1)
    kv = _c(kv_len, np.int32).copy()
    acc = np.empty(B, np.int32)
    nodes = np.empty((B, n_steps), np.int32)
    out = np.empty((B, n_steps + 1), np.int32)
    _load().orc_accept_tree(B, m, n_steps, tt.ctypes.data, tp.ctypes.data, tn.ctypes.data,
                            _c(n_new, np.int32).ctypes.data, kv.ctypes.data, acc.ctypes.data,
                            nodes.ctypes.data, out.ctypes.data)
    return {"accept_len": acc, "accept_nodes": nodes, "out_tokens": out, "kv_len": kv}
