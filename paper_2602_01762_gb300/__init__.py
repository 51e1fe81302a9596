"""PRISM draft round on GB300 (sm_103a): Python binding of ``libprism.so``.

The binding only marshals arguments: it checks torch tensors' dtype, shape,
device and contiguity, and passes their device pointers and the current CUDA
stream to the C ABI declared in ``include/prism.h``.  Every step of the draft
round runs in the library's CUDA kernels; there is no CPU fallback, and a
missing library raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

__all__ = ["Drafter", "PrismError", "library", "lm_head_topk_static", "STEP_TENSORS", "KERNEL_KINDS"]

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.environ.get("PRISM_LIB") or os.path.join(_HERE, "libprism.so")
STEP_TENSORS = ("w_fuse", "g_attn", "w_qkv", "w_o", "g_mlp", "w_gate_up", "w_down", "g_final")
KERNEL_KINDS = ("fusion", "qkv", "rope_append", "attention", "o_proj", "gate_up", "down", "lm_head", "sample",
                "tree_gather", "tree_lse_select")
_STATUS = ["OK", "INVALID_ARG", "SHAPE", "CAPACITY", "NOT_LOADED", "CUDA", "OOM", "DEVICE_FLAG", "TIMEOUT"]


class PrismError(RuntimeError):
    def __init__(self, status: int, msg: str):
        name = _STATUS[status] if 0 <= status < len(_STATUS) else str(status)
        super().__init__(f"PRISM_{name}: {msg}")
        self.status = status


class _Config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "hidden", "n_q_heads", "n_kv_heads", "head_dim", "ffn", "vocab", "n_steps", "dtype",
        "max_batch", "max_ctx", "max_new", "topk")] + [
        ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float), ("final_norm", ctypes.c_int32),
        ("max_tree_width", ctypes.c_int32)]


class _TreeOutputs(ctypes.Structure):
    _fields_ = [("tokens", ctypes.c_void_p), ("parents", ctypes.c_void_p), ("depths", ctypes.c_void_p),
                ("scores", ctypes.c_void_p), ("pool_tokens", ctypes.c_void_p), ("pool_parents", ctypes.c_void_p),
                ("pool_scores", ctypes.c_void_p), ("frontier", ctypes.c_void_p), ("row_logits", ctypes.c_void_p)]


class _StepWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in STEP_TENSORS]


_lib = None


def library() -> ctypes.CDLL:
    """Load libprism.so (built in-tree by ``build.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2602_01762_gb300.build` (nvcc, sm_103a)")
        lib = ctypes.CDLL(LIB_PATH)
        vp, i32 = ctypes.c_void_p, ctypes.c_int32
        P = ctypes.POINTER
        lib.prism_create.argtypes = [P(_Config), i32, P(vp)]
        lib.prism_destroy.argtypes = [vp]
        lib.prism_load_shared_weights.argtypes = [vp, vp, vp]
        lib.prism_load_step_weights.argtypes = [vp, i32, P(_StepWeights)]
        lib.prism_draft_round.argtypes = [vp, i32] + [vp] * 12
        lib.prism_accept_greedy.argtypes = [vp, i32] + [vp] * 7
        lib.prism_sync_status.argtypes = [vp, vp, P(i32)]
        lib.prism_set_option.argtypes = [vp, ctypes.c_char_p, i32]
        lib.prism_profile_round.argtypes = [vp, i32] + [vp] * 10 + [P(ctypes.c_float), P(i32), i32, P(i32)]
        lib.prism_lm_head_topk_static.argtypes = [i32] * 5 + [ctypes.c_float] + [vp] * 9
        lib.prism_get_error.argtypes = [vp]
        lib.prism_round_launches.argtypes = [vp, P(i32)]
        flt = ctypes.c_float
        lib.prism_draft_round_sampled.argtypes = [vp, i32] + [vp] * 6 + [flt] + [vp] * 8
        lib.prism_accept_sampled.argtypes = [vp, i32, vp, vp, vp, flt] + [vp] * 7
        lib.prism_draft_tree.argtypes = [vp, i32] + [vp] * 6 + [i32, i32, P(_TreeOutputs), vp]
        lib.prism_accept_tree.argtypes = [vp, i32, i32] + [vp] * 9
        lib.prism_draft_loop.argtypes = [vp, i32, i32] + [vp] * 11
        lib.prism_profile_tree.argtypes = [vp, i32] + [vp] * 6 + [i32, i32, P(_TreeOutputs), vp,
                                                                P(ctypes.c_float), P(i32), i32, P(i32)]
        lib.prism_get_error.restype = ctypes.c_char_p
        lib.prism_version.restype = ctypes.c_char_p
        for f in ("prism_create", "prism_destroy", "prism_load_shared_weights", "prism_load_step_weights",
                  "prism_draft_round", "prism_accept_greedy", "prism_sync_status", "prism_set_option",
                  "prism_profile_round", "prism_lm_head_topk_static", "prism_round_launches",
                  "prism_draft_round_sampled", "prism_accept_sampled", "prism_draft_tree", "prism_accept_tree",
                  "prism_profile_tree", "prism_draft_loop"):
            getattr(lib, f).restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, device=None):
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


class Drafter:
    """One PRISM drafter on one GPU: K draft steps, each bound to a module
    (fusion + transformer layer), a shared embedding and LM head."""

    def __init__(self, *, hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab, n_steps,
                 dtype="bf16", max_batch=1, max_ctx=4096, max_new=1, topk=1,
                 rope_theta=10000.0, rms_eps=1e-5, final_norm=True, max_tree_width=0, device=0):
        self.lib = library()
        self.dtype = dtype
        self.tdtype = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.device = torch.device("cuda", device)
        self.cfg = _Config(hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab, n_steps,
                           1 if dtype == "bf16" else 0, max_batch, max_ctx, max_new, topk,
                           rope_theta, rms_eps, int(final_norm), int(max_tree_width))
        self.hidden, self.n_steps, self.vocab, self.topk = hidden, n_steps, vocab, topk
        self.max_batch, self.max_ctx, self.max_new = max_batch, max_ctx, max_new
        self.n_kv_heads, self.head_dim = n_kv_heads, head_dim
        self.max_tree_width = max_tree_width
        self._shapes = {
            "w_fuse": (hidden, 2 * hidden), "g_attn": (hidden,),
            "w_qkv": ((n_q_heads + 2 * n_kv_heads) * head_dim, hidden),
            "w_o": (hidden, n_q_heads * head_dim), "g_mlp": (hidden,),
            "w_gate_up": (2 * ffn, hidden), "w_down": (hidden, ffn), "g_final": (hidden,),
        }
        self._keep = {}
        h = ctypes.c_void_p()
        self._check(self.lib.prism_create(ctypes.byref(self.cfg), device, ctypes.byref(h)), None)
        self.h = h

    @classmethod
    def from_shape(cls, shape, *, max_batch, max_ctx, max_new, topk=1, final_norm=True, max_tree_width=0,
                   device=0):
        return cls(hidden=shape.hidden, n_q_heads=shape.n_q_heads, n_kv_heads=shape.n_kv_heads,
                   head_dim=shape.head_dim, ffn=shape.ffn, vocab=shape.vocab, n_steps=shape.n_steps,
                   dtype=shape.dtype, max_batch=max_batch, max_ctx=max_ctx, max_new=max_new,
                   topk=topk, rope_theta=shape.rope_theta, rms_eps=shape.rms_eps,
                   final_norm=final_norm, max_tree_width=max_tree_width, device=device)

    # ------------------------------------------------------------ helpers
    def _check(self, status, h="self"):
        if status != 0:
            handle = self.h if h == "self" else None
            msg = self.lib.prism_get_error(handle).decode()
            raise PrismError(status, msg)

    def _tensor(self, t, shape, dtype, name):
        if not isinstance(t, torch.Tensor):
            raise TypeError(f"{name}: expected a torch.Tensor")
        if t.device != self.device:
            raise ValueError(f"{name}: expected device {self.device}, got {t.device}")
        if t.dtype != dtype:
            raise ValueError(f"{name}: expected {dtype}, got {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{name}: must be contiguous")
        if shape is not None and tuple(t.shape) != tuple(shape):
            raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")
        return t

    # ------------------------------------------------------------ weights
    def load_shared_weights(self, embed, lm_head):
        shp = (self.vocab, self.hidden)
        self._tensor(embed, shp, self.tdtype, "embed")
        self._tensor(lm_head, shp, self.tdtype, "lm_head")
        self._keep["shared"] = (embed, lm_head)
        self._check(self.lib.prism_load_shared_weights(self.h, _ptr(embed), _ptr(lm_head)))

    def load_step_weights(self, step: int, weights: dict):
        for n in STEP_TENSORS:
            self._tensor(weights[n], self._shapes[n], self.tdtype, n)
        sw = _StepWeights(*[weights[n].data_ptr() for n in STEP_TENSORS])
        self._keep[("step", step)] = dict(weights)
        self._check(self.lib.prism_load_step_weights(self.h, step, ctypes.byref(sw)))

    def set_option(self, name: str, value: int):
        self._check(self.lib.prism_set_option(self.h, name.encode(), int(value)))

    # ------------------------------------------------------------ round
    def _round_args(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                    topk_ids, topk_logits):
        B = tokens.shape[0]
        i32 = torch.int32
        self._tensor(tokens, (B, self.max_new), i32, "tokens")
        self._tensor(hidden, (B, self.max_new, self.hidden), self.tdtype, "hidden")
        self._tensor(n_new, (B,), i32, "n_new")
        self._tensor(kv_len, (B,), i32, "kv_len")
        cshape = (k_cache.shape[0], self.n_kv_heads, self.max_ctx, self.head_dim)
        if k_cache.shape[0] < B:
            raise ValueError("k_cache holds fewer sequences than the batch")
        self._tensor(k_cache, cshape, self.tdtype, "k_cache")
        self._tensor(v_cache, cshape, self.tdtype, "v_cache")
        if draft_ids is not None:
            self._tensor(draft_ids, (B, self.n_steps), i32, "draft_ids")
        if topk_ids is not None:
            self._tensor(topk_ids, (B, self.n_steps, self.topk), i32, "topk_ids")
        if topk_logits is not None:
            self._tensor(topk_logits, (B, self.n_steps, self.topk), torch.float32, "topk_logits")
        return B

    def draft_round(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                    topk_ids=None, topk_logits=None, logits=None, hidden_out=None, stream=None):
        B = self._round_args(tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                             topk_ids, topk_logits)
        if logits is not None:
            self._tensor(logits, (B, self.n_steps, self.vocab), torch.float32, "logits")
        if hidden_out is not None:
            self._tensor(hidden_out, (B, self.n_steps, self.hidden), torch.float32, "hidden_out")
        self._check(self.lib.prism_draft_round(
            self.h, B, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache),
            _ptr(v_cache), _ptr(draft_ids), _ptr(topk_ids), _ptr(topk_logits), _ptr(logits),
            _ptr(hidden_out), _stream(stream)))

    def draft_round_sampled(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, temperature: float, seed,
                            draft_ids, logits, draft_lse, topk_ids=None, topk_logits=None, hidden_out=None,
                            stream=None):
        """Draft round with every x^_k drawn from softmax(z / temperature).
        ``seed``: uint64 device tensor of one element (int64 storage), read when
        the round runs; ``logits`` [B, K, V] and ``draft_lse`` [B, K] are required."""
        B = self._round_args(tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                             topk_ids, topk_logits)
        self._tensor(logits, (B, self.n_steps, self.vocab), torch.float32, "logits")
        self._tensor(draft_lse, (B, self.n_steps), torch.float32, "draft_lse")
        self._tensor(seed, (1,), torch.int64, "seed")
        if hidden_out is not None:
            self._tensor(hidden_out, (B, self.n_steps, self.hidden), torch.float32, "hidden_out")
        self._check(self.lib.prism_draft_round_sampled(
            self.h, B, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache),
            _ptr(v_cache), float(temperature), _ptr(seed), _ptr(draft_ids), _ptr(topk_ids), _ptr(topk_logits),
            _ptr(logits), _ptr(draft_lse), _ptr(hidden_out), _stream(stream)))

    def accept_sampled(self, draft, logits, draft_lse, temperature: float, target_probs, seed, n_new, kv_len,
                       accept_len, out_tokens, stream=None):
        """Speculative-sampling acceptance against target_probs [B, K + 1, V]."""
        B = draft.shape[0]
        K, V = self.n_steps, self.vocab
        i32 = torch.int32
        self._tensor(draft, (B, K), i32, "draft")
        self._tensor(logits, (B, K, V), torch.float32, "logits")
        self._tensor(draft_lse, (B, K), torch.float32, "draft_lse")
        self._tensor(target_probs, (B, K + 1, V), torch.float32, "target_probs")
        self._tensor(seed, (1,), torch.int64, "seed")
        self._tensor(n_new, (B,), i32, "n_new")
        self._tensor(kv_len, (B,), i32, "kv_len")
        self._tensor(accept_len, (B,), i32, "accept_len")
        self._tensor(out_tokens, (B, K + 1), i32, "out_tokens")
        self._check(self.lib.prism_accept_sampled(
            self.h, B, _ptr(draft), _ptr(logits), _ptr(draft_lse), float(temperature), _ptr(target_probs),
            _ptr(seed), _ptr(n_new), _ptr(kv_len), _ptr(accept_len), _ptr(out_tokens), _stream(stream)))

    def draft_loop(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, target, draft_ids, accept_len, out_tokens,
                   stream=None):
        """``prism_draft_loop``: R greedy rounds on the device, each followed by
        acceptance that writes the next round's tokens and n_new.  hidden
        [R, B, max_new, d]; target [R, B, K + 1]; draft_ids [R, B, K];
        accept_len [R, B]; out_tokens [R, B, K + 1]; tokens, n_new and kv_len
        are updated in place."""
        R, B = hidden.shape[0], tokens.shape[0]
        K = self.n_steps
        i32 = torch.int32
        self._round_args(tokens, hidden[0], n_new, kv_len, k_cache, v_cache, None, None, None)
        self._tensor(hidden, (R, B, self.max_new, self.hidden), self.tdtype, "hidden")
        for t, shp, name in ((target, (R, B, K + 1), "target"), (draft_ids, (R, B, K), "draft_ids"),
                             (accept_len, (R, B), "accept_len"), (out_tokens, (R, B, K + 1), "out_tokens")):
            self._tensor(t, shp, i32, name)
        self._check(self.lib.prism_draft_loop(
            self.h, B, R, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache), _ptr(v_cache),
            _ptr(target), _ptr(draft_ids), _ptr(accept_len), _ptr(out_tokens), _stream(stream)))

    def tree_pool_size(self, width: int) -> int:
        """Candidates of one tree round of this width: w + (K - 1) w^2."""
        return width + (self.n_steps - 1) * width * width

    def draft_tree(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, width: int, tree_tokens, tree_parents,
                   tree_depths, tree_scores, pool_tokens=None, pool_parents=None, pool_scores=None, frontier=None,
                   row_logits=None, stream=None):
        """Tree-drafting round (``prism_draft_tree``): the verified tree goes to
        tree_tokens / tree_parents / tree_depths (int32 [B, n]) and tree_scores
        (fp32 [B, n]), n = tree_tokens.shape[1]; the candidate pool
        ([B, P]), the frontiers ([B, K, w]) and every row's logits
        ([K, B, w, V]) are optional outputs."""
        B = self._round_args(tokens, hidden, n_new, kv_len, k_cache, v_cache, None, None, None)
        n = tree_tokens.shape[1]
        P = self.tree_pool_size(width)
        i32, f32 = torch.int32, torch.float32
        for t, shp, dt, name in ((tree_tokens, (B, n), i32, "tree_tokens"), (tree_parents, (B, n), i32, "tree_parents"),
                                 (tree_depths, (B, n), i32, "tree_depths"), (tree_scores, (B, n), f32, "tree_scores"),
                                 (pool_tokens, (B, P), i32, "pool_tokens"), (pool_parents, (B, P), i32, "pool_parents"),
                                 (pool_scores, (B, P), f32, "pool_scores"),
                                 (frontier, (B, self.n_steps, width), i32, "frontier"),
                                 (row_logits, (self.n_steps, B, width, self.vocab), f32, "row_logits")):
            if t is not None:
                self._tensor(t, shp, dt, name)
        out = _TreeOutputs(*[None if t is None else t.data_ptr() for t in (
            tree_tokens, tree_parents, tree_depths, tree_scores, pool_tokens, pool_parents, pool_scores, frontier,
            row_logits)])
        self._check(self.lib.prism_draft_tree(
            self.h, B, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache), _ptr(v_cache),
            int(width), int(n), ctypes.byref(out), _stream(stream)))

    def profile_tree(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, width: int, tree_tokens, tree_parents,
                     tree_depths, tree_scores, stream=None):
        """Eager tree round with a CUDA event around every kernel; returns a
        list of (kind, milliseconds) in launch order."""
        B = self._round_args(tokens, hidden, n_new, kv_len, k_cache, v_cache, None, None, None)
        n = tree_tokens.shape[1]
        for t, dt, name in ((tree_tokens, torch.int32, "tree_tokens"), (tree_parents, torch.int32, "tree_parents"),
                            (tree_depths, torch.int32, "tree_depths"), (tree_scores, torch.float32, "tree_scores")):
            self._tensor(t, (B, n), dt, name)
        out = _TreeOutputs(tree_tokens.data_ptr(), tree_parents.data_ptr(), tree_depths.data_ptr(),
                           tree_scores.data_ptr(), None, None, None, None, None)
        cap = 12 * self.n_steps + 8
        ms = (ctypes.c_float * cap)()
        kinds = (ctypes.c_int32 * cap)()
        cnt = ctypes.c_int32(0)
        self._check(self.lib.prism_profile_tree(
            self.h, B, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache), _ptr(v_cache),
            int(width), int(n), ctypes.byref(out), _stream(stream), ms, kinds, cap, ctypes.byref(cnt)))
        return [(KERNEL_KINDS[kinds[i]], float(ms[i])) for i in range(cnt.value)]

    def accept_tree(self, tree_tokens, tree_parents, target_next, n_new, kv_len, accept_len, accept_nodes,
                    out_tokens, stream=None):
        """Greedy tree acceptance (``prism_accept_tree``); target_next int32 [B, n + 1]."""
        B, n = tree_tokens.shape
        K = self.n_steps
        i32 = torch.int32
        for t, shp, name in ((tree_tokens, (B, n), "tree_tokens"), (tree_parents, (B, n), "tree_parents"),
                             (target_next, (B, n + 1), "target_next"), (n_new, (B,), "n_new"),
                             (kv_len, (B,), "kv_len"), (accept_len, (B,), "accept_len"),
                             (accept_nodes, (B, K), "accept_nodes"), (out_tokens, (B, K + 1), "out_tokens")):
            self._tensor(t, shp, i32, name)
        self._check(self.lib.prism_accept_tree(
            self.h, B, n, _ptr(tree_tokens), _ptr(tree_parents), _ptr(target_next), _ptr(n_new), _ptr(kv_len),
            _ptr(accept_len), _ptr(accept_nodes), _ptr(out_tokens), _stream(stream)))

    def round_launches(self) -> int:
        """Kernel launches of the last round replayed from a CUDA graph."""
        n = ctypes.c_int32(0)
        self._check(self.lib.prism_round_launches(self.h, ctypes.byref(n)))
        return int(n.value)

    def profile_round(self, tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                      topk_ids=None, topk_logits=None, stream=None):
        """Eager round with a CUDA event around every kernel; returns a list of
        (kind, milliseconds) in launch order."""
        B = self._round_args(tokens, hidden, n_new, kv_len, k_cache, v_cache, draft_ids,
                             topk_ids, topk_logits)
        cap = 12 * self.n_steps + 8
        ms = (ctypes.c_float * cap)()
        kinds = (ctypes.c_int32 * cap)()
        n = ctypes.c_int32(0)
        self._check(self.lib.prism_profile_round(
            self.h, B, _ptr(tokens), _ptr(hidden), _ptr(n_new), _ptr(kv_len), _ptr(k_cache),
            _ptr(v_cache), _ptr(draft_ids), _ptr(topk_ids), _ptr(topk_logits), _stream(stream),
            ms, kinds, cap, ctypes.byref(n)))
        return [(KERNEL_KINDS[kinds[i]], float(ms[i])) for i in range(n.value)]

    def accept_greedy(self, draft, target, n_new, kv_len, accept_len, out_tokens, stream=None):
        B, K = draft.shape
        i32 = torch.int32
        self._tensor(draft, (B, self.n_steps), i32, "draft")
        self._tensor(target, (B, self.n_steps + 1), i32, "target")
        self._tensor(n_new, (B,), i32, "n_new")
        self._tensor(kv_len, (B,), i32, "kv_len")
        self._tensor(accept_len, (B,), i32, "accept_len")
        self._tensor(out_tokens, (B, self.n_steps + 1), i32, "out_tokens")
        self._check(self.lib.prism_accept_greedy(
            self.h, B, _ptr(draft), _ptr(target), _ptr(n_new), _ptr(kv_len), _ptr(accept_len),
            _ptr(out_tokens), _stream(stream)))

    def sync_status(self, stream=None) -> int:
        """Synchronise and return the device error word (0 when clean); raises
        on CUDA errors.  A set word is returned, not raised (the C status,
        PRISM_ERR_DEVICE_FLAG or PRISM_ERR_TIMEOUT, is kept in
        ``last_status``)."""
        flags = ctypes.c_int32(0)
        st = self.lib.prism_sync_status(self.h, _stream(stream), ctypes.byref(flags))
        self.last_status = st
        if st not in (0, 7, 8):
            self._check(st)
        return int(flags.value)

    def close(self):
        if getattr(self, "h", None):
            self.lib.prism_destroy(self.h)
            self.h = None
            self._keep.clear()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def lm_head_topk_static(h, g_final, lm_head, draft, topk_ids=None, topk_logits=None, logits=None,
                        dev_flags=None, rms_eps=1e-5, stream=None):
    """Final norm + LM head + top-k of the rows of ``h`` through
    ``prism_lm_head_topk_static``, the entry point that allocates no device
    memory (its scratch is a static array inside the library; for callers
    that cannot call cudaMalloc).  ``h`` fp32 [B, d]; ``g_final`` [d] or None;
    ``lm_head`` [V, d] (bf16 or fp32); ``draft`` int32 [B]; ``topk_ids`` int32
    [B, k], ``topk_logits`` fp32 [B, k], ``logits`` fp32 [B, V] and
    ``dev_flags`` int32 [1] optional outputs.  B <= 64; calls that may overlap
    on the GPU race on the shared scratch."""
    lib = library()
    V, d = lm_head.shape
    B = h.shape[0]
    dt = {torch.bfloat16: 1, torch.float32: 0}.get(lm_head.dtype)
    if dt is None:
        raise TypeError("lm_head must be bfloat16 or float32")
    topk = 1 if topk_ids is None and topk_logits is None else (topk_ids if topk_ids is not None else topk_logits).shape[1]
    want = [(h, (B, d), torch.float32, "h"), (lm_head, (V, d), lm_head.dtype, "lm_head"),
            (draft, (B,), torch.int32, "draft")]
    if g_final is not None:
        want.append((g_final, (d,), lm_head.dtype, "g_final"))
    for t, shape, dtype, name in ((topk_ids, (B, topk), torch.int32, "topk_ids"),
                                  (topk_logits, (B, topk), torch.float32, "topk_logits"),
                                  (logits, (B, V), torch.float32, "logits"),
                                  (dev_flags, (1,), torch.int32, "dev_flags")):
        if t is not None:
            want.append((t, shape, dtype, name))
    for t, shape, dtype, name in want:
        if tuple(t.shape) != shape or t.dtype != dtype or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name}: expected contiguous CUDA {dtype} {shape}, got {t.dtype} {tuple(t.shape)}")
        if t.device != h.device:
            raise ValueError(f"{name} is on {t.device}, h on {h.device}: every tensor must be on one device")
    # the library launches on the current device: make it the tensors' device
    with torch.cuda.device(h.device):
        st = lib.prism_lm_head_topk_static(dt, d, V, B, topk, float(rms_eps), _ptr(h), _ptr(g_final),
                                           _ptr(lm_head), _ptr(draft), _ptr(topk_ids), _ptr(topk_logits),
                                           _ptr(logits), _ptr(dev_flags), _stream(stream, h.device))
    if st != 0:
        raise PrismError(st, (lib.prism_get_error(None) or b"").decode())
