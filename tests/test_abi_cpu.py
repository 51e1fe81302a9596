"""The C ABI library builds, loads without a GPU and exports every entry
point that include/prism.h declares; host-side argument checks that need no
device answer correctly."""
from __future__ import annotations

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "prism.h")


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(prism_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2602_01762_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_round_entry_points():
    syms = declared_symbols()
    for s in ("prism_load_step_weights", "prism_draft_round", "prism_accept_greedy", "prism_create",
              "prism_destroy", "prism_load_shared_weights", "prism_sync_status", "prism_get_error"):
        assert s in syms


def test_library_exports_every_declared_symbol(lib):
    missing = [s for s in declared_symbols() if not hasattr(lib, s)]
    assert not missing, f"not exported: {missing}"


def test_version_and_error_strings(lib):
    lib.prism_version.restype = ctypes.c_char_p
    assert b"sm_103a" in lib.prism_version()
    lib.prism_get_error.restype = ctypes.c_char_p
    lib.prism_get_error.argtypes = [ctypes.c_void_p]
    assert isinstance(lib.prism_get_error(None), bytes)


def test_create_rejects_bad_configuration_before_touching_cuda(lib):
    from paper_2602_01762_gb300 import _Config
    bad = _Config(256, 4, 3, 64, 688, 4096, 3, 1, 1, 64, 1, 1, 10000.0, 1e-5, 1)  # 4 % 3 != 0
    out = ctypes.c_void_p()
    lib.prism_create.argtypes = [ctypes.POINTER(_Config), ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]
    assert lib.prism_create(ctypes.byref(bad), 0, ctypes.byref(out)) == 1
    assert not out.value
    bad = _Config(256, 4, 4, 96, 688, 4096, 3, 1, 1, 64, 1, 1, 10000.0, 1e-5, 1)  # head_dim 96
    assert lib.prism_create(ctypes.byref(bad), 0, ctypes.byref(out)) == 1
    bad = _Config(256, 4, 4, 64, 688, 4096, 3, 1, 1, 64, 1, 9, 10000.0, 1e-5, 1)  # topk 9
    assert lib.prism_create(ctypes.byref(bad), 0, ctypes.byref(out)) == 1
    assert lib.prism_create(None, 0, ctypes.byref(out)) == 1


def test_null_context_calls_return_invalid_arg(lib):
    for name, n in (("prism_draft_round", 14), ("prism_accept_greedy", 9)):
        f = getattr(lib, name)
        f.argtypes = [ctypes.c_void_p, ctypes.c_int32] + [ctypes.c_void_p] * (n - 2)
        assert f(None, 1, *([None] * (n - 2))) == 1
    vp, f32 = ctypes.c_void_p, ctypes.c_float
    f = lib.prism_draft_round_sampled
    f.argtypes = [vp, ctypes.c_int32] + [vp] * 6 + [f32] + [vp] * 8
    assert f(None, 1, *([None] * 6), 0.8, *([None] * 8)) == 1
    f = lib.prism_accept_sampled
    f.argtypes = [vp, ctypes.c_int32, vp, vp, vp, f32] + [vp] * 7
    assert f(None, 1, None, None, None, 0.8, *([None] * 7)) == 1
    assert lib.prism_destroy(None) == 0


def test_tree_entry_points_reject_null_context(lib):
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    f = lib.prism_draft_tree
    f.argtypes = [vp, i32] + [vp] * 6 + [i32, i32, vp, vp]
    assert f(None, 1, *([None] * 6), 4, 16, None, None) == 1
    f = lib.prism_accept_tree
    f.argtypes = [vp, i32, i32] + [vp] * 9
    assert f(None, 1, 16, *([None] * 9)) == 1


def test_create_rejects_tree_width_above_eight(lib):
    from paper_2602_01762_gb300 import _Config
    bad = _Config(256, 4, 4, 64, 688, 4096, 3, 1, 1, 64, 1, 1, 10000.0, 1e-5, 1, 9)
    out = ctypes.c_void_p()
    lib.prism_create.argtypes = [ctypes.POINTER(_Config), ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]
    assert lib.prism_create(ctypes.byref(bad), 0, ctypes.byref(out)) == 1


def test_loop_entry_point_rejects_null_context(lib):
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    f = lib.prism_draft_loop
    f.argtypes = [vp, i32, i32] + [vp] * 11
    assert f(None, 1, 2, *([None] * 11)) == 1


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No fallback: without the built library every entry of the binding raises."""
    import paper_2602_01762_gb300 as pkg
    monkeypatch.setattr(pkg, "LIB_PATH", str(tmp_path / "libprism.so"))
    monkeypatch.setattr(pkg, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        pkg.library()
    with pytest.raises(RuntimeError, match="missing"):
        pkg.Drafter(hidden=64, n_q_heads=4, n_kv_heads=2, head_dim=16, ffn=96, vocab=300, n_steps=3)


def test_product_path_does_not_reach_the_oracle():
    """The package and its CUDA sources name neither the oracle nor the test
    helpers; only the tests, the smoke check and the benchmark's CPU legs may."""
    pkg = os.path.join(ROOT, "paper_2602_01762_gb300")
    offenders = []
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if not f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                continue
            text = open(os.path.join(dirpath, f)).read()
            if re.search(r"^\s*(import|from)\s+(oracle|tests|synth)\b", text, flags=re.M) or "orc_" in text:
                offenders.append(f)
    assert not offenders, offenders


def test_oracle_is_independent_of_the_product():
    """The oracle includes only system headers and imports nothing of the
    package: the two sides share no code."""
    odir = os.path.join(ROOT, "oracle")
    for f in os.listdir(odir):
        path = os.path.join(odir, f)
        if f.endswith((".c", ".h")):
            incs = re.findall(r'^\s*#\s*include\s*([<"][^>"]+[>"])', open(path).read(), flags=re.M)
            assert all(i.startswith("<") for i in incs), (f, incs)
        elif f.endswith(".py"):
            text = open(path).read()
            assert not re.search(r"^\s*(import|from)\s+paper_2602_01762_gb300\b", text, flags=re.M), f
            assert "libprism" not in text and "csrc" not in text, f


def test_host_marshalling_round_trips_bit_patterns():
    """bf16 tensors travel as their uint16 bit patterns (NaN and -0 included);
    other dtypes unchanged."""
    import numpy as np
    from paper_2602_01762_gb300.host import to_device, to_numpy
    bits = np.array([0x0000, 0x8000, 0x3F80, 0xBF80, 0x7F80, 0xFF80, 0x7FC1, 0x0001, 0xFFFF], np.uint16)
    t = to_device(bits.reshape(3, 3), device="cpu")
    assert str(t.dtype) == "torch.bfloat16" and tuple(t.shape) == (3, 3)
    assert np.array_equal(to_numpy(t), bits.reshape(3, 3))
    assert float(t[0, 2]) == 1.0 and float(t[1, 0]) == -1.0 and float(t[1, 1]) == float("inf")
    for a in (np.arange(12, dtype=np.int32).reshape(3, 4), np.linspace(-2, 2, 7, dtype=np.float32)):
        assert np.array_equal(to_numpy(to_device(a, device="cpu")), a)
