"""The benchmark's host-side accounting, on the CPU.

The roofline fraction the benchmark reports divides algorithmic bytes by a
measured duration, so the byte counts are pinned here against figures
derived by hand from the Llama-3-8B architecture (one matrix at a time, not
through the shape's own parameter count).  The clock record and the check
that ties the committed traffic figure to the kernel source it was captured
on are host logic too; they run here on canned input."""
from __future__ import annotations

import hashlib
import json
import os

import pytest

import bench
from synth.workloads import WORKLOADS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# Llama-3-8B drafter module, matrix by matrix (bf16 elements)
D, HQ, HKV, HD, FF, V = 4096, 32, 8, 128, 14336, 128256
FUSE = D * 2 * D
QKV = (HQ + 2 * HKV) * HD * D
O = D * HQ * HD
GATE_UP = 2 * FF * D
DOWN = D * FF
GAINS = 3 * D
LM = V * D
KV_ROW = 2 * HKV * HD * 2          # K and V of one position, bf16


def test_module_and_head_sizes_of_the_llama3_8b_shape():
    s = WORKLOADS["l3-8b-b1"].shape
    assert s.module_params() == FUSE + QKV + O + GATE_UP + DOWN + GAINS
    assert abs((FUSE + QKV + O + GATE_UP + DOWN) / 1e6 - 251.66) < 0.01
    assert abs(LM / 1e6 - 525.34) < 0.01


def test_round_bytes_of_the_batch1_round():
    """K = 5 steps at batch 1, context 2048, one accepted token: every step
    streams its module and the LM head; step 1 attends over 2049 positions,
    step k >= 2 over 2048 + k."""
    w = WORKLOADS["l3-8b-b1"]
    K = 5
    weights = K * (FUSE + QKV + O + GATE_UP + DOWN + GAINS + LM) * 2
    emb = K * D * 2                   # one embedding row per step (the prefill's and the K - 1 drafted)
    hid = D * 2                       # the one target hidden state
    kv_read = sum(2049 if k == 1 else 2048 + k for k in range(1, K + 1)) * KV_ROW
    kv_write = K * KV_ROW             # the prefill row and K - 1 draft rows
    got = bench.round_bytes(w, [2048])
    assert got == weights + emb + hid + kv_read + kv_write
    assert abs(got / 1e9 - 7.81) < 0.005          # 7.770 GB of weights + 0.042 GB of KV


def test_round_bytes_grow_by_one_kv_row_per_step_per_position():
    w = WORKLOADS["l3-8b-b16"]
    K = w.shape.n_steps
    base = bench.round_bytes(w, [1000] * w.batch)
    longer = bench.round_bytes(w, [1000] * (w.batch - 1) + [1001])
    assert longer - base == K * KV_ROW


def test_tree_round_bytes_of_the_papers_tree():
    """6 steps, 4 branches, batch 1, context 2048: step 1 reads the 2049
    committed and prefill positions; step k >= 2 also reads the (k - 1) * 4
    draft slots written so far; 1 + 5 * 4 rows are written."""
    w = WORKLOADS["l3-8b-b1-tree"]
    K, tw = 6, 4
    weights = K * (FUSE + QKV + O + GATE_UP + DOWN + GAINS + LM) * 2
    emb = (1 + (K - 1) * tw) * D * 2
    hid = D * 2
    kv_read = (2049 + sum(2049 + (k - 1) * tw for k in range(2, K + 1))) * KV_ROW
    kv_write = (1 + (K - 1) * tw) * KV_ROW
    got = bench.tree_round_bytes(w, [2048])
    assert got == weights + emb + hid + kv_read + kv_write
    assert abs(got / 1e9 - 9.37) < 0.005


def test_lm_head_bytes_are_the_head_plus_its_activations():
    w = WORKLOADS["l3-8b-b1"]
    assert bench.lm_head_bytes(w) == LM * 2 + D * 4 + bench.kTOP * 8


def test_committed_traffic_figure_is_tied_to_its_kernel_source(tmp_path):
    src = os.path.join(ROOT, "paper_2602_01762_gb300", "csrc", "gemv_tc.cu")
    with open(os.path.join(ROOT, "profiles", "lm_head_traffic.json")) as f:
        rec = json.load(f)
    with open(src, "rb") as f:
        current = hashlib.sha256(f.read()).hexdigest() == rec["kernel_sha256"]
    got = bench.traffic_from_profile(src, rec["workload"])
    if current:
        assert got == rec["dram_bytes_per_launch_full_size"]
        # DRAM traffic of the capture is the algorithmic bytes, plus the next
        # step's first 16 MiB of fusion weights that the kernel requests into
        # L2 (option prefetch_next_kb), plus well under 1 %
        w = WORKLOADS[rec["workload"]]
        assert 1.0 <= got / (bench.lm_head_bytes(w) + 16 * 1024 * 1024) < 1.01
    else:
        assert got is None
    other = tmp_path / "edited.cu"
    other.write_bytes(b"// another kernel\n")
    assert bench.traffic_from_profile(str(other), rec["workload"]) is None
    assert bench.traffic_from_profile(src, "tiny-bf16") is None


class _FakeSmi:
    def __init__(self, out):
        self.out = out

    def terminate(self):
        pass

    def communicate(self, timeout=None):
        return self.out, ""


def _row(sm, util, hw="Not Active", thermal="Not Active", sw_thermal="Not Active", cap="Not Active"):
    return f"0, {sm}, 2070, 900.5, {util}, 0x0, {hw}, {thermal}, {sw_thermal}, {cap}"


def test_clock_record_takes_the_median_under_load_and_names_reasons():
    rows = [_row(2070, 0), _row(1980, 100, cap="Active"), _row(2070, 100), _row(2055, 95), "garbled line"]
    cs = bench.ClockSampler(0)
    cs.proc = _FakeSmi("\n".join(rows) + "\n")
    got = cs.stop()
    assert got["sm_mhz"] == 2055 and got["sm_max_mhz"] == 2070
    assert got["reasons"] == ["sw_power_cap"] and got["samples"] == 3


def test_clock_record_flags_thermal_slowdown():
    cs = bench.ClockSampler(0)
    cs.proc = _FakeSmi(_row(1500, 100, hw="Active", thermal="Active") + "\n")
    got = cs.stop()
    assert got["reasons"] == ["hw_slowdown", "hw_thermal_slowdown"]


def test_clock_record_without_nvidia_smi():
    cs = bench.ClockSampler(0)
    assert cs.stop()["reasons"] == ["nvidia-smi unavailable"]
    cs.proc = _FakeSmi("")
    assert cs.stop()["reasons"] == ["no samples"]


@pytest.mark.parametrize("name", ["l3-8b-b1", "l3-8b-b1-tree"])
def test_config_names_the_workload_and_its_l2_policy(name):
    c = bench.config_of(WORKLOADS[name])
    assert c["workload"] == name and "larger than L2" in c["l2"]
    assert ("tree_width" in c) == name.endswith("tree")


def _fake_smi(tmp_path, monkeypatch, script: str):
    exe = tmp_path / "nvidia-smi"
    exe.write_text("#!/bin/sh\n" + script)
    exe.chmod(0o755)
    monkeypatch.setenv("PATH", f"{tmp_path}:{os.environ.get('PATH', '')}")


def test_clock_sampler_finds_the_device_by_uuid(tmp_path, monkeypatch):
    """CUDA device 0 may be nvidia-smi's GPU 5 when only some GPUs are visible:
    the sampler asks nvidia-smi for the index of the device's UUID."""
    _fake_smi(tmp_path, monkeypatch, 'case "$1" in --id=GPU-abc) echo 5 ;; *) exit 6 ;; esac\n')
    assert bench.smi_index(0, "abc") == "5"
    assert bench.smi_index(0, "GPU-abc") == "5"
    assert bench.smi_index(2, "GPU-other") == "2"          # unknown UUID: CUDA's index
    _fake_smi(tmp_path, monkeypatch, "echo 'No devices were found'\n")
    assert bench.smi_index(1, "abc") == "1"


def test_clock_sampler_without_nvidia_smi_keeps_the_index(tmp_path, monkeypatch):
    monkeypatch.setenv("PATH", str(tmp_path))
    assert bench.smi_index(3, "abc") == "3"
