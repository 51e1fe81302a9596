"""Benchmark of the PRISM draft round on GB300.

A step is one draft round (all K draft steps: fusion, QKV, RoPE + KV append,
attention, O projection, gate/up + SwiGLU, down projection, LM head + top-k)
over one batch of synthetic inputs.  Default workload: the Llama-3-8B-shaped
drafter at batch 1, KV context 2048, K = 5 (inputs are 7.8 GB of weights per
round, far larger than L2, so no flush is needed between rounds).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl reference]

Prints one JSON line (rank 0).  Under torchrun each rank runs an independent
replica on its own GPU (the round has no cross-sequence exchange), timing is
bracketed by a barrier and synchronisation, the max over ranks is taken and
`value` counts the tokens of all ranks.  `--impl reference` times the CPU
oracle (fp64 C, all host cores) on the same workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "draft tokens/s and K-step round latency (µs) at 1 GB300; % of HBM roofline"
UNIT = "draft tokens/s"
TREE_UNIT = "draft tree tokens/s (verified tree nodes)"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
LM_KIND = "lm_head"


# ----------------------------------------------------------------------------- helpers

def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def round_bytes(w, kv_len):
    """Algorithmic bytes one round must move: every step's module weights, the
    LM head, embedding rows gathered, target hidden states read, KV rows read
    over each query's causal window and KV rows written."""
    s = w.shape
    es = 2 if s.dtype == "bf16" else 4
    K, B, n = s.n_steps, w.batch, w.n_new
    weights = K * (s.module_params() + s.vocab * s.hidden) * es
    emb = K * B * s.hidden * es + (n - 1) * B * s.hidden * es
    hid = B * n * s.hidden * es
    kv_row = 2 * s.n_kv_heads * s.head_dim * es          # K and V of one position
    kv_read = 0
    for L in kv_len:
        for k in range(1, K + 1):
            p = L + n - 1 if k == 1 else L + n + k - 2
            kv_read += (p + 1) * kv_row
    kv_write = B * (n + K - 1) * kv_row
    return weights + emb + hid + kv_read + kv_write


def tree_round_bytes(w, kv_len):
    """Algorithmic bytes of one tree round: every step's module weights and
    the LM head, embedding rows gathered and target hidden states read, the
    KV rows each step's attention must read once per sequence (the committed
    rows plus the tree's draft slots so far) and the KV rows written."""
    s = w.shape
    es = 2 if s.dtype == "bf16" else 4
    K, B, n, tw = s.n_steps, w.batch, w.n_new, w.tree_width
    weights = K * (s.module_params() + s.vocab * s.hidden) * es
    emb = B * n * s.hidden * es + B * (K - 1) * tw * s.hidden * es
    hid = B * n * s.hidden * es
    kv_row = 2 * s.n_kv_heads * s.head_dim * es
    kv_read = 0
    for L in kv_len:
        kv_read += (L + n) * kv_row                      # step 1: the causal window of the last prefill row
        for k in range(2, K + 1):
            kv_read += (L + n + (k - 1) * tw) * kv_row   # committed rows + the draft slots up to this step
    kv_write = B * (n + (K - 1) * tw) * kv_row
    return weights + emb + hid + kv_read + kv_write


def lm_head_bytes(w):
    s = w.shape
    es = 2 if s.dtype == "bf16" else 4
    return s.vocab * s.hidden * es + w.batch * s.hidden * 4 + w.batch * kTOP * 8


kTOP = 8


def smi_index(local: int, uuid: str | None = None) -> str:
    """nvidia-smi's index of CUDA device `local`, matched by the device's UUID
    (CUDA's device numbering need not be nvidia-smi's when only some GPUs are
    visible); `local` itself when the UUID or nvidia-smi is unavailable."""
    try:
        if uuid is None:
            import torch
            uuid = str(torch.cuda.get_device_properties(local).uuid)
        if not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
        r = subprocess.run(["nvidia-smi", f"--id={uuid}", "--query-gpu=index", "--format=csv,noheader"],
                           capture_output=True, text=True, timeout=20)
        out = r.stdout.strip()
        if r.returncode == 0 and out.isdigit():
            return out
    except Exception:
        pass
    return str(local)


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, uuid: str | None = None):
        self.idx = gpu_index
        self.uuid = uuid
        self.proc = None

    def start(self):
        try:
            self.idx = smi_index(self.idx, self.uuid)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 10:
                continue
            try:
                rows.append({"sm": float(f[1]), "max": float(f[2]), "util": float(f[4]),
                             "hw": f[6], "hw_thermal": f[7], "sw_thermal": f[8], "power_cap": f[9]})
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        busy = [r for r in rows if r["util"] > 0] or rows
        reasons = set()
        for r in busy:
            for key, name in (("hw", "hw_slowdown"), ("hw_thermal", "hw_thermal_slowdown"),
                              ("sw_thermal", "sw_thermal_slowdown"), ("power_cap", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in busy), "sm_max_mhz": max(r["max"] for r in rows),
                "reasons": sorted(reasons), "samples": len(busy)}


def dist_setup():
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def dist_barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def dist_reduce(x: float, op: str, world: int, device=None) -> float:
    """max or sum of a host scalar over ranks (plain host-side bookkeeping)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def traffic_from_profile(kernel_src: str, workload: str):
    """dram bytes per LM-head launch from the committed ncu summary, or None
    when the kernel source changed since that capture or the summary is of
    another workload."""
    path = os.path.join(ROOT, "profiles", "lm_head_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        with open(kernel_src, "rb") as f:
            digest = hashlib.sha256(f.read()).hexdigest()
        if rec.get("kernel_sha256") != digest or rec.get("workload") != workload:
            return None
        return float(rec["dram_bytes_per_launch_full_size"])
    except Exception:
        return None


# ----------------------------------------------------------------------------- CPU oracle leg

def time_oracle(w, W, I, budget_s: float, max_rounds: int | None = None):
    """Time whole oracle rounds on sequence 0 until `budget_s` of CPU work (at
    least one round).  Returns (draft tokens/s, seconds per round, rounds)."""
    import oracle
    times = []
    t_end = time.perf_counter() + budget_s
    while True:
        t0 = time.perf_counter()
        oracle.draft_round(w.shape, W, I, topk=max(1, w.topk), want_hidden=False, seqs=[0])
        times.append(time.perf_counter() - t0)
        if time.perf_counter() >= t_end or (max_rounds and len(times) >= max_rounds):
            break
    per_round = statistics.median(times)
    return w.shape.n_steps / per_round, per_round, len(times)


# ----------------------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="l3-8b-b1")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=10.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--temperature", type=float, default=0.0,
                    help="> 0: sampled drafting (prism_draft_round_sampled) at this temperature")
    ap.add_argument("--loop", type=int, default=0, metavar="R",
                    help="> 0: time prism_draft_loop, R rounds with acceptance per step")
    ap.add_argument("--opt", action="append", default=[], metavar="NAME=VALUE",
                    help="drafter option (prism_set_option), repeatable")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    import synth
    w = synth.WORKLOADS[args.workload]
    if args.impl == "reference":
        # CPU oracle: rank 0 alone runs and prints; other ranks exit at once
        if int(os.environ.get("RANK", "0")) == 0:
            run_reference(args, w)
        return
    world, rank, local = dist_setup()
    if w.tree_width > 0:
        run_tree(args, w, world, rank, local)
    elif args.loop > 0:
        run_loop(args, w, world, rank, local)
    else:
        run_ours(args, w, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_reference(args, w):
    """The oracle as it stands, on this host's cores.  One step is a bounded
    sample of the workload: the first draft step (fusion, block, LM head and
    selection: one draft token) of sequence 0, so that the default step count
    finishes in about a minute."""
    from dataclasses import replace

    import oracle
    import synth
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    shape1 = replace(w.shape, n_steps=1)
    W1 = dict(W, f_map=tuple(W["f_map"])[:1])

    def sample():
        oracle.draft_round(shape1, W1, I, topk=max(1, w.topk, w.tree_width), want_hidden=False, seqs=[0])

    for _ in range(args.warmup):
        sample()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        sample()
        times.append(time.perf_counter() - t0)
    total = sum(times)
    value = args.steps / total                      # one draft token per sample
    cores = oracle.num_threads()
    desc = (f"per step, the first draft step of sequence 0 of workload {w.name} (one draft token: "
            f"fusion, transformer block, LM head, selection), fp64 oracle")
    unit = UNIT
    if w.tree_width > 0:
        # a tree round processes 1 + (K - 1) w such rows and yields n_nodes tree tokens
        rows = 1 + (w.shape.n_steps - 1) * w.tree_width
        value *= w.tree_nodes / rows
        unit = TREE_UNIT
        desc += (f"; scaled to tree tokens: {w.tree_nodes} tokens per round of {rows} processed rows, "
                 f"each row costing one such step")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": unit, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(w),
        "cpu_baseline": {"value": value, "unit": unit, "cores": cores, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def config_of(w):
    s = w.shape
    return {"workload": w.name, "shape": s.name, "hidden": s.hidden, "q_heads": s.n_q_heads,
            "kv_heads": s.n_kv_heads, "head_dim": s.head_dim, "ffn": s.ffn, "vocab": s.vocab,
            "draft_steps": s.n_steps, "batch": w.batch, "kv_context": [w.ctx_lo, w.ctx_hi],
            "accepted_tokens_in": w.n_new, "topk": w.topk, "modules": len(set(w.modules())),
            "seed": w.seed, "l2": "inputs larger than L2 (whole weight set streamed every round)",
            "parallelism": "replicas",
            **({"tree_width": w.tree_width, "tree_nodes": w.tree_nodes} if w.tree_width else {})}


def eager_round_us(dr, one_round, stream, steps, dev):
    """Round latency with the graph off: every kernel launched from the host,
    one event pair around the rounds (after 3 untimed rounds).  Reported next
    to the replayed round as evidence of what the graph saves; the option is
    restored afterwards (the graph is captured again on the next call)."""
    import torch
    n = max(3, min(20, steps))
    dr.set_option("use_graph", 0)
    try:
        for _ in range(3):
            one_round()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        e0.record(stream)
        for _ in range(n):
            one_round()
        e1.record(stream)
        torch.cuda.synchronize(dev)
    finally:
        dr.set_option("use_graph", 1)
    return e0.elapsed_time(e1) * 1e3 / n


def run_ours(args, w, world, rank, local):
    import numpy as np
    import torch

    import synth
    from paper_2602_01762_gb300 import Drafter
    from paper_2602_01762_gb300.host import bind_weights, to_device

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s = w.shape
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    B, K = w.batch, s.n_steps
    max_new = I["tokens"].shape[1]
    dr = Drafter.from_shape(s, max_batch=B, max_ctx=int(I["max_ctx"]), max_new=max_new, topk=w.topk,
                            device=local)
    weights_dev = bind_weights(dr, W, device=dev)
    options = {}
    for kv in args.opt:
        name, value = kv.split("=", 1)
        options[name] = int(value)
        dr.set_option(name, int(value))
    t = {n: to_device(I[n], dev) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
    ids = torch.empty((B, K), dtype=torch.int32, device=dev)
    tk_ids = torch.empty((B, K, w.topk), dtype=torch.int32, device=dev)
    tk_val = torch.empty((B, K, w.topk), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    sampled = args.temperature > 0
    if sampled:
        logits_buf = torch.empty((B, K, s.vocab), dtype=torch.float32, device=dev)
        lse_buf = torch.empty((B, K), dtype=torch.float32, device=dev)
        seed_buf = torch.tensor([12345], dtype=torch.int64, device=dev)

    def one_round():
        if sampled:
            dr.draft_round_sampled(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"],
                                   args.temperature, seed_buf, ids, logits_buf, lse_buf, tk_ids, tk_val,
                                   stream=stream)
        else:
            dr.draft_round(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"],
                           ids, tk_ids, tk_val, stream=stream)

    # ---- device-resident timing (graph replay) ---------------------------------
    for _ in range(args.warmup):
        one_round()
    assert dr.sync_status(stream) == 0
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.2)
    dist_barrier(world)
    torch.cuda.synchronize(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        one_round()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    dist_barrier(world)
    clk = clocks.stop()
    ms_local = ev0.elapsed_time(ev1)
    ms = dist_reduce(ms_local, "max", world, dev if world > 1 else None)
    flags = dr.sync_status(stream)
    launches_per_round = dr.round_launches()

    # per-replay latency distribution (after the timed region: an event pair around each replay)
    n_pct = min(200, args.steps)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_pct)]
    for e0, e1 in evs:
        e0.record(stream)
        one_round()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    lat = sorted(e0.elapsed_time(e1) * 1e3 for e0, e1 in evs)
    pct = {"p10": lat[len(lat) // 10], "p50": lat[len(lat) // 2], "p90": lat[(len(lat) * 9) // 10],
           "replays": n_pct}
    tokens_total = B * K * args.steps * world
    value = tokens_total / (ms / 1e3)
    per_round_ms = ms / args.steps

    # ---- the same round without the graph (eager launches, evidence only) -------
    eager_us = eager_round_us(dr, one_round, stream, args.steps, dev)

    # ---- per-kernel durations (eager launches, an event around each kernel) -----
    prof = []
    for _ in range(max(3, min(20, args.steps))):
        prof.append(dr.profile_round(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"],
                                     t["v_cache"], ids, tk_ids, tk_val, stream=stream))
    by_kind = {}
    for rnd in prof[1:]:
        for kind, kms in rnd:
            by_kind.setdefault(kind, []).append(kms)
    kind_total = {k: sum(v) / (len(prof) - 1) for k, v in by_kind.items()}
    lm = by_kind.get(LM_KIND, [float("nan")])
    lm_ms = statistics.mean(lm)
    peak, peak_src = hbm_peak()
    lm_b = lm_head_bytes(w)
    achieved = lm_b / (lm_ms / 1e3) / 1e9
    kernel_src = os.path.join(ROOT, "paper_2602_01762_gb300", "csrc", "gemv_tc.cu")

    # ---- end to end through the public API with host buffers --------------------
    pin = {n: torch.from_numpy(np.ascontiguousarray(
        I[n].view(np.int16) if I[n].dtype == np.uint16 else I[n])).pin_memory()
        for n in ("tokens", "hidden", "n_new", "kv_len")}
    if I["hidden"].dtype == np.uint16:
        pin["hidden"] = pin["hidden"].view(torch.bfloat16)
    ids_host = torch.empty((B, K), dtype=torch.int32).pin_memory()
    h2d = sum(p.numel() * p.element_size() for p in pin.values())
    d2h = ids_host.numel() * ids_host.element_size()

    def e2e_round():
        for n, p in pin.items():
            t[n].copy_(p, non_blocking=True)
        one_round()
        ids_host.copy_(ids, non_blocking=True)

    for _ in range(args.warmup):
        e2e_round()
    torch.cuda.synchronize(dev)
    dist_barrier(world)
    e0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_round()
    torch.cuda.synchronize(dev)
    e_s = dist_reduce(time.perf_counter() - e0, "max", world, dev if world > 1 else None)
    e2e_value = tokens_total / e_s

    # ---- CPU baseline: the oracle on a bounded sample (rank 0, N = 1 only) -------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        tps, sec, n_rounds = time_oracle(w, W, I, args.cpu_budget)
        cpu = {"value": tps, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
               "sample": (f"{n_rounds} full {K}-step rounds of sequence 0 of {w.name} "
                          f"(median {sec:.3f} s per round), fp64 oracle on all host cores")}

    total_bytes = round_bytes(w, [int(x) for x in I["kv_len"]])
    if rank == 0:
        shares = {k: v / sum(kind_total.values()) for k, v in kind_total.items()}
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": per_round_ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if s.dtype == "bf16" else "f32",
            "data": "synthetic", "config": dict(config_of(w), options=options,
                                                **({"temperature": args.temperature} if sampled else {})),
            "round_latency_us": per_round_ms * 1e3,
            "round_latency_percentiles_us": pct,
            "round_latency_eager_us": eager_us,
            "hbm": {"bytes_per_round": total_bytes,
                    "achieved_gbs": total_bytes / (per_round_ms / 1e3) / 1e9,
                    "frac_of_8tbs": total_bytes / (per_round_ms / 1e3) / 1e9 / NOMINAL_HBM_GBS,
                    "frac_of_measured": total_bytes / (per_round_ms / 1e3) / 1e9 / peak},
            "roofline": {"kernel": "LM head GEMV + top-k selection", "bound": "hbm", "achieved": achieved,
                         "peak": peak, "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic_from_profile(kernel_src, w.name), "bytes_per_launch": lm_b,
                         "avg_launch_ms": lm_ms},
            "kernel_time_share": shares,
            **({"kernel_time_share_note": "from the greedy round: the sampled draws are not in it"}
               if sampled else {}),
            "kernel_ms_per_round": kind_total,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": launches_per_round * args.steps,
            "clocks": clk,
            "device_error_word": flags,
        }
        print(json.dumps(out), flush=True)
    dr.close()
    del weights_dev


def run_tree(args, w, world, rank, local):
    """Tree-drafting rounds (prism_draft_tree): the same timing contract as
    the chain; `value` counts verified tree tokens (n_nodes per sequence)."""
    import numpy as np
    import torch

    import synth
    from paper_2602_01762_gb300 import Drafter
    from paper_2602_01762_gb300.host import bind_weights, to_device

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s = w.shape
    W, I = synth.make_weights(w), synth.make_round_inputs(w)
    B, K, tw, m = w.batch, s.n_steps, w.tree_width, w.tree_nodes
    dr = Drafter.from_shape(s, max_batch=B, max_ctx=int(I["max_ctx"]), max_new=I["tokens"].shape[1], topk=1,
                            max_tree_width=tw, device=local)
    weights_dev = bind_weights(dr, W, device=dev)
    options = {}
    for kv in args.opt:
        name, value = kv.split("=", 1)
        options[name] = int(value)
        dr.set_option(name, int(value))
    t = {n: to_device(I[n], dev) for n in ("tokens", "hidden", "n_new", "kv_len", "k_cache", "v_cache")}
    tt = torch.empty((B, m), dtype=torch.int32, device=dev)
    tp = torch.empty((B, m), dtype=torch.int32, device=dev)
    td = torch.empty((B, m), dtype=torch.int32, device=dev)
    ts = torch.empty((B, m), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def one_round():
        dr.draft_tree(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], tw,
                      tt, tp, td, ts, stream=stream)

    for _ in range(args.warmup):
        one_round()
    assert dr.sync_status(stream) == 0
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.2)
    dist_barrier(world)
    torch.cuda.synchronize(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        one_round()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    dist_barrier(world)
    clk = clocks.stop()
    ms = dist_reduce(ev0.elapsed_time(ev1), "max", world, dev if world > 1 else None)
    flags = dr.sync_status(stream)
    launches_per_round = dr.round_launches()
    tokens_total = B * m * args.steps * world
    value = tokens_total / (ms / 1e3)
    per_round_ms = ms / args.steps
    eager_us = eager_round_us(dr, one_round, stream, args.steps, dev)

    prof = [dr.profile_tree(t["tokens"], t["hidden"], t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], tw,
                            tt, tp, td, ts, stream=stream) for _ in range(max(3, min(20, args.steps)))]
    by_kind = {}
    for rnd in prof[1:]:
        for kind, kms in rnd:
            by_kind.setdefault(kind, []).append(kms)
    kind_total = {k: sum(v) / (len(prof) - 1) for k, v in by_kind.items()}
    lm_ms = statistics.mean(by_kind.get(LM_KIND, [float("nan")]))
    es = 2 if s.dtype == "bf16" else 4
    # LM-head launches of a round: step 1 on B rows, steps 2..K on B * w rows
    lm_b = s.vocab * s.hidden * es + (B + (K - 1) * B * tw) / K * (s.hidden * 4 + kTOP * 8)
    peak, peak_src = hbm_peak()
    achieved = lm_b / (lm_ms / 1e3) / 1e9

    pin = {n: torch.from_numpy(np.ascontiguousarray(
        I[n].view(np.int16) if I[n].dtype == np.uint16 else I[n])).pin_memory()
        for n in ("tokens", "hidden", "n_new", "kv_len")}
    if I["hidden"].dtype == np.uint16:
        pin["hidden"] = pin["hidden"].view(torch.bfloat16)
    host_out = [torch.empty((B, m), dtype=torch.int32).pin_memory() for _ in range(2)]
    h2d = sum(p.numel() * p.element_size() for p in pin.values())
    d2h = sum(h.numel() * h.element_size() for h in host_out)

    def e2e_round():
        for n, p in pin.items():
            t[n].copy_(p, non_blocking=True)
        one_round()
        host_out[0].copy_(tt, non_blocking=True)
        host_out[1].copy_(tp, non_blocking=True)

    for _ in range(args.warmup):
        e2e_round()
    torch.cuda.synchronize(dev)
    dist_barrier(world)
    e0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_round()
    torch.cuda.synchronize(dev)
    e_s = dist_reduce(time.perf_counter() - e0, "max", world, dev if world > 1 else None)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        times = []
        t_end = time.perf_counter() + args.cpu_budget
        while True:
            c0 = time.perf_counter()
            oracle.draft_tree(s, W, I, width=tw, n_nodes=m, want_logits=False, seqs=[0])
            times.append(time.perf_counter() - c0)
            if time.perf_counter() >= t_end:
                break
        sec = statistics.median(times)
        cpu = {"value": m / sec, "unit": TREE_UNIT, "cores": oracle.num_threads(), "kind": "oracle",
               "sample": (f"{len(times)} full tree rounds of sequence 0 of {w.name} "
                          f"(median {sec:.3f} s per round), fp64 oracle on all host cores")}

    total_bytes = tree_round_bytes(w, [int(x) for x in I["kv_len"]])
    if rank == 0:
        shares = {k: v / sum(kind_total.values()) for k, v in kind_total.items()}
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": TREE_UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": per_round_ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if s.dtype == "bf16" else "f32",
            "data": "synthetic", "config": dict(config_of(w), options=options),
            "round_latency_us": per_round_ms * 1e3,
            "round_latency_eager_us": eager_us,
            "hbm": {"bytes_per_round": total_bytes,
                    "achieved_gbs": total_bytes / (per_round_ms / 1e3) / 1e9,
                    "frac_of_8tbs": total_bytes / (per_round_ms / 1e3) / 1e9 / NOMINAL_HBM_GBS,
                    "frac_of_measured": total_bytes / (per_round_ms / 1e3) / 1e9 / peak},
            "roofline": {"kernel": "LM head GEMV + top-w selection", "bound": "hbm", "achieved": achieved,
                         "peak": peak, "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": None, "bytes_per_launch": lm_b, "avg_launch_ms": lm_ms},
            "kernel_time_share": shares,
            "kernel_ms_per_round": kind_total,
            "cpu_baseline": cpu,
            "e2e": {"value": B * m * args.steps * world / e_s, "unit": TREE_UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": launches_per_round * args.steps,
            "clocks": clk,
            "device_error_word": flags,
        }), flush=True)
    dr.close()
    del weights_dev

def run_loop(args, w, world, rank, local):
    """prism_draft_loop: a step is one call of R greedy rounds with acceptance
    on the device.  Targets agree with the drafts of a first pass per position
    with probability 1/2 (round 0's agreement is exact; later rounds' inputs
    follow the acceptances, so their agreement is incidental); every step
    starts from the same tokens, n_new and kv_len."""
    import numpy as np
    import torch

    import synth
    from paper_2602_01762_gb300 import Drafter
    from paper_2602_01762_gb300.host import bind_weights, to_device, to_numpy

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s = w.shape
    B, K, R = w.batch, s.n_steps, args.loop
    W = synth.make_weights(w)
    I = synth.make_round_inputs(w, max_new=K + 1)
    mc = (w.ctx_hi + (R + 1) * (K + 1) + K + 15) // 16 * 16
    for key in ("k_cache", "v_cache"):
        a = I[key]
        pad = np.zeros(a.shape[:2] + (mc,) + a.shape[3:], a.dtype)
        pad[:, :, :a.shape[2]] = a
        I[key] = pad
    hid = np.stack([synth.normal(w.seed, f"loop_hidden_{r}", I["hidden"].shape, 1.0, s.dtype) for r in range(R)])
    dr = Drafter.from_shape(s, max_batch=B, max_ctx=mc, max_new=K + 1, topk=1, device=local)
    weights_dev = bind_weights(dr, W, device=dev)
    options = {}
    for kv in args.opt:
        name, value = kv.split("=", 1)
        options[name] = int(value)
        dr.set_option(name, int(value))
    t0 = {n: to_device(I[n], dev) for n in ("tokens", "n_new", "kv_len")}
    t = {n: to_device(I[n], dev) for n in ("tokens", "n_new", "kv_len", "k_cache", "v_cache")}
    hd = to_device(hid, dev)
    i32 = torch.int32
    draft = torch.empty((R, B, K), dtype=i32, device=dev)
    acc = torch.empty((R, B), dtype=i32, device=dev)
    out = torch.empty((R, B, K + 1), dtype=i32, device=dev)
    rnd = synth.uniform_int(w.seed, "loop_target_tok", (R, B, K + 1), 0, s.vocab - 1)
    target = to_device(rnd, dev)
    stream = torch.cuda.current_stream(dev)

    def one_step():
        for n in ("tokens", "n_new", "kv_len"):
            t[n].copy_(t0[n], non_blocking=True)
        dr.draft_loop(t["tokens"], hd, t["n_new"], t["kv_len"], t["k_cache"], t["v_cache"], target, draft, acc,
                      out, stream=stream)

    one_step()
    torch.cuda.synchronize(dev)
    u = synth.uniform01(w.seed, "loop_target_u", (R, B, K))
    tg = rnd.copy()
    tg[:, :, :K] = np.where(u < 0.5, to_numpy(draft), rnd[:, :, :K])
    target.copy_(to_device(tg.astype(np.int32), dev))
    for _ in range(args.warmup):
        one_step()
    assert dr.sync_status(stream) == 0
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.2)
    dist_barrier(world)
    torch.cuda.synchronize(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        one_step()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    dist_barrier(world)
    clk = clocks.stop()
    ms = dist_reduce(ev0.elapsed_time(ev1), "max", world, dev if world > 1 else None)
    flags = dr.sync_status(stream)
    accepted = to_numpy(acc)
    value = B * K * R * args.steps * world / (ms / 1e3)
    per_round_ms = ms / args.steps / R
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if s.dtype == "bf16" else "f32", "data": "synthetic",
            "config": dict(config_of(w), loop_rounds=R, max_new=K + 1, options=options),
            "round_latency_us": per_round_ms * 1e3,
            "loop": {"rounds_per_step": R, "mean_accept_len": float(accepted.mean()),
                     "accepted_tokens_per_s": float((accepted + 1).sum()) * args.steps * world / (ms / 1e3)},
            "cpu_baseline": None, "e2e": None,
            "gpu_launches": None,
            "clocks": clk, "device_error_word": flags,
        }), flush=True)
    dr.close()
    del weights_dev

if __name__ == "__main__":
    main()
