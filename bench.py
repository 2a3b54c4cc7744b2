"""Benchmark of the GBLA layer-core forward on GB300 (one JSON line on rank 0).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--backward | --layer | --hybrid]

A step is one GBLA forward (Conv1D, phi, key gate, state reduction, readout,
gated RMSNorm) over the paper's headline length: B=2, H=8, N=32768, D=64,
bf16 inputs (synthetic, seeded).  `value` is whole-job tokens/s (valid tokens
over all ranks, each token carrying all H heads) with the inputs resident in
HBM; `e2e` is the same metric through the host-memory C-ABI entry point with
the host<->device copies inside the timed region.  `roofline` reports the
dominant kernel's algorithmic bytes per launch over its CUDA-event duration
against the measured HBM copy bandwidth; `cpu_baseline` is the fp64 oracle
timed on this machine's host cores.

Under torchrun each rank runs its own copy of the workload (the (batch, head)
pairs are independent, so the path shards with no collective): weak scaling.
`--impl reference` times the fp64 oracle instead (on rank 0 only), a
deliberately slow program; the GPU/CPU ratio says nothing about kernel quality.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2606_07317_gb300.workloads import (HEADLINE, WORKLOADS, make_inputs,  # noqa: E402
                                              make_layer_inputs)

METRIC = "GBLA fwd tokens/sec and % of GB300 HBM roofline at N=32768, 1 GPU"
UNIT = "tokens/s"
L2_BYTES = 129 * 1024 * 1024
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e data-sheet bandwidth, reported beside the measured peak


# --------------------------------------------------------------------------- helpers

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def init_dist(ws, backend):
    if ws > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group(backend=backend)


def barrier(ws):
    if ws > 1:
        torch.distributed.barrier()


def max_over_ranks(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash() -> str:
    """Hash of the sources of the forward's tensor-core kernels (the ones whose DRAM
    traffic profiles/traffic.json records)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2606_07317_gb300", "csrc")
    for name in ("gbla_tc.cu", "gbla_sm100.cuh"):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on the
    current kernel sources (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel, {}).get(workload)
    if not e or e.get("source_hash") != kernel_source_hash():
        return None
    return e.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=self.f, stderr=subprocess.DEVNULL)
            self.t0 = time.time()
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.t1 = time.time()
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- our arm

def bench_ours(args, ws, rank, local):
    from paper_2606_07317_gb300 import gbla

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(ws, "nccl")
    lib = gbla.load()  # fails loudly if the CUDA library is missing
    w = WORKLOADS[args.workload]
    tokens = w.valid_tokens
    inp0 = make_inputs(w, dev)
    # Two input sets rotated between steps (each larger than L2 at the headline size).
    sets = [inp0, {k: (v.clone() if v is not None else None) for k, v in inp0.items()}]
    outs = [torch.empty_like(inp0["q"]) for _ in sets]
    step_bytes = w.valid_tokens * w.H * w.bytes_per_token_head
    if args.flags:  # an ablation does not need out_gate (no norm) or the gate logits
        e_el = 2 if w.dtype == "bf16" else 4
        step_bytes -= w.valid_tokens * w.H * e_el * (
            (w.D if args.flags & 4 else 0) + (1 if args.flags & 2 else 0))
    stream = torch.cuda.current_stream(dev)

    def step(i):
        s = sets[i % 2]
        gbla.forward(s["q"], s["k"], s["v"], s["gate"], s["out_gate"], s["conv_w"],
                     s["norm_w"], s["seq_lens"], out=outs[i % 2], algo=args.algo, stream=stream,
                     flags=args.flags)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize(dev)

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.1)
    n0 = gbla.launch_count()
    barrier(ws)
    torch.cuda.synchronize(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for i in range(args.steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(ws)
    launches = gbla.launch_count() - n0
    clocks = sampler.stop()
    ms = ev0.elapsed_time(ev1) / args.steps
    ms = max_over_ranks(ms, ws, dev)
    value = tokens * ws / (ms * 1e-3)

    # Per-phase durations (state reduction vs readout) with CUDA events on the
    # launching stream, over the same number of steps (full core only; an
    # ablation reports the whole step against its own algorithmic bytes).
    nph = min(args.steps, 500) if not args.flags else 0
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(nph)]
    st_bufs = [torch.empty((w.B, w.H, w.D * w.D + w.D), dtype=torch.float32, device=dev)
               for _ in sets]
    torch.cuda.synchronize(dev)
    for i in range(nph):
        s = sets[i % 2]
        evs[i][0].record(stream)
        gbla.state(s["k"], s["v"], s["gate"], s["conv_w"], s["seq_lens"], out=st_bufs[i % 2],
                   algo=args.algo, stream=stream)
        evs[i][1].record(stream)
        gbla.readout(s["q"], s["out_gate"], s["conv_w"], s["norm_w"], st_bufs[i % 2],
                     s["seq_lens"], out=outs[i % 2], algo=args.algo, stream=stream)
        evs[i][2].record(stream)
    torch.cuda.synchronize(dev)
    t_state = sum(e[0].elapsed_time(e[1]) for e in evs) / nph if nph else 0.0
    t_read = sum(e[1].elapsed_time(e[2]) for e in evs) / nph if nph else 0.0
    e_el = 2 if w.dtype == "bf16" else 4
    per_th = w.valid_tokens * w.H
    bytes_state = per_th * e_el * (2 * w.D + 1)   # k, v, gate
    bytes_read = per_th * e_el * (3 * w.D)        # q, out_gate, o
    if t_read >= t_state:
        dom, dom_ms, dom_bytes = "readout", t_read, bytes_read
    else:
        dom, dom_ms, dom_bytes = "state", t_state, bytes_state
    if not nph:
        dom, dom_ms, dom_bytes = "whole step (ablation)", ms, step_bytes
    peak, peak_kind = measured_peaks()
    achieved = dom_bytes / (dom_ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                "unit": "GB/s", "frac": round(achieved / peak, 4),
                "traffic": recorded_traffic(dom, w.name),
                "kernel": dom, "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"
                if peak_kind == "measured" else "fallback 6.8 TB/s",
                "alg_bytes_per_launch": dom_bytes, "launch_ms": round(dom_ms, 5),
                "phases_ms": {"state": round(t_state, 5), "readout": round(t_read, 5)},
                "whole_step_frac": round(step_bytes / (ms * 1e-3) / 1e9 / peak, 4),
                "peak_nominal": NOMINAL_HBM_GBS,
                "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                "whole_step_frac_of_nominal":
                    round(step_bytes / (ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS, 4)}

    e2e = None
    if not args.no_e2e and not args.flags:  # the host-buffer entry point runs the full core
        e2e = bench_e2e(args, w, inp0, dev, gbla, tokens, ws)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, inp0)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic (seeded N(0,1) inputs of the workload's shape)",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "D": w.D,
                       "conv_width": 4, "tokens_per_step": tokens,
                       "alg_bytes_per_step": step_bytes,
                       "l2": "inputs larger than L2 (%.0f MB per set vs 129 MB), two sets rotated"
                             % (step_bytes / 1e6),
                       "algo": {0: "auto", 1: "simt", 2: "tc"}[args.algo],
                       "flags": args.flags,
                       "parallelism": f"replicas x{ws}" if ws > 1 else "1 GPU"},
            "roofline": roofline,
            "e2e": e2e,
            "gpu_launches": launches,
            "clocks": clocks,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def bench_backward(args, ws, rank, local):
    """--backward: the backward (gradients of sum(dy * o) for every input) on the
    workload; tokens/s and the whole-step roofline (bf16: q, k, v, out_gate, dy, gate
    read and dq, dk, dv, dout_gate, dgate written, 18 D + 4 bytes per token-head).
    The line's value is gbla_backward_from_state, given the state and gate statistics
    the forward keeps (gbla_state_stats of each input set, made before the timed
    region); `recompute` times gbla_backward, which runs the state pass again."""
    from paper_2606_07317_gb300 import gbla

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(ws, "nccl")
    gbla.load()
    w = WORKLOADS[args.workload]
    tokens = w.valid_tokens
    inp0 = make_inputs(w, dev)
    sets = [inp0, {k: (v.clone() if v is not None else None) for k, v in inp0.items()}]
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed + 1000)
    dys = [torch.randn(inp0["q"].shape, generator=gen, device=dev).to(inp0["q"].dtype)
           for _ in sets]
    saved = [gbla.state_stats(s["k"], s["v"], s["gate"], s["conv_w"], s["seq_lens"])
             for s in sets]
    e_el = 2 if w.dtype == "bf16" else 4
    step_bytes = w.valid_tokens * w.H * e_el * (9 * w.D + 2)
    stream = torch.cuda.current_stream(dev)

    def step(i, from_state):
        s = sets[i % 2]
        kw = dict(state=saved[i % 2][0], stats=saved[i % 2][1]) if from_state else {}
        gbla.backward(s["q"], s["k"], s["v"], s["gate"], s["out_gate"], s["conv_w"],
                      s["norm_w"], s["seq_lens"], dys[i % 2], stream=stream, **kw)

    def timed(from_state):
        for i in range(args.warmup):
            step(i, from_state)
        torch.cuda.synchronize(dev)
        n0 = gbla.launch_count()
        barrier(ws)
        torch.cuda.synchronize(dev)
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for i in range(args.steps):
            step(i, from_state)
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(ws)
        return (max_over_ranks(ev0.elapsed_time(ev1) / args.steps, ws, dev),
                gbla.launch_count() - n0)

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.1)
    ms, launches = timed(True)
    ms_re, launches_re = timed(False)
    clocks = sampler.stop()
    peak, peak_kind = measured_peaks()
    achieved = step_bytes / (ms * 1e-3) / 1e9
    achieved_re = step_bytes / (ms_re * 1e-3) / 1e9
    if rank == 0:
        print(json.dumps({
            "metric": "GBLA bwd tokens/sec (gradients of every input)", "value":
            round(tokens * ws / (ms * 1e-3), 1), "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic (seeded N(0,1) inputs and dy)",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "D": w.D,
                       "alg_bytes_per_step": step_bytes,
                       "state": "the forward's, kept (gbla_backward_from_state)",
                       "l2": "inputs larger than L2, two sets rotated"},
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                         "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": None,
                         "kernel": "whole backward step",
                         "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"},
            "recompute": {"entry": "gbla_backward (state pass included)",
                          "ms_per_step": round(ms_re, 6),
                          "value": round(tokens * ws / (ms_re * 1e-3), 1),
                          "frac": round(achieved_re / peak, 4), "gpu_launches": launches_re},
            "gpu_launches": launches, "clocks": clocks}), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def measured_bf16_peak():
    """Dense bf16 tensor peak (TFLOP/s): the burst figure of MEASURED_PEAKS.json for a
    kernel timed on its own, else the fallback."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        if "bf16_tflops" in d:
            return float(d["bf16_tflops"]), "measured"
    return 1900.0, "fallback"


def bench_layer(args, ws, rank, local):
    """--layer: the whole GBLA layer from the embedded sequence X (gbla_layer_forward:
    X-space Conv1D and the stacked projections on tensor cores, then the core with its
    Conv1D off) on the workload's B, N, H, D with model width d = H D; tokens/s of the
    layer, and the front-end kernel (gbla_project) against the bf16 tensor peak:
    2 d (4 H D + H) flops per token."""
    from paper_2606_07317_gb300 import gbla

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(ws, "nccl")
    gbla.load()
    w = WORKLOADS[args.workload]
    d = args.model_dim or w.H * w.D
    F = 4 * w.H * w.D + w.H
    tokens = w.valid_tokens
    sets = [make_layer_inputs(w.B, w.N, d, w.H, w.D, seed=w.seed + i, seq_lens=w.seq_lens,
                              device=dev) for i in range(2)]
    outs = [torch.empty((w.B, w.N, w.H, w.D), dtype=torch.bfloat16, device=dev) for _ in sets]
    pouts = [{n: torch.empty((w.B, w.N, w.H, w.D), dtype=torch.bfloat16, device=dev)
              for n in ("q", "k", "v", "out_gate")} for _ in sets]
    for po in pouts:
        po["gate"] = torch.empty((w.B, w.N, w.H), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    def layer_step(i):
        s = sets[i % 2]
        gbla.layer_forward(s["x"], s["conv_x"], s["w_proj"], s["norm_w"], w.H, w.D,
                           seq_lens=s["seq_lens"], out=outs[i % 2], stream=stream)

    def project_step(i):
        s = sets[i % 2]
        gbla.project(s["x"], s["conv_x"], s["w_proj"], w.H, w.D, seq_lens=s["seq_lens"],
                     out=pouts[i % 2], stream=stream)

    def timed(fn, steps):
        for i in range(args.warmup):
            fn(i)
        torch.cuda.synchronize(dev)
        barrier(ws)
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for i in range(steps):
            fn(i)
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(ws)
        return max_over_ranks(ev0.elapsed_time(ev1) / steps, ws, dev)

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.1)
    n0 = gbla.launch_count()
    ms = timed(layer_step, args.steps)
    launches = gbla.launch_count() - n0
    ms_proj = timed(project_step, args.steps)
    clocks = sampler.stop()
    assert gbla.device_error() == 0
    flops = 2.0 * d * F * tokens
    tf_peak, tf_kind = measured_bf16_peak()
    achieved = flops / (ms_proj * 1e-3) / 1e12
    hbm_peak, _ = measured_peaks()
    proj_bytes = tokens * 2 * (d + F)
    if rank == 0:
        print(json.dumps({
            "metric": "GBLA layer fwd tokens/sec (X-space Conv1D + fused projections + core)",
            "value": round(tokens * ws / (ms * 1e-3), 1), "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic (seeded N(0,1) x, N(0,1/d) weights)",
            "config": {"workload": w.name + f"_layer_d{d}", "B": w.B, "H": w.H, "N": w.N,
                       "D": w.D, "d": d, "F": F, "tokens_per_step": tokens,
                       "l2": "two input sets rotated; each step writes 4 B N H D bf16 "
                             "intermediates (%.0f MB, above L2)" % (8 * tokens * w.H * w.D / 1e6)},
            "roofline": {"bound": "tensor", "achieved": round(achieved, 1), "peak": tf_peak,
                         "unit": "TFLOP/s", "frac": round(achieved / tf_peak, 4),
                         "traffic": None, "kernel": "tc_project_kernel",
                         "peak_source": f"{tf_kind} (MEASURED_PEAKS.json bf16_tflops, burst)",
                         "flops_per_launch": flops, "launch_ms": round(ms_proj, 5),
                         "hbm_gbs": round(proj_bytes / (ms_proj * 1e-3) / 1e9, 1),
                         "hbm_frac": round(proj_bytes / (ms_proj * 1e-3) / 1e9 / hbm_peak, 4),
                         "phases_ms": {"project": round(ms_proj, 5),
                                       "core": round(ms - ms_proj, 5)}},
            "gpu_launches": launches, "clocks": clocks}), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def bench_hybrid(args, ws, rank, local):
    """--hybrid: the paper's hybrid encoder block [SA, LA, LA] (Sec. 3) against an
    all-softmax block [SA, SA, SA], core only (the mixing of given q, k, v, and for
    GBLA the gate and out-gate inputs): batch 8, 16 heads of 64 (Table 5), L from
    2048 to 32768.  Each stack is its three calls back to back on one stream;
    per-layer latencies of both layers and the SA / GBLA ratio (Table 5's
    columns) are printed per L.  SA is this library's tcgen05 kernel
    (gbla_attention_forward), timed against the bf16 tensor peak."""
    from paper_2606_07317_gb300 import gbla
    from paper_2606_07317_gb300.workloads import custom

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(ws, "nccl")
    gbla.load()
    B, H, D = 8, 16, 64
    stream = torch.cuda.current_stream(dev)
    tf_peak, tf_kind = measured_bf16_peak()
    rows = []
    sampler = ClockSampler(local)
    sampler.start()
    n0 = gbla.launch_count()
    for L in args.hybrid_lengths:
        inp = make_inputs(custom(B=B, H=H, N=L, D=D, dtype="bf16", seed=L), dev)
        o_sa = torch.empty_like(inp["q"])
        o_la = torch.empty_like(inp["q"])

        def sa():
            gbla.attention(inp["q"], inp["k"], inp["v"], None, out=o_sa, stream=stream)

        def la():
            gbla.forward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                         inp["conv_w"], inp["norm_w"], None, out=o_la, stream=stream)

        def timed(fn, budget_s=4.0):
            for _ in range(args.warmup):
                fn()
            torch.cuda.synchronize(dev)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            one = e0.elapsed_time(e1)
            n = max(1, min(args.steps, int(budget_s * 1e3 / max(one, 1e-3))))
            barrier(ws)
            e0.record(stream)
            for _ in range(n):
                fn()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            return max_over_ranks(e0.elapsed_time(e1) / n, ws, dev), n

        t_sa, n_sa = timed(sa)
        t_la, n_la = timed(la)
        t_hyb, _ = timed(lambda: (sa(), la(), la()))
        t_all, _ = timed(lambda: (sa(), sa(), sa()))
        flops = 4.0 * B * H * L * L * D
        rows.append({"L": L, "sa_ms": round(t_sa, 4), "gbla_ms": round(t_la, 4),
                     "sa_over_gbla": round(t_sa / t_la, 2),
                     "block_sa_la_la_ms": round(t_hyb, 4), "block_sa_sa_sa_ms": round(t_all, 4),
                     "block_speedup": round(t_all / t_hyb, 2),
                     "sa_tflops": round(flops / (t_sa * 1e-3) / 1e12, 1),
                     "sa_frac_of_bf16_peak": round(flops / (t_sa * 1e-3) / 1e12 / tf_peak, 4),
                     "gbla_tokens_per_s": round(B * L / (t_la * 1e-3), 1),
                     "timed_calls": {"sa": n_sa, "gbla": n_la}})
        del inp, o_sa, o_la
        torch.cuda.empty_cache()
    clocks = sampler.stop()
    assert gbla.device_error() == 0
    if rank == 0:
        last = rows[-1]
        print(json.dumps({
            "metric": "hybrid encoder block [SA, LA, LA] vs [SA, SA, SA]: per-layer latency "
                      "(core), batch 8, 16 heads of 64",
            "value": last["block_speedup"], "unit": "x (block [SA,SA,SA] / [SA,LA,LA] time) "
                                                     "at the longest L",
            "n_gpus": ws, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic (seeded N(0,1) inputs)",
            "config": {"workload": "hybrid_block_b8_h16_d64", "B": B, "H": H, "D": D,
                       "lengths": args.hybrid_lengths,
                       "note": "core only: SA = softmax mixing of q, k, v; LA = the GBLA core "
                               "(Conv1D, key gate, state, readout, gated RMSNorm); no "
                               "projections in either"},
            "per_length": rows,
            "sa_peak": {"bf16_tflops": tf_peak, "source": tf_kind},
            "gpu_launches": gbla.launch_count() - n0, "clocks": clocks}), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def bench_e2e(args, w, inp, dev, gbla, tokens, ws):
    host = {k: (v.cpu().pin_memory() if v is not None else None) for k, v in inp.items()}
    out = torch.empty_like(host["q"]).pin_memory()
    n = max(3, min(args.steps, 30))

    def call():
        gbla.forward_host(host["q"], host["k"], host["v"], host["gate"], host["out_gate"],
                          host["conv_w"], host["norm_w"], host["seq_lens"], out=out)

    for _ in range(2):
        call()
    barrier(ws)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for _ in range(n):
        call()
    torch.cuda.synchronize(dev)
    dt = (time.perf_counter() - t0) / n
    dt = max_over_ranks(dt, ws, dev)
    e_el = 2 if w.dtype == "bf16" else 4
    th = w.valid_tokens * w.H
    h2d = th * e_el * (4 * w.D + 1) + 4 * (3 * w.H * w.D * 4 + w.H * w.D)
    if w.seq_lens is not None:
        h2d += 4 * w.B
    d2h = th * e_el * w.D
    return {"value": round(tokens * ws / dt, 1), "unit": UNIT, "steps": n,
            "ms_per_step": round(dt * 1e3, 4),
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "api": "gbla_forward_host (pinned host buffers)"}


# --------------------------------------------------------------------------- oracle (CPU)

def _oracle_inputs(inp, pairs, lens):
    """float64 slices of the valid tokens of each (b, h) pair, taken outside any
    timing; lens[i] is the number of tokens used for pairs[i]."""
    f64 = lambda t: t.detach().cpu().double().numpy()  # noqa: E731
    cw, nw = f64(inp["conv_w"]), f64(inp["norm_w"])
    out = []
    for (b, h), L in zip(pairs, lens):
        sl = lambda n: np.ascontiguousarray(f64(inp[n][b, :L, h]))  # noqa: E731
        out.append(dict(q=sl("q"), k=sl("k"), v=sl("v"), a=sl("gate"), og=sl("out_gate"),
                        wq=cw[0, h], wk=cw[1, h], wv=cw[2, h], nw=nw[h]))
    return out


def _oracle_run(heads, n_threads):
    import concurrent.futures as cf

    import oracle
    lib = oracle.load()

    def one(x):
        return oracle.gbla_head(x["q"], x["k"], x["v"], x["a"], x["og"], x["wq"], x["wk"],
                                x["wv"], x["nw"], lib=lib)
    if n_threads == 1:
        for x in heads:
            one(x)
    else:  # ctypes releases the GIL, so threads run the C oracle in parallel
        with cf.ThreadPoolExecutor(n_threads) as ex:
            list(ex.map(one, heads))


def _sample_pairs(w):
    """The workload's (b, h) pairs with a non-empty sequence, heads outermost, so
    that any prefix of the list spans the batch's length mix."""
    lens = w.lengths()
    return [(b, h) for h in range(w.H) for b in range(w.B) if lens[b] > 0]


def cpu_baseline(w, inp, budget_s: float = 10.0):
    """The oracle on the host cores over a bounded sample of the workload: batches of
    (b, h) sequences, each over its own valid length, one thread per sequence, until
    about `budget_s` seconds of oracle time; plus a single-thread rate on one
    sequence.  Only the oracle calls are timed."""
    cores = os.cpu_count() or 1
    lens = w.lengths()
    pairs = _sample_pairs(w)
    threads = min(cores, len(pairs))
    done_tok_heads, dt, npairs, i = 0, 0.0, 0, 0
    while dt < budget_s:
        batch = [pairs[(i + j) % len(pairs)] for j in range(threads)]
        i += threads
        heads = _oracle_inputs(inp, batch, [lens[b] for b, _ in batch])
        t0 = time.perf_counter()
        _oracle_run(heads, threads)
        dt += time.perf_counter() - t0
        done_tok_heads += sum(lens[b] for b, _ in batch)
        npairs += len(batch)
    # single thread: the median-length sequence of the first batch
    first = sorted(pairs[:threads], key=lambda bh: lens[bh[0]])
    b1, h1 = first[len(first) // 2]
    one = _oracle_inputs(inp, [(b1, h1)], [lens[b1]])
    t0 = time.perf_counter()
    _oracle_run(one, 1)
    dt1 = time.perf_counter() - t0
    return {"value": round(done_tok_heads / w.H / dt, 1), "unit": UNIT, "cores": threads,
            "host_cores": cores, "kind": "oracle", "seconds": round(dt, 3),
            "single_thread_value": round(lens[b1] / w.H / dt1, 1),
            "sample": f"{npairs} (batch, head) sequences of {w.name} (cycling heads-outer over "
                      f"all {len(pairs)} non-empty ones), each over its own valid length, "
                      f"fp64 C oracle, {threads} threads (one per sequence) on "
                      f"{cores} host cores; tokens = token-heads / H; single thread: one "
                      f"{lens[b1]}-token sequence"}


def bench_reference(args, ws, rank):
    """--impl reference: the fp64 oracle on the host cores (rank 0 only)."""
    if rank != 0:
        return
    w = WORKLOADS[args.workload]
    inp = make_inputs(w, "cpu")
    cores = os.cpu_count() or 1
    lens = w.lengths()
    pairs = _sample_pairs(w)
    # calibrate the sample so that (warmup + steps) fit in ~120 s
    probe_L = min(1024, max(lens))
    bp = max(range(w.B), key=lambda b: lens[b])
    heads = _oracle_inputs(inp, [(bp, 0)], [probe_L])
    t0 = time.perf_counter()
    _oracle_run(heads, 1)
    per_tok = (time.perf_counter() - t0) / probe_L
    n_pairs = min(len(pairs), cores)
    batch = pairs[:n_pairs]
    step_budget = 120.0 / max(1, args.steps + args.warmup)
    # each sequence over its own length, capped so that the slowest thread fits
    cap = int(max(64, step_budget / per_tok))
    use = [min(lens[b], cap) for b, _ in batch]
    heads = _oracle_inputs(inp, batch, use)
    for _ in range(args.warmup):
        _oracle_run(heads, n_pairs)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _oracle_run(heads, n_pairs)
    dt = (time.perf_counter() - t0) / args.steps
    tok = sum(use) / w.H
    value = tok / dt
    capped = sum(1 for b, _ in batch if lens[b] > cap)
    sample = (f"per step: {n_pairs} (batch, head) sequences of {w.name} (heads outer), each "
              f"over its own valid length" + (f", {capped} of them capped at {cap} tokens"
                                              if capped else "") +
              f"; fp64 C oracle, one thread per sequence on {cores} host cores; "
              f"tokens = token-heads / H")
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT,
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(dt * 1e3, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "D": w.D},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": n_pairs,
                             "host_cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=HEADLINE, choices=sorted(WORKLOADS))
    ap.add_argument("--algo", type=int, default=0, help="0 auto, 1 simt, 2 tc")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--flags", type=int, default=0,
                    help="ablation (gbla_flags): 1 no Conv1D, 2 uniform gate, 4 no gated "
                         "RMSNorm, 7 BLA; 0 (default) is the full core")
    ap.add_argument("--backward", action="store_true",
                    help="time gbla_backward instead of the forward")
    ap.add_argument("--layer", action="store_true",
                    help="time the whole layer from X (gbla_layer_forward) and its front end")
    ap.add_argument("--model-dim", type=int, default=0,
                    help="--layer: model width d (default H * D)")
    ap.add_argument("--hybrid", action="store_true",
                    help="time the hybrid block [SA, LA, LA] against [SA, SA, SA] (Table 5's "
                         "shapes: batch 8, 16 heads of 64) over --hybrid-lengths")
    ap.add_argument("--hybrid-lengths", type=int, nargs="+",
                    default=[2048, 4096, 8192, 16384, 32768])
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    ws, rank, local = dist_env()
    if args.gpus != ws:
        sys.exit(f"bench.py: --gpus {args.gpus} but WORLD_SIZE is {ws}; for N > 1 launch one "
                 f"process per GPU with torch.distributed.run --nproc-per-node N")
    if args.impl == "reference":
        bench_reference(args, ws, rank)
        return
    if args.backward:
        bench_backward(args, ws, rank, local)
        return
    if args.layer:
        bench_layer(args, ws, rank, local)
        return
    if args.hybrid:
        bench_hybrid(args, ws, rank, local)
        return
    bench_ours(args, ws, rank, local)


if __name__ == "__main__":
    main()
