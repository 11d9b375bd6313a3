#!/usr/bin/env python3
"""Throughput of the LUNA attention hot path on GB300 (one JSON line on stdout).

A step is one pass of the whole path over one batch of synthetic input: the
feature-map table is prepared from the parameters, the forward pass runs
(saving the key statistics) and the backward pass produces dQ, dK, dV and the
parameter gradients.  The default workload is the long-context streaming form
(causal_long: B=2, H=32, n=65536, d=128, D=128, bf16 I/O, fwd+bwd); the
Long-Range-Arena-shaped encoder attention (lra: B=32, H=4, n=4096, d=32, D=64,
valid lengths uniform in [2048, 4096], non-causal) is measured in the same run
and reported under its own key.  Tokens per step = B * n.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--also NAMES] [--impl reference]

Every kernel's roofline fraction counts only the method's own tensors that it
reads or writes (Q, K, V, dO, O, dQ, dK, dV and the per-head key statistics);
rows that one stage hands to the next are traffic, not algorithmic bytes.

Multi-GPU (torchrun): every rank runs an independent replica of the workload
(the (batch, head) units are independent; there is no data-path collective),
so scaling is weak and value = all ranks' tokens / max-over-ranks time.
`--impl reference` times the fp64 CPU oracle instead (rank 0 only), on a
bounded sample of the same workload (the first 4096 tokens of each sequence
for the streaming form), and reports the rate of that sample.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402
from synth.workloads import WORKLOADS  # noqa: E402

METRIC = "LUNA attn tokens/sec fwd & fwd+bwd on 1 GB300; % of HBM/tensor roofline"
L2_BYTES = 129 * 1024 * 1024


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="causal_long", choices=sorted(WORKLOADS))
    ap.add_argument("--also", default="lra",
                    help="comma-separated workloads also measured in the same run, each under its own key "
                         "(empty: none)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU work of the oracle sample")
    ap.add_argument("--seq-len", type=int, default=0,
                    help="shorter sequence length n for profiler captures of a small case (the JSON line reports it)")
    ap.add_argument("--ch-rms-target", type=float, default=0.0,
                    help="channel RMS normalisation of the feature map with this target (non-causal workloads)")
    args = ap.parse_args()
    if args.ch_rms_target < 0:
        ap.error("--ch-rms-target must be >= 0")
    if args.ch_rms_target > 0 and WORKLOADS[args.workload].decode:
        ap.error("--ch-rms-target: the channel normalisation is a batch statistic, not defined for a decode step")
    args.also = [a for a in args.also.split(",") if a]
    for a in args.also:
        if a not in WORKLOADS or WORKLOADS[a].decode:
            ap.error(f"--also: unknown or decode workload {a}")
    if args.seq_len > 0 or args.ch_rms_target > 0:
        args.also = []
    return args


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def max_over_ranks(value: float, device, world: int) -> float:
    """The largest of the ranks' values (a replicated step takes as long as its slowest rank);
    the value itself on one rank."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as tdist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, ms: float) -> float:
    """Whole-job rate: the units every rank processed, over the slowest rank's time (ms)."""
    return units_per_rank * world / (ms * 1e-3)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


# --------------------------------------------------------------------------
# algorithmic bytes and flops of the method's own inputs and outputs

def row_counts(w, lengths):
    valid = int(np.sum(lengths)) * w.H if lengths is not None else w.B * w.H * w.n
    return valid, w.B * w.H * w.n


def kernel_bytes(w, lengths, kernel: str) -> float:
    """Algorithmic HBM bytes of one launch of a kernel: the method's own tensors
    that the kernel reads or writes (Q, K, V, dO read on their valid rows; O,
    dQ, dK, dV written on every row, padded rows as zeros) and, for the
    non-causal passes, the (D x dv + D) fp32 key statistics per head that the
    method hands from the key pass to the query pass.  Rows that one stage of
    the streaming-form backward writes for the next one (dphi, phi(k),
    phi(q)/den) are this implementation's staging, not the method's: they count
    as traffic (ncu), never as algorithmic bytes."""
    eb = 4 if w.io == "f32" else 2
    valid, total = row_counts(w, lengths)
    stats = w.B * w.H * (w.D * w.dv + w.D) * 4
    rd, rv = w.d * eb, w.dv * eb
    table = {
        "keystats": valid * (rd + rv) + stats,
        "query": valid * rd + total * rv + stats,
        "bwd_query": valid * (rd + rv) + total * rd + 2 * stats,
        "bwd_key": valid * (rd + rv) + total * (rd + rv) + stats,
        "causal_out": valid * (2 * rd + rv) + total * rv,
        # streaming-form backward on tensor cores: the method's tensors each stage touches
        "tcc_query": valid * (2 * rd + 2 * rv),   # Q, K, V, dO
        "tcc_dstats": 0,                          # staging rows only
        "tcc_key": valid * 2 * rv + total * rv,   # V, dO; dV
        "tc_phi_bwd": valid * rd + total * rd,    # Q (or K); dQ (or dK)
        # channel normalisation, both sides per launch: the statistics read every valid row of Q and K;
        # the scale-term pass reads them and reads and writes the same rows of dQ and dK
        "chrms_stats": 2 * valid * rd,
        "tc_chstats": 2 * valid * rd,             # the same statistics with the projections on tensor cores
        "chrms_kterm": 2 * valid * 3 * rd,
        "tc_kterm": 2 * valid * 3 * rd,           # the same scale term on tensor cores
    }
    # the tensor-core kernels move the same tensors as their generic counterparts
    for tc, generic in (("tc_keys", "keystats"), ("tc_query", "query"), ("tc_bwd_query", "bwd_query"),
                        ("tc_bwd_key", "bwd_key"), ("tc_causal", "causal_out")):
        table[tc] = table[generic]
    if w.causal:  # the streaming form's key pass per state segment reads K and V; its statistics are staging
        table["tc_keys"] = valid * (rd + rv)
    return float(table.get(kernel, 0.0))


CSRC = os.path.join(ROOT, "paper_2512_08061_gb300", "csrc")


def _includes(name: str, seen: set) -> None:
    """`name` and the library headers it includes, transitively."""
    if name in seen or not os.path.exists(os.path.join(CSRC, name)):
        return
    seen.add(name)
    with open(os.path.join(CSRC, name)) as fh:
        for line in fh:
            m = re.match(r'\s*#\s*include\s+"([^"]+)"', line)
            if m:
                _includes(m.group(1), seen)


def kernel_source(kernel: str):
    """The CUDA source file that defines `k_<kernel>`, or None."""
    pat = re.compile(r"\bk_" + re.escape(kernel) + r"\s*\(")
    for f in sorted(os.listdir(CSRC)):
        if f.endswith(".cu"):
            with open(os.path.join(CSRC, f)) as fh:
                if any(pat.search(line) and "__global__" in line for line in fh):
                    return f
    for f in sorted(os.listdir(CSRC)):  # definitions whose __global__ sits on the line before the name
        if f.endswith(".cu"):
            with open(os.path.join(CSRC, f)) as fh:
                if pat.search(fh.read()):
                    return f
    return None


def csrc_digest(kernel: str | None = None) -> str:
    """sha256 over CUDA sources (file names and contents): the file that defines k_<kernel> and the
    library headers it includes; with no kernel, every source of the library."""
    files = set()
    if kernel is not None:
        src = kernel_source(kernel)
        if src is not None:
            _includes(src, files)
    if not files:
        files = {f for f in os.listdir(CSRC) if f.endswith((".cu", ".cuh"))}
    h = hashlib.sha256()
    for f in sorted(files):
        h.update(f.encode())
        with open(os.path.join(CSRC, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def measured_traffic(kernel: str, workload: str):
    """DRAM bytes (read + write) per launch of `kernel` from the committed ncu
    summaries (lines `traffic <workload> k_<kernel> <bytes> <sources sha256>`, the digest over the
    kernel's own source file and the headers it includes), or None when no summary was taken on the
    current sources."""
    pdir = os.path.join(ROOT, "profiles")
    digest = csrc_digest(kernel)
    try:
        names = sorted(os.listdir(pdir))
    except OSError:
        return None, None
    for f in names:
        if not f.endswith(".md"):
            continue
        with open(os.path.join(pdir, f)) as fh:
            for line in fh:
                parts = line.strip().strip("`").split()
                if len(parts) == 5 and parts[0] == "traffic" and parts[1] == workload and parts[2] == "k_" + kernel:
                    if parts[4] == digest:
                        return float(parts[3]), "profiles/" + f
    return None, None


def step_bytes(w, lengths) -> float:
    eb = 4 if w.io == "f32" else 2
    valid, total = row_counts(w, lengths)
    fwd = valid * (2 * w.d + w.dv) * eb + total * w.dv * eb
    bwd = valid * (2 * w.d + 2 * w.dv) * eb + total * (2 * w.d + w.dv) * eb
    return float(fwd + bwd) if w.backward else float(fwd)


def step_flops(w, lengths) -> float:
    """Tensor-core flops of the recurrent minimum per valid row (Sec. 4 runtime
    model): forward 4Md + 4Dd + 4D, backward 12Md + 10Dd + 6D (both sides)."""
    valid, _ = row_counts(w, lengths)
    f = 4 * w.M * w.d + 4 * w.D * w.dv + 4 * w.D
    b = 12 * w.M * w.d + 10 * w.D * w.dv + 6 * w.D
    return float(valid * (f + (b if w.backward else 0)))


# --------------------------------------------------------------------------
# clocks during the timed region

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: str):
        self.proc = None
        self.path = None
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-i", gpu_index, "-lms", "50"], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 8:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        smax = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------
# the GPU arm

def host_inputs(w):
    inp = synth.attn_inputs(w.seed, w.B, w.H, w.n, w.d, w.dv, w.io, w.qkv_scale, w.len_range, with_grad=w.backward)
    params = synth.phi_params(w.seed, w.d, w.M, w.L, w.hidden)
    return inp, params


def workload_label(w, ch_rms_target=0.0) -> str:
    return (f"{w.name}: B={w.B} H={w.H} n={w.n} d={w.d} D={w.D} (M={w.M}, L={w.L}), {w.io}, "
            f"{'causal' if w.causal else 'non-causal'}, {'fwd+bwd' if w.backward else 'fwd'}"
            + (f", lengths U[{w.len_range[0]},{w.len_range[1]}]" if w.len_range else "")
            + (f", channel RMS normalisation target {ch_rms_target:g}" if ch_rms_target > 0 else ""))


def measure_workload(args, w, dev, world, steps, ch_rms_target=0.0, with_e2e=True):
    """Times `steps` steps of workload w on this rank's GPU (after the warm-up), the forward alone, every
    library kernel of a step (live CUDA events on the launching stream) and, with_e2e, the step end to end
    from pinned host buffers.  Returns the measurements of this rank (times are max over ranks)."""
    import torch
    import paper_2512_08061_gb300.luna as L

    inp, params = host_inputs(w)
    io_dtype = torch.float32 if w.io == "f32" else torch.bfloat16

    def pinned(t):
        if t.io == "f32":
            h = torch.from_numpy(np.ascontiguousarray(t.raw))
        else:
            h = torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).view(torch.bfloat16)
        return h.pin_memory()

    host = {k: pinned(inp[k]) for k in ("Q", "K", "V", "dO") if k in inp}
    lengths_h = None if inp["lengths"] is None else torch.from_numpy(inp["lengths"]).pin_memory()
    devt = {k: v.to(dev, non_blocking=True) for k, v in host.items()}
    lengths_d = None if lengths_h is None else lengths_h.to(dev)
    params_d = {k: torch.from_numpy(v).to(dev) for k, v in params.items()}
    lu = L.Luna(w.B, w.H, w.n, w.d, w.dv, w.M, w.L, w.hidden, w.causal, w.eps, io_dtype, w.chunk, dev,
                ch_rms_target=ch_rms_target)
    O = torch.empty_like(devt["V"])
    grads = None
    f32 = dict(dtype=torch.float32, device=dev)

    def grad_buffers():
        return {"dQ": torch.empty_like(devt["Q"]), "dK": torch.empty_like(devt["K"]),
                "dV": torch.empty_like(devt["V"]), "dW": torch.empty(w.M, w.d, **f32),
                "db": torch.empty(w.M, **f32), "dw1": torch.empty(w.L, w.hidden, **f32),
                "db1": torch.empty(w.L, w.hidden, **f32), "dw2": torch.empty(w.L, w.hidden, **f32),
                "db2": torch.empty(w.L, **f32)}

    if w.backward:
        grads = grad_buffers()
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(t, backward=w.backward):
        lu.prepare(params_d)
        lu.forward(t["Q"], t["K"], t["V"], lengths_d, O=O, save_state=True)
        if backward:
            lu.backward(t["Q"], t["K"], t["V"], t["dO"], lengths_d, use_state=True, out=grads)

    def timed(n_steps, fn):
        """Per-step CUDA-event times with an L2 flush (outside the events) before each step."""
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_steps)]
        for s0, s1 in evs:
            flush.zero_()
            s0.record(stream)
            fn()
            s1.record(stream)
        torch.cuda.synchronize()
        return sum(s0.elapsed_time(s1) for s0, s1 in evs)

    for _ in range(max(args.warmup, 3)):
        step(devt)
    torch.cuda.synchronize()

    # every library kernel of one step, timed live with CUDA events on its launching stream
    kernels = ["phi_prepare", "keystats", "query", "bwd_query", "bwd_key", "grad_sum", "mlp_grads",
               "causal_out", "causal_bwd_seg", "causal_dq", "causal_dkv"] + L.TC_KERNELS
    if ch_rms_target > 0:
        kernels += ["chrms_stats", "tc_chstats", "chrms_scales", "chrms_scale", "chrms_dstate", "chrms_kappa",
                    "chrms_kterm", "tc_kterm"]
    per_kernel = {}
    for k in kernels:
        L.luna_profile_start(k)
        step(devt)
        ms, n = L.luna_profile_stop()
        if n:
            per_kernel[k] = (ms, n)
    dominant = max(per_kernel, key=lambda k: per_kernel[k][0]) if per_kernel else None

    # timed region
    if world > 1:
        import torch.distributed as tdist
        tdist.barrier()
    torch.cuda.synchronize()
    uuid = str(getattr(torch.cuda.get_device_properties(dev), "uuid", "") or "")
    clocks = ClockSampler(("GPU-" + uuid if uuid and not uuid.startswith("GPU-") else uuid) or str(dev.index))
    if dominant:
        L.luna_profile_start(dominant)
    n0 = L.luna_launch_count()
    ms_total = timed(steps, lambda: step(devt))
    launches = L.luna_launch_count() - n0
    dom_ms, dom_n = L.luna_profile_stop() if dominant else (0.0, 0)
    clk = clocks.stop()
    torch.cuda.synchronize()
    ms_step = max_over_ranks(ms_total / steps, dev, world)

    # forward-only throughput (same flush discipline)
    fwd_ms = max_over_ranks(timed(steps, lambda: step(devt, backward=False)) / steps, dev, world)

    # End to end through the public API with host buffers: every step copies its inputs in from pinned host
    # memory and reads all of its results back (O; with the backward also dQ, dK, dV and the parameter
    # gradients).  Steps are pipelined two deep on three streams (copy-in, compute, copy-out) with
    # double-buffered device inputs and outputs, so that step i+1's inputs arrive and step i-1's results
    # leave while step i computes.  Events keep every dependency: a step computes after its own inputs have
    # landed, its results leave after it has computed, and a buffer is refilled only after the step that
    # last used it is done with it.
    e2e = None
    if with_e2e:
        nb = 2
        dev_in = [{k: torch.empty_like(devt[k]) for k in host} for _ in range(nb)]
        len_in = [None if lengths_h is None else torch.empty_like(lengths_d) for _ in range(nb)]
        dev_out = [dict({"O": torch.empty_like(O)}, **(grad_buffers() if grads else {})) for _ in range(nb)]
        result_keys = list(dev_out[0].keys())
        host_out = [{k: torch.empty(dev_out[0][k].shape, dtype=dev_out[0][k].dtype).pin_memory() for k in result_keys}
                    for _ in range(nb)]
        bi = sum(v.numel() * v.element_size() for v in host.values()) + (
            lengths_h.numel() * 4 if lengths_h is not None else 0)
        bo = sum(v.numel() * v.element_size() for v in host_out[0].values())
        s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
        ev_in = [torch.cuda.Event() for _ in range(nb)]
        ev_c = [torch.cuda.Event() for _ in range(nb)]
        ev_out = [torch.cuda.Event() for _ in range(nb)]

        def compute(t, ln, out):
            lu.prepare(params_d)
            lu.forward(t["Q"], t["K"], t["V"], ln, O=out["O"], save_state=True)
            if w.backward:
                lu.backward(t["Q"], t["K"], t["V"], t["dO"], ln, use_state=True, out=out)

        def e2e_run(n_steps, t_start=None, t_end=None):
            for i in range(n_steps):
                b = i % nb
                with torch.cuda.stream(s_in):
                    if i >= nb:
                        s_in.wait_event(ev_c[b])  # step i-2 has read these inputs
                    if i == 0 and t_start is not None:
                        t_start.record(s_in)
                    for k in host:
                        dev_in[b][k].copy_(host[k], non_blocking=True)
                    if lengths_h is not None:
                        len_in[b].copy_(lengths_h, non_blocking=True)
                    ev_in[b].record(s_in)
                stream.wait_event(ev_in[b])
                if i >= nb:
                    stream.wait_event(ev_out[b])  # step i-2's results have left these buffers
                compute(dev_in[b], len_in[b], dev_out[b])
                ev_c[b].record(stream)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(ev_c[b])
                    for k in result_keys:
                        host_out[b][k].copy_(dev_out[b][k], non_blocking=True)
                    ev_out[b].record(s_out)
            if t_end is not None:
                s_out.wait_stream(s_in)
                s_out.wait_stream(stream)
                t_end.record(s_out)

        e2e_run(2 * nb)
        torch.cuda.synchronize()
        n_e2e = max(8, steps // 2)
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e2e_run(n_e2e, t0, t1)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(t0.elapsed_time(t1) / n_e2e, dev, world)
        e2e = {"value": job_throughput(w.tokens, world, e2e_ms), "unit": "tokens/s", "h2d_bytes_per_step": int(bi),
               "d2h_bytes_per_step": int(bo), "ms_per_step": e2e_ms,
               "pipelining": "copy-in of step i+1 and copy-out of step i-1 overlap the compute of step i",
               "result": ", ".join(result_keys) + " read back every step"}
        del dev_in, dev_out, host_out

    hbm, tflops, peak_src = peaks()
    lengths = inp["lengths"]
    kern = {}
    for k, (ms, n) in per_kernel.items():
        byts = kernel_bytes(w, lengths, k)
        launch_ms = ms / n
        kern[k] = {"launch_ms": launch_ms, "launches_per_step": n, "share": ms / max(1e-12, sum(
            v[0] for v in per_kernel.values())), "algorithmic_bytes": byts,
            "frac": (byts / (launch_ms * 1e-3) / 1e9 / hbm) if byts else 0.0}
    roof = None
    if dominant and dom_n:
        byts = kernel_bytes(w, lengths, dominant)
        dur = dom_ms / dom_n * 1e-3
        achieved = byts / dur / 1e9 if byts else None
        traffic, traffic_src = measured_traffic(dominant, w.name) if args.seq_len <= 0 else (None, None)
        roof = {"bound": "hbm", "kernel": dominant, "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": (achieved / hbm) if achieved else None, "traffic": traffic, "traffic_source": traffic_src,
                "peak_source": peak_src, "algorithmic_bytes": byts, "launch_ms": dom_ms / dom_n, "launches": dom_n,
                "of": f"{peak_src} HBM copy bandwidth"}
    sb, sf = step_bytes(w, lengths), step_flops(w, lengths)
    t_roof = max(sb / (hbm * 1e9), sf / (tflops * 1e12))
    out = {"workload": workload_label(w, ch_rms_target), "value": job_throughput(w.tokens, world, ms_step),
           "ms_per_step": ms_step, "fwd": {"value": job_throughput(w.tokens, world, fwd_ms), "unit": "tokens/s",
                                           "ms_per_step": fwd_ms},
           "step_roofline": {"bytes": sb, "tensor_flops": sf, "time_ms": t_roof * 1e3, "frac": t_roof * 1e3 / ms_step,
                             "bound": "hbm" if sb / (hbm * 1e9) >= sf / (tflops * 1e12) else "tensor"},
           "roofline": roof, "kernels": kern, "e2e": e2e, "gpu_launches": int(launches), "clocks": clk,
           "steps": steps}
    del lu, devt, O, grads, flush
    torch.cuda.empty_cache()
    return out


def run_gpu(args, w):
    import torch
    import torch.distributed as tdist

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    from paper_2512_08061_gb300 import build
    if rank == 0 or world == 1:
        build.build()
    if world > 1:
        tdist.barrier()

    dev = torch.device("cuda", local_rank)
    head = measure_workload(args, w, dev, world, args.steps, args.ch_rms_target, not args.no_e2e)
    # the other long-sequence workload (LRA-shaped, non-causal), measured in the same run and reported under
    # its own key
    also = {}
    for name in args.also:
        if name and name != w.name:
            w2 = WORKLOADS[name]
            also[name] = measure_workload(args, w2, dev, world, max(3, min(args.steps, 50)), 0.0, not args.no_e2e)
    result = {
        "metric": METRIC,
        "value": head["value"],
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": head["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": w.io,
        "data": "synthetic",
        "config": {"workload": head["workload"], "global_batch": w.B * world, "seq_len": w.n,
                   "parallelism": f"replicas{world}",
                   "l2": "flushed before every timed step (2x L2 buffer written outside the events)"},
        "fwd": head["fwd"],
        "step_roofline": head["step_roofline"],
        "roofline": head["roofline"],
        "kernels": head["kernels"],
        "per_kernel_ms": {k: v["launch_ms"] for k, v in head["kernels"].items()},
        "e2e": head["e2e"],
        "gpu_launches": head["gpu_launches"],
        "clocks": head["clocks"],
    }
    for name, m in also.items():
        result[name] = {k: m[k] for k in ("workload", "value", "ms_per_step", "fwd", "step_roofline", "roofline",
                                          "kernels", "e2e", "gpu_launches", "clocks", "steps")}
        result[name]["unit"] = "tokens/s"
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds, args.ch_rms_target)
    if world > 1:
        tdist.destroy_process_group()
    return result if rank == 0 else None


# --------------------------------------------------------------------------
# the CPU oracle (reported baseline, and the --impl reference arm)

def sample_rows(w) -> int:
    """Rows per (batch, head) unit that one oracle sample takes: the whole sequence for the non-causal
    workloads (every query reads every key), the first 4096 tokens of each sequence for the streaming form,
    whose cost per token is the same at every position (a prefix of a causal sequence is its own causal
    problem)."""
    return min(w.n, 4096) if w.causal else w.n


def oracle_run(w, units: int, ch_rms_target: float = 0.0, rows: int | None = None) -> float:
    """Runs the fp64 oracle (fwd, and bwd for training workloads) on the first `units` (batch, head) units of
    the workload's own input streams, on their first `rows` tokens (default: all); returns the wall time in
    seconds."""
    import oracle
    n = w.n if rows is None else rows
    ln = None
    if w.len_range is not None:
        ln = synth.randint(w.seed, "attn.lengths", (w.B,), w.len_range[0], w.len_range[1]).astype(np.int32)
    # the first `units` heads of (B, H, n, d) in flat order, their first n tokens drawn directly
    def draw(name, width, scale):
        idx = ((np.arange(units)[:, None, None] * w.n + np.arange(n)[None, :, None]) * width
               + np.arange(width)[None, None, :]).ravel()
        x = synth.normal_at(w.seed, name, idx).reshape(units, 1, n, width) * scale
        return np.ascontiguousarray(synth.IOTensor(x, w.io).value)

    Q, K = draw("attn.Q", w.d, w.qkv_scale), draw("attn.K", w.d, w.qkv_scale)
    V = draw("attn.V", w.dv, w.qkv_scale)
    dO = draw("attn.dO", w.dv, 1.0) if w.backward else None
    lengths = None if ln is None else np.array([min(n, ln[(u // w.H) % w.B]) for u in range(units)], dtype=np.int32)
    p = oracle.PhiParams(synth.phi_params(w.seed, w.d, w.M, w.L, w.hidden), ch_rms_target)
    t0 = time.perf_counter()
    oracle.attn_fwd(p, Q, K, V, lengths, w.causal, w.eps)
    if w.backward:
        oracle.attn_bwd(p, Q, K, V, dO, lengths, w.causal, w.eps)
    return time.perf_counter() - t0


def tokens_per_s(w, units, seconds, rows=None) -> float:
    """Tokens per second of a sample of `units` (batch, head) units of `rows` tokens each: one token of the
    workload is one position of one sequence over all H heads."""
    rows = w.n if rows is None else rows
    return units * rows / (w.H * seconds)


def cpu_baseline(w, target_s, ch_rms_target=0.0):
    import oracle
    threads = oracle.max_threads()
    rows = sample_rows(w)
    t1 = oracle_run(w, threads, ch_rms_target, rows)
    units = int(min(max(threads, threads * round(target_s / max(t1, 1e-3))), 4 * w.B * w.H))
    t = oracle_run(w, units, ch_rms_target, rows) if units != threads else t1
    return {"value": tokens_per_s(w, units, t, rows), "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": f"{units} (batch, head) units of {rows} tokens"
                      + (f" (the first {rows} of each {w.n}-token sequence)" if rows < w.n else "")
                      + f", fwd{'+bwd' if w.backward else ''}, {t:.1f} s on {threads} threads; tokens/s scaled "
                        f"from the sample (value = units * rows / H / seconds)"}


def run_reference(args, w):
    rank, _, world = dist_env()
    if rank != 0:
        return None
    import oracle
    threads = oracle.max_threads()
    rows = sample_rows(w)
    if args.warmup > 0:
        oracle_run(w, 1, args.ch_rms_target, min(rows, 256))
    per, secs = [], []
    for _ in range(args.steps):
        t = oracle_run(w, threads, args.ch_rms_target, rows)
        secs.append(t)
        per.append(tokens_per_s(w, threads, t, rows))
    value = statistics.median(per)
    sample = (f"{threads} (batch, head) units of {rows} tokens per step"
              + (f" (the first {rows} of each {w.n}-token sequence)" if rows < w.n else "")
              + f" on {threads} threads, {statistics.median(secs):.2f} s each")
    return {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": w.tokens / value * 1e3, "higher_is_better": True,
            "ms_per_step_kind": "extrapolated: the time the oracle would take for one whole step (B*H units of "
                                "n tokens) at the sample's rate; each timed step ran the sample only",
            "sample_seconds_per_step": statistics.median(secs),
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": workload_label(w, args.ch_rms_target) + ", fp64 CPU oracle",
                       "global_batch": w.B, "seq_len": w.n, "parallelism": "cpu"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


DECODE_METRIC = "LUNA decode tokens/sec (one token per sequence per step) on 1 GB300; % of HBM roofline"


def decode_oracle_run(w, units: int) -> float:
    """One decode step of the first `units` (batch, head) units by the fp64 oracle as it stands: it keeps
    no state between calls, so each unit's output for the new token is its causal output at position
    n + 1, recomputed over the prefill and the token.  Returns the wall time in seconds."""
    import oracle
    tensors = {}
    for name, tok, width in (("Q", "q", w.d), ("K", "k", w.d), ("V", "v", w.dv)):
        pre = synth.normal(w.seed, f"attn.{name}", (units, 1, w.n, width)) * w.qkv_scale
        new = synth.normal(w.seed, f"decode.{tok}", (units, 1, 1, width)) * w.qkv_scale
        tensors[name] = synth.IOTensor(np.concatenate([pre, new], axis=2), w.io).value
    p = oracle.PhiParams(synth.phi_params(w.seed, w.d, w.M, w.L, w.hidden))
    t0 = time.perf_counter()
    oracle.attn_fwd(p, tensors["Q"], tensors["K"], tensors["V"], None, True, w.eps)
    return time.perf_counter() - t0


def decode_tokens_per_s(w, units, seconds) -> float:
    # one step = one token for each of the B sequences = B*H units
    return units / (w.H * seconds)


def decode_cpu_baseline(w, target_s):
    import oracle
    threads = oracle.max_threads()
    t1 = decode_oracle_run(w, threads)
    units = int(min(max(threads, threads * round(target_s / max(t1, 1e-3))), w.B * w.H))
    t = decode_oracle_run(w, units) if units != threads else t1
    return {"value": decode_tokens_per_s(w, units, t), "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": f"{units} (batch, head) units, each recomputing its causal output over the {w.n}-token "
                      f"prefill and the new token (the oracle keeps no state), {t:.1f} s on {threads} threads, "
                      f"scaled to B*H={w.B * w.H} units per step"}


def run_reference_decode(args, w):
    rank, _, world = dist_env()
    if rank != 0:
        return None
    import oracle
    threads = oracle.max_threads()
    if args.warmup > 0:
        decode_oracle_run(w, 1)
    per = [decode_tokens_per_s(w, threads, decode_oracle_run(w, threads)) for _ in range(args.steps)]
    value = statistics.median(per)
    sample = (f"{threads} (batch, head) units per step on {threads} threads, each recomputing its causal output "
              f"over the {w.n}-token prefill and the new token")
    return {"metric": DECODE_METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": w.B / value * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": f"{w.name}: B={w.B} H={w.H}, one token per sequence per step after a causal "
                                   f"prefill of n={w.n}, d={w.d} D={w.D}, fp64 CPU oracle",
                       "global_batch": w.B, "seq_len": w.n, "parallelism": "cpu"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def decode_bytes(w) -> float:
    """Bytes of one decode step: every fp32 state element read and written once, and the
    token's q, k, v read and o written."""
    eb = 4 if w.io == "f32" else 2
    return float(w.B * w.H * (2 * (w.D * w.dv + w.D) * 4 + (2 * w.d + 2 * w.dv) * eb))


def run_decode(args, w):
    """Streaming inference: a causal prefill of w.n tokens saves the state, then every step
    advances all B x H heads by one token through luna_attn_decode (state updated in place)."""
    import torch
    import torch.distributed as tdist

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    from paper_2512_08061_gb300 import build
    if rank == 0 or world == 1:
        build.build()
    if world > 1:
        tdist.barrier()
    import paper_2512_08061_gb300.luna as L

    dev = torch.device("cuda", local_rank)
    io_dtype = torch.float32 if w.io == "f32" else torch.bfloat16
    inp, params = host_inputs(w)

    def pinned(t):
        if t.io == "f32":
            return torch.from_numpy(np.ascontiguousarray(t.raw)).pin_memory()
        return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).view(torch.bfloat16).pin_memory()

    pre = {k: pinned(inp[k]).to(dev) for k in ("Q", "K", "V")}
    lu = L.Luna(w.B, w.H, w.n, w.d, w.dv, w.M, w.L, w.hidden, True, w.eps, io_dtype, w.chunk, dev)
    lu.prepare({k: torch.from_numpy(v).to(dev) for k, v in params.items()})
    lu.forward(pre["Q"], pre["K"], pre["V"], None, save_state=True)
    host = {k: pinned(synth.IOTensor(synth.normal(w.seed, f"decode.{k}", (w.B, w.H, n)) * w.qkv_scale, w.io))
            for k, n in (("q", w.d), ("k", w.d), ("v", w.dv))}
    tok = {k: v.to(dev) for k, v in host.items()}
    o = torch.empty(w.B, w.H, w.dv, dtype=io_dtype, device=dev)
    S, Ss, z, zs = L.luna_state_final(lu.ad, lu.pd, lu.state)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(t):
        L.luna_attn_decode(lu.ad, lu.pd, lu.table, t["q"], t["k"], t["v"], o, S, Ss, z, zs)

    def timed(n_steps, fn):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_steps)]
        for s0, s1 in evs:
            flush.zero_()
            s0.record(stream)
            fn()
            s1.record(stream)
        torch.cuda.synchronize()
        return sum(s0.elapsed_time(s1) for s0, s1 in evs)

    for _ in range(max(args.warmup, 3)):
        step(tok)
    torch.cuda.synchronize()
    if world > 1:
        tdist.barrier()
    uuid = str(getattr(torch.cuda.get_device_properties(local_rank), "uuid", "") or "")
    clocks = ClockSampler(("GPU-" + uuid if uuid and not uuid.startswith("GPU-") else uuid) or str(local_rank))
    L.luna_profile_start("decode")
    n0 = L.luna_launch_count()
    ms_step = timed(args.steps, lambda: step(tok)) / args.steps
    launches = L.luna_launch_count() - n0
    dom_ms, dom_n = L.luna_profile_stop()
    clk = clocks.stop()
    ms_step = max_over_ranks(ms_step, dev, world)
    e2e = None
    if not args.no_e2e:
        o_host = torch.empty(o.shape, dtype=o.dtype).pin_memory()

        def e2e_step():
            step({k: v.to(dev, non_blocking=True) for k, v in host.items()})
            o_host.copy_(o, non_blocking=True)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        e2e_ms = timed(max(3, args.steps // 4), e2e_step) / max(3, args.steps // 4)
        e2e_ms = max_over_ranks(e2e_ms, dev, world)
        e2e = {"value": job_throughput(w.B, world, e2e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": int(sum(v.numel() * v.element_size() for v in host.values())),
               "d2h_bytes_per_step": int(o_host.numel() * o_host.element_size()), "ms_per_step": e2e_ms}
    hbm, _, peak_src = peaks()
    byts = decode_bytes(w)
    roof = None
    if dom_n:
        achieved = byts / (dom_ms / dom_n * 1e-3) / 1e9
        traffic, traffic_src = measured_traffic("decode", w.name) if args.seq_len <= 0 else (None, None)
        roof = {"bound": "hbm", "kernel": "decode", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "traffic": traffic, "traffic_source": traffic_src, "peak_source": peak_src,
                "algorithmic_bytes": byts, "launch_ms": dom_ms / dom_n, "launches": dom_n}
    result = {
        "metric": DECODE_METRIC, "value": job_throughput(w.B, world, ms_step), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.io, "data": "synthetic",
        "config": {"workload": f"{w.name}: B={w.B} H={w.H}, one token per sequence per step after a causal "
                               f"prefill of n={w.n}, d={w.d} D={w.D} (M={w.M}, L={w.L}), {w.io}, fp32 state",
                   "global_batch": w.B * world, "seq_len": w.n, "parallelism": f"replicas{world}",
                   "l2": "flushed before every timed step (2x L2 buffer written outside the events)"},
        "step_roofline": {"bytes": byts, "time_ms": byts / (hbm * 1e9) * 1e3,
                          "frac": byts / (hbm * 1e9) * 1e3 / ms_step},
        "roofline": roof, "per_kernel_ms": {"decode": dom_ms / dom_n if dom_n else None},
        "e2e": e2e, "gpu_launches": int(launches), "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = decode_cpu_baseline(w, args.cpu_seconds)
    if world > 1:
        tdist.destroy_process_group()
    return result if rank == 0 else None


def main():
    args = parse()
    w = WORKLOADS[args.workload]
    if args.seq_len > 0:
        n = args.seq_len
        w = dataclasses.replace(w, n=n, len_range=None if w.len_range is None else
                                (min(w.len_range[0], n), min(w.len_range[1], n)))
    if w.decode:
        res = run_reference_decode(args, w) if args.impl == "reference" else run_decode(args, w)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    res = run_reference(args, w) if args.impl == "reference" else run_gpu(args, w)
    if res is not None:
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
