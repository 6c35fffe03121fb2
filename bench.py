"""Benchmark of the packed ternary linear layer on GB300.

Default workload: one Qwen3-8B decode step, linear layers only, batch M = 1
(36 layers x {q, k, v, o, gate, up, down} = 252 packed projections, 10 % of
groups salient), seeded synthetic weights and activations resident in HBM.
One step = one pass over all 252 projections (tq_linear_batched: one kernel
launch).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl tq|reference]
  python bench.py --prefill      (one Qwen3-8B layer at M = 2048 tokens)
  python bench.py --ternarize    (E2M-ATQ ternarization of one Qwen3-8B layer)

--impl reference times the CPU oracle on the host cores (the reference arm
of this project: a plain fp64 implementation of the same layer) on a
bounded sample of the same workload.  --prefill measures the prefill tile
path (tensor-core bound) and times dense fp16 cuBLAS on the same shapes as
context.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Qwen3-8B W1.58A16 GEMV: packed GB/s vs HBM peak; linear-layer tokens/s"
HBM_FALLBACK_GBS = 6800.0


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return HBM_FALLBACK_GBS, "fallback"


def measured_tensor_peak():
    """fp16 dense tensor peak (TFLOP/s): the measured sustained bf16 cuBLAS
    rate (fp16 and bf16 share the nominal rate), else the fallback."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured sustained bf16 (= fp16 rate)"
    return 1700.0, "fallback sustained"


def max_over_ranks(value: float, pg, device) -> float:
    """The largest of every rank's value (the job's time is its slowest
    rank's); the value itself without a process group."""
    if pg is None:
        return float(value)
    import torch

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, ms: float, scale: float = 1e9) -> float:
    """Units all ranks processed per second (divided by `scale`), over the
    slowest rank's time `ms`: each of `world` replicas does the same work."""
    return world * units_per_rank / (ms * 1e-3) / scale


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi sampling (every 20 ms) of SM clocks and throttle reasons.
    Enter it before the warm-up, call ready() before the timed region, and
    mark() its start and end: summary() then counts the samples read during
    the timed region (and, when the region is shorter than the interval,
    the samples of the whole sampled span, saying so)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []  # (host time read, line)
        self.marks = []

    def __enter__(self):
        try:
            # a pseudo-terminal as stdout, so that nvidia-smi writes each sample
            # as it takes it (into a pipe it would buffer them until exit)
            import pty

            self.master, slave = pty.openpty()
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=slave, stderr=subprocess.DEVNULL, close_fds=True)
            os.close(slave)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        buf = b""
        while True:
            try:
                chunk = os.read(self.master, 4096)
            except OSError:
                break
            if not chunk:
                break
            buf += chunk
            *full, buf = buf.split(b"\n")
            now = time.perf_counter()
            for ln in full:
                self.lines.append((now, ln.decode(errors="replace").strip()))

    def ready(self, timeout=5.0):
        """Wait (bounded) until the first sample has arrived."""
        t = time.perf_counter()
        while self.proc and not self.lines and time.perf_counter() - t < timeout:
            time.sleep(0.005)

    def mark(self):
        self.marks.append(time.perf_counter())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.t.join(timeout=2)
            try:
                os.close(self.master)
            except OSError:
                pass

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        lines = [ln for _, ln in self.lines]
        window = "whole sampled span"
        if len(self.marks) >= 2:
            # a sample is read within a few ms of being taken
            inside = [ln for t, ln in self.lines if self.marks[0] <= t <= self.marks[-1] + 0.01]
            if inside:
                lines, window = inside, "timed region"
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm),
                "window": window}


# ---------------------------------------------------------------- workload
def build_step(M, device, seed0=0, layers=None, on_codes=None):
    """Pack the 252 projections of the Qwen3-8B step on the device.  Every
    projection's activations and outputs are views of one contiguous x / y
    buffer (so a step's inputs move host<->device in one copy each).
    on_codes(projection, drawn tensors, packed weight), if given, sees each
    projection's drawn codes and parameters before they are freed (the
    full-size parity test packs them again with the oracle).
    Returns (items, x_all, y_all, packed_bytes, weights)."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    projs = wl.config_projections(2)
    if layers is not None:
        projs = [p for p in projs if p.layer < layers]
    x_all = torch.empty(sum(M * p.K for p in projs), dtype=torch.float16, device=device)
    y_all = torch.empty(sum(M * p.N for p in projs), dtype=torch.float16, device=device)
    items, total_bytes, total_w, xo, yo = [], 0, 0, 0, 0
    for p in projs:
        seed = seed0 * 100003 + p.layer * 16 + p.proj
        g = wl.gen_weights_torch(p.N, p.K, 0.1, device, seed)
        pw = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"] if g["nnz"] else None)
        if on_codes is not None:
            on_codes(p, g, pw)
        del g
        x = x_all[xo:xo + M * p.K].view(M, p.K)
        x.copy_(wl.gen_x_torch(M, p.K, device, seed + 7))
        y = y_all[yo:yo + M * p.N].view(M, p.N)
        xo += M * p.K
        yo += M * p.N
        items.append((pw, x, y))
        total_bytes += pw.packed_bytes()
        total_w += p.N * p.K
    torch.cuda.synchronize()
    return items, x_all, y_all, total_bytes, total_w


# the sources the decode-step kernels are compiled from
DECODE_SOURCES = ("tq_common.cuh", "tq_decode_ops.cuh", "tq_gemv_g4.cu", "tq_gemv_mma.cu", "tq_p2_tile.cuh", "tq_sm100.cuh")


def kernel_hash():
    """sha256 (16 hex digits) of the decode kernels' sources without their
    // comments and blank lines, so that a comment edit keeps the counters"""
    import hashlib

    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_09240_gb300", "csrc")
    for f in DECODE_SOURCES:
        for line in open(os.path.join(csrc, f), encoding="utf-8"):
            code = line.split("//", 1)[0].rstrip()
            if code:
                h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def ncu_traffic():
    """dram bytes per launch of the decode kernel from the committed ncu
    summary, or None if the kernel changed since it was captured."""
    p = os.path.join(ROOT, "profiles", "gemv_qwen3_8b_step_traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    if d.get("kernel_hash") != kernel_hash():
        return None
    return d.get("dram_bytes_per_launch")


# ------------------------------------------------------------ cpu baseline
class OracleLayer:
    """Layer 0 of the Qwen3-8B step (its seven projections, every row, M=1,
    10 % salient groups), drawn with numpy and packed by the oracle, so that
    the CPU oracle can be timed on a bounded sample of the same workload."""

    def __init__(self):
        import oracle
        import workloads as wl

        oracle.build()
        self.oracle = oracle
        self.projs = []
        for p in wl.config_projections(4):  # the seven shapes of one Qwen3-8B layer
            w = wl.gen_weights(p.N, p.K, 0.1, config=2, layer=0, proj=p.proj)
            x = wl.gen_x(1, p.K, config=2, layer=0, proj=p.proj)
            rp, _ = oracle.rowptr(p.N, p.K, w.sal)
            p1, p2, _ = oracle.pack(p.N, p.K, w.T1, w.T2, w.sal, rp)
            G = p.K // 128
            # packed bytes a row owns: plane 1, s1 + off, salience words,
            # its rowptr entry, its plane-2 records and their s2
            row_fixed = oracle.row_bytes(p.K) + 4 * G + 4 * oracle.sal_words(p.K) + 4
            row_bytes = row_fixed + 28 * np.diff(rp.astype(np.int64))
            self.projs.append(dict(N=p.N, K=p.K, p1=p1, p2=p2, sal=w.sal, s1=w.s1, off=w.off, s2=w.s2, x=x,
                                   cum=np.concatenate([[0], np.cumsum(row_bytes)])))
            del w
        self.cores = os.cpu_count() or 1

    def run(self, frac=1.0, nthreads=None):
        """One oracle pass over the first `frac` of every projection's rows;
        returns (packed bytes covered, seconds)."""
        nbytes, t = 0, 0.0
        for d in self.projs:
            R = max(1, int(round(d["N"] * frac)))
            rows = None if R >= d["N"] else np.arange(R, dtype=np.int32)
            t0 = time.perf_counter()
            self.oracle.linear(1, d["N"], d["K"], d["p1"], d["p2"], d["sal"], d["s1"], d["off"], d["s2"], d["x"],
                               rows=rows, nthreads=nthreads or self.cores)
            t += time.perf_counter() - t0
            nbytes += int(d["cum"][min(R, d["N"])])
        return nbytes, t


def cpu_baseline(budget_s):
    """Whole passes of the oracle over layer 0 until `budget_s` seconds of
    CPU work have been timed."""
    L = OracleLayer()
    nbytes, t, passes = 0, 0.0, 0
    while t < budget_s and passes < 1000:
        b, dt = L.run()
        nbytes += b
        t += dt
        passes += 1
    desc = (f"{passes} full passes over layer 0 of the Qwen3-8B step (q, k, v, o, gate, up, down: every row, "
            f"M=1, 10% salient), {nbytes / 1e9:.2f} GB of packed bytes in {t:.1f} s")
    return nbytes / t / 1e9, L.cores, desc, t


# ------------------------------------------------------------------- prefill
def run_prefill(args, ws, rank, local):
    """One Qwen3-8B layer (its seven projections) at M = 2048 tokens through
    the prefill tile path, one tq_linear_batched call per layer (every
    projection's tiles in one launch); dense fp16 cuBLAS on the same shapes
    is timed beside it as context."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    M = 2048
    items, flops, packed = [], 0, 0
    for p in wl.config_projections(4):
        g = wl.gen_weights_torch(p.N, p.K, 0.1, dev, 500 + p.proj)
        pw = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"] if g["nnz"] else None)
        del g
        x = wl.gen_x_torch(M, p.K, dev, 600 + p.proj)
        y = torch.empty((M, p.N), dtype=torch.float16, device=dev)
        wsb = tq.workspace(tq.tq_workspace_bytes(M, p.N, p.K), dev)
        items.append((pw, x, y, wsb))
        flops += 2 * M * p.N * p.K
        packed += pw.packed_bytes()
    stream = torch.cuda.current_stream()
    batch = tq.Batch(M, [(pw, x, y) for pw, x, y, _ in items])

    def step():
        tq.tq_linear_batched(batch, stream=stream)

    steps = max(1, min(args.steps, 100))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        clk.ready()
        for _ in range(max(args.warmup, 3)):
            step()
        torch.cuda.synchronize()
        clk.mark()
        e0.record(stream)
        for _ in range(steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        clk.mark()
    ms = e0.elapsed_time(e1) / steps
    # context: dense fp16 matmul (cuBLAS) with a dense W of the same shapes
    dense = [torch.randn((pw.N, pw.K), device=dev, dtype=torch.float16) for pw, _, _, _ in items]

    def dstep():
        for (pw, x, y, _), W in zip(items, dense):
            torch.matmul(x, W.t(), out=y)

    for _ in range(3):
        dstep()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(steps):
        dstep()
    e1.record(stream)
    torch.cuda.synchronize()
    ms_dense = e0.elapsed_time(e1) / steps
    peak, kind = measured_tensor_peak()
    tflops = flops / (ms * 1e-3) / 1e12
    out = {
        "metric": "Qwen3-8B W1.58A16 prefill: TFLOP/s of one layer at M=2048", "value": tflops,
        "unit": "TFLOP/s", "n_gpus": 1, "steps": steps, "warmup": max(args.warmup, 3), "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": "qwen3-8b prefill, one layer's 7 projections, M=2048 tokens",
                   "flops_per_step": flops, "packed_bytes_per_step": packed,
                   "l2": "no flush: 2048-token activations and outputs of a layer exceed L2 per step"},
        "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s", "frac": tflops / peak,
                     "peak_kind": kind, "traffic": None,
                     "kernel": "prefill tile kernel (one launch per step: every projection's tiles)"},
        "dense_fp16_cublas": {"ms_per_step": ms_dense, "tflops": flops / (ms_dense * 1e-3) / 1e12},
        "gpu_launches": steps,
        "clocks": clk.summary(),
    }
    if rank == 0:
        print(json.dumps(out), flush=True)
    return 0


# ----------------------------------------------------------------- ternarize
# fp32 operations per weight that the computation needs (a product with a
# trit counts as one; the refinement sweeps are scalar work per block):
#   statistics 15 (mean 1, mean |c| 3, support 3, first scale 3, energy 5);
#   planes 5 for a block without second plane (support 3, moments 2), 16 for
#   a salient block (support and moments 5, residual mean 5, second support
#   and its moment 6).
TERN_OPS_STATS, TERN_OPS_PLAIN, TERN_OPS_SALIENT = 15, 5, 16
# fp32 lanes per SM on sm_100-class parts; the ALU peak for single fp32
# operations is lanes x the device's SM count x its maximum SM clock
FP32_LANES_PER_SM = 128


def alu_peak_tops(dev, sm_max_mhz=None):
    """Single-fp32-operation peak of `dev` in Top/s: lanes x SMs x maximum clock.

    The SM count is the device's own; the clock is the maximum that the clock
    sampler read during the run, else 2070 MHz (the part's maximum SM clock).
    """
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    mhz = sm_max_mhz if sm_max_mhz else 2070.0
    return FP32_LANES_PER_SM * sms * mhz * 1e6 / 1e12, sms, mhz


def run_ternarize(args, ws, rank, local):
    """E2M-ATQ ternarization (tq_ternarize) of one Qwen3-8B layer: its seven
    dense fp16 projections (seeded synthetic weights resident in HBM) into
    packed weights with 10 % salient groups and 4 refinement sweeps."""
    import ctypes

    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    L = tq.lib()
    stream = torch.cuda.current_stream()
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    sweeps, frac = 4, 0.1
    jobs, n_weights, ops = [], 0, 0.0
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    for i, (nm, N, K) in enumerate(wl.QWEN3_8B):
        W = wl.gen_dense_weights_torch(N, K, dev, seed=700 + i)
        G = K // 128
        nnz = int(round(frac * N * G))
        out = dict(plane1=torch.empty((N, tq.tq_row_bytes(K)), dtype=torch.uint8, device=dev),
                   sal=torch.empty((N, tq.tq_sal_words(K)), dtype=torch.int32, device=dev),
                   rowptr=torch.empty(N + 1, dtype=torch.int32, device=dev),
                   plane2=torch.empty((nnz, 26), dtype=torch.uint8, device=dev),
                   s1=torch.empty((N, G), dtype=torch.float16, device=dev),
                   off=torch.empty((N, G), dtype=torch.float16, device=dev),
                   s2=torch.empty(nnz, dtype=torch.float16, device=dev))
        wsb = tq.workspace(tq.tq_ternarize_workspace_bytes(N, K), dev)
        jobs.append((N, K, nnz, W, out, wsb))
        n_weights += N * K
        ops += N * K * (TERN_OPS_STATS + (1 - nnz / (N * G)) * TERN_OPS_PLAIN + nnz / (N * G) * TERN_OPS_SALIENT)

    def call(N, K, nnz, W, o, wsb):
        rc = L.tq_ternarize(N, K, P(W), nnz, sweeps, P(o["plane1"]), P(o["sal"]), P(o["rowptr"]), P(o["plane2"]),
                            P(o["s1"]), P(o["off"]), P(o["s2"]), P(wsb), wsb.numel(), P(st),
                            ctypes.c_void_p(stream.cuda_stream))
        assert rc == 0, rc

    def step():
        for j in jobs:
            call(*j)

    steps = max(1, min(args.steps, 50))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        clk.ready()
        for _ in range(max(args.warmup, 3)):
            step()
        torch.cuda.synchronize()
        clk.mark()
        e0.record(stream)
        for _ in range(steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        clk.mark()
    ms = e0.elapsed_time(e1) / steps
    assert int(st.item()) == 0
    # end to end: fp16 weights from pinned host memory, packed outputs back to pinned host memory
    hostW = [j[3].cpu().pin_memory() for j in jobs]
    hostO = [{k: v.cpu().pin_memory() for k, v in j[4].items()} for j in jobs]
    h2d = sum(h.numel() * 2 for h in hostW)
    d2h = sum(v.numel() * v.element_size() for o in hostO for v in o.values())

    def e2e_step():
        for (N, K, nnz, W, o, wsb), hw, ho in zip(jobs, hostW, hostO):
            W.copy_(hw, non_blocking=True)
            call(N, K, nnz, W, o, wsb)
            for k, v in o.items():
                ho[k].copy_(v, non_blocking=True)

    e2e_step()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / steps
    achieved = ops / (ms * 1e-3) / 1e12
    clocks = clk.summary()
    peak, sms, mhz = alu_peak_tops(torch.cuda.current_device(), clocks.get("sm_max_mhz"))
    out = {
        "metric": "Qwen3-8B E2M-ATQ ternarization into the packed format: weights/s", "value": n_weights / (ms * 1e-3) / 1e9,
        "unit": "Gweights/s", "n_gpus": 1, "steps": steps, "warmup": max(args.warmup, 3), "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "E2M-ATQ of one Qwen3-8B layer's 7 projections (fp16 in, packed out), "
                               "10% salient groups, 4 sweeps", "weights_per_step": n_weights,
                   "l2": "no flush: a layer's 386 MB of fp16 weights exceed L2 per step"},
        "roofline": {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "Top/s",
                     "frac": achieved / peak, "traffic": None,
                     "peak_kind": f"{FP32_LANES_PER_SM} fp32 lanes x {sms} SMs x {mhz:.0f} MHz (derived, not measured)",
                     "kernel": "whole tq_ternarize call (nine launches per projection, 63 per step)",
                     "ops_per_step": ops},
        "e2e": {"value": n_weights / (e2e_ms * 1e-3) / 1e9, "unit": "Gweights/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": 9 * 7 * steps,
        "clocks": clocks,
    }
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = ternarize_cpu_baseline(10.0)
    if rank == 0:
        print(json.dumps(out), flush=True)
    return 0


def ternarize_cpu_baseline(budget_s):
    """The oracle (numpy float32) on whole projections of the same layer, in
    order, until `budget_s` seconds have been timed."""
    import workloads as wl
    from oracle import ternarize as tz

    n, t, names = 0, 0.0, []
    for i, (nm, N, K) in enumerate(wl.QWEN3_8B):
        if t >= budget_s:
            break
        W = wl.gen_dense_weights(N, K, config=9, proj=700 + i)
        t0 = time.perf_counter()
        tz.ternarize(W, int(round(0.1 * N * K / 128)), sweeps=4)
        t += time.perf_counter() - t0
        n += N * K
        names.append(nm)
    return {"value": n / t / 1e9, "unit": "Gweights/s", "cores": 1, "kind": "oracle",
            "sample": f"the oracle on whole projections {', '.join(names)} of one Qwen3-8B layer "
                      f"({n / 1e6:.1f} M weights, {t:.1f} s, numpy on one core)"}


# ------------------------------------------------- the other configurations
L2_BYTES = 129 * 2 ** 20


def graph_ms(fn, reps, warmup=2):
    """Device time per replay of a CUDA graph that captured fn() (the calls
    go to the current stream, which is the capture stream while capturing):
    launch gaps of the host loop are not part of the number."""
    import torch

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(warmup):
            fn()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fn()
    for _ in range(warmup):
        graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def _clone_weight(pw):
    from paper_2609_09240_gb300 import tq

    c = lambda t: None if t is None else t.clone()
    return tq.PackedWeight(pw.N, pw.K, c(pw.plane1), c(pw.salience), c(pw.rowptr), c(pw.plane2), c(pw.scale1),
                           c(pw.offset), c(pw.scale2), pw.nnz, c(pw.p2index))


def sub_config0(dev, peak):
    """Config 0: one 512 x 1024 ternary linear at M = 1 (no second plane),
    one tq_linear call at a time over rotated copies whose bytes total more
    than 4 x L2, so that every call reads its weight from HBM."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    N, K, M = 512, 1024, 1
    g = wl.gen_weights_torch(N, K, 0.0, dev, 11)
    pw0 = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], None)
    ws_bytes = tq.tq_workspace_bytes(M, N, K)
    per = pw0.packed_bytes() + ws_bytes + 2 * (K + N)
    R = -(-4 * L2_BYTES // per)
    copies = [(_clone_weight(pw0), wl.gen_x_torch(M, K, dev, 100 + r), torch.empty((M, N), dtype=torch.float16,
                                                                              device=dev),
               tq.workspace(ws_bytes, dev)) for r in range(R)]

    def calls():
        for pw, x, y, wsb in copies:
            tq.tq_linear(x, pw, y=y, ws=wsb)

    ms = graph_ms(calls, reps=5) / R
    gbs = pw0.packed_bytes() / (ms * 1e-3) / 1e9
    return {"workload": "single ternary linear 512 x 1024, M=1, no second plane (config 0)",
            "us_per_call": ms * 1e3, "packed_bytes": pw0.packed_bytes(), "packed_gbs": gbs, "frac_of_hbm_peak": gbs / peak,
            "tokens_per_s": 1.0 / (ms * 1e-3),
            "timing": f"{R} rotated copies of weight, x, y and workspace ({R * per / 2 ** 20:.0f} MiB > 4 x L2), "
                      "one tq_linear call each, replayed as one CUDA graph (2 launches per call)"}


def sub_config1(dev, peak):
    """Config 1: one Qwen3-4B decoder layer's seven projections at M = 1,
    10 % salient groups; a layer as one batched call and as seven tq_linear
    calls, over rotated copies of the layer (more than 4 x L2 in total)."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    M = 1
    base = []
    for p in wl.config_projections(1):
        g = wl.gen_weights_torch(p.N, p.K, 0.1, dev, 700 + p.proj)
        base.append(tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"] if g["nnz"] else None))
        del g
    layer_bytes = sum(pw.packed_bytes() for pw in base)
    R = -(-4 * L2_BYTES // layer_bytes)
    layers, batches = [], []
    for r in range(R):
        items = [(pw if r == 0 else _clone_weight(pw), wl.gen_x_torch(M, pw.K, dev, 800 + 8 * r + i),
                  torch.empty((M, pw.N), dtype=torch.float16, device=dev)) for i, pw in enumerate(base)]
        layers.append(items)
        batches.append(tq.Batch(M, items))
    wss = [tq.workspace(tq.tq_workspace_bytes(M, pw.N, pw.K), dev) for pw in base]

    def batched():
        for b in batches:
            tq.tq_linear_batched(b)

    def unbatched():
        for items in layers:
            for (pw, x, y), wsb in zip(items, wss):
                tq.tq_linear(x, pw, y=y, ws=wsb)

    ms_b = graph_ms(batched, reps=10) / R
    ms_u = graph_ms(unbatched, reps=10) / R
    gbs = layer_bytes / (ms_b * 1e-3) / 1e9
    return {"workload": "qwen3-4b one decoder layer (q, k, v, o, gate, up, down), M=1, 10% salient (config 1)",
            "us_per_layer": ms_b * 1e3, "packed_bytes": layer_bytes, "packed_gbs": gbs, "frac_of_hbm_peak": gbs / peak,
            "us_per_layer_unbatched": ms_u * 1e3,
            "timing": f"{R} rotated copies of the layer ({R * layer_bytes / 2 ** 20:.0f} MiB of packed weights > "
                      "4 x L2); one tq_linear_batched call per layer (3 launches), or seven tq_linear calls; "
                      "replayed as CUDA graphs"}


def sub_skinny(items, M, dev, peak, packed_bytes, steps):
    """Config 3: the Qwen3-8B step at M tokens (same packed weights as the
    M = 1 step, fresh activations)."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    its = [(pw, wl.gen_x_torch(M, pw.K, dev, 900 + i), torch.empty((M, pw.N), dtype=torch.float16, device=dev))
           for i, (pw, _, _) in enumerate(items)]
    batch = tq.Batch(M, its)
    stream = torch.cuda.current_stream()
    for _ in range(3):
        tq.tq_linear_batched(batch, stream)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        tq.tq_linear_batched(batch, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    gbs = packed_bytes / (ms * 1e-3) / 1e9
    return {"M": M, "ms_per_step": ms, "packed_gbs": gbs, "frac_of_hbm_peak": gbs / peak,
            "tokens_per_s": M / (ms * 1e-3), "steps": steps}


def sub_unbatched_8b(items, dev, batched_ms):
    """The Qwen3-8B step's projections called one tq_linear at a time (M = 1),
    every layer in turn (the step's 1.79 GB rotate through L2)."""
    from paper_2609_09240_gb300 import tq

    shapes = {}
    for pw, _, _ in items:
        shapes.setdefault((pw.N, pw.K), tq.workspace(tq.tq_workspace_bytes(1, pw.N, pw.K), pw.plane1.device))

    def calls():
        for pw, x, y in items:
            tq.tq_linear(x, pw, y=y, ws=shapes[(pw.N, pw.K)])

    ms = graph_ms(calls, reps=5)
    layers = len(items) // 7
    return {"workload": "qwen3-8b step, each projection its own tq_linear call, M=1",
            "us_per_layer": ms * 1e3 / layers, "us_per_layer_batched": batched_ms * 1e3 / layers,
            "ratio_to_batched": ms / batched_ms,
            "timing": f"{len(items)} tq_linear calls (3 launches each) replayed as one CUDA graph"}


def sub_prefill(dev, steps=20):
    """Config 4: one Qwen3-8B layer's seven projections at M = 2048 tokens
    (tensor-core tile path); dense fp16 cuBLAS on the same shapes beside it."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    M = 2048
    items, flops = [], 0
    for p in wl.config_projections(4):
        g = wl.gen_weights_torch(p.N, p.K, 0.1, dev, 500 + p.proj)
        pw = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"] if g["nnz"] else None)
        del g
        items.append((pw, wl.gen_x_torch(M, p.K, dev, 600 + p.proj), torch.empty((M, p.N), dtype=torch.float16,
                                                                                  device=dev),
                      tq.workspace(tq.tq_workspace_bytes(M, p.N, p.K), dev)))
        flops += 2 * M * p.N * p.K
    stream = torch.cuda.current_stream()
    batch = tq.Batch(M, [(pw, x, y) for pw, x, y, _ in items])

    def step():
        tq.tq_linear_batched(batch, stream=stream)

    def calls():
        for pw, x, y, wsb in items:
            tq.tq_linear(x, pw, y=y, ws=wsb, stream=stream)

    dense = [torch.randn((pw.N, pw.K), device=dev, dtype=torch.float16) for pw, _, _, _ in items]

    def dstep():
        for (pw, x, y, _), W in zip(items, dense):
            torch.matmul(x, W.t(), out=y)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps

    ms, ms_calls, ms_dense = timed(step), timed(calls), timed(dstep)
    peak, kind = measured_tensor_peak()
    tflops = flops / (ms * 1e-3) / 1e12
    return {"workload": "qwen3-8b prefill: one layer's 7 projections at M=2048 tokens (config 4), one "
                        "tq_linear_batched call",
            "ms_per_layer": ms, "ms_per_layer_seven_calls": ms_calls, "flops_per_layer": flops, "tflops": tflops,
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s", "frac": tflops / peak,
                         "peak_kind": kind},
            "dense_fp16_cublas": {"ms_per_layer": ms_dense, "tflops": flops / (ms_dense * 1e-3) / 1e12},
            "l2": "no flush: a layer's 2048-token activations and outputs (~234 MB) exceed L2",
            "gpu_launches_per_layer": 1, "steps": steps}


def sub_sequence(dev, peak, steps=30):
    """The dependency-ordered Qwen3-8B step (M = 1): per layer q/k/v fused
    (6144 x 4096), o, gate/up fused (24576 x 4096), down -- 144 problems run
    in order by tq_linear_sequence (one persistent launch, a grid barrier
    between problems) -- beside the same 144 problems as one independent
    tq_linear_batched call."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    fused = [("qkv", 6144, 4096), ("o", 4096, 4096), ("gate_up", 24576, 4096), ("down", 4096, 12288)]
    items, packed = [], 0
    for layer in range(wl.QWEN3_8B_LAYERS):
        for j, (name, N, K) in enumerate(fused):
            seed = 7_000_000 + layer * 16 + j
            g = wl.gen_weights_torch(N, K, 0.1, dev, seed)
            pw = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"] if g["nnz"] else None)
            del g
            items.append((pw, wl.gen_x_torch(1, K, dev, seed + 7), torch.empty((1, N), dtype=torch.float16,
                                                                               device=dev)))
            packed += pw.packed_bytes()
    batch = tq.Batch(1, items)
    stream = torch.cuda.current_stream()

    def timed(fn):
        for _ in range(3):
            fn(batch, stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            fn(batch, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps

    ms_seq = timed(tq.tq_linear_sequence)
    ms_ind = timed(tq.tq_linear_batched)
    st = tq.tq_get_device_status(clear=True)
    gbs = packed / (ms_seq * 1e-3) / 1e9
    return {"workload": "qwen3-8b decode step, M=1, q/k/v and gate/up fused: 144 problems in layer order",
            "ms_per_step": ms_seq, "packed_bytes": packed, "packed_gbs": gbs, "frac_of_hbm_peak": gbs / peak,
            "tokens_per_s": 1.0 / (ms_seq * 1e-3),
            "independent_ms_per_step": ms_ind, "ordering_cost_ms": ms_seq - ms_ind,
            "gpu_launches_per_step": 2, "device_status": st, "steps": steps}


def sub_codec(dev, peak, reps=5):
    """The codec and conversion kernels over one Qwen3-8B layer's seven
    projections (HBM-bound): tq_pack (int8 codes -> planes), tq_unpack
    (planes -> int8 codes), tq_plane2_index (the group-ordered second-plane
    index) and tq_dequantize (packed -> dense fp16 W-hat).  Algorithmic bytes
    = what each must read and write once; GB/s against the measured copy
    bandwidth."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    L = tq.lib()
    items = []
    bytes_ = {"pack": 0, "unpack": 0, "plane2_index": 0, "dequantize": 0}
    for p in wl.config_projections(4):
        g = wl.gen_weights_torch(p.N, p.K, 0.1, dev, 700 + p.proj)
        pw = tq.pack_weight(g["T1"], g["T2"], g["sal"], g["s1"], g["off"], g["s2"])
        N, K, nnz = p.N, p.K, pw.nnz
        T1o = torch.empty_like(g["T1"])
        T2o = torch.empty_like(g["T2"])
        Wd = torch.empty((N, K), dtype=torch.float16, device=dev)
        idx = torch.empty(int(L.tq_plane2_index_bytes(N, K, nnz)) // 4, dtype=torch.int32, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        items.append((pw, g["T1"], g["T2"], T1o, T2o, Wd, idx, st))
        side = pw.salience.numel() * 4 + pw.rowptr.numel() * 4
        planes = pw.plane1.numel() + nnz * 26
        bytes_["pack"] += 2 * N * K + side + planes
        bytes_["unpack"] += planes + side + 2 * N * K
        bytes_["plane2_index"] += nnz * 26 + nnz * 2 + side + idx.numel() * 4
        bytes_["dequantize"] += pw.packed_bytes() + 2 * N * K
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream

    def run(kind):
        for pw, T1, T2, T1o, T2o, Wd, idx, st in items:
            if kind == "pack":
                tq.tq_pack(pw.N, pw.K, T1, T2, pw.salience, pw.rowptr, pw.plane1, pw.plane2, st, stream)
            elif kind == "unpack":
                tq.tq_unpack(pw.N, pw.K, pw.plane1, pw.plane2, pw.salience, pw.rowptr, T1o, T2o, st, stream)
            elif kind == "plane2_index":
                L.tq_plane2_index(pw.N, pw.K, pw.salience.data_ptr(), pw.rowptr.data_ptr(), pw.nnz,
                                  pw.plane2.data_ptr(), pw.scale2.data_ptr(), idx.data_ptr(), sp)
            else:
                tq.tq_dequantize(pw, out=Wd, d_status=st, stream=stream)

    out = {}
    for kind in bytes_:
        for _ in range(2):
            run(kind)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            run(kind)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        gbs = bytes_[kind] / (ms * 1e-3) / 1e9
        out[kind] = {"ms_per_layer": ms, "bytes_per_layer": bytes_[kind], "gbs": gbs, "frac_of_hbm_peak": gbs / peak}
    status = sum(int(it[-1].item()) for it in items)
    return {"workload": "qwen3-8b one layer's 7 projections (193 M weights, 10 % salient groups)",
            "kernels": out, "data_status": status,
            "bytes": "algorithmic: pack reads the int8 T1 and T2 codes (all of T2: codes outside the salient groups "
                     "must be checked to be zero), salience and rowptr and writes plane 1 and plane 2; unpack the "
                     "reverse with full int8 T1 and T2; the index reads "
                     "plane 2, s2, salience and rowptr and writes the index; dequantize reads the packed weight "
                     "and writes fp16 W-hat",
            "l2": "no flush: a layer's int8 codes (386 MB) and fp16 W-hat (386 MB) exceed L2"}


def sub_elementwise(dev, peak):
    """The element-wise four-mask form (orders [2, 2, 1, 1], the paper's
    recorded coverages) of one Qwen3-8B layer at M = 1: seven tq_ew_linear
    calls per layer over rotated copies (more than 4 x L2 of packed bytes),
    replayed as a CUDA graph."""
    import torch

    import workloads as wl
    from paper_2609_09240_gb300 import tq

    base, layer_bytes, index_bytes = [], 0, 0
    for p in wl.config_projections(4):
        g = torch.Generator(device=dev)
        g.manual_seed(900 + p.proj)
        N, K = p.N, p.K
        u = torch.rand((N, K), generator=g, device=dev)
        mask = ((u >= 0.005).to(torch.uint8) + (u >= 0.036).to(torch.uint8) + (u >= 0.136).to(torch.uint8))
        u0 = torch.rand((N, K), generator=g, device=dev)
        T0 = ((u0 >= 0.3).to(torch.int8) + (u0 >= 0.7).to(torch.int8) - 1)
        u1 = torch.rand((N, K), generator=g, device=dev)
        T1 = ((u1 >= 0.3).to(torch.int8) + (u1 >= 0.7).to(torch.int8) - 1) * (mask <= 1).to(torch.int8)
        mu = (torch.randn((N, 4), generator=g, device=dev) * 1e-3).half()
        a0 = torch.empty((N, 4), device=dev).log_normal_(-4.0, 0.5, generator=g).half()
        a1 = torch.empty((N, 2), device=dev).log_normal_(-4.0, 0.5, generator=g).half()
        w = tq.ew_index(tq.pack_ew_weight(T0, T1, mask, mu, a0, a1))
        del u, u0, u1, T0, T1, mask
        base.append(w)
        layer_bytes += w.packed_bytes()
        index_bytes += w.index_bytes()
    R = -(-4 * L2_BYTES // layer_bytes)
    clone = lambda w: tq.EwWeight(w.N, w.K, w.mask.clone(), w.plane1.clone(), w.p2rowptr.clone(), w.plane2.clone(),
                                  w.mu.clone(), w.alpha0.clone(), w.alpha1.clone(), w.idx_off.clone(), w.idx.clone())
    layers = [[(w if r == 0 else clone(w), wl.gen_x_torch(1, w.K, dev, 950 + 8 * r + i),
                torch.empty((1, w.N), dtype=torch.float16, device=dev)) for i, w in enumerate(base)] for r in range(R)]
    wss = [tq.workspace(int(tq.lib().tq_ew_workspace_bytes(1, w.N, w.K)), dev) for w in base]
    batches = [tq.EwBatch(1, items) for items in layers]
    plain = [tq.EwBatch(1, [(dataclasses.replace(w, idx_off=None, idx=None), x, y) for w, x, y in items])
             for items in layers]

    def batched():
        for b in batches:
            tq.tq_ew_linear_batched(b)

    def batched_plain():
        for b in plain:
            tq.tq_ew_linear_batched(b)

    def calls():
        for items in layers:
            for (w, x, y), wsb in zip(items, wss):
                tq.tq_ew_linear(x, w, y=y, ws=wsb)

    ms = graph_ms(batched, reps=5) / R
    ms_plain = graph_ms(batched_plain, reps=5) / R
    ms_unb = graph_ms(calls, reps=5) / R
    gbs = layer_bytes / (ms * 1e-3) / 1e9
    n_w = sum(w.N * w.K for w in base)
    return {"workload": "qwen3-8b one layer in the element-wise four-mask form (coverages 0.5/3.1/10/86.4 %), M=1",
            "us_per_layer": ms * 1e3, "us_per_layer_without_index": ms_plain * 1e3,
            "us_per_layer_unbatched": ms_unb * 1e3, "packed_bytes": layer_bytes, "index_bytes": index_bytes,
            "bits_per_weight": 8 * layer_bytes / n_w, "packed_gbs": gbs, "frac_of_hbm_peak": gbs / peak,
            "timing": f"{R} rotated copies of the layer ({R * layer_bytes / 2 ** 20:.0f} MiB > 4 x L2); one "
                      "tq_ew_linear_batched call per layer (views, prep, plane 1, correction: 4 launches) with the "
                      "correction index, the same without it (mask-plane correction), and (unbatched) seven "
                      "tq_ew_linear calls per layer with the index; each replayed as a CUDA graph"}


def cpu_baseline_single(budget_s):
    """The oracle on one host core over a prefix of layer 0's rows."""
    L = OracleLayer()
    frac, nbytes, t = 0.02, 0, 0.0
    while t < budget_s and frac <= 1.0:
        b, dt = L.run(frac, nthreads=1)
        nbytes, t = nbytes + b, t + dt
        frac *= 2
    return nbytes / t / 1e9, f"the first rows of layer 0's seven projections on 1 core, {nbytes / 1e6:.1f} MB in {t:.1f} s"


# ------------------------------------------------------------------- main
def run_reference(args, ws, rank):
    """The oracle timed on the host cores.  A step is one pass of the oracle
    over a fixed sample of the workload (the first rows of each of layer 0's
    seven projections), sized so that the whole run stays within about two
    minutes of CPU work; ms_per_step is that pass's measured time and value
    its packed bytes over that time."""
    if rank != 0:
        return 0
    L = OracleLayer()
    _, t_full = L.run()  # calibration pass (untimed)
    n = args.warmup + args.steps
    frac = min(1.0, 120.0 / max(n, 1) / max(t_full, 1e-6))
    times, nbytes_step = [], 0
    for i in range(n):
        b, t = L.run(frac)
        if i >= args.warmup:
            times.append(t)
            nbytes_step = b
    t_step = float(np.median(times))
    value = nbytes_step / t_step / 1e9
    bytes_full = 1_792_241_424
    desc = (f"per step one oracle pass over the first {frac:.3f} of the rows of each projection of layer 0 of the "
            f"Qwen3-8B step ({nbytes_step / 1e6:.1f} MB of packed bytes, M=1, 10% salient); ms_per_step is "
            "that pass's measured time")
    out = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_step * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "impl": "reference",
        "config": {"workload": "qwen3-8b decode step, linear layers only, M=1: a fixed row sample of layer 0 per step",
                   "sample_packed_bytes": nbytes_step, "global_batch": 1, "seq_len": 1,
                   "parallelism": "none (host CPU)"},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": L.cores, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "tokens_per_s_full_step": value * 1e9 / bytes_full,
    }
    print(json.dumps(out), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="tq", choices=["tq", "reference"])
    ap.add_argument("--M", type=int, default=1, help="tokens per step (1 = batch-1 decode)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=None, help="profile a smaller step (first L layers)")
    ap.add_argument("--prefill", action="store_true", help="one Qwen3-8B layer at M = 2048 tokens")
    ap.add_argument("--ternarize", action="store_true", help="E2M-ATQ ternarization of one Qwen3-8B layer")
    ap.add_argument("--no-configs", action="store_true",
                    help="time only the Qwen3-8B M=1 step (skip configs 0, 1, 3, 4 and the unbatched calls)")
    args = ap.parse_args()
    ws, rank, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, ws, rank)
    if args.prefill:
        return run_prefill(args, ws, rank, local)
    if args.ternarize:
        return run_ternarize(args, ws, rank, local)

    import torch

    assert torch.cuda.is_available(), "bench.py needs a GPU"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    from paper_2609_09240_gb300 import tq

    tq.lib()
    items, x_all, y_all, packed_bytes, n_weights = build_step(args.M, dev, seed0=0, layers=args.layers)
    batch = tq.Batch(args.M, items)
    stream = torch.cuda.current_stream()
    # activation prep, second plane (when any projection has one), first plane
    launches_per_step = 3 if any(pw.nnz > 0 for pw, _, _ in items) else 2

    def step():
        tq.tq_linear_batched(batch, stream)

    def barrier():
        if pg:
            pg.barrier()
        torch.cuda.synchronize()

    # device-timed region: inputs resident in HBM (1.79 GB of packed weights
    # per step, larger than the 129 MB L2, so no flush is needed)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(torch.cuda.current_device()) as clk:
        clk.ready()
        for _ in range(max(args.warmup, 3)):
            step()
        barrier()
        clk.mark()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(args.steps):
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
        t1.record(stream)
        barrier()
        clk.mark()
    total_ms = t0.elapsed_time(t1)
    launch_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = max_over_ranks(total_ms, pg, dev)
    ms_per_step = total_ms / args.steps
    value = whole_job_rate(packed_bytes, ws, ms_per_step)
    launch_avg = float(np.mean(launch_ms))

    # end to end through the C ABI with host buffers: per step, H2D of every
    # projection's activations from pinned memory, the step, D2H of outputs
    x_host = x_all.cpu().pin_memory()
    y_host = torch.empty(y_all.shape, dtype=y_all.dtype).pin_memory()
    h2d = x_host.numel() * x_host.element_size()
    d2h = y_host.numel() * y_host.element_size()

    def e2e_step():
        x_all.copy_(x_host, non_blocking=True)
        step()
        y_host.copy_(y_all, non_blocking=True)

    for _ in range(2):
        e2e_step()
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    e1.record(stream)
    barrier()
    e2e_ms = e0.elapsed_time(e1) / args.steps
    e2e_ms = max_over_ranks(e2e_ms, pg, dev)
    e2e_value = whole_job_rate(packed_bytes, ws, e2e_ms)

    peak, peak_kind = measured_peaks()
    achieved = packed_bytes / (launch_avg * 1e-3) / 1e9
    out = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "accumulate": "f32", "data": "synthetic",
        "config": {"workload": f"qwen3-8b decode step, linear layers only, M={args.M} (252 packed projections)",
                   "model": "Qwen3-8B projection shapes, random ternary weights", "global_batch": args.M * ws,
                   "seq_len": 1, "parallelism": f"replicas x{ws}" if ws > 1 else "none",
                   "packed_bytes_per_step": packed_bytes, "weights_per_step": n_weights,
                   "p2index_bytes_per_step": sum(pw.p2index.numel() * 4 for pw, _, _ in items
                                                 if pw.p2index is not None),
                   "l2": "no flush: 1.79 GB of packed weights per step > 129 MB L2"},
        "tokens_per_s": ws * args.M / (ms_per_step * 1e-3),
        "us_per_step": ms_per_step * 1e3,
        "frac_of_8TBps_nominal": value / ws / 8000.0,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": f"{peak_kind} copy bandwidth",
                     "traffic": ncu_traffic(),
                     "kernel": "decode step: activation prep + second plane (group-ordered index) + first plane "
                               "(one-group-per-lane kernel); 3 launches per step, timed together (the first-plane "
                               "kernel is ~84 % of it)",
                     "launch_ms_avg": launch_avg},
        "e2e": {"value": e2e_value, "unit": "GB/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms},
        "gpu_launches": args.steps * launches_per_step,
        "clocks": clk.summary(),
    }
    if not args.no_configs and args.layers is None and args.M == 1:
        # the other configurations, each with its own timing (after the
        # headline's timed region)
        with ClockSampler(torch.cuda.current_device()) as clk2:
            clk2.ready()
            clk2.mark()
            cfg = {"config0": sub_config0(dev, peak), "config1": sub_config1(dev, peak),
                   "config3": [sub_skinny(items, M, dev, peak, packed_bytes, steps=50) for M in (2, 4, 8, 16)],
                   "unbatched_calls": sub_unbatched_8b(items, dev, ms_per_step)}
            cfg["config4"] = sub_prefill(dev)
            cfg["dependency_ordered"] = sub_sequence(dev, peak)
            cfg["elementwise"] = sub_elementwise(dev, peak)
            cfg["codec"] = sub_codec(dev, peak)
            clk2.mark()
        cfg["clocks"] = clk2.summary()
        out["configs"] = cfg
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        gbs, cores, desc, t = cpu_baseline(budget_s=15.0)
        gbs1, desc1 = cpu_baseline_single(budget_s=5.0)
        out["cpu_baseline"] = {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
                               "sample": desc, "seconds": t,
                               "single_core": {"value": gbs1, "unit": "GB/s", "cores": 1, "sample": desc1}}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if pg:
        pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
