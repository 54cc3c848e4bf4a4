#!/usr/bin/env python
"""Throughput of the rotated-hypercube mixing stack on GB300, forward + backward.

One step = one hcw_stack_train_step call (the work of hcw_stack_fwd +
hcw_stack_bwd) over one batch of the char-LM window-256 workload: B = 64
sequences of n = 256 positions, d = 512,
16 rotated causal layers (dimensions 0..7 twice), residual, ReLU, bias, with
per-layer weight gradients (Sec. 3.1 wiring, Eq. (1) maps).  Inputs are
synthetic (Zipf(1.1) byte ids embedded to d; see paper_2609_18145_gb300.synth)
and resident in HBM when the timed region starts; L2 is flushed (a 256 MiB
write) before every timed step, outside the timed events.

Prints ONE JSON line (rank 0).  --impl reference times the fp64 CPU oracle
instead (the reference arm of this build: there is no reference code).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
  torchrun --nproc-per-node N bench.py --gpus N ...   (N independent replicas)
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "HypercubeMix fwd+bwd tokens/s at n=256,d=512 bf16; % of roofline"
WORKLOAD = "charlm_w256_d512"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20
STACK_KERNELS = {"auto": 0, "resident": 1, "streaming": 2}   # hcw_set_stack_kernels modes
# Layer schedules (hcw_stack_fwd_dims): None = the rotated stack of the workload.
# hy256 = the near and jump layers of the paper's window-256 hybrid (App. A:
# near jump128 near [attn] near jump32 near jump16 near [attn] near jump4 near
# jump2 near jump1, the two attention layers left out); -1 = near (shift by 1).
SCHEDULES = {"rot": None, "hy256": [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0]}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def workload():
    from paper_2609_18145_gb300 import synth
    w = dict(synth.WORKLOADS[WORKLOAD])
    w["flags"] = 1 | 2 | 4          # causal, residual, ReLU
    return w


def step_flops(B, n, d, L, dims=None):
    """Algorithmic flops of one fwd+bwd step (causal): per token and layer
    3d^2 forward (half the positions use both maps), 3d^2 input gradient,
    3d^2 weight gradients (flop = 2 MAC).  With a schedule, a shift layer by
    k uses both maps on the n - k positions that have a predecessor k back."""
    if dims is None:
        return 9.0 * d * d * B * n * L
    per_token = 0.0
    for s in dims:
        frac = 0.5 if s >= 0 else (n + s) / n
        per_token += 3.0 * (2.0 * d * d + 2.0 * d * d * frac)
    return per_token * B * n


class ClockSampler:
    """SM clock and clock-event reasons sampled while a timed region runs:
    read-only NVML queries polled every ~2 ms from a thread (a timed region can
    be a few milliseconds long), else nvidia-smi every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, local_rank: int):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        ids = [v.strip() for v in vis.split(",")] if vis else []
        self.gpu = ids[local_rank] if local_rank < len(ids) else str(local_rank)
        self.proc = None
        self.file = None
        self.nvml = None
        self.samples = []
        self.stop = None
        self.thread = None

    def _open_nvml(self):
        import ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        handle = ctypes.c_void_p()
        if self.gpu.isdigit():
            rc = lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(int(self.gpu)),
                                                   ctypes.byref(handle))
        else:
            rc = lib.nvmlDeviceGetHandleByUUID(self.gpu.encode(), ctypes.byref(handle))
        if rc != 0:
            raise OSError("no NVML handle")
        reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons
        mx = ctypes.c_uint()
        lib.nvmlDeviceGetMaxClockInfo(handle, 1, ctypes.byref(mx))   # 1 = SM clock
        self.nvml = (lib, handle, reasons, mx.value)

    def _sample(self):
        import ctypes
        lib, handle, reasons, mx = self.nvml
        sm = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        if lib.nvmlDeviceGetClockInfo(handle, 1, ctypes.byref(sm)) == 0 and \
                reasons(handle, ctypes.byref(r)) == 0:
            self.samples.append((sm.value, mx, r.value))

    def _poll(self):
        while not self.stop.is_set():
            self._sample()
            time.sleep(0.002)

    def __enter__(self):
        import threading
        try:
            self._open_nvml()
            self.stop = threading.Event()
            self._sample()
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
            return self
        except (OSError, AttributeError):
            self.nvml = None
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.thread is not None:
            self._sample()
            self.stop.set()
            self.thread.join(timeout=5)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.nvml is not None:
            if not self.samples:
                return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
            reasons = sorted({name for _, _, r in self.samples
                              for bit, name in self.REASONS.items() if r & bit})
            return {"sm_mhz": statistics.median(sm for sm, _, _ in self.samples),
                    "sm_max_mhz": max(mx for _, mx, _ in self.samples), "reasons": reasons,
                    "samples": len(self.samples), "source": "nvml"}
        if self.proc is None or self.file is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.file.flush()
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def kernel_source_sha():
    h = hashlib.sha256()
    for f in ("hcw_tc.cu", "hcw_res.cu", "hcw_ptx.cuh", "hcw_api.cu"):
        with open(os.path.join(ROOT, "paper_2609_18145_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, or None
    when the kernel sources changed since those counters were taken."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    e = rec.get(kernel)
    if not e or e.get("src_sha") != kernel_source_sha():
        return None
    return e.get("bytes_per_launch")


# ---------------------------------------------------------------- oracle timing

def time_oracle(w, seconds_target: float, seed: int = 0, max_seqs: int = 64, dims=None):
    """Time the fp64 oracle's stack forward + backward on a bounded sample of
    the workload (whole sequences), on the layer schedule dims if given;
    returns (tokens/s, seconds, sequences, threads)."""
    from oracle import oracle as O
    from paper_2609_18145_gb300 import synth
    n, d, L = w["n"], w["d"], w["L"] if dims is None else len(dims)

    def run(seqs):
        pr = synth.problem(seqs, n, d, L=L, seed=seed, w_std=(1 / (2 * d)) ** 0.5,
                           x_ids="zipf256")
        _, x = synth.to_bf16_exact(pr.x)
        _, Ws = synth.to_bf16_exact(pr.W_self)
        _, Wn = synth.to_bf16_exact(pr.W_nbr)
        _, dy = synth.to_bf16_exact(pr.dy)
        t0 = time.perf_counter()
        _, acts, zs = O.stack_fwd(x, Ws, Wn, pr.bias.astype(np.float64), 0, L, -1, w["flags"],
                                  round_bf16=True, dims=dims)
        O.stack_bwd(acts, zs, dy, Ws, Wn, 0, L, -1, w["flags"], round_bf16=True, dims=dims)
        return time.perf_counter() - t0

    t1 = run(1)
    seqs = 1
    total = t1
    if t1 < seconds_target:
        seqs = int(min(max_seqs, max(1, round(seconds_target / max(t1, 1e-3)))))
        if seqs > 1:
            total = run(seqs)
    return seqs * n / total, total, seqs, O.num_threads()


# ---------------------------------------------------------------- reference arm

def run_reference(args):
    from paper_2609_18145_gb300 import replicas
    rank, _, world = replicas.env_world()
    if rank != 0:
        return 0
    w = workload()
    n, d, L = w["n"], w["d"], w["L"]
    from oracle import oracle as O
    from paper_2609_18145_gb300 import synth
    # one bounded sample per step: whole sequences, sized to about 2 s of CPU work
    _, t1, seqs, threads = time_oracle(w, 2.0, max_seqs=8)
    pr = synth.problem(seqs, n, d, L=L, seed=0, w_std=(1 / (2 * d)) ** 0.5, x_ids="zipf256")
    _, x = synth.to_bf16_exact(pr.x)
    _, Ws = synth.to_bf16_exact(pr.W_self)
    _, Wn = synth.to_bf16_exact(pr.W_nbr)
    _, dy = synth.to_bf16_exact(pr.dy)
    bias = pr.bias.astype(np.float64)

    def step():
        _, acts, zs = O.stack_fwd(x, Ws, Wn, bias, 0, L, -1, w["flags"], round_bf16=True)
        O.stack_bwd(acts, zs, dy, Ws, Wn, 0, L, -1, w["flags"], round_bf16=True)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    tokens = seqs * n
    value = tokens * args.steps / el
    sample = "%d sequence(s) of n=%d (of the 64-sequence batch) per step, 16 layers fwd+bwd" % (
        seqs, n)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * el / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "n": n, "d": d, "layers": L, "batch": w["B"],
                   "sample_sequences_per_step": seqs, "causal": True, "residual": True,
                   "act": "relu", "bias": True},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- our arm

def run_ours(args):
    import torch

    from paper_2609_18145_gb300 import hcw as H
    from paper_2609_18145_gb300 import replicas, synth

    rank, local_rank, world = replicas.env_world()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the compute path has no CPU fallback)")
    torch.cuda.set_device(local_rank)
    replicas.init("nccl")
    dev = torch.device("cuda", local_rank)
    H.lib()
    H.hcw_set_stack_kernels(STACK_KERNELS[args.stack_kernels])

    w = workload()
    B, n, d, L, flags = w["B"], w["n"], w["d"], w["L"], w["flags"]
    dims = SCHEDULES[args.schedule]
    if dims is not None:
        L = len(dims)
    tokens = B * n
    peaks, peak_src = load_peaks()

    # ---- inputs: weights shared by all replicas, activations per rank
    wstd = (1 / (2 * d)) ** 0.5
    pw = synth.problem(1, n, d, L=L, seed=0, w_std=wstd)
    px = synth.problem(B, n, d, L=1, seed=replicas.batch_seed(0, rank), x_ids="zipf256")
    x = torch.from_numpy(px.x).to(torch.bfloat16).to(dev)
    dy = torch.from_numpy(px.dy).to(torch.bfloat16).to(dev)
    Ws = torch.from_numpy(pw.W_self).to(torch.bfloat16).to(dev)
    Wn = torch.from_numpy(pw.W_nbr).to(torch.bfloat16).to(dev)
    bias = torch.from_numpy(pw.bias).to(dev)
    act_shape = (L - 1, B, n, d)
    y = torch.empty_like(x)
    acts = torch.empty(act_shape, dtype=torch.bfloat16, device=dev)
    masks = torch.empty((L, B, n, d // 32), dtype=torch.int32, device=dev)
    dx = torch.empty_like(x)
    gWs = torch.empty((L, d, d), dtype=torch.float32, device=dev)
    gWn = torch.empty((L, d, d), dtype=torch.float32, device=dev)
    gb = torch.empty((L, d), dtype=torch.float32, device=dev)
    ws = torch.empty(H.hcw_stack_workspace_bytes(B, n, d, H.HCW_BF16, flags, L), dtype=torch.uint8,
                     device=dev)
    fws = torch.empty(max(1, H.hcw_stack_fwd_workspace_bytes(B, n, d, H.HCW_BF16, flags, L)),
                      dtype=torch.uint8, device=dev)
    tws = torch.empty(max(1, H.hcw_stack_train_step_workspace_bytes(B, n, d, H.HCW_BF16, flags,
                                                                    L)),
                      dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step_calls(xin, dyin, outs=None):
        oWs, oWn, ob = outs if outs is not None else (gWs, gWn, gb)
        # one training-step call (on the schedule dims if given): the forward and
        # the input gradient in one launch where the shape allows it, then the
        # weight gradients
        H.hcw_stack_train_step(xin, Ws, Wn, bias, dyin, 0, -1, flags, y=y, acts=acts,
                               masks=masks, dx=dx, dW_self=oWs, dW_nbr=oWn, dbias=ob,
                               workspace=tws, dims=dims)

    def capture(xin, dyin, outs=None):
        # the step's launches, recorded once and replayed: no host work per step
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            step_calls(xin, dyin, outs)    # first call on this stream: one-time set-up
            with torch.cuda.graph(g, stream=side):
                step_calls(xin, dyin, outs)
        torch.cuda.current_stream().wait_stream(side)
        return g

    for _ in range(args.warmup):
        step_calls(x, dy)
    graph = capture(x, dy) if not args.no_graph else None
    step_launches = H.hcw_launch_count()
    step_calls(x, dy)
    step_launches = H.hcw_launch_count() - step_launches

    def step(xin, dyin):
        if graph is not None and xin is x:
            graph.replay()
        else:
            step_calls(xin, dyin)

    for _ in range(args.warmup):
        step(x, dy)
    torch.cuda.synchronize()
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error during warm-up")

    # ---- timed region: K steps, device time by CUDA events, L2 flushed before each
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    replicas.barrier()
    torch.cuda.synchronize()
    launches0 = H.hcw_launch_count()
    with ClockSampler(local_rank) as clk:
        for i in range(args.steps):
            flush.fill_(i & 0xFF)
            starts[i].record(stream)
            step(x, dy)
            ends[i].record(stream)
        torch.cuda.synchronize()
    launches = H.hcw_launch_count() - launches0
    if graph is not None:
        launches = step_launches * args.steps     # graph replays launch the captured kernels
    replicas.barrier()
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error during the timed region")
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    ms_local = sum(step_ms) / len(step_ms)
    ms = replicas.max_over_ranks(ms_local, dev)
    value = world * tokens / (ms * 1e-3)
    clocks = clk.summary()

    # ---- per-kernel device time (each kernel kind launched alone, same inputs)
    def time_calls(fn, reps):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(reps)]
        for i in range(reps):
            flush.fill_(i & 0xFF)
            evs[i][0].record(stream)
            fn(i)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in evs) / reps

    # the step's three tensor-core launches, each timed alone on the same inputs:
    # the stacked forward, the stacked input gradient (with the top layer's
    # ReLU-gradient pass in front) and the batched weight gradient (bias off)
    dz_all = torch.empty((L, B, n, d), dtype=torch.bfloat16, device=dev)
    dws = torch.empty(max(1, H.hcw_stack_bwd_data_workspace_bytes(B, n, d, H.HCW_BF16, flags, L)),
                      dtype=torch.uint8, device=dev)
    wws = torch.empty(max(1, H.hcw_stack_bwd_weight_workspace_bytes(B, n, d, H.HCW_BF16, flags,
                                                                    L)),
                      dtype=torch.uint8, device=dev)
    reps = 5
    family = H.hcw_stack_kernels_used(B, n, d)
    has_shift = dims is not None and any(v < 0 for v in dims)
    fused = (family == H.HCW_STACK_STREAMING and d % 256 == 0 and L <= 16 and
             (not has_shift or (n >= 128 and (B * n) % 256 == 0)))
    if dims is not None and not fused:
        # a schedule the one-launch step does not take: time its forward and its
        # backward (input and weight gradients) as two launch sequences
        f_ms = time_calls(lambda i: H.hcw_stack_fwd(x, Ws, Wn, bias, 0, -1, flags, y=y,
                                                    acts=acts, masks=masks, workspace=fws,
                                                    dims=dims), reps)
        b_ms = time_calls(lambda i: H.hcw_stack_bwd(x, acts, masks, dy, Ws, Wn, 0, -1, flags,
                                                    dx=dx, dW_self=gWs, dW_nbr=gWn, dbias=gb,
                                                    workspace=ws, dims=dims), reps)
        f_flops = step_flops(B, n, d, L, dims) / 3.0
        kflops = {"forward of the %s schedule" % args.schedule: f_flops,
                  "backward of the %s schedule (input and weight gradients)"
                  % args.schedule: 2.0 * f_flops}
        kernels = dict(zip(kflops, (f_ms, b_ms)))
        dwb_ms = dw_ms = 0.0
    if dims is None and not fused:
        kflops = None
        fwd_ms = time_calls(lambda i: H.hcw_stack_fwd(x, Ws, Wn, bias, 0, -1, flags, y=y,
                                                      acts=acts, masks=masks, workspace=fws),
                            reps)
    if fused:
        # the step's two launches: the forward and the input gradient in one
        # launch (the training step without weight gradients), and the batched
        # weight gradient (bias off), each timed alone on the same inputs
        fdx_ms = time_calls(lambda i: H.hcw_stack_train_step(x, Ws, Wn, bias, dy, 0, -1, flags,
                                                             y=y, acts=acts, masks=masks, dx=dx,
                                                             want_dw=False, workspace=tws,
                                                             dims=dims),
                            reps)
        dz_step = tws[:L * x.numel() * 2].view(torch.bfloat16).view(L, B, n, d)
        dw_ms = time_calls(lambda i: H.hcw_stack_bwd_weight(x, acts, dz_step, 0, -1, flags,
                                                            dW_self=gWs, dW_nbr=gWn,
                                                            want_dbias=False, workspace=wws,
                                                            dims=dims),
                           reps)
        dwb_ms = time_calls(lambda i: H.hcw_stack_bwd_weight(x, acts, dz_step, 0, -1, flags,
                                                             dW_self=gWs, dW_nbr=gWn, dbias=gb,
                                                             workspace=wws, dims=dims), reps)
        fdx_name = ("hcw_tc_kernel<FDX,256,%d> (stacked forward and input gradient in one "
                    "launch on SM pairs, top dz written by the last forward layer)" % (2 * L))
        dw_name = ("hcw_dwp_kernel<256> (weight and bias gradients on SM pairs, a unit per "
                   "layer and 256 x 256 output tile)")
        kernels = {fdx_name: fdx_ms, dw_name: dw_ms}
        third = step_flops(B, n, d, L, dims) / 3.0   # one of forward, input and weight gradient
        kflops = {fdx_name: 2.0 * third, dw_name: third}
    elif dims is None:
        dx_ms = time_calls(lambda i: H.hcw_stack_bwd_data(masks, dy, Ws, Wn, 0, -1, flags,
                                                          dx=dx, dz=dz_all, workspace=dws), reps)
        dw_ms = time_calls(lambda i: H.hcw_stack_bwd_weight(x, acts, dz_all, 0, -1, flags,
                                                            dW_self=gWs, dW_nbr=gWn,
                                                            want_dbias=False, workspace=wws),
                           reps)
        dwb_ms = time_calls(lambda i: H.hcw_stack_bwd_weight(x, acts, dz_all, 0, -1, flags,
                                                             dW_self=gWs, dW_nbr=gWn, dbias=gb,
                                                             workspace=wws), reps)
        if family == H.HCW_STACK_RESIDENT:
            fwd_name = ("hcw_res_kernel<FWD,%d> (resident stacked forward: 256 tokens per SM "
                        "pair through all layers)" % d)
            dx_name = ("hcw_res_kernel<DX,%d> (resident stacked input gradient, top dz "
                       "included)" % d)
        else:
            fwd_name = "hcw_tc_kernel<FWD,256,16> (stacked forward on SM pairs)"
            dx_name = ("hcw_tc_kernel<DX,256,16> (stacked input gradient on SM pairs, top dz "
                       "included)")
        kernels = {fwd_name: fwd_ms, dx_name: dx_ms,
                   "hcw_dwp_kernel<256> (weight and bias gradients on SM pairs, a unit per "
                   "layer and 256 x 256 output tile)": dw_ms}
        # per stacked launch, 16 causal layers
        kflops = {k: 3.0 * d * d * tokens * L for k in kernels}
    dominant = max(kernels, key=kernels.get)
    dom_ms = kernels[dominant]
    launch_flops = kflops[dominant]
    peak = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    achieved = launch_flops / (dom_ms * 1e-3) / 1e12
    per_kernel = {k: {"ms": v, "tflops": kflops[k] / (v * 1e-3) / 1e12,
                      "frac": kflops[k] / (v * 1e-3) / 1e12 / peak} for k, v in kernels.items()}
    step_tflops = step_flops(B, n, d, L, dims) / (ms * 1e-3) / 1e12
    peak_sus = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    traffic = recorded_traffic(dominant.split(" ")[0])

    # ---- end to end through the public API with host buffers: every step
    # copies its inputs (x, dy) in from pinned host memory and its result (the
    # weight and bias gradients) out to pinned host memory.  Steps are
    # pipelined as a training loop would run them: step i + 1's inputs come in
    # on one copy stream and step i's gradients go out on another while step i
    # (or i + 1) computes, with double-buffered inputs and gradient outputs
    # (two graphs); the timed span runs from the first input copy to the last
    # gradient copy, and each step still flushes L2 (inside the span).
    x_h = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
    dy_h = torch.empty(dy.shape, dtype=dy.dtype, pin_memory=True)
    x_h.copy_(x)
    dy_h.copy_(dy)
    outs = (gWs, gWn, gb)
    outs_h = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs]
    h2d = x_h.numel() * x_h.element_size() + dy_h.numel() * dy_h.element_size()
    d2h = sum(t.numel() * t.element_size() for t in outs_h)
    e2e_steps = max(4, args.steps)
    ins = [(x.clone(), dy.clone()) for _ in range(2)]
    res = [tuple(torch.empty_like(t) for t in outs) for _ in range(2)]
    graphs = [capture(*ins[b], res[b]) if not args.no_graph else None for b in range(2)]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in", "used", "out", "sent")}
    replicas.barrier()
    torch.cuda.synchronize()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s_in.record_event(e_start)

    def load(i):
        b = i % 2
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev["used"][b])      # step i - 2 has read this pair
            ins[b][0].copy_(x_h, non_blocking=True)
            ins[b][1].copy_(dy_h, non_blocking=True)
            s_in.record_event(ev["in"][b])

    load(0)
    for i in range(e2e_steps):
        b = i % 2
        if i + 1 < e2e_steps:
            load(i + 1)
        stream.wait_event(ev["in"][b])
        if i >= 2:
            stream.wait_event(ev["sent"][b])        # step i - 2's gradients have left
        flush.fill_(i & 0xFF)
        if graphs[b] is not None:
            graphs[b].replay()
        else:
            step_calls(*ins[b], res[b])
        stream.record_event(ev["used"][b])
        stream.record_event(ev["out"][b])
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["out"][b])
            for th, t in zip(outs_h, res[b]):
                th.copy_(t, non_blocking=True)
            s_out.record_event(ev["sent"][b])
    s_out.wait_stream(s_in)
    s_out.wait_stream(stream)
    s_out.record_event(e_end)
    torch.cuda.synchronize()
    e2e_ms = replicas.max_over_ranks(e_start.elapsed_time(e_end) / e2e_steps, dev)
    e2e_value = world * tokens / (e2e_ms * 1e-3)
    last = res[(e2e_steps - 1) % 2]
    if not all(torch.equal(th.to(dev), t) for th, t in zip(outs_h, last)):
        raise SystemExit("end-to-end gradients differ from the ones on the device")
    if not all(torch.equal(a, b2) for a, b2 in zip(last, outs)):
        raise SystemExit("end-to-end gradients differ from the device-timed step's")

    # ---- the oracle on the host cores, bounded sample (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, secs, seqs, threads = time_oracle(w, 10.0, dims=dims)
        cpu = {"value": v, "unit": "tokens/s", "cores": threads, "kind": "oracle",
               "sample": "%d of the 64 sequences (n=256), %d layers (%s) fwd+bwd, fp64, %.1f s"
                         % (seqs, L, args.schedule, secs)}

    replicas.barrier()
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "n": n, "d": d, "layers": L, "batch": B,
                       "tokens_per_step_per_gpu": tokens, "causal": True, "residual": True,
                       "act": "relu", "bias": True,
                       "l2": "flushed before every timed step (256 MiB write, untimed)",
                       "parallelism": "replicas" if world > 1 else "single",
                       "stack_kernels": ("one-launch forward + input gradient" if fused else
                                         "schedule: forward and backward calls" if dims is not None else
                                         "resident" if family == H.HCW_STACK_RESIDENT
                                         else "streaming"),
                       "schedule": args.schedule,
                       "launch": "host calls" if args.no_graph else "CUDA graph of the step's calls"},
            "roofline": {"bound": "tensor", "kernel": dominant, "achieved": achieved,
                         "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                         "traffic": traffic, "peak_source": peak_src + " bf16 burst",
                         "flops_per_launch": launch_flops, "avg_launch_ms": dom_ms,
                         "kernels": per_kernel, "dbias_ms": dwb_ms - dw_ms},
            "step_roofline": {"achieved": step_tflops, "peak": peak_sus, "unit": "TFLOP/s",
                              "frac": step_tflops / peak_sus,
                              "peak_source": peak_src + " bf16 sustained",
                              "flops_per_step": step_flops(B, n, d, L, dims)},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                    "copies": "pinned host buffers; step i+1's inputs and step i's gradients "
                              "copied on two streams while the steps compute (double-buffered "
                              "inputs and outputs); L2 flushed every step inside the span"},
            "gpu_launches": launches,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    replicas.finish()
    return 0


# ---------------------------------------------------------------- other workloads
# The other configurations of the mixing stack, one JSON line each (--workload):
# the synthetic reachability shape (rotated, and its fixed-dimension control),
# the character-LM window-64 shape, and the 2^20-token scaling sweep at
# d = 1024 (L = log2 n), fwd+bwd and forward only.  Same timing rules as the
# headline line: warm-up, L2 flushed before every timed step, CUDA events.
WORKLOADS_EXTRA = {
    # name: (synth.WORKLOADS entry, dim_override, forward only)
    "reach_n64_d128": ("reach_n64_d128", -1, False),
    "reach_n64_d128_fixed": ("reach_n64_d128", 0, False),
    "charlm_w64_d512": ("charlm_w64_d512", -1, False),
    "scale_n256_d1024": ("scale_n256_d1024", -1, False),
    "scale_n4096_d1024": ("scale_n4096_d1024", -1, False),
    "scale_n65536_d1024": ("scale_n65536_d1024", -1, False),
    "scale_n256_d1024_fwd": ("scale_n256_d1024", -1, True),
    "scale_n4096_d1024_fwd": ("scale_n4096_d1024", -1, True),
    "scale_n65536_d1024_fwd": ("scale_n65536_d1024", -1, True),
}


def workload_bytes(d, L, causal, relu, fwd_only):
    """Algorithmic HBM bytes per token of one step (bf16 activations, each
    tensor moved once): per layer the forward reads x and writes y (4d), the
    backward reads the layer input and the output gradient and writes the
    input gradient (6d); with ReLU one mask bit per feature is written and read
    back.  Weights (4 d^2 bytes per layer) are amortised over the batch."""
    m = d / 8.0 if relu else 0.0
    if fwd_only:
        return (4.0 * d + m) * L
    return (10.0 * d + 2.0 * m) * L


def workload_flops(d, L, causal, fwd_only):
    per = (3.0 if causal else 4.0) * d * d      # flop = 2 MAC; causal: half the rows
    return per * L * (1 if fwd_only else 3)


def run_workload(args):
    import torch

    from oracle import oracle as O
    from paper_2609_18145_gb300 import hcw as H
    from paper_2609_18145_gb300 import replicas, synth

    rank, local_rank, world = replicas.env_world()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the compute path has no CPU fallback)")
    torch.cuda.set_device(local_rank)
    replicas.init("nccl")
    dev = torch.device("cuda", local_rank)
    H.lib()
    key, dim_over, fwd_only = WORKLOADS_EXTRA[args.workload]
    w = synth.WORKLOADS[key]
    B, n, d, L, causal = w["B"], w["n"], w["d"], w["L"], w["causal"]
    flags = (H.HCW_CAUSAL if causal else 0) | H.HCW_RESIDUAL | H.HCW_ACT_RELU
    tokens = B * n
    peaks, peak_src = load_peaks()
    wstd = (1 / (2 * d)) ** 0.5
    seed = replicas.batch_seed(0, rank)
    # inputs: weights from the host generator, activations of the 2^20-token
    # shapes drawn on the device (4 GiB each in fp32)
    Ws = torch.from_numpy(synth.normal((L, d, d), 2, wstd)).to(torch.bfloat16).to(dev)
    Wn = torch.from_numpy(synth.normal((L, d, d), 3, wstd)).to(torch.bfloat16).to(dev)
    bias = torch.from_numpy(synth.normal((L, d), 4, 0.1)).to(dev)
    if tokens * d <= (1 << 24):
        px = synth.problem(B, n, d, L=1, seed=seed, x_ids=w.get("x_ids"))
        x = torch.from_numpy(px.x).to(torch.bfloat16).to(dev)
        dy = torch.from_numpy(px.dy).to(torch.bfloat16).to(dev)
    else:
        x = synth.device_normal((B, n, d), seed + 1, dev).to(torch.bfloat16)
        dy = synth.device_normal((B, n, d), seed + 5, dev).to(torch.bfloat16)
    y = torch.empty_like(x)
    acts = torch.empty((L - 1, B, n, d), dtype=torch.bfloat16, device=dev)
    masks = torch.empty((L, B, n, (d + 31) // 32), dtype=torch.int32, device=dev)
    dx = torch.empty_like(x)
    gWs = torch.empty((L, d, d), dtype=torch.float32, device=dev)
    gWn = torch.empty((L, d, d), dtype=torch.float32, device=dev)
    gb = torch.empty((L, d), dtype=torch.float32, device=dev)
    if fwd_only:
        ws = torch.empty(max(1, H.hcw_stack_fwd_workspace_bytes(B, n, d, H.HCW_BF16, flags, L)),
                         dtype=torch.uint8, device=dev)
    else:
        ws = torch.empty(max(1, H.hcw_stack_train_step_workspace_bytes(B, n, d, H.HCW_BF16,
                                                                       flags, L)),
                         dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(xin, dyin):
        if fwd_only:
            H.hcw_stack_fwd(xin, Ws, Wn, bias, 0, dim_over, flags, y=y, acts=acts, masks=masks,
                            workspace=ws)
        else:
            H.hcw_stack_train_step(xin, Ws, Wn, bias, dyin, 0, dim_over, flags, y=y, acts=acts,
                                   masks=masks, dx=dx, dW_self=gWs, dW_nbr=gWn, dbias=gb,
                                   workspace=ws)

    for _ in range(args.warmup):
        step(x, dy)
    torch.cuda.synchronize()
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error during warm-up")
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    replicas.barrier()
    torch.cuda.synchronize()
    launches0 = H.hcw_launch_count()
    with ClockSampler(local_rank) as clk:
        for i in range(args.steps):
            flush.fill_(i & 0xFF)
            starts[i].record(stream)
            step(x, dy)
            ends[i].record(stream)
        torch.cuda.synchronize()
    launches = H.hcw_launch_count() - launches0
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error during the timed region")
    ms_local = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / args.steps
    ms = replicas.max_over_ranks(ms_local, dev)
    value = world * tokens / (ms * 1e-3)
    clocks = clk.summary()

    # roofline of the whole step: the slower of the flops at the bf16 peak and
    # the algorithmic bytes at the copy bandwidth
    flops = workload_flops(d, L, causal, fwd_only) * tokens
    nbytes = workload_bytes(d, L, causal, True, fwd_only) * tokens
    peak_t = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    peak_b = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    t_flop, t_byte = flops / (peak_t * 1e12), nbytes / (peak_b * 1e9)
    sec = ms * 1e-3
    if t_flop >= t_byte:
        roof = {"bound": "tensor", "achieved": flops / sec / 1e12, "peak": peak_t,
                "unit": "TFLOP/s", "frac": t_flop / sec,
                "peak_source": peak_src + " bf16 burst"}
    else:
        roof = {"bound": "hbm", "achieved": nbytes / sec / 1e9, "peak": peak_b, "unit": "GB/s",
                "frac": t_byte / sec, "peak_source": peak_src + " copy bandwidth"}
    roof.update({"kernel": "the whole step (%s launches)" % (launches // args.steps),
                 "traffic": None, "flops_per_step": flops, "algorithmic_bytes_per_step": nbytes})

    # end to end through the public API with host buffers: every step copies
    # x and dy in from pinned memory and its result out (the weight and bias
    # gradients, or y for the forward), pipelined as a training loop runs
    # them: step i + 1's inputs come in on one copy stream and step i's result
    # goes out on another while the steps compute (double-buffered inputs and
    # results); the span runs from the first input copy to the last result
    # copy, and each step still flushes L2 inside it
    x_h = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
    dy_h = torch.empty(dy.shape, dtype=dy.dtype, pin_memory=True)
    x_h.copy_(x)
    dy_h.copy_(dy)
    outs = (y,) if fwd_only else (gWs, gWn, gb)
    outs_h = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs]
    h2d = x_h.numel() * 2 + (0 if fwd_only else dy_h.numel() * 2)
    d2h = sum(t.numel() * t.element_size() for t in outs_h)
    e_steps = max(4, min(args.steps, 20))
    ins = [(torch.empty_like(x), torch.empty_like(dy)) for _ in range(2)]
    res = [tuple(torch.empty_like(t) for t in outs) for _ in range(2)]

    def step_into(xin, dyin, out):
        if fwd_only:
            H.hcw_stack_fwd(xin, Ws, Wn, bias, 0, dim_over, flags, y=out[0], acts=acts,
                            masks=masks, workspace=ws)
        else:
            H.hcw_stack_train_step(xin, Ws, Wn, bias, dyin, 0, dim_over, flags, y=y, acts=acts,
                                   masks=masks, dx=dx, dW_self=out[0], dW_nbr=out[1],
                                   dbias=out[2], workspace=ws)

    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in", "used", "out", "sent")}
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s_in.record_event(a)

    def load(i):
        k = i % 2
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev["used"][k])       # step i - 2 has read this pair
            ins[k][0].copy_(x_h, non_blocking=True)
            if not fwd_only:
                ins[k][1].copy_(dy_h, non_blocking=True)
            s_in.record_event(ev["in"][k])

    load(0)
    for i in range(e_steps):
        k = i % 2
        if i + 1 < e_steps:
            load(i + 1)
        stream.wait_event(ev["in"][k])
        if i >= 2:
            stream.wait_event(ev["sent"][k])         # step i - 2's result has left
        flush.fill_(i & 0xFF)
        step_into(ins[k][0], ins[k][1], res[k])
        stream.record_event(ev["used"][k])
        stream.record_event(ev["out"][k])
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["out"][k])
            for th, t in zip(outs_h, res[k]):
                th.copy_(t, non_blocking=True)
            s_out.record_event(ev["sent"][k])
    s_out.wait_stream(s_in)
    s_out.wait_stream(stream)
    s_out.record_event(b)
    torch.cuda.synchronize()
    e2e_ms = a.elapsed_time(b) / e_steps
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error during the end-to-end run")
    if not all(torch.equal(th.to(dev), t) for th, t in zip(outs_h, res[(e_steps - 1) % 2])):
        raise SystemExit("end-to-end results differ from the ones on the device")

    # the oracle on the host cores, a bounded sample: whole sequences of the
    # workload for n <= 256, else one layer of one n = 256 sequence (the cost
    # per token and layer does not depend on n) scaled to the L layers
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_s, L_s = (n, L) if n <= 256 else (256, 1)
        seqs = 1
        pr = synth.problem(seqs, n_s, d, L=L_s, seed=0, w_std=wstd, x_ids=w.get("x_ids"))
        _, xo = synth.to_bf16_exact(pr.x)
        _, wso = synth.to_bf16_exact(pr.W_self)
        _, wno = synth.to_bf16_exact(pr.W_nbr)
        _, dyo = synth.to_bf16_exact(pr.dy)
        t0 = time.perf_counter()
        _, oa, oz = O.stack_fwd(xo, wso, wno, pr.bias.astype(np.float64), 0, L_s, dim_over,
                                flags, round_bf16=True)
        if not fwd_only:
            O.stack_bwd(oa, oz, dyo, wso, wno, 0, L_s, dim_over, flags, round_bf16=True)
        secs = time.perf_counter() - t0
        v = seqs * n_s / secs * L_s / L
        cpu = {"value": v, "unit": "tokens/s", "cores": O.num_threads(), "kind": "oracle",
               "sample": "%d sequence(s) of n=%d through %d layer(s), %s, fp64, %.1f s%s"
                         % (seqs, n_s, L_s, "forward" if fwd_only else "fwd+bwd", secs,
                            "" if L_s == L else "; scaled to %d layers" % L)}

    replicas.barrier()
    if rank == 0:
        print(json.dumps({
            "metric": "HypercubeMix %s tokens/s at %s bf16; %% of roofline"
                      % ("forward" if fwd_only else "fwd+bwd", args.workload),
            "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "n": n, "d": d, "layers": L, "batch": B,
                       "tokens_per_step_per_gpu": tokens, "causal": causal, "residual": True,
                       "act": "relu", "bias": True,
                       "schedule": "fixed dimension 0" if dim_over == 0 else "rotated",
                       "l2": "flushed before every timed step (256 MiB write, untimed)",
                       "parallelism": "replicas" if world > 1 else "single",
                       "launch": "host calls"},
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": world * tokens / (e2e_ms * 1e-3), "unit": "tokens/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms,
                    "copies": "pinned host buffers; step i+1's inputs and step i's result "
                              "copied on two streams while the steps compute "
                              "(double-buffered); L2 flushed every step inside the span"},
            "gpu_launches": launches,
            "clocks": clocks,
        }), flush=True)
    replicas.finish()
    return 0


def run_kernel_only(args):
    """Launch one kernel kind alone (for profiler captures): the layer
    forward, input-gradient or weight-gradient pass of the workload's shape
    with --batch sequences, --warmup untimed and --steps timed launches."""
    import torch

    from paper_2609_18145_gb300 import hcw as H
    from paper_2609_18145_gb300 import synth

    w = workload()
    B, n, d, flags = args.batch, w["n"], w["d"], w["flags"]
    dev = torch.device("cuda", 0)
    H.lib()
    H.hcw_set_stack_kernels(STACK_KERNELS[args.stack_kernels])
    pr = synth.problem(B, n, d, L=1, seed=0, w_std=(1 / (2 * d)) ** 0.5, x_ids="zipf256")
    x = torch.from_numpy(pr.x).to(torch.bfloat16).to(dev)
    dz = torch.from_numpy(pr.dy).to(torch.bfloat16).to(dev)
    Ws = torch.from_numpy(pr.W_self[0]).to(torch.bfloat16).to(dev)
    Wn = torch.from_numpy(pr.W_nbr[0]).to(torch.bfloat16).to(dev)
    bias = torch.from_numpy(pr.bias[0]).to(dev)
    y = torch.empty_like(x)
    z = torch.empty_like(x)
    gWs = torch.empty((d, d), dtype=torch.float32, device=dev)
    gWn = torch.empty_like(gWs)
    wws = torch.empty(max(1, H.hcw_layer_bwd_weight_workspace_bytes(B, n, d, H.HCW_BF16, flags)),
                      dtype=torch.uint8, device=dev)
    layer = 3
    if args.kernel == "decode":
        return run_decode(args, w, dev)
    if args.kernel == "block":
        return run_block(args, w, dev)
    if args.kernel == "step":
        # one whole step (stack forward + stack backward) of --batch sequences
        L = w["L"]
        ps = synth.problem(1, n, d, L=L, seed=0, w_std=(1 / (2 * d)) ** 0.5)
        SWs = torch.from_numpy(ps.W_self).to(torch.bfloat16).to(dev)
        SWn = torch.from_numpy(ps.W_nbr).to(torch.bfloat16).to(dev)
        Sb = torch.from_numpy(ps.bias).to(dev)
        acts = torch.empty((L - 1, B, n, d), dtype=torch.bfloat16, device=dev)
        masks = torch.empty((L, B, n, d // 32), dtype=torch.int32, device=dev)
        sWs = torch.empty((L, d, d), dtype=torch.float32, device=dev)
        sWn = torch.empty_like(sWs)
        sb = torch.empty((L, d), dtype=torch.float32, device=dev)
        dxs = torch.empty_like(x)
        tws = torch.empty(H.hcw_stack_train_step_workspace_bytes(B, n, d, H.HCW_BF16, flags, L),
                          dtype=torch.uint8, device=dev)

        def fn():
            # the bench step: one training-step call (forward + input gradient in one
            # launch, then the weight gradients)
            H.hcw_stack_train_step(x, SWs, SWn, Sb, dz, 0, -1, flags, y=y, acts=acts,
                                   masks=masks, dx=dxs, dW_self=sWs, dW_nbr=sWn, dbias=sb,
                                   workspace=tws)
    elif args.kernel == "fwd":
        fn = lambda: H.hcw_layer_fwd(x, Ws, Wn, bias, layer, -1, flags, y=y, z_save=z)
    elif args.kernel == "dx":
        fn = lambda: H.hcw_layer_bwd_data(dz, dz, Ws, Wn, layer, -1, flags, dx=y)
    else:
        fn = lambda: H.hcw_layer_bwd_weight(x, dz, layer, -1, flags, dW_self=gWs, dW_nbr=gWn,
                                            want_dbias=False, workspace=wws)
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        fn()
    b.record()
    torch.cuda.synchronize()
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error")
    ms = a.elapsed_time(b) / args.steps
    flops = step_flops(B, n, d, w["L"]) if args.kernel == "step" else 3.0 * d * d * B * n
    print(json.dumps({"kernel": args.kernel, "batch": B, "n": n, "d": d, "avg_ms": ms,
                      "tflops": flops / (ms * 1e-3) / 1e12}), flush=True)
    return 0


def run_decode(args, w, dev):
    """Decode one whole window of --batch sequences position by position
    (hcw_decode_step, Sec. 6) with the workload's layers, issued from the host
    and as one CUDA graph of the window, and print the time per position."""
    import torch

    from paper_2609_18145_gb300 import hcw as H
    from paper_2609_18145_gb300 import synth

    B, n, d, L, flags = args.batch, w["n"], w["d"], w["L"], w["flags"]
    dims = SCHEDULES[args.schedule]
    if dims is not None:
        L = len(dims)
    ps = synth.problem(B, n, d, L=L, seed=0, w_std=(1 / (2 * d)) ** 0.5, x_ids="zipf256")
    xs = torch.from_numpy(ps.x).to(torch.bfloat16).transpose(0, 1).contiguous().to(dev)  # [n,B,d]
    Ws = torch.from_numpy(ps.W_self).to(torch.bfloat16).to(dev)
    Wn = torch.from_numpy(ps.W_nbr).to(torch.bfloat16).to(dev)
    bias = torch.from_numpy(ps.bias).to(dev)
    cache = torch.zeros(max(1, H.hcw_decode_cache_bytes(L, B, n, d, dims=dims)), dtype=torch.uint8,
                        device=dev)
    ys = torch.empty_like(xs)

    def window():
        for t in range(n):
            H.hcw_decode_step(xs[t], Ws, Wn, bias, t, n, cache, flags, dims=dims, y=ys[t])

    def timed(fn, reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record()
        for _ in range(reps):
            fn()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    def graph_time():
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            window()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                window()
        torch.cuda.synchronize()
        g.replay()
        return timed(g.replay, max(1, args.steps))

    for _ in range(max(1, args.warmup)):
        window()
    c0 = H.hcw_launch_count()
    host_ms = timed(window, max(1, args.steps))
    launches = (H.hcw_launch_count() - c0) / max(1, args.steps) / n
    graph_ms = graph_time()
    # the same window with the tcgen05 contraction (hcw_set_decode_kernel)
    prev = H.hcw_set_decode_kernel(H.HCW_DECODE_TCGEN05)
    try:
        window()
        tc_ms = graph_time()
    finally:
        H.hcw_set_decode_kernel(prev)
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error")
    wbytes = 2.0 * L * d * d * 2
    peaks, _ = load_peaks()
    us = graph_ms * 1e3 / n
    print(json.dumps({
        "kernel": "decode", "batch": B, "n": n, "d": d, "L": L, "schedule": args.schedule,
        "cache_bytes": cache.numel(), "launches_per_position": launches,
        "us_per_position_host_issued": round(host_ms * 1e3 / n, 2),
        "us_per_position_graph": round(us, 2),
        "us_per_position_graph_tcgen05": round(tc_ms * 1e3 / n, 2),
        "tokens_per_s_graph": round(B / (us * 1e-6)),
        "weight_bytes_per_position": wbytes,
        "weight_gbs_graph": round(wbytes / (us * 1e-6) / 1e9, 1),
        "hbm_peak_gbs": peaks.get("hbm_gbs")}), flush=True)
    return 0


BLOCK_BF16 = {"E", "P", "W_self", "W_nbr", "W1", "W2", "Wh"}


def run_block(args, w, dev):
    """Time one training step (forward, loss, backward) of the character-LM
    block around the workload's stack (hcw_block_step: hidden 2d, 256 symbols)
    for --batch sequences, issued from the host and as a CUDA graph."""
    import torch

    from paper_2609_18145_gb300 import hcw as H
    from paper_2609_18145_gb300 import synth

    B, n, d, L = args.batch, w["n"], w["d"], w["L"]
    h, V = 2 * d, 256
    pr = synth.block_problem(B, n, d, h, V, L, seed=0)
    params = {f: torch.from_numpy(getattr(pr, f)).to(
        torch.bfloat16 if f in BLOCK_BF16 else torch.float32).to(dev).contiguous()
        for f in H.BLOCK_FIELDS}
    ids = torch.from_numpy(pr.ids.astype("int32")).to(dev)
    grads = {f: torch.empty(tuple(params[f].shape), dtype=torch.float32, device=dev)
             for f in H.BLOCK_FIELDS}
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    ws = torch.empty(H.hcw_block_workspace_bytes(B, n, d, h, V, L), dtype=torch.uint8, device=dev)

    def step():
        H.hcw_block_step(ids, params, grads, loss=loss, workspace=ws)

    def timed(fn, reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record()
        for _ in range(reps):
            fn()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    for _ in range(max(1, args.warmup)):
        step()
    c0 = H.hcw_launch_count()
    host_ms = timed(step, max(1, args.steps))
    launches = (H.hcw_launch_count() - c0) / max(1, args.steps)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            step()
    torch.cuda.synchronize()
    g.replay()
    graph_ms = timed(g.replay, max(1, args.steps))
    if H.hcw_sync_status() != H.HCW_OK:
        raise SystemExit("device error")
    T = B * n
    flops = T * (L * (9.0 * d * d + 12.0 * d * h) + 6.0 * d * V)
    print(json.dumps({
        "kernel": "block", "batch": B, "n": n, "d": d, "hidden": h, "vocab": V, "L": L,
        "loss": float(loss.item()), "launches_per_step": launches,
        "ms_per_step_host_issued": round(host_ms, 4), "ms_per_step_graph": round(graph_ms, 4),
        "tokens_per_s_graph": round(T / (graph_ms * 1e-3)),
        "flops_per_step": flops, "tflops_graph": round(flops / (graph_ms * 1e-3) / 1e12, 1)}),
        flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-graph", action="store_true",
                    help="issue every step's launches from the host instead of replaying a "
                         "CUDA graph of them")
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="skip timing the CPU oracle (it is only timed at N = 1 anyway)")
    ap.add_argument("--kernel", choices=("fwd", "dx", "dw", "step", "decode", "block"),
                    help="launch only this kernel kind, one whole step of --batch sequences "
                         "(profiler captures), decode one window of --batch sequences "
                         "token by token, or one training step of the character-LM block "
                         "around the stack; no bench line")
    ap.add_argument("--batch", type=int, default=64, help="sequences for --kernel runs")
    ap.add_argument("--schedule", choices=tuple(SCHEDULES), default="rot",
                    help="layer schedule of the stack: rot (the workload's rotated stack) or "
                         "hy256 (the near and jump layers of the paper's window-256 hybrid)")
    ap.add_argument("--workload", choices=("charlm_w256_d512",) + tuple(WORKLOADS_EXTRA),
                    default="charlm_w256_d512",
                    help="configuration of the bench line: the metric's char-LM window-256 "
                         "shape (default), or one of the other configurations")
    ap.add_argument("--stack-kernels", choices=tuple(STACK_KERNELS), default="auto",
                    help="kernel family of the stacked forward and input gradient "
                         "(hcw_set_stack_kernels); auto is the streaming family")
    args = ap.parse_args()
    if args.kernel:
        return run_kernel_only(args)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.steps < 1:
        ap.error("--steps must be at least 1")
    if args.impl == "reference":
        return run_reference(args)
    if args.workload != WORKLOAD:
        return run_workload(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
