#!/usr/bin/env python3
"""Benchmark of the GB300 Frac scan (one JSON line on rank 0).

Headline: the training-shaped layer step (forward + backward of the chunked scan) on
B8 L4096 H64 P64 N128 K8 bf16 inputs, in tokens/s (whole job, all ranks), with the roofline
fraction of its dominant kernel and of the whole step, an end-to-end number through host
buffers, and the fp64 CPU oracle on a bounded sample of the same workload.  The same line
carries every other workload of the metric, each with its own roofline and oracle baseline:
  configs.c1  float32 forward, B1 L256 H2 P32 N16 K4 (latency-bound; microseconds)
  configs.c2  bf16 forward, B4 L2048 H16 P64 N64 K8
  configs.c4  long-context prefill, B1 L65536 H64 P64 N128 K8, Delta skewed small
  configs.c5  decode, B128 H64 P64 N128 K8, float32 state, 1024 steps after a 512-token prefill
  paper_shape the paper's layer (H16, head dim 256, N 1, K 16): batch-1 prefill at 1K/4K/16K
              tokens, batch-1 decode
  mixer       the scan-parameter and mixer-glue kernels at the training shape (HBM-bound)

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {gb300,reference}]
Under torchrun (N > 1) every rank runs an independent replica of the workload (the scan
shards over batch with no exchange) and rank 0 prints the line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Frac scan tokens/s (prefill, fwd+bwd) and % of GB300 roofline; decode tok/s"
TRAIN = "train_bf16_b8_l4096"
F32 = "fwd_f32_small"
FWD = "fwd_bf16_b4_l2048"
DECODE = "decode_b128"
PREFILL = "prefill_bf16_l65536"
FALLBACK_PEAKS = dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0,
                      sm_max_mhz=2070.0)
NUM_SMS = 152
L2_BYTES = 129 * 2 ** 20


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--decode-steps", type=int, default=1024)
    ap.add_argument("--no-configs", action="store_true", help="headline training step only")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the training workload's batch (small profiling captures)")
    ap.add_argument("--only", default="",
                    help="comma list of sections to run (train, c1, c2, c4, c5, paper, mixer); "
                         "for profiling captures")
    return ap.parse_args()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        p["source"] = "measured"
        return p
    p = dict(FALLBACK_PEAKS)
    p["source"] = "fallback"
    return p


def alu_peak_tflops(peaks):
    """CUDA-core float32 FMA peak: SMs x 128 lanes x 2 flops x max SM clock."""
    return NUM_SMS * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="frac_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", self.gpu_id], stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        sm, mx, reasons = [], [], set()
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for name, v in zip(self.NAMES, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


def gpu_id_for(dev_index: int) -> str:
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev_index).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            return vis.split(",")[dev_index]
        return str(dev_index)


# ----------------------------------------------------------------------------- work counts
def shape_of(name):
    from paper_2609_36314_gb300 import synth
    return synth.WORKLOADS[name]


def kpn(s):
    return s.nmodes * s.headdim * s.dstate


def fwd_flops_per_token_head(s, q=128):
    """The forward's algorithmic flops: state update 2KPN + readout 2KPN + the causal
    intra-chunk products Q P (times X) and Q N G / H (C B^T, shared by the group's heads)."""
    return 4 * kpn(s) + q * s.headdim + q * s.dstate * s.ngroups / s.nheads


def train_flops_per_token_head(s, q=128):
    """Forward + backward: 14KPN + 3QP + 2QN G/H (forward above; backward: reverse pass 2KPN,
    inter-chunk readout and dx 4KPN, dC and dB 4KPN, the intra products 2QP + QN G/H)."""
    return 14 * kpn(s) + 3 * q * s.headdim + 2 * q * s.dstate * s.ngroups / s.nheads


def intra_pair_flops_per_token_head(s, q=128):
    """FP32 work of the intra-chunk backward by its definition: for each pair k <= t of a chunk
    ((q + 1) / 2 pairs per token) and each mode, the decay factor's contributions to Gamma,
    Gamma', the read-weight gradient and the kappa gradient, one multiply-add (2 flops) each."""
    return (q + 1) / 2 * s.nmodes * 8


def fwd_bytes_per_token_head(s):
    """Algorithmic bytes of the forward per token-head: x and y, the three controls, the two
    weight rows, and B, C shared by the group's heads."""
    es = 2 if s.dtype == "bf16" else 4
    return 2 * s.headdim * es + 12 + 2 * s.nmodes * es + 2 * s.dstate * es * s.ngroups / s.nheads


# DRAM bytes (read + write) per launch of each tensor-core kernel from one ncu capture of the
# training shape at batch 2 (dram__bytes_read.sum + dram__bytes_write.sum of every launch of the
# step, averaged; the summary is kept under profiles/); the per-chunk state traffic grows in
# proportion to the batch, so a run at batch B reports bytes x B / 2.  A figure is used only while
# the kernel's sources hash to the digest they had when they were profiled.
PROFILED_TRAFFIC_BATCH = 2
PROFILED_TRAFFIC = {
    "coef_tc": ("scan_tc.cu", "6165989fffff61ad", 23.10e6 + 38.93e6),
    "state_pass_fwd_tc": ("scan_tc.cu", "6165989fffff61ad", 138.87e6 + 479.23e6),
    "chunk_fwd_tc": ("scan_tc.cu", "6165989fffff61ad", 717.33e6 + 57.85e6),
    "state_pass_rev_tc": ("scan_tc.cu", "6165989fffff61ad", 139.00e6 + 479.77e6),
    "bwd_intra_tc": ("scan_tc_bwd.cu", "0352bc18c55c4601", 183.02e6 + 122.53e6),
    "bwd_state_tc": ("scan_tc_bwd.cu", "0352bc18c55c4601", 1467.70e6 + 167.03e6),
    "bwd_final_tc": ("scan_tc_bwd.cu", "0352bc18c55c4601", 323.47e6 + 67.30e6),
}

# DRAM bytes (read + write) per launch of the scan-parameter and mixer-glue kernels at the
# benchmark's training shape (B8 L4096), from one ncu capture of bench.py's mixer section.
PROFILED_MIXER_TRAFFIC = {
    "param_prep_fwd": ("param_prep.cu", "60ecfacdc7d4a027", 92.31e6 + 43.81e6),
    "param_prep_bwd": ("param_prep.cu", "60ecfacdc7d4a027", 184.63e6 + 60.37e6),
    "conv1d_fwd": ("mixer_glue.cu", "c05c49b825953b57", 285.36e6 + 233.22e6),
    "conv1d_bwd": ("mixer_glue.cu", "c05c49b825953b57", 570.67e6 + 252.29e6),
    "gated_rmsnorm_fwd": ("mixer_glue.cu", "c05c49b825953b57", 536.95e6 + 235.98e6),
    "gated_rmsnorm_bwd": ("mixer_glue.cu", "c05c49b825953b57", 805.43e6 + 491.07e6),
}

# DRAM bytes (read + write) of one decode_step launch of the decode workload (B128 H64 P64 N128
# K8, float32 state), from one ncu capture (summarised under profiles/); used only while
# decode.cu hashes to the digest it had when profiled.
PROFILED_DECODE_TRAFFIC = ("decode.cu", "853bdd0b44e394c4", 2151.50e6 + 2098.02e6)


def source_digest(fname: str) -> str:
    import hashlib
    src = os.path.join(ROOT, "paper_2609_36314_gb300", "csrc")
    m = hashlib.sha256()
    for f in (fname, "tc.cuh", "tc_util.cuh", "common.cuh", "kernels.h"):
        with open(os.path.join(src, f), "rb") as fh:
            m.update(fh.read())
    return m.hexdigest()[:16]


def profiled_traffic(kernel: str, batch: int):
    """DRAM bytes per launch at this batch from the committed ncu capture, or None."""
    entry = PROFILED_TRAFFIC.get(kernel)
    if entry is None or source_digest(entry[0]) != entry[1]:
        return None
    return entry[2] * batch / PROFILED_TRAFFIC_BATCH


def algorithmic_work(kernel: str, s, per_launch_units: float):
    """Algorithmic flops or bytes of one launch of a scan kernel over `per_launch_units`
    token-heads: state contractions count 2 K P N flops per token-head each."""
    per_th = {
        "state_pass_fwd_simt": 2, "state_pass_rev_simt": 2, "chunk_fwd_simt": 2,
        "chunk_bwd_simt": 8, "state_pass_fwd_tc": 2, "state_pass_rev_tc": 2,
    }
    if kernel in per_th:
        return "flops", per_th[kernel] * kpn(s) * per_launch_units
    # kernels with the intra-chunk terms: the readout (2 K P N) plus the causal intra-chunk
    # products (Q P per token-head, and Q N per token for the C B^T shared by the heads of a group)
    q = 128
    if kernel == "chunk_fwd_tc":
        return "flops", (2 * kpn(s) + q * s.headdim + q * s.dstate * s.ngroups / s.nheads) * per_launch_units
    if kernel == "bwd_state_tc":  # Z, U, dC, dB contractions + the head-summed intra dC, dB
        return "flops", (8 * kpn(s) + 4 * q * s.dstate * s.ngroups / s.nheads) * per_launch_units
    if kernel == "bwd_intra_tc":
        return "flops", (2 * q * s.headdim + q * s.dstate * s.ngroups / s.nheads) * per_launch_units
    if kernel == "coef_tc":  # dt, alpha, lam, w_read, w_write in; f, s, u, exp(-E/tau), E, kappa out
        return "bytes", (12 + 4 * s.nmodes + 16 * s.nmodes + 4 * (16 if s.nmodes == 8 else 8)) * per_launch_units
    if kernel == "bwd_final_tc":  # per-position terms, dx_acc, dy, x in; dx and the scalar grads out
        return "bytes", (36 + 14 * s.nmodes + 10 * s.headdim) * per_launch_units
    if kernel == "decode_step":
        return "bytes", 2.0 * 4 * kpn(s) * per_launch_units
    return None, None


def roofline_of(kernel, kind, work, avg_ms, peaks, traffic=None):
    """The roofline object of one kernel (or of a whole call when `kernel` says so)."""
    s = avg_ms / 1e3
    if kind == "flops_tc":
        peak = peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops"))
        ach = work / s / 1e12
        return {"kernel": kernel, "bound": "tensor", "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak, "traffic": traffic,
                "peak_source": peaks["source"] + " (bf16, sustained)"}
    if kind == "flops_alu":
        peak = alu_peak_tflops(peaks)
        ach = work / s / 1e12
        return {"kernel": kernel, "bound": "alu", "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak, "traffic": traffic,
                "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 x max SM clock"}
    ach = work / s / 1e9
    return {"kernel": kernel, "bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"],
            "unit": "GB/s", "frac": ach / peaks["hbm_gbs"], "traffic": traffic,
            "peak_source": peaks["source"]}


# ----------------------------------------------------------------------------- CPU baselines
def cpu_scan(s, sample, nthreads, backward=False, seed=1):
    """The oracle (fp64, OpenMP over (batch, head) streams) on `sample` = (batch rows, heads,
    seqlen) of workload s; tokens/s in full-layer tokens (the cost is linear in token-heads:
    heads are independent streams)."""
    from oracle import oracle
    from paper_2609_36314_gb300 import synth
    rows, heads, L = sample
    sub = s.replace(batch=rows, nheads=heads, seqlen=L)
    d = {k: synth.to_f64(v) for k, v in synth.make_scan_inputs(sub, seed=seed, with_dy=backward).items()}
    t0 = time.perf_counter()
    oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"], d["w_read"],
               d["w_write"], d["D"], nthreads=nthreads)
    if backward:
        oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"], d["w_read"],
                   d["w_write"], d["D"], d["dy"], nthreads=nthreads)
    dt = time.perf_counter() - t0
    tokens = rows * L * heads / s.nheads
    return {"value": tokens / dt, "unit": "tokens/s", "cores": nthreads, "kind": "oracle",
            "sample": f"{'fwd+bwd' if backward else 'fwd'} of {rows} batch row(s) x {heads}/{s.nheads} "
                      f"heads x {L} tokens ({dt:.1f} s), in full-layer tokens"}


def cpu_decode(s, rows, steps, seed=2):
    """The oracle's decode step on `rows` batch rows (all heads) for `steps` steps, one core.
    The rows are independent streams, so the rate in rows x steps / s scales with the batch."""
    import numpy as np

    from oracle import oracle
    from paper_2609_36314_gb300 import synth
    sub = s.replace(batch=rows)
    dec = {k: synth.to_f64(v) for k, v in synth.make_decode_inputs(sub, steps, seed=seed).items()}
    st = np.zeros((rows, s.nheads, s.nmodes, s.headdim, s.dstate))
    t0 = time.perf_counter()
    for t in range(steps):
        _, st = oracle.decode(dec["x"][t], dec["dt"][t], dec["alpha"][t], dec["lam"][t], dec["tau"],
                              dec["B"][t], dec["C"][t], dec["w_read"][t], dec["w_write"][t],
                              dec["D"], st)
    dt = time.perf_counter() - t0
    return {"value": rows * steps / dt, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"{rows} batch row(s) (all {s.nheads} heads) x {steps} decode steps ({dt:.1f} s)"}


def cpu_baselines(nthreads):
    """Oracle baselines of every workload: all host cores and one core, on bounded samples."""
    s1, s2, s3, s4 = shape_of(F32), shape_of(FWD), shape_of(TRAIN), shape_of(PREFILL)
    return {
        "c1": [cpu_scan(s1, (1, 2, 256), nthreads), cpu_scan(s1, (1, 2, 256), 1)],
        "c2": [cpu_scan(s2, (4, 16, 2048), nthreads), cpu_scan(s2, (1, 2, 2048), 1)],
        "c3": [cpu_scan(s3, (2, 64, 4096), nthreads, backward=True),
               cpu_scan(s3, (1, 1, 1024), 1, backward=True)],
        "c4": [cpu_scan(s4, (1, 16, 8192), nthreads), cpu_scan(s4, (1, 1, 4096), 1)],
        "c5": [cpu_decode(shape_of(DECODE), 1, 32)],
    }


def run_reference(args, rank):
    """The fp64 CPU oracle on a bounded sample of the training workload, per step."""
    if rank != 0:
        return
    from oracle import oracle
    from paper_2609_36314_gb300 import synth
    s = shape_of(TRAIN)
    heads = 4
    sub = s.replace(batch=1, nheads=heads)
    host = synth.make_scan_inputs(sub, seed=0, with_dy=True)
    d = {k: synth.to_f64(v) for k, v in host.items()}

    def step():
        oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                   d["w_read"], d["w_write"], d["D"])
        oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                   d["w_read"], d["w_write"], d["D"], d["dy"])

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    tokens = sub.seqlen * heads / s.nheads  # token-heads of the sample in full-layer tokens
    value = tokens * args.steps / dt
    cores = oracle.max_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{TRAIN} sample: batch row 0, heads 0-{heads - 1}, L={s.seqlen}, "
                               "fwd+bwd", "global_batch": 1, "seq_len": s.seqlen},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"1 x {s.seqlen} tokens x {heads}/{s.nheads} heads per step"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU helpers
class Ctx:
    """Device, peaks, rank plumbing and the L2 flush buffer shared by the measurements."""

    def __init__(self, dev, world, peaks):
        import torch
        import torch.distributed as dist
        self.torch, self.dist = torch, dist
        self.dev, self.world, self.peaks = dev, world, peaks
        self._flush = None

    def barrier(self):
        if self.world > 1:
            self.dist.barrier()

    def max_over_ranks(self, v):
        if self.world == 1:
            return v
        t = self.torch.tensor([v], device=self.dev, dtype=self.torch.float64)
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def flush_l2(self):
        """Writes a buffer twice the size of L2 (evicts the inputs of small workloads)."""
        if self._flush is None:
            self._flush = self.torch.empty(2 * L2_BYTES, dtype=self.torch.uint8, device=self.dev)
        self._flush.zero_()

    def time(self, fn, iters, flush=False, warmup=3):
        """Mean device milliseconds of fn() (CUDA events on the current stream, a synchronize
        and a barrier on both sides), max over ranks; with flush, L2 is flushed before every
        call (outside its timed span).  Also returns {kernel: (launches, total ms)} from the
        library's launch tracing."""
        from paper_2609_36314_gb300 import _lib
        torch = self.torch
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        _lib.trace_reset()
        _lib.trace_enable(True)
        self.barrier()
        stream = torch.cuda.current_stream()
        total = 0.0
        if flush:
            for _ in range(iters):
                self.flush_l2()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                fn()
                e1.record(stream)
                torch.cuda.synchronize()
                total += e0.elapsed_time(e1)
        else:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(iters):
                fn()
            e1.record(stream)
            torch.cuda.synchronize()
            total = e0.elapsed_time(e1)
        self.barrier()
        _lib.trace_enable(False)
        trace = _lib.trace_collect()
        return self.max_over_ranks(total / iters), trace


def kernel_table(trace, iters):
    tot = sum(t for _, t in trace.values()) or 1.0
    return {k: {"launches_per_call": n / iters, "avg_ms": t / max(n, 1), "share": t / tot}
            for k, (n, t) in trace.items()}


def dominant(trace):
    return max(trace.items(), key=lambda kv: kv[1][1])[0] if trace else None


# ----------------------------------------------------------------------------- C3 headline
def bench_train(args, ctx, rank, local):
    import torch

    from paper_2609_36314_gb300 import scan_bwd, scan_fwd, synth
    from paper_2609_36314_gb300.api import bwd_workspace_size, fwd_workspace_size, make_dims
    dev, peaks = ctx.dev, ctx.peaks
    s = shape_of(TRAIN)
    if args.batch:
        s = s.replace(batch=args.batch)
    inp = synth.make_scan_inputs_torch(s, seed=1000 + rank, device=dev, with_dy=True)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    # one workspace for both calls: the backward reuses the per-chunk states of the forward
    ws = torch.empty(max(bwd_workspace_size(dims), fwd_workspace_size(dims)), dtype=torch.uint8,
                     device=dev)
    y = torch.empty_like(inp["x"])
    grads = dict(dx=torch.empty_like(inp["x"]), ddt=torch.empty_like(inp["dt"]),
                 dalpha=torch.empty_like(inp["alpha"]), dlam=torch.empty_like(inp["lam"]),
                 dB=torch.empty_like(inp["B"]), dC=torch.empty_like(inp["C"]),
                 dw_read=torch.empty_like(inp["w_read"]), dw_write=torch.empty_like(inp["w_write"]),
                 dD=torch.empty_like(inp["D"]), dh0=None)

    def train_step_on(a, y, grads):
        scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], want_final_state=False, y=y, workspace=ws)
        scan_bwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], a["dy"], workspace=ws, out=grads, reuse_fwd_states=True)

    clocks = ClockSampler(gpu_id_for(local)) if rank == 0 else None
    if clocks:
        clocks.start()
    ms, trace = ctx.time(lambda: train_step_on(inp, y, grads), args.steps,
                         warmup=max(args.warmup, 3))
    clk = clocks.stop() if clocks else None
    tokens_per_step = s.batch * s.seqlen
    value = ctx.world * tokens_per_step / (ms / 1e3)
    units = s.batch * s.seqlen * s.nheads
    kern = kernel_table(trace, args.steps)
    for k in kern:
        tb = profiled_traffic(k, s.batch)
        if tb is not None and kern[k]["avg_ms"] > 0:  # DRAM bytes of the ncu capture / launch time
            kern[k]["dram_gbs"] = tb / (kern[k]["avg_ms"] / 1e3) / 1e9
            kern[k]["dram_frac_of_peak"] = kern[k]["dram_gbs"] / peaks["hbm_gbs"]
        kind, work = algorithmic_work(k, s, units)
        if kind == "flops":
            kern[k]["achieved_tflops"] = work / (kern[k]["avg_ms"] / 1e3) / 1e12
            kern[k]["frac_of_bf16_sustained"] = kern[k]["achieved_tflops"] / peaks.get(
                "bf16_tflops_sustained", peaks.get("bf16_tflops"))
        elif kind == "bytes":
            kern[k]["achieved_gbs"] = work / (kern[k]["avg_ms"] / 1e3) / 1e9
    if "bwd_intra_tc" in kern:  # its real bound: the per-pair FP32 work on the CUDA cores
        kern["bwd_intra_tc"]["roofline_alu"] = roofline_of(
            "bwd_intra_tc", "flops_alu", intra_pair_flops_per_token_head(s) * units,
            kern["bwd_intra_tc"]["avg_ms"], peaks)
    dom = dominant(trace)
    roofline = None
    if dom:
        kind, work = algorithmic_work(dom, s, units)
        if dom == "bwd_intra_tc":  # bound by its per-pair FP32 work, not by its small tensor-core products
            roofline = dict(kern[dom]["roofline_alu"], traffic=profiled_traffic(dom, s.batch))
        elif kind == "flops":
            roofline = roofline_of(dom, "flops_tc" if dom.endswith("_tc") else "flops_alu", work,
                                   kern[dom]["avg_ms"], peaks, profiled_traffic(dom, s.batch))
        elif kind == "bytes":
            roofline = roofline_of(dom, "bytes", work, kern[dom]["avg_ms"], peaks)
    step_roof = roofline_of("whole training step", "flops_tc",
                            train_flops_per_token_head(s) * units, ms, peaks)
    launches = sum(n for n, _ in trace.values())
    e2e = None if args.no_e2e else bench_e2e(args, ctx, inp, y, grads, train_step_on, tokens_per_step)
    del ws
    torch.cuda.empty_cache()
    return dict(s=s, ms=ms, value=value, kern=kern, roofline=roofline, step_roof=step_roof,
                launches=launches, clk=clk, e2e=e2e,
                dtype="bf16" if any(k.endswith("_tc") for k in trace) else "f32")


def bench_e2e(args, ctx, inp, y, grads, train_step_on, tokens_per_step):
    """End to end through pinned host buffers: every step copies its inputs host -> device and
    all its results device -> host inside the timed region, pipelined over two buffer sets the
    way a training loop with a prefetching loader runs (step s's inputs copy in on one stream
    while step s - 1 computes, its results copy out on another while step s + 1 computes)."""
    import torch
    hin = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True).copy_(v) for k, v in inp.items()}
    hout = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True)
            for k, v in grads.items() if v is not None}
    hout["y"] = torch.empty(y.shape, dtype=y.dtype, pin_memory=True)
    h2d = sum(v.numel() * v.element_size() for v in hin.values())
    d2h = sum(v.numel() * v.element_size() for v in hout.values())
    sets_in = [inp, {k: torch.empty_like(v) for k, v in inp.items()}]
    sets_out = [(y, grads), (torch.empty_like(y),
                             {k: (torch.empty_like(v) if v is not None else None) for k, v in grads.items()})]
    comp = torch.cuda.current_stream()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event(), torch.cuda.Event()]    # inputs of set i on the device
    ev_done = [torch.cuda.Event(), torch.cuda.Event()]  # the step that used set i has finished
    ev_out = [torch.cuda.Event(), torch.cuda.Event()]   # results of set i read back

    def copy_in(st):
        i = st % 2
        with torch.cuda.stream(s_in):
            if st >= 2:
                s_in.wait_event(ev_done[i])
            for k, v in hin.items():
                sets_in[i][k].copy_(v, non_blocking=True)
            ev_in[i].record(s_in)

    def compute(st):
        i = st % 2
        comp.wait_event(ev_in[i])
        if st >= 2:
            comp.wait_event(ev_out[i])
        train_step_on(sets_in[i], sets_out[i][0], sets_out[i][1])
        ev_done[i].record(comp)

    def copy_out(st):
        i = st % 2
        y_i, g_i = sets_out[i]
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_done[i])
            for k, v in hout.items():
                v.copy_(g_i[k] if k != "y" else y_i, non_blocking=True)
            ev_out[i].record(s_out)

    def e2e_run(nsteps):
        copy_in(0)
        for st in range(nsteps):
            if st + 1 < nsteps:
                copy_in(st + 1)
            compute(st)
            copy_out(st)
        comp.wait_event(ev_out[(nsteps - 1) % 2])

    e2e_run(2)
    torch.cuda.synchronize()
    ctx.barrier()
    n = max(2, args.steps)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(comp)
    s_in.wait_event(ev0)
    e2e_run(n)
    ev1.record(comp)
    torch.cuda.synchronize()
    ctx.barrier()
    ms = ctx.max_over_ranks(ev0.elapsed_time(ev1) / n)
    return {"value": ctx.world * tokens_per_step / (ms / 1e3), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms}


# ----------------------------------------------------------------------------- other workloads
def bench_forward(ctx, name, iters, flush, seed, tensor_bound):
    """Forward scan of workload `name` (final state kept)."""
    import torch

    from paper_2609_36314_gb300 import scan_fwd, synth
    from paper_2609_36314_gb300.api import fwd_workspace_size, make_dims
    s = shape_of(name)
    a = synth.make_scan_inputs_torch(s, seed=seed, device=ctx.dev)
    dty = torch.bfloat16 if s.dtype == "bf16" else torch.float32
    chunk = s.chunk if s.dtype == "f32" else 0
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes, dty,
                     chunk=chunk)
    ws = torch.empty(fwd_workspace_size(dims), dtype=torch.uint8, device=ctx.dev)
    y = torch.empty_like(a["x"])
    hf = torch.empty((s.batch, s.nheads, s.nmodes, s.headdim, s.dstate), dtype=torch.float32,
                     device=ctx.dev)

    def fwd():
        scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], y=y, h_final=hf, workspace=ws, chunk=chunk)

    ms, trace = ctx.time(fwd, iters, flush=flush)
    units = s.batch * s.seqlen * s.nheads
    work = fwd_flops_per_token_head(s, 128 if tensor_bound else (s.chunk or 64)) * units
    out = {"workload": f"{name}: forward of B{s.batch} L{s.seqlen} H{s.nheads} P{s.headdim} "
                       f"N{s.dstate} K{s.nmodes} G{s.ngroups}, {s.dtype} inputs, final state kept",
           "ms_per_forward": ms, "us_per_forward": 1e3 * ms,
           "value": ctx.world * s.batch * s.seqlen / (ms / 1e3), "unit": "tokens/s",
           "l2": "flushed before every timed call" if flush else "inputs larger than L2, no flush",
           "gpu_launches_per_call": sum(n for n, _ in trace.values()) / iters,
           "kernels": kernel_table(trace, iters),
           "roofline": roofline_of("whole forward", "flops_tc" if tensor_bound else "flops_alu",
                                   work, ms, ctx.peaks)}
    dom = dominant(trace)
    if dom:
        kind, kw = algorithmic_work(dom, s, units)
        if kind == "flops":
            out["roofline_dominant"] = roofline_of(dom, "flops_tc" if dom.endswith("_tc") else "flops_alu",
                                                   kw, out["kernels"][dom]["avg_ms"], ctx.peaks)
    del a, ws, y, hf
    torch.cuda.empty_cache()
    return out


def bench_decode(args, ctx):
    import torch

    from paper_2609_36314_gb300 import decode_step, scan_fwd, synth
    s = shape_of(DECODE)
    pre = synth.make_scan_inputs_torch(s, seed=7, device=ctx.dev)
    _, state = scan_fwd(pre["x"], pre["dt"], pre["alpha"], pre["lam"], pre["tau"], pre["B"],
                        pre["C"], pre["w_read"], pre["w_write"], pre["D"])
    del pre
    T = args.decode_steps
    stp = synth.make_scan_inputs_torch(s.replace(seqlen=T), seed=8, device=ctx.dev)
    # [B, T, ...] -> [T, B, ...] so that every step reads contiguous inputs
    stp = {k: (v.transpose(0, 1).contiguous() if k not in ("tau", "D") else v)
           for k, v in stp.items()}
    ybuf = torch.empty((T, s.batch, s.nheads, s.headdim), dtype=torch.bfloat16, device=ctx.dev)

    def steps():
        for t in range(T):
            decode_step(stp["x"][t], stp["dt"][t], stp["alpha"][t], stp["lam"][t], stp["tau"],
                        stp["B"][t], stp["C"][t], stp["w_read"][t], stp["w_write"][t],
                        stp["D"], state, y_t=ybuf[t])

    steps()  # warm-up
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        steps()
    ms, _ = ctx.time(g.replay, 2, warmup=1)
    ms_step = ms / T
    work = 2.0 * 4 * s.batch * s.nheads * kpn(s)
    traffic = (PROFILED_DECODE_TRAFFIC[2]
               if source_digest(PROFILED_DECODE_TRAFFIC[0]) == PROFILED_DECODE_TRAFFIC[1] else None)
    out = {"workload": f"{DECODE}: B{s.batch} H{s.nheads} P{s.headdim} N{s.dstate} K{s.nmodes}, "
                       f"float32 state, 512-token prefill then {T} steps in one CUDA graph",
           "value": ctx.world * s.batch / (ms_step / 1e3), "unit": "tokens/s",
           "us_per_step": 1e3 * ms_step, "gpu_launches_per_step": 1,
           "l2": "state 2.15 GB, larger than L2",
           "roofline": roofline_of("decode_step", "bytes", work, ms_step, ctx.peaks, traffic)}
    del stp, ybuf, state, g
    torch.cuda.empty_cache()
    return out


def bench_paper_shape(ctx):
    """The paper's own layer shape (H16, head dim 256, N = 1, K = 16 modes on the 1 .. 2^17
    bank): batch-1 prefill at 1K, 4K and 16K tokens (forward), and batch-1 decode (one CUDA
    graph of 64 steps, the length the paper averages its decode rate over)."""
    import torch

    from paper_2609_36314_gb300 import decode_step, scan_fwd, synth
    pts = []
    for L in (1024, 4096, 16384):
        s = synth.Shape(1, L, 16, 256, 1, 1, 16, 0, "bf16")
        a = synth.make_scan_inputs_torch(s, seed=13, device=ctx.dev)
        y = torch.empty_like(a["x"])

        def fwd():
            scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                     a["w_write"], a["D"], y=y)

        ms, trace = ctx.time(fwd, 10, flush=True)
        work = fwd_bytes_per_token_head(s) * L * s.nheads
        pts.append({"seqlen": L, "ms_per_forward": ms, "tokens_per_s": L / (ms / 1e3),
                    "kernels": kernel_table(trace, 10),
                    "roofline": roofline_of("whole forward", "bytes", work, ms, ctx.peaks)})
        del a, y
    # training-shaped step at the paper's layer: forward + backward over 4 packed 4K sequences
    from paper_2609_36314_gb300 import scan_bwd
    from paper_2609_36314_gb300.api import bwd_workspace_size, make_dims
    s = synth.Shape(4, 4096, 16, 256, 1, 1, 16, 0, "bf16")
    a = synth.make_scan_inputs_torch(s, seed=15, device=ctx.dev, with_dy=True)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    ws = torch.empty(bwd_workspace_size(dims), dtype=torch.uint8, device=ctx.dev)
    y = torch.empty_like(a["x"])

    def train():
        scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], y=y, want_final_state=False, workspace=ws)
        scan_bwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], a["dy"], workspace=ws, reuse_fwd_states=True)

    ms, trace = ctx.time(train, 5)
    tr = {"workload": "B4 L4096 H16 P256 N1 K16 bf16, forward + backward (the backward reuses "
                      "the forward's per-chunk states)",
          "ms_per_step": ms, "tokens_per_s": s.batch * s.seqlen / (ms / 1e3),
          "kernels": kernel_table(trace, 5)}
    del a, ws, y
    torch.cuda.empty_cache()
    s = synth.Shape(1, 64, 16, 256, 1, 1, 16, 0, "bf16")
    stp = synth.make_scan_inputs_torch(s, seed=14, device=ctx.dev)
    stp = {k: (v.transpose(0, 1).contiguous() if k not in ("tau", "D") else v) for k, v in stp.items()}
    state = torch.zeros((1, 16, 16, 256, 1), dtype=torch.float32, device=ctx.dev)
    ybuf = torch.empty((64, 1, 16, 256), dtype=torch.bfloat16, device=ctx.dev)

    def steps():
        for t in range(64):
            decode_step(stp["x"][t], stp["dt"][t], stp["alpha"][t], stp["lam"][t], stp["tau"],
                        stp["B"][t], stp["C"][t], stp["w_read"][t], stp["w_write"][t], stp["D"],
                        state, y_t=ybuf[t])

    steps()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        steps()
    ms, _ = ctx.time(g.replay, 20, warmup=2)
    us = 1e3 * ms / 64
    dec = {"us_per_step": us, "tokens_per_s": 1e6 / us, "batch": 1,
           "note": "64 steps in one CUDA graph; the state is 256 KB, so a step is launch-latency "
                   "bound, not bandwidth bound"}
    return {"workload": "paper layer shape: B1 H16 P256 N1 K16, tau geometric in [1, 2^17], bf16 "
                        "inputs; prefill = forward with L2 flushed before each call",
            "unit": "tokens/s", "prefill": pts, "decode": dec, "train": tr}


def bench_mixer(ctx):
    """The scan-parameter and mixer-glue kernels at the training shape (B8 L4096): each timed
    alone (inputs larger than L2), HBM roofline on its algorithmic bytes (inputs and outputs
    once)."""
    import torch

    from paper_2609_36314_gb300 import (conv1d_bwd, conv1d_fwd, gated_rmsnorm_bwd,
                                        gated_rmsnorm_fwd, param_prep_bwd, param_prep_fwd)
    dev = ctx.dev
    g = torch.Generator(device=dev)
    g.manual_seed(17)

    def n(*shape, dtype=torch.bfloat16):
        return torch.randn(shape, generator=g, device=dev, dtype=torch.float32).to(dtype)

    out = {}
    B, L, H, K = 8, 4096, 64, 8
    f32 = torch.float32
    raw = dict(dt_raw=n(B, L, H, dtype=f32), alpha_raw=n(B, L, H, dtype=f32),
               lam_raw=n(B, L, H, dtype=f32), g_read=0.5 * n(B, L, H, K), g_write=0.5 * n(B, L, H, K),
               tau=(2.0 ** (17.0 * torch.arange(K, device=dev) / (K - 1))).repeat(H, 1).contiguous(),
               dt_bias=torch.full((H,), -1.0, device=dev))
    up = dict(ddt=n(B, L, H, dtype=f32), dalpha=n(B, L, H, dtype=f32), dlam=n(B, L, H, dtype=f32),
              dw_read=n(B, L, H, K), dw_write=n(B, L, H, K))
    rows = B * L * H

    def add(name, fn, nbytes):
        # the call's time through the Python API, and the kernel's own device time (CUDA events
        # around its launch on the stream), which the roofline takes
        ms, trace = ctx.time(fn, 10)
        entry = PROFILED_MIXER_TRAFFIC.get(name)
        traffic = entry[2] if entry and source_digest(entry[0]) == entry[1] else None
        kms = trace[name][1] / max(trace[name][0], 1) if name in trace else ms
        out[name] = {"ms": ms, "kernel_ms": kms,
                     "gpu_launches_per_call": sum(c for c, _ in trace.values()) / 10,
                     "roofline": roofline_of(name, "bytes", nbytes, kms, ctx.peaks, traffic)}

    # prep: 3 float32 controls + 2 K bf16 logits in, 3 controls + 2 K weights out
    add("param_prep_fwd", lambda: param_prep_fwd(raw["dt_raw"], raw["alpha_raw"], raw["lam_raw"],
                                                 raw["g_read"], raw["g_write"], raw["tau"],
                                                 raw["dt_bias"]), rows * (24 + 8 * K))
    # backward: raw controls, logits, the 5 upstream gradients in; 3 + 2 K gradients out
    add("param_prep_bwd", lambda: param_prep_bwd(raw["dt_raw"], raw["alpha_raw"], raw["lam_raw"],
                                                 raw["g_read"], raw["g_write"], raw["tau"], up["ddt"],
                                                 up["dalpha"], up["dlam"], up["dw_read"], up["dw_write"],
                                                 raw["dt_bias"]), rows * (36 + 12 * K))
    del raw, up
    C, W = 4352, 4
    x, du = n(B, L, C), n(B, L, C)
    w = n(C, W, dtype=f32) * 0.5
    bias = n(C, dtype=f32) * 0.1
    add("conv1d_fwd", lambda: conv1d_fwd(x, w, bias, silu=True), B * L * C * 4)
    add("conv1d_bwd", lambda: conv1d_bwd(x, w, du, bias, silu=True), B * L * C * 6)
    del x, du
    D = 4096
    y, z, dout = n(B * L, D), n(B * L, D), n(B * L, D)
    wt = torch.ones(D, device=dev)
    add("gated_rmsnorm_fwd", lambda: gated_rmsnorm_fwd(y, z, wt), B * L * D * 6)
    add("gated_rmsnorm_bwd", lambda: gated_rmsnorm_bwd(y, z, wt, dout), B * L * D * 10)
    del y, z, dout
    torch.cuda.empty_cache()
    out["workload"] = ("training shape B8 L4096: prep over H64 K8 (bf16 logits); conv1d over 4352 "
                       "channels (d_inner 4096 + B, C of 128), width 4, SiLU; gated RMSNorm over "
                       "4096 features, one group; algorithmic bytes = inputs and outputs once")
    return out


# ----------------------------------------------------------------------------- main
def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank)
        return

    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", rank=rank, world_size=world, device_id=dev)
    ctx = Ctx(dev, world, load_peaks())
    only = set(x for x in args.only.split(",") if x)

    def want(sec):
        return (not only or sec in only) and (sec == "train" or not args.no_configs)

    tr = bench_train(args, ctx, rank, local) if want("train") else None
    configs = {}
    if want("c1"):
        configs["c1"] = bench_forward(ctx, F32, 50, True, 21, tensor_bound=False)
    if want("c2"):
        configs["c2"] = bench_forward(ctx, FWD, 20, True, 22, tensor_bound=True)
    if want("c4"):
        configs["c4"] = bench_forward(ctx, PREFILL, 5, False, 11, tensor_bound=True)
        configs["c4"]["workload"] += ("; chunk 128 (the tensor-core kernels' chunk; results are "
                                      "chunk-independent)")
    if want("c5"):
        configs["c5"] = bench_decode(args, ctx)
    paper = bench_paper_shape(ctx) if want("paper") else None
    mixer = bench_mixer(ctx) if want("mixer") else None

    if rank == 0:
        line = {"metric": METRIC, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "data": "synthetic", "peaks_source": ctx.peaks["source"]}
        if tr:
            s = tr["s"]
            line.update({
                "value": tr["value"], "unit": "tokens/s", "ms_per_step": tr["ms"],
                "dtype": tr["dtype"],
                "config": {"workload": f"{TRAIN}: forward + backward of the chunked scan, B{s.batch} "
                                       f"L{s.seqlen} H{s.nheads} P{s.headdim} N{s.dstate} K{s.nmodes} "
                                       f"G{s.ngroups}, bf16 inputs; tensor-core products take bf16 "
                                       "operands with float32 accumulation, the rest is float32",
                           "global_batch": s.batch * world, "seq_len": s.seqlen,
                           "parallelism": f"replicas{world}" if world > 1 else "single",
                           "l2": "inputs larger than L2 (0.78 GB per step), no flush"},
                "roofline": tr["roofline"], "roofline_step": tr["step_roof"],
                "kernels": tr["kern"], "gpu_launches": tr["launches"], "e2e": tr["e2e"],
                "clocks": tr["clk"]})
            if args.batch:
                line["config"]["workload"] += f" (batch overridden to {args.batch})"
        line["configs"] = configs
        if paper:
            line["paper_shape"] = paper
        if mixer:
            line["mixer"] = mixer
        if world == 1 and not args.no_cpu_baseline and not only:
            from oracle import oracle
            cb = cpu_baselines(oracle.max_threads())
            if tr:
                line["cpu_baseline"] = cb["c3"][0]
                line["cpu_baseline_1core"] = cb["c3"][1]
            for key in ("c1", "c2", "c4", "c5"):
                if key in configs:
                    configs[key]["cpu_baseline"] = cb[key][0]
                    if len(cb[key]) > 1:
                        configs[key]["cpu_baseline_1core"] = cb[key][1]
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
