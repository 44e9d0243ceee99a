#!/usr/bin/env python3
"""Benchmark of the GB300 Frac scan (one JSON line on rank 0).

Headline: the training-shaped layer step (forward + backward of the chunked scan) on
B8 L4096 H64 P64 N128 K8 bf16 inputs, in tokens/s (whole job, all ranks).  Also
reported: the decode step (B128 H64 P64 N128 K8, float32 state, 512-token prefill then
1024 single-token steps) in tokens/s, per-kernel device times, the roofline fraction of
the dominant kernel, an end-to-end number through host buffers, and the fp64 CPU oracle
timed on a bounded sample of the same workload.

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
DECODE = "decode_b128"
PREFILL = "prefill_bf16_l65536"
FALLBACK_PEAKS = dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0,
                      sm_max_mhz=2070.0)
NUM_SMS = 152


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--decode-steps", type=int, default=1024)
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--no-paper-shape", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the training workload's batch (small profiling captures)")
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


# ----------------------------------------------------------------------------- helpers
def shape_of(name):
    from paper_2609_36314_gb300 import synth
    return synth.WORKLOADS[name]


def kpn(s):
    return s.nmodes * s.headdim * s.dstate


# DRAM bytes (read + write) per launch of each tensor-core kernel from one ncu capture of the
# training shape at batch 2 (the ncu summary of these kernels kept under profiles/); the per-chunk state traffic
# grows in proportion to the batch, so a run at batch B reports bytes x B / 2.  A figure is used
# only while the kernel's sources hash to the digest they had when they were profiled.
PROFILED_TRAFFIC_BATCH = 2
PROFILED_TRAFFIC = {
    "coef_tc": ("scan_tc.cu", "900e85af153e741a", 23.101e6 + 41.631e6),
    "state_pass_fwd_tc": ("scan_tc.cu", "900e85af153e741a", 138.760e6 + 481.840e6),
    "chunk_fwd_tc": ("scan_tc.cu", "900e85af153e741a", 717.318e6 + 60.756e6),
    "state_pass_rev_tc": ("scan_tc.cu", "900e85af153e741a", 139.129e6 + 482.585e6),
    "bwd_intra_tc": ("scan_tc_bwd.cu", "a135ecad70d3c440", 182.952e6 + 126.667e6),
    "bwd_state_tc": ("scan_tc_bwd.cu", "a135ecad70d3c440", 1464.175e6 + 165.234e6),
    "bwd_final_tc": ("scan_tc_bwd.cu", "a135ecad70d3c440", 323.524e6 + 70.281e6),
}


# DRAM bytes (read + write) of one decode_step launch of the decode workload (B128 H64 P64 N128
# K8, float32 state), from one ncu capture (summarised under profiles/); used only while
# decode.cu hashes to the digest it had when profiled.
PROFILED_DECODE_TRAFFIC = ("decode.cu", "5a6ee76a91d8f3d2", 2151.500e6 + 2097.820e6)


def source_digest(fname: str) -> str:
    import hashlib
    src = os.path.join(os.path.dirname(os.path.abspath(__file__)), "paper_2609_36314_gb300", "csrc")
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
    """Algorithmic flops or bytes of one launch of `kernel` (the per-kernel counts below):
    state contractions count 2 K P N flops per token-head each."""
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


def cpu_baseline(rows=2):
    """The oracle (fp64, OpenMP over (batch, head) streams) on `rows` full batch rows of the
    training workload: all heads, the full sequence, forward + backward (about 10-15 s on 16
    cores)."""
    from oracle import oracle
    from paper_2609_36314_gb300 import synth
    s = shape_of(TRAIN)
    sub = s.replace(batch=rows)
    host = synth.make_scan_inputs(sub, seed=1, with_dy=True)
    d = {k: synth.to_f64(v) for k, v in host.items()}
    t0 = time.perf_counter()
    oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"], d["w_read"],
               d["w_write"], d["D"])
    oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"], d["w_read"],
               d["w_write"], d["D"], d["dy"])
    dt = time.perf_counter() - t0
    tokens = sub.batch * sub.seqlen
    return {"value": tokens / dt, "unit": "tokens/s", "cores": oracle.max_threads(),
            "kind": "oracle",
            "sample": f"fwd+bwd of batch rows 0-{rows - 1} (all {s.nheads} heads, L={s.seqlen}; "
                      f"{rows}/{s.batch} of the workload), {dt:.1f} s"}


# ----------------------------------------------------------------------------- GPU arm
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

    from paper_2609_36314_gb300 import _lib, scan_bwd, scan_fwd, synth
    from paper_2609_36314_gb300.api import bwd_workspace_size, fwd_workspace_size, make_dims

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", rank=rank, world_size=world, device_id=dev)
    peaks = load_peaks()

    def barrier():
        if world > 1:
            dist.barrier()

    def max_over_ranks(v):
        if world == 1:
            return v
        t = torch.tensor([v], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    s = shape_of(TRAIN)
    if args.batch:
        s = s.replace(batch=args.batch)
    inp = synth.make_scan_inputs_torch(s, seed=1000 + rank, device=dev, with_dy=True)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    # one workspace for both calls: the backward reuses the per-chunk states of the forward
    ws_b = torch.empty(max(bwd_workspace_size(dims), fwd_workspace_size(dims)), dtype=torch.uint8,
                       device=dev)
    ws_f = ws_b
    y = torch.empty_like(inp["x"])
    grads = dict(dx=torch.empty_like(inp["x"]), ddt=torch.empty_like(inp["dt"]),
                 dalpha=torch.empty_like(inp["alpha"]), dlam=torch.empty_like(inp["lam"]),
                 dB=torch.empty_like(inp["B"]), dC=torch.empty_like(inp["C"]),
                 dw_read=torch.empty_like(inp["w_read"]), dw_write=torch.empty_like(inp["w_write"]),
                 dD=torch.empty_like(inp["D"]), dh0=None)
    a = inp

    def train_step_on(a, y, grads):
        scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], want_final_state=False, y=y, workspace=ws_f)
        scan_bwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], a["dy"], workspace=ws_b, out=grads, reuse_fwd_states=True)

    def train_step():
        train_step_on(a, y, grads)

    for _ in range(max(args.warmup, 3)):
        train_step()
    torch.cuda.synchronize()

    clocks = ClockSampler(gpu_id_for(local)) if rank == 0 else None
    if clocks:
        clocks.start()
    _lib.trace_reset()
    _lib.trace_enable(True)
    barrier()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        train_step()
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    _lib.trace_enable(False)
    ms = ev0.elapsed_time(ev1) / args.steps
    trace = _lib.trace_collect()
    clk = clocks.stop() if clocks else None
    ms_max = max_over_ranks(ms)
    tokens_per_step = s.batch * s.seqlen
    value = world * tokens_per_step / (ms_max / 1e3)

    # per-kernel device time and the dominant kernel's roofline
    kern = {k: {"launches": n, "avg_ms": t / max(n, 1), "share": 0.0} for k, (n, t) in trace.items()}
    tot = sum(t for _, t in trace.values()) or 1.0
    for k, (n, t) in trace.items():
        kern[k]["share"] = t / tot
        tb = profiled_traffic(k, s.batch)
        if tb is not None and kern[k]["avg_ms"] > 0:  # DRAM bytes of the ncu capture / launch time
            kern[k]["dram_gbs"] = tb / (kern[k]["avg_ms"] / 1e3) / 1e9
            kern[k]["dram_frac_of_peak"] = kern[k]["dram_gbs"] / peaks["hbm_gbs"]
    launches = sum(n for n, _ in trace.values())
    dom = max(trace.items(), key=lambda kv: kv[1][1])[0] if trace else None
    roofline = None
    if dom:
        kind, work = algorithmic_work(dom, s, s.batch * s.seqlen * s.nheads)
        avg_s = kern[dom]["avg_ms"] / 1e3
        if kind == "flops" and dom.endswith("_tc"):
            # tensor-core kernel timed inside a long step: sustained bf16 peak
            peak = peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops"))
            ach = work / avg_s / 1e12
            roofline = {"kernel": dom, "bound": "tensor", "achieved": ach, "peak": peak,
                        "unit": "TFLOP/s", "frac": ach / peak,
                        "traffic": profiled_traffic(dom, s.batch),
                        "peak_source": peaks["source"] + " (bf16, sustained)"}
        elif kind == "flops":
            # CUDA-core float32 FMA peak: SMs x 128 lanes x 2 flops x max SM clock
            peak = NUM_SMS * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
            ach = work / avg_s / 1e12
            roofline = {"kernel": dom, "bound": "alu", "achieved": ach, "peak": peak,
                        "unit": "TFLOP/s", "frac": ach / peak, "traffic": None,
                        "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 x max SM clock"}
        elif kind == "bytes":
            ach = work / avg_s / 1e9
            roofline = {"kernel": dom, "bound": "hbm", "achieved": ach,
                        "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "frac": ach / peaks["hbm_gbs"], "traffic": None,
                        "peak_source": peaks["source"]}

    # end to end through host buffers (pinned), copies inside the timed region
    e2e = None
    if not args.no_e2e:
        hin = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True).copy_(v)
               for k, v in inp.items()}
        hout = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True)
                for k, v in grads.items() if v is not None}
        hout["y"] = torch.empty(y.shape, dtype=y.dtype, pin_memory=True)
        h2d = sum(v.numel() * v.element_size() for v in hin.values())
        d2h = sum(v.numel() * v.element_size() for v in hout.values())

        # Steps pipelined over two device copies of the inputs and of the results: step s copies
        # its inputs (pinned host -> set s % 2) on one stream while step s - 1 computes, and
        # reads its results back (set s % 2 -> pinned host) on another while step s + 1
        # computes.  Every step's copies lie inside the timed region.
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
        barrier()
        n_e2e = max(2, args.steps)
        ev0.record(comp)
        s_in.wait_event(ev0)
        e2e_run(n_e2e)
        ev1.record(comp)
        torch.cuda.synchronize()
        barrier()
        ms_e2e = max_over_ranks(ev0.elapsed_time(ev1) / n_e2e)
        e2e = {"value": world * tokens_per_step / (ms_e2e / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e}
        del hin, hout

    decode = None
    if not args.no_decode:
        decode = bench_decode(args, dev, peaks, world, max_over_ranks, barrier)
    prefill = None
    if not args.no_prefill:
        prefill = bench_prefill(args, dev, world, max_over_ranks, barrier)
    paper_shape = None
    if not args.no_paper_shape:
        paper_shape = bench_paper_shape(dev, max_over_ranks, barrier)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if any(k.endswith("_tc") for k in trace) else "f32",
            "data": "synthetic",
            "config": {"workload": f"{TRAIN}: forward + backward of the chunked scan, B{s.batch} "
                                   f"L{s.seqlen} H{s.nheads} P{s.headdim} N{s.dstate} "
                                   f"K{s.nmodes} G{s.ngroups}, bf16 inputs; tensor-core products "
                                   "take bf16 operands with float32 accumulation, the rest is "
                                   "float32",
                       "global_batch": s.batch * world, "seq_len": s.seqlen,
                       "parallelism": f"replicas{world}" if world > 1 else "single",
                       "l2": "inputs larger than L2 (0.78 GB per step), no flush"},
            "roofline": roofline, "kernels": kern, "gpu_launches": launches,
            "e2e": e2e, "decode": decode, "prefill": prefill, "paper_shape_prefill": paper_shape,
            "clocks": clk,
            "peaks_source": peaks["source"],
        }
        if args.batch:
            line["config"]["workload"] += f" (batch overridden to {args.batch})"
        if world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline()
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def bench_prefill(args, dev, world, max_over_ranks, barrier):
    """Long-context prefill: the forward scan of B1 L65536 H64 P64 N128 K8 (Delta skewed small),
    final state kept; tokens/s over the timed forwards (inputs resident, 1.3 GB > L2)."""
    import torch

    from paper_2609_36314_gb300 import _lib, scan_fwd, synth
    from paper_2609_36314_gb300.api import fwd_workspace_size, make_dims
    s = shape_of(PREFILL)
    a = synth.make_scan_inputs_torch(s, seed=11, device=dev)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    ws = torch.empty(fwd_workspace_size(dims), dtype=torch.uint8, device=dev)
    y = torch.empty_like(a["x"])
    hf = torch.empty((s.batch, s.nheads, s.nmodes, s.headdim, s.dstate), dtype=torch.float32, device=dev)

    def fwd():
        scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                 a["w_write"], a["D"], y=y, h_final=hf, workspace=ws)

    for _ in range(3):
        fwd()
    torch.cuda.synchronize()
    _lib.trace_reset()
    _lib.trace_enable(True)
    barrier()
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n = 5
    ev0.record(stream)
    for _ in range(n):
        fwd()
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    _lib.trace_enable(False)
    ms = max_over_ranks(ev0.elapsed_time(ev1) / n)
    kern = {k: {"launches": c, "avg_ms": t / max(c, 1)} for k, (c, t) in _lib.trace_collect().items()}
    del a, ws, y, hf
    torch.cuda.empty_cache()
    return {"workload": f"{PREFILL}: forward of B{s.batch} L{s.seqlen} H{s.nheads} P{s.headdim} "
                        f"N{s.dstate} K{s.nmodes}, Delta = softplus(z - {s.dt_shift}), final state "
                        "kept; chunk 128 (results are chunk-independent)",
            "value": world * s.batch * s.seqlen / (ms / 1e3), "unit": "tokens/s", "ms_per_forward": ms,
            "kernels": kern}


def bench_paper_shape(dev, max_over_ranks, barrier):
    """The paper's own layer shape (H16, head dim 256, N = 1, K = 16 modes on the 1 .. 2^17
    bank), batch-1 prefill at 1K, 4K and 16K tokens: forward tokens/s per length (inputs
    resident; CUDA-core path, these shapes are outside the tensor-core kernels)."""
    import torch

    from paper_2609_36314_gb300 import scan_fwd, synth
    pts = []
    for L in (1024, 4096, 16384):
        s = synth.Shape(1, L, 16, 256, 1, 1, 16, 0, "bf16")
        a = synth.make_scan_inputs_torch(s, seed=13, device=dev)
        y = torch.empty_like(a["x"])

        def fwd():
            scan_fwd(a["x"], a["dt"], a["alpha"], a["lam"], a["tau"], a["B"], a["C"], a["w_read"],
                     a["w_write"], a["D"], y=y)

        for _ in range(3):
            fwd()
        torch.cuda.synchronize()
        barrier()
        stream = torch.cuda.current_stream()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n = 10
        ev0.record(stream)
        for _ in range(n):
            fwd()
        ev1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ms = max_over_ranks(ev0.elapsed_time(ev1) / n)
        pts.append({"seqlen": L, "ms_per_forward": ms, "tokens_per_s": L / (ms / 1e3)})
        del a, y
    return {"workload": "paper layer shape: B1 H16 P256 N1 K16, tau geometric in [1, 2^17], bf16 "
                        "inputs, forward only", "unit": "tokens/s", "points": pts}


def bench_decode(args, dev, peaks, world, max_over_ranks, barrier):
    import torch

    from paper_2609_36314_gb300 import decode_step, scan_fwd, synth
    s = shape_of(DECODE)
    pre = synth.make_scan_inputs_torch(s, seed=7, device=dev)
    _, state = scan_fwd(pre["x"], pre["dt"], pre["alpha"], pre["lam"], pre["tau"], pre["B"],
                        pre["C"], pre["w_read"], pre["w_write"], pre["D"])
    del pre
    T = args.decode_steps
    stp = synth.make_scan_inputs_torch(s.replace(seqlen=T), seed=8, device=dev)
    # [B, T, ...] -> [T, B, ...] so that every step reads contiguous inputs
    stp = {k: (v.transpose(0, 1).contiguous() if k not in ("tau", "D") else v)
           for k, v in stp.items()}
    ybuf = torch.empty((T, s.batch, s.nheads, s.headdim), dtype=torch.bfloat16, device=dev)

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
    g.replay()
    torch.cuda.synchronize()
    barrier()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 2
    e0.record(stream)
    for _ in range(reps):
        g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms_step = max_over_ranks(e0.elapsed_time(e1) / (reps * T))
    state_bytes = 2.0 * 4 * s.batch * s.nheads * kpn(s)
    gbs = state_bytes / (ms_step / 1e3) / 1e9
    return {"workload": f"{DECODE}: B{s.batch} H{s.nheads} P{s.headdim} N{s.dstate} K{s.nmodes}, "
                        f"float32 state, 512-token prefill then {T} steps in one CUDA graph",
            "value": world * s.batch / (ms_step / 1e3), "unit": "tokens/s",
            "us_per_step": 1e3 * ms_step,
            "roofline": {"kernel": "decode_step", "bound": "hbm", "achieved": gbs,
                         "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"],
                         "traffic": (PROFILED_DECODE_TRAFFIC[2]
                                     if source_digest(PROFILED_DECODE_TRAFFIC[0]) == PROFILED_DECODE_TRAFFIC[1]
                                     else None),
                         "peak_source": peaks["source"]}}


if __name__ == "__main__":
    main()
