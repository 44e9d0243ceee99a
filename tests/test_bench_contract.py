"""bench.py's CPU-side contract: the reference arm (the oracle on a bounded sample) prints one
JSON line with the keys the benchmark driver reads, and the roofline helpers give positive
algorithmic work and traffic only for the kernels they describe (CPU only)."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_36314_gb300 import synth  # noqa: E402


def test_reference_arm_prints_one_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0"],
                         cwd=ROOT, capture_output=True, text=True, timeout=300, check=True).stdout
    lines = [ln for ln in out.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "dtype", "config", "cpu_baseline", "e2e"):
        assert k in d
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "tokens/s"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0


def test_roofline_helpers():
    s = synth.WORKLOADS["train_bf16_b8_l4096"]
    units = s.batch * s.seqlen * s.nheads
    for k in ("state_pass_fwd_tc", "chunk_fwd_tc", "bwd_state_tc", "bwd_intra_tc"):
        kind, work = bench.algorithmic_work(k, s, units)
        assert kind == "flops" and work > 0
    for k in ("coef_tc", "bwd_final_tc"):
        kind, work = bench.algorithmic_work(k, s, units)
        assert kind == "bytes" and work > 0
    assert bench.algorithmic_work("no_such_kernel", s, units) == (None, None)
    assert bench.profiled_traffic("no_such_kernel", 8) is None
    for k, (src, digest, _) in bench.PROFILED_TRAFFIC.items():
        t = bench.profiled_traffic(k, 8)
        # a figure is reported only while the kernel's sources are the ones that were profiled
        assert (t is not None) == (bench.source_digest(src) == digest)
        if t is not None:
            assert t > 0


def test_algorithmic_flops_match_the_products_of_the_chunked_form():
    """The roofline numerators, recounted from the products of one chunk (Q = 128 positions of
    one head; mm(m, k, n) = the flops of an (m x k) x (k x n) product, causal products counted
    at half): the state update K (P x Q)(Q x N), the readout K (Q x N)(N x P), the intra term
    (Q x Q)(Q x P) and C B^T (Q x N)(N x Q) once per B/C group; the backward's state terms four
    contractions per mode (Z, U, dC, dB) plus the head-summed intra dC = M B, dB = M^T C, and
    its intra kernel H = dY X^T, dx = (Gamma o G)^T dY and G = C B^T.  The whole step's count
    takes the C B^T-type terms at their algorithmic (causal, shared) size, which the kernels
    exceed by their dense or recomputed products (0.1% of the training step, 0.4% at H16 N64)."""
    q = 128
    for name in ("train_bf16_b8_l4096", "fwd_bf16_b4_l2048"):
        s = synth.WORKLOADS[name]
        K, P, N, G, H = s.nmodes, s.headdim, s.dstate, s.ngroups, s.nheads

        def mm(m, k, n):
            return 2 * m * k * n

        per_chunk = {
            "state_pass_fwd_tc": K * mm(P, q, N),
            "state_pass_rev_tc": K * mm(P, q, N),
            "chunk_fwd_tc": K * mm(q, N, P) + mm(q, q, P) / 2 + mm(q, N, q) / 2 * G / H,
            "bwd_state_tc": 4 * K * mm(q, N, P) + 2 * mm(q, q, N) * G / H,
            "bwd_intra_tc": 2 * mm(q, P, q) / 2 + mm(q, N, q) / 2 * G / H,
        }
        for k, flops in per_chunk.items():
            kind, work = bench.algorithmic_work(k, s, q)  # one chunk of one head = q token-heads
            assert kind == "flops"
            assert work == pytest.approx(flops), k
        step = sum(per_chunk.values())
        assert bench.train_flops_per_token_head(s) * q == pytest.approx(step, rel=5e-3)
        assert bench.train_flops_per_token_head(s) * q < step
        fwd = per_chunk["state_pass_fwd_tc"] + per_chunk["chunk_fwd_tc"]
        assert bench.fwd_flops_per_token_head(s) * q == pytest.approx(fwd)
