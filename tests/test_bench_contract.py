"""bench.py's CPU-side contract: the reference arm (the oracle on a bounded sample) prints one
JSON line with the keys the benchmark driver reads, and the roofline helpers give positive
algorithmic work and traffic only for the kernels they describe (CPU only)."""
import json
import os
import subprocess
import sys

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
