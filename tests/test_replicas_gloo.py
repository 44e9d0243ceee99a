"""The N > 1 plumbing of bench.py on the CPU: the scan has no exchange step here (each GPU runs an
independent replica of the workload), so the only cross-rank work is the barrier around the timed
region and the maximum of the per-rank times, from which rank 0 reports the whole job's
throughput.  Two gloo ranks (world size 2, 127.0.0.1) run that code; the reference arm under
torchrun prints from rank 0 only."""
import json
import os
import socket
import subprocess
import sys
import tempfile

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ctx = bench.Ctx(torch.device("cpu"), world, {"source": "test"})
        ctx.barrier()
        ms = 2.0 + 3.0 * rank  # rank 1 is the slower replica
        worst = ctx.max_over_ranks(ms)
        tokens_per_step = 1000
        value = world * tokens_per_step / (worst / 1e3)  # as bench_train: all ranks' tokens / max time
        ctx.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"worst": worst, "value": value}, f)
    finally:
        dist.destroy_process_group()


def test_replica_ranks_agree_on_the_slowest_time():
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_rank_main, args=(world, _free_port(), d), nprocs=world, join=True,
                           start_method="spawn")
        res = [json.load(open(os.path.join(d, f"rank{r}.json"))) for r in range(world)]
    assert [r["worst"] for r in res] == [5.0, 5.0]
    assert res[0]["value"] == pytest.approx(2 * 1000 / 5e-3)


def test_single_rank_needs_no_process_group():
    ctx = bench.Ctx(torch.device("cpu"), 1, {"source": "test"})
    ctx.barrier()
    assert ctx.max_over_ranks(1.25) == 1.25


@pytest.mark.parametrize("rank", [0, 1])
def test_reference_arm_runs_on_rank_0_only(rank):
    env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
               MASTER_ADDR="127.0.0.1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--gpus", "2", "--steps", "1", "--warmup", "0"],
                         cwd=ROOT, env=env, capture_output=True, text=True, timeout=300, check=True).stdout
    lines = [ln for ln in out.splitlines() if ln.strip().startswith("{")]
    if rank == 0:
        assert len(lines) == 1
        d = json.loads(lines[0])
        assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    else:
        assert lines == []
