"""Host logic of the multi-process benchmark, on CPU with the gloo backend and
two ranks.  Units are independent, so the ranks exchange nothing on the data
path; the only collective is the all-gather of per-rank timings that the
whole-job throughput (all frames of all ranks over the slowest rank) needs."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank r took (r + 1) seconds for 100 frames and 2 (r + 1) seconds end to end
    gathered = bench.allgather_floats([float(rank + 1), 2.0 * (rank + 1)], world)
    value, tmax = bench.aggregate([100.0] * world, [g[0] for g in gathered])
    e2e, _ = bench.aggregate([100.0] * world, [g[1] for g in gathered])
    with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
        json.dump({"gathered": gathered, "value": value, "tmax": tmax, "e2e": e2e}, f)
    dist.barrier()
    dist.destroy_process_group()


def test_aggregate_over_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn", join=True)
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(2)]
    for r in res:
        assert r["gathered"] == [[1.0, 2.0], [2.0, 4.0]]
        assert r["tmax"] == 2.0
        assert r["value"] == pytest.approx(200.0 / 2.0)    # both ranks' frames / slowest rank
        assert r["e2e"] == pytest.approx(200.0 / 4.0)


def test_aggregate_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.allgather_floats([3.0, 1.0], 1) == [[3.0, 1.0]]
    assert bench.aggregate([60.0], [0.5]) == (120.0, 0.5)


def test_reference_arm_prints_on_rank_zero_only(tmp_path):
    """torchrun with two CPU ranks: rank 0 times the oracle on one frame and
    prints one JSON line; rank 1 exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, p.stdout
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == 2
    assert rec["cpu_baseline"]["kind"] == "oracle" and rec["value"] > 0
    assert rec["e2e"]["h2d_bytes_per_step"] == 0 and rec["e2e"]["d2h_bytes_per_step"] == 0
