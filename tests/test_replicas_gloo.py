"""The multi-GPU mode of the benchmark is replicas only: N ranks decode
independent sequences, with no collective on the data path.  Its host logic
(the slowest rank's time, the tokens of all ranks; the reference arm printing
on rank 0 only) runs here as two gloo processes on the CPU."""
import json
import os
import socket
import subprocess
import sys

import pytest

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, world: int, port: int, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, REPO)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, tok = bench.aggregate_replicas(100.0 + 50.0 * rank, 256.0 + rank, "cpu")
    q.put((rank, ms, tok))
    dist.barrier()
    dist.destroy_process_group()


def test_replica_aggregation_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, ms, tok in res:
        assert ms == 150.0 and tok == 513.0  # max of the times, sum of the tokens


def test_single_process_aggregation_is_identity():
    sys.path.insert(0, REPO)
    import bench
    assert bench.aggregate_replicas(12.5, 7, "cpu") == (12.5, 7.0)


@pytest.mark.slow
def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` under a 2-rank launch: rank 0 alone times
    the oracle and prints one JSON line; rank 1 exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl",
           "reference", "--workload", "tiny", "--steps", "1", "--warmup", "0", "--ref-prompt", "8",
           "--ref-new", "2"]
    r = subprocess.run(cmd, cwd=REPO, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
