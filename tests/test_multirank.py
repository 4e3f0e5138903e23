"""The multi-rank host logic of bench.py on CPU (gloo, world size 2): every
rank routes its own seeded batch (no data-path collective, weak scaling), the
job's time is the slowest rank's, and the job's throughput counts every
rank's tokens. The reference arm under torchrun prints one line from rank 0
and the other rank exits without work."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # the slowest rank's time is the job's time
    out.put((rank, "max", bench.max_over_ranks(1.5 + rank, dist)))
    # each rank draws a different batch
    from paper_2608_04401_gb300 import synth
    x = synth.layer_inputs(T=8, d=256, N=64, I=128, seed=bench.rank_seed(1003, rank),
                           with_experts=False)["x"]
    out.put((rank, "x0", int(x[0, 0])))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = {}
    while not q.empty():
        r, key, v = q.get()
        got[(r, key)] = v
    assert got[(0, "max")] == got[(1, "max")] == 2.5
    assert got[(0, "x0")] != got[(1, "x0")]


def test_job_throughput_counts_every_rank():
    import bench
    assert bench.job_tokens_per_s(16384, 1, 1.0) == pytest.approx(16384e3)
    assert bench.job_tokens_per_s(16384, 4, 1.0) == pytest.approx(4 * 16384e3)
    assert bench.rank_seed(1003, 0) == 1003 and bench.rank_seed(1003, 1) != 1003
    assert bench.max_over_ranks(3.0, None) == 3.0


def test_reference_arm_under_torchrun():
    """bench.py --impl reference with two ranks (gloo): one JSON line, from rank 0."""
    env = dict(os.environ, BENCH_BACKEND="gloo", OMP_NUM_THREADS="2")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "1",
           "--warmup", "1"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["n_gpus"] == 2 and j["value"] > 0
    assert j["e2e"]["h2d_bytes_per_step"] == 0
