"""Multi-rank host logic of bench.py on the CPU (gloo, world size 2).

The verify step does not shard (one batch-1 step per GPU), so N > 1 runs
are independent replicas: each rank times its own steps, the job's time is
the slowest rank's, and the value counts the units of every rank.  These
tests run that reduction over a real gloo process group, and the reference
arm under torchrun, where rank 0 alone prints its line."""
import json
import os
import socket
import subprocess
import sys

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _replica(rank, world, port, seconds, units, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    slowest = bench.max_over_ranks(seconds[rank], world, "cpu")
    value = bench.whole_job_rate(units, slowest, world)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, slowest, value))


def _run_replicas(seconds, units):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_replica, args=(r, len(seconds), port, seconds, units, q))
             for r in range(len(seconds))]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    return out


def test_replicas_take_the_slowest_rank_and_count_every_rank():
    out = _run_replicas([0.5, 2.0], units=300.0)
    assert [o[1] for o in out] == [2.0, 2.0]
    # 2 ranks x 300 units in the slowest rank's 2 s
    assert all(abs(o[2] - 300.0) < 1e-9 for o in out)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(1.25, 1) == 1.25
    assert bench.whole_job_rate(10.0, 0.5, 1) == 20.0


def test_reference_arm_under_torchrun_prints_one_line():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "2",
           "--warmup", "1", "--workload", "tiny-f32-chain8"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
