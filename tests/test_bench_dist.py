"""The multi-rank leg of bench.py on CPU: two gloo ranks (replicas) agree on
the job time (max over ranks) and on the whole-job throughput, and the
barrier lets both through.  The GPU run uses the same functions over NCCL."""
import multiprocessing as mp
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    w, r, loc = bench.dist_setup()
    ms = [10.0, 12.5][rank]
    m = bench.reduce_max(ms, w, device="cpu")
    bench.barrier(w)
    q.put((r, loc, m, bench.job_tokens_per_s(512, 3, w, m)))
    dist.destroy_process_group()


def test_two_replicas_reduce_to_the_slowest():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1] and [o[1] for o in out] == [0, 1]
    assert all(o[2] == 12.5 for o in out)
    assert all(o[3] == pytest.approx(512 * 3 * 2 / 0.0125) for o in out)


def test_single_rank_is_local():
    import bench
    assert bench.reduce_max(3.0, 1) == 3.0
    assert bench.job_tokens_per_s(512, 3, 1, 1000.0) == pytest.approx(1536.0)


def test_gpus_flag_starts_the_replicas():
    """`bench.py --gpus 2` starts two ranks itself (torch.distributed.run on
    127.0.0.1) and reports the ranks that ran; on a machine without GPUs the
    ranks rendezvous over gloo.  --launch-only decodes nothing."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    if not torch.cuda.is_available():
        env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--gpus", "2", "--launch-only"],
                       capture_output=True, text=True, timeout=300, env=env, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(l) for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    assert lines[0]["n_gpus"] == 2 and lines[0]["max_rank"] == 1
    if not torch.cuda.is_available():
        assert lines[0]["backend"] == "gloo"
