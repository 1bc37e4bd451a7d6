"""The multi-GPU benchmark path (independent replicas, max-over-ranks timing)
on two CPU processes over gloo: no GPU, no data-path collective."""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2606_09905_gb300 import replicas


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, times, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = replicas.rank_world_local()
        replicas.barrier()
        ms_max = replicas.max_over_ranks(times[rank])
        rate = replicas.whole_job_rate(units_per_rank=1000.0, seconds_max=ms_max / 1e3, world=w)
        out.put((r, w, local, replicas.replica_seed(r), ms_max, rate))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_replicas_time_is_the_slowest_rank(world):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    times = [12.5, 20.0]                              # ms per rank: rank 1 is slower
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, times, out)) for r in range(world)]
    for p in procs:
        p.start()
    results = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[0] for r in results] == [0, 1] and all(r[1] == world for r in results)
    assert [r[2] for r in results] == [0, 1]
    assert len({r[3] for r in results}) == world          # distinct seeds per replica
    for r in results:
        assert r[4] == 20.0                               # every rank sees the maximum
        assert r[5] == pytest.approx(world * 1000.0 / 0.020)


def test_single_process_needs_no_group():
    assert replicas.max_over_ranks(3.5) == 3.5
    assert replicas.whole_job_rate(10.0, 2.0, 1) == 5.0
    with pytest.raises(ValueError):
        replicas.whole_job_rate(1.0, 0.0, 1)


def test_reference_arm_runs_on_rank0_only():
    """Under torchrun the CPU reference arm does its work on rank 0 alone; any
    other rank exits 0 at once, printing nothing."""
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "3", "--warmup", "3"],
                       env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == ""
