"""Several GPUs as independent replicas (no exchange step): the rank bookkeeping of the bench,
run as world-size-2 gloo process groups on the CPU.

A stream cannot be split across GPUs (its chunks are sequential through the cache, Algorithm 1);
separate streams share only the weights, so ranks decode disjoint streams and the job's
throughput is every rank's frames over the slowest rank's time."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from paper_2607_14898_gb300.replicas import (RankGroup, job_frames_per_second,  # noqa: E402
                                             stream_seeds)


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_stream_seeds_are_disjoint_across_ranks():
    for S in (1, 3, 8):
        seen = set()
        for rank in range(4):
            seeds = stream_seeds(7, rank, S)
            assert len(seeds) == S
            assert not seen & set(seeds)
            seen |= set(seeds)
        assert seen == set(range(7, 7 + 4 * S))  # no stream skipped either
    with pytest.raises(ValueError):
        stream_seeds(0, 0, 0)


def test_single_process_group_is_the_identity():
    g = RankGroup(None)
    assert g.world == 1
    g.barrier()
    assert g.max(3.5) == 3.5 and g.sum(2.0) == 2.0
    value, frames, ms = g.throughput(64, 80.0)
    assert (frames, ms) == (64.0, 80.0)
    assert value == pytest.approx(800.0)
    with pytest.raises(ValueError):
        job_frames_per_second(64, 0.0)


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        g = RankGroup(dist, "cpu")
        g.barrier()
        # rank r: 64 (r + 1) frames in 100 + 50 r ms
        value, frames_all, ms_max = g.throughput(64 * (rank + 1), 100.0 + 50.0 * rank)
        seeds = stream_seeds(0, rank, 8)
        gathered = [None] * world
        dist.all_gather_object(gathered, seeds)
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as fh:
            json.dump({"value": value, "frames_all": frames_all, "ms_max": ms_max,
                       "world": g.world, "seeds": gathered}, fh)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_job_throughput(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    for r in res:
        assert r["world"] == world
        assert r["frames_all"] == 64 + 128
        assert r["ms_max"] == 150.0  # the slowest rank's time, not the mean
        assert r["value"] == pytest.approx(192 / 0.150)
        s0, s1 = r["seeds"]
        assert not set(s0) & set(s1)


def test_bench_reference_arm_under_torchrun_prints_once(tmp_path):
    """`bench.py --impl reference` under torchrun: rank 0 alone times the oracle and prints
    one JSON line; the other rank exits 0 without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
           "--workload", "tiny", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    p = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=str(tmp_path),
                       env=env)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, p.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["unit"] == "frames/s"
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0


def test_bench_attention_traffic_is_the_launch_weighted_capture_mean():
    """The roofline's traffic is per attention launch over the same launch mix as its achieved
    rate: the committed backbone and refinement captures weighted by launch counts."""
    import bench
    tb = bench.ncu_traffic("fd_attn.cu", "480p", "backbone")
    tr = bench.ncu_traffic("fd_attn.cu", "480p", "refine")
    prof = {"attn_backbone": (24, 1.0), "attn_refine": (2, 1.0)}
    if tb is None or tr is None:  # the kernel changed since the captures: no traffic claimed
        assert bench.attention_traffic("480p", prof) is None
        return
    assert tr > tb > 0
    assert bench.attention_traffic("480p", prof) == round((24 * tb + 2 * tr) / 26)
    assert bench.attention_traffic("720p", prof) is None          # no capture for 720p
    assert bench.attention_traffic("480p", {"attn_backbone": (0, 0.0),
                                            "attn_refine": (0, 0.0)}) is None


def _rank_dies(rank, world, port, out_dir):
    import datetime
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=10))
    if rank == 1:
        os._exit(3)  # the rank is lost between steps, without any goodbye
    g = RankGroup(dist, "cpu")
    try:
        g.barrier()
        g.max(1.0)
        outcome = "no error"
    except Exception as e:  # the survivors learn of it through the failed collective
        outcome = "error: " + type(e).__name__
    with open(os.path.join(out_dir, "rank0.txt"), "w") as fh:
        fh.write(outcome)
    os._exit(0)


def test_a_lost_rank_fails_the_next_collective_instead_of_hanging(tmp_path):
    """Failure detection of the replica bookkeeping, on the host: a rank that dies between
    steps makes the surviving rank's next barrier / reduction raise (connection loss or the
    process group's timeout) rather than wait forever."""
    import multiprocessing
    ctx = multiprocessing.get_context("spawn")
    port = free_port()
    procs = [ctx.Process(target=_rank_dies, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()
    assert not alive, "a rank hung"
    assert procs[1].exitcode == 3
    assert (tmp_path / "rank0.txt").read_text().startswith("error")
