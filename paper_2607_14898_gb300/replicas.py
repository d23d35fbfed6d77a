"""Several GPUs as independent replicas.

Chunks of one stream are strictly sequential through the rolling cache (Algorithm 1: chunk t
attends to the cache that chunk t-1 left), so one stream cannot be split across GPUs. Separate
streams share nothing but the weights (the batch dimension B of the cache in Eq. 2 keeps them
apart), so each rank decodes whole streams of its own with a weight replica, and no tensor of
the decode path crosses ranks. The process group carries only host bookkeeping: a barrier around the timed
region and the max / sum of two scalars, so that the whole job's throughput is

    frames decoded by all ranks / the slowest rank's time.

`RankGroup` wraps that bookkeeping over any `torch.distributed` backend (NCCL with one GPU per
rank, gloo on the CPU) or none at all (one process).
"""
from __future__ import annotations

import os
from dataclasses import dataclass


def stream_seeds(base_seed: int, rank: int, streams_per_rank: int) -> list[int]:
    """Latent seeds of the streams one rank decodes: rank r owns streams
    r*S .. r*S + S - 1 of the job, so no two ranks decode the same stream."""
    if rank < 0 or streams_per_rank < 1:
        raise ValueError("rank must be >= 0 and streams_per_rank >= 1")
    first = base_seed + rank * streams_per_rank
    return list(range(first, first + streams_per_rank))


def job_frames_per_second(frames_all_ranks: float, ms_slowest_rank: float) -> float:
    """Whole-job throughput: every rank's frames over the slowest rank's time."""
    if ms_slowest_rank <= 0:
        raise ValueError("the timed region must have a positive duration")
    return frames_all_ranks / (ms_slowest_rank * 1e-3)


@dataclass
class RankEnv:
    rank: int
    world: int
    local_rank: int


def rank_env() -> RankEnv:
    """RANK / WORLD_SIZE / LOCAL_RANK as torchrun sets them (one process: 0 / 1 / 0)."""
    return RankEnv(int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
                   int(os.environ.get("LOCAL_RANK", "0")))


class RankGroup:
    """Barrier and scalar reductions across the replicas.

    `dist` is `torch.distributed` with an initialised default group, or None for a single
    process (every call is then the identity). `device` is where the reduction tensors live:
    "cuda" under NCCL, "cpu" under gloo."""

    def __init__(self, dist=None, device: str = "cpu"):
        self.dist = dist
        self.device = device

    @property
    def world(self) -> int:
        return 1 if self.dist is None else self.dist.get_world_size()

    def barrier(self) -> None:
        if self.dist is not None:
            self.dist.barrier()

    def _reduce(self, x: float, op) -> float:
        import torch
        t = torch.tensor([float(x)], dtype=torch.float64, device=self.device)
        self.dist.all_reduce(t, op=op)
        return float(t.item())

    def max(self, x: float) -> float:
        return float(x) if self.dist is None else self._reduce(x, self.dist.ReduceOp.MAX)

    def sum(self, x: float) -> float:
        return float(x) if self.dist is None else self._reduce(x, self.dist.ReduceOp.SUM)

    def throughput(self, frames_this_rank: float, ms_this_rank: float) -> tuple[float, float, float]:
        """(frames/s of the whole job, frames of all ranks, slowest rank's ms)."""
        ms_max = self.max(ms_this_rank)
        frames_all = self.sum(frames_this_rank)
        return job_frames_per_second(frames_all, ms_max), frames_all, ms_max
