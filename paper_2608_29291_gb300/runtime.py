"""Host-side run-time helpers: rank discovery, weak-scaling replica seeds and
the max-over-ranks reduction used for timing.  The routed block shards by
sequence with no data-path exchange (each sequence's top-K is local), so ranks
only meet for a barrier and for the timing reduction.
"""
from __future__ import annotations

import dataclasses
import os


@dataclasses.dataclass(frozen=True)
class RankInfo:
    rank: int
    world: int
    local_rank: int

    @property
    def is_root(self) -> bool:
        return self.rank == 0


def rank_info() -> RankInfo:
    return RankInfo(int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
                    int(os.environ.get("LOCAL_RANK", "0")))


def replica_seed(base_seed: int, rank: int) -> int:
    """Each rank draws its own batch of sequences (weak scaling)."""
    return base_seed + 1000003 * rank


def init_group(info: RankInfo, backend: str):
    """Initialise torch.distributed when world > 1 (env:// rendezvous)."""
    import torch.distributed as dist
    if info.world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist if info.world > 1 else None


def barrier(dist) -> None:
    if dist is not None:
        dist.barrier()


def max_over_ranks(dist, value: float, device="cpu") -> float:
    """The slowest rank's value (every rank gets it)."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(dist, value: float, device="cpu") -> float:
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())
