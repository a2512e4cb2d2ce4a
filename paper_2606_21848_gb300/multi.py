"""Host logic of the multi-GPU paths (one process per GPU, torch.distributed).

The decode shards without any exchange: sequences and value heads are independent, so N GPUs
run N replicas, each on its own batch, and a step's time is the slowest rank's. A single long
sequence can also be cut across GPUs by token range; each GPU then produces split states
(o, m, l) for its range (kl_decode_attention_ex with partial_o / partial_ml) and one all-gather
plus kl_combine merges them -- the one real exchange step of the path.

Only host-side bookkeeping lives here (ranks, seeds, reductions of timings, token ranges,
gathering states); every number a GPU computes comes from the CUDA library.
"""
from __future__ import annotations

import os

import torch


def dist_env() -> tuple[int, int, int]:
    """(rank, world_size, local_rank) from the launcher's environment (1 process: 0, 1, 0)."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def replica_seed(base_seed: int, rank: int) -> int:
    """Seed of rank `rank`'s batch: replicas draw distinct inputs of the same shapes."""
    return base_seed + rank


def max_over_ranks(values, device=None) -> list[float]:
    """Element-wise maximum of per-rank timings over all ranks (identity with one process).
    `device` is where the reduction tensor lives: CPU for gloo, the rank's GPU for NCCL."""
    vals = [float(v) for v in values]
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return vals
    t = torch.tensor(vals, dtype=torch.float64, device=device or "cpu")
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def job_throughput(units_per_rank: int, world: int, seconds: float) -> float:
    """Whole-job rate: the units every rank processed in one step over the slowest rank's time."""
    return units_per_rank * world / seconds


def shard_token_range(seq_len: int, rank: int, world: int, quantum: int = 128) -> tuple[int, int]:
    """Contiguous token range [t0, t1) of rank `rank` when one sequence of `seq_len` tokens is
    cut across `world` GPUs; boundaries fall on multiples of `quantum` (the decode's tile)."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError("rank must lie in [0, world)")
    per = -(-seq_len // world)
    per = -(-per // quantum) * quantum
    t0 = min(seq_len, rank * per)
    t1 = min(seq_len, t0 + per)
    return t0, t1


def gather_split_states(part_o: torch.Tensor, part_ml: torch.Tensor):
    """All-gather every rank's split states and concatenate them along the split axis, rank
    order: [B, Hq, S, D] and [B, Hq, S, 2] per rank -> [B, Hq, world * S, D] and
    [B, Hq, world * S, 2], ready for kl_combine (empty splits carry l = 0 and drop out)."""
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return part_o, part_ml
    world = torch.distributed.get_world_size()
    os_ = [torch.empty_like(part_o) for _ in range(world)]
    ms_ = [torch.empty_like(part_ml) for _ in range(world)]
    torch.distributed.all_gather(os_, part_o.contiguous())
    torch.distributed.all_gather(ms_, part_ml.contiguous())
    return torch.cat(os_, dim=2), torch.cat(ms_, dim=2)
