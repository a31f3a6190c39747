"""Data-parallel replicas of the rollout-collection step: one process per GPU.

The step shards by prompt.  A prompt's posterior, decisions, KV cache and decode are
independent of every other prompt's, so rank r runs the whole step (`Handle.collect_step`)
on its own prompt stream -- the workload's seeds shifted by `seed_offset(r)` -- with its own
budget N and target B.  Nothing is exchanged on the data path; the only collective is the
final reduction of the step counters (sum) and of the step time (max over ranks), so the
job's throughput is the sum of the replicas' work over the slowest replica's time.

Exact global semantics (one budget and one target shared by all ranks) would need a small
all-reduce per round; the replicas here keep per-rank budgets instead, which is the weak-
scaling reading of the multi-GPU step.
"""
from __future__ import annotations

import numpy as np

# Step counters reduced across ranks (sara_result / Handle.collect_step counters).
COUNTER_KEYS = ("rollouts", "gen_tokens", "prefill_tokens", "decode_steps", "rounds", "committed", "abandoned",
                "incomplete", "prompts_drawn")

SEED_STRIDE = 1000  # rank r's prompt stream: every seed + 1000 r


def seed_offset(rank: int) -> int:
    """Seed shift of rank `rank`'s prompt stream (rank 0 runs the unshifted workload)."""
    if rank < 0:
        raise ValueError("rank must be >= 0")
    return SEED_STRIDE * rank


def reduce_counters(counters: dict, device=None, group=None) -> dict:
    """Sum the step counters over the ranks of `group` (torch.distributed, initialised)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(counters[k]) for k in COUNTER_KEYS], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return {k: int(round(v)) for k, v in zip(COUNTER_KEYS, t.tolist())}


def reduce_max(values, device=None, group=None) -> list:
    """Element-wise maximum over the ranks (step times: the job ends with its slowest rank)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(np.asarray(values, dtype=np.float64), device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return t.tolist()


def reduce_sum(values, device=None, group=None) -> list:
    """Element-wise sum over the ranks."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(np.asarray(values, dtype=np.float64), device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return t.tolist()
