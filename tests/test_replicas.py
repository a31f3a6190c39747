"""Host logic of the multi-GPU path (replicas over prompt-stream shards), on CPU with gloo.

Two ranks each take their own shard of the prompt stream and run the Algorithm 1 schedule
on it (the oracle stands in for the GPU step here); the counters they reduce must equal the
sum of the per-shard schedules computed in one process, the step time reduces to the
maximum, and the shards must be distinct streams.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import synth
from oracle import controller as oc
from paper_2607_26253_gb300 import replicas


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = synth.WORKLOADS["tiny"].with_seed_offset(replicas.seed_offset(rank))
        res = oc.collect_workload(w)
        counters = {k: int(res.counters[k]) for k in replicas.COUNTER_KEYS}
        total = replicas.reduce_counters(counters)
        tmax = replicas.reduce_max([10.0 * (rank + 1), -rank])
        out.put((rank, counters, total, tmax, int(res.status.sum())))
    finally:
        dist.destroy_process_group()


def test_two_replicas_reduce_to_the_sum_of_their_shards():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    got.sort(key=lambda g: g[0])
    per_rank = [g[1] for g in got]
    expect = {k: sum(c[k] for c in per_rank) for k in replicas.COUNTER_KEYS}
    for _, _, total, tmax, _ in got:
        assert total == expect                     # every rank sees the same job total
        assert tmax == [20.0, 0.0]                 # max over ranks, element-wise
    # the shards are the single-process schedules of the shifted streams
    for r, c in enumerate(per_rank):
        ref = oc.collect_workload(synth.WORKLOADS["tiny"].with_seed_offset(replicas.seed_offset(r)))
        for k in ("rollouts", "gen_tokens", "committed", "abandoned", "rounds"):
            assert c[k] == ref.counters[k]
    assert got[0][4] != got[1][4] or per_rank[0] != per_rank[1]  # distinct streams


def test_seed_offset_rank0_is_the_unsharded_workload():
    w = synth.WORKLOADS["tiny"]
    assert w.with_seed_offset(replicas.seed_offset(0)) == w
    s1 = synth.step_inputs(w.with_seed_offset(replicas.seed_offset(1)))
    s0 = synth.step_inputs(w)
    assert not np.array_equal(s0.tokens, s1.tokens)
    with pytest.raises(ValueError):
        replicas.seed_offset(-1)
