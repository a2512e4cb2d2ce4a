"""The multi-process host logic on CPU: two `gloo` ranks (world size 2), no GPU.

Covers what `bench.py --gpus N` relies on (distinct replica inputs, the slowest rank's time,
the whole-job rate) and the exchange step of a sequence cut across GPUs by token range: each
rank holds the split states of its own range, one all-gather brings them together, and the
merge equals the decode of the whole sequence. The fp64 oracle stands in for each rank's
GPU kernels here (CPU test infrastructure)."""
from __future__ import annotations

import math
import os
import queue
import socket
import time

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2606_21848_gb300 import multi

WORLD = 2


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _init(rank: int, port: int):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)


def _timing_worker(rank: int, port: int, q):
    _init(rank, port)
    try:
        # rank 1 is the slower one in the first value, rank 0 in the second
        mine = [10.0 + 5.0 * rank, 7.0 - 3.0 * rank]
        q.put((rank, multi.max_over_ranks(mine), multi.replica_seed(4, rank)))
    finally:
        dist.destroy_process_group()


def _shard_worker(rank: int, port: int, q):
    _init(rank, port)
    try:
        import oracle
        from paper_2606_21848_gb300.workloads import bf16_bits
        from tests._inputs import tiny
        x = tiny(B=2, Hq=8, Hkv=2, D=64, P=16, lens=(900, 300), seed=81)
        qb, wb, vb = bf16_bits(x["q"]), bf16_bits(x["w_r"]), bf16_bits(x["v_cache"])
        bt, sl = x["block_table"].numpy(), x["seq_lens"].numpy()
        scale = 1.0 / math.sqrt(64)
        # every rank cuts both sequences at the same boundary: its own range is one split of
        # `chunk` tokens (rank 1's is empty for the shorter sequence)
        L = int(sl.max())
        t0, t1 = multi.shard_token_range(L, rank, WORLD)
        chunk = multi.shard_token_range(L, 0, WORLD)[1]
        po, pml = oracle.decode_partial(qb, wb, vb, bt, sl, scale=scale, chunk=chunk,
                                        num_splits=WORLD)
        own_o = torch.from_numpy(po[:, :, rank:rank + 1].copy())
        own_ml = torch.from_numpy(pml[:, :, rank:rank + 1].copy())
        all_o, all_ml = multi.gather_split_states(own_o, own_ml)
        merged = oracle.combine(all_o.numpy(), all_ml.numpy())
        full = oracle.decode(qb, wb, vb, bt, sl, scale=scale)
        q.put((rank, (t0, t1), tuple(all_o.shape), float(np.abs(merged - full).max())))
    finally:
        dist.destroy_process_group()


def _run(worker):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=worker, args=(r, port, q)) for r in range(WORLD)]
    for p in procs:
        p.start()
    # A spawned rank imports torch afresh; in a cold container that alone can take minutes, so
    # the wait is long but ends early when a rank dies without reporting.
    out, deadline = [], time.monotonic() + 900
    while len(out) < WORLD:
        try:
            out.append(q.get(timeout=5))
        except queue.Empty:
            dead = [p.exitcode for p in procs if p.exitcode not in (None, 0)]
            assert not dead, f"a rank exited with {dead} before reporting"
            assert time.monotonic() < deadline, "ranks did not report within 900 s"
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    return sorted(out)


def test_slowest_rank_time_and_distinct_replica_seeds():
    out = _run(_timing_worker)
    for rank, maxed, seed in out:
        assert maxed == [15.0, 7.0]          # element-wise max over the two ranks
    assert [seed for _, _, seed in out] == [4, 5]
    assert multi.job_throughput(256, 2, 0.5) == 1024.0


def test_sharded_sequence_states_gather_and_merge_to_the_full_decode():
    out = _run(_shard_worker)
    (r0, rng0, shape0, err0), (r1, rng1, shape1, err1) = out
    assert rng0 == (0, 512) and rng1 == (512, 900)
    assert shape0 == shape1 == (2, 8, 2, 64)   # both ranks' splits, rank order
    assert err0 < 1e-12 and err1 < 1e-12


def test_shard_token_ranges_cover_the_sequence_once():
    for L in (1, 127, 128, 129, 4096, 131072, 100003):
        for world in (1, 2, 3, 8):
            got = [multi.shard_token_range(L, r, world) for r in range(world)]
            assert got[0][0] == 0 and got[-1][1] == L
            for (a0, a1), (b0, b1) in zip(got, got[1:]):
                assert a1 == b0 and a0 <= a1
            assert all(t0 % 128 == 0 or t0 == L for t0, _ in got)   # tile boundaries
    with pytest.raises(ValueError):
        multi.shard_token_range(10, 2, 2)


def test_single_process_helpers_are_identity():
    assert multi.max_over_ranks([1.5, 2.0]) == [1.5, 2.0]
    o, ml = torch.zeros(1, 2, 3, 4), torch.zeros(1, 2, 3, 2)
    go, gml = multi.gather_split_states(o, ml)
    assert go is o and gml is ml
