"""World-size-2 gloo tests (CPU) of the multi-rank paths.

1. Vocabulary-parallel split: each rank holds half of the LM head's rows,
   reduces every position to a (max, sum of exponentials, lowest argmax)
   partial over its shard, the partials are all-gathered, and the merge rule
   the library applies across CTAs (and would apply across GPUs) must give
   the oracle's full-vocabulary token and confidence.
2. bench.py's weak-scaling aggregation: slowest rank's time, every rank's
   positions.
"""

import math
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _merge(parts):
    """(m, s, a) partials -> (m, s, a): max, rescaled sum, lowest index on ties."""
    m = max(p[0] for p in parts)
    s = sum(p[1] * math.exp(p[0] - m) for p in parts if p[0] > -math.inf)
    a = min(p[2] for p in parts if p[0] == m)
    return m, s, a


def _vocab_parallel_worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        from workloads import B8X2X32_BF16, generate, scaled
        from workloads.rawio import raw_numpy

        cfg = scaled(B8X2X32_BF16, n_seq=1, n_slots=2, d=64, V=1001, mask_token_id=500)
        wl = generate(cfg)
        h = oracle.commit_oracle.hidden_f64(raw_numpy(wl.hidden), "bf16")
        w_raw = raw_numpy(wl.weight)
        V = cfg.V
        lo, hi = rank * V // world, (rank + 1) * V // world
        shard = oracle.lm_head_logits(h, w_raw[lo:hi], "bf16")  # this rank's rows of the head
        parts = np.zeros((cfg.P, 3))
        for p in range(cfg.P):
            l = shard[p].copy()
            if lo <= cfg.mask_token_id < hi:
                l[cfg.mask_token_id - lo] = -np.inf
            m = l.max()
            parts[p] = (m, np.exp(l - m).sum(), lo + int(np.flatnonzero(l == m)[0]))
        gathered = [torch.zeros((cfg.P, 3), dtype=torch.float64) for _ in range(world)]
        dist.all_gather(gathered, torch.from_numpy(parts))
        if rank == 0:
            full = oracle.lm_head_logits(h, w_raw, "bf16")
            bad = 0
            for p in range(cfg.P):
                m, s, a = _merge([tuple(g[p].tolist()) for g in gathered])
                tok, conf, _ = oracle.row_confidence(full[p], cfg.mask_token_id)
                bad += int(a != tok) + int(abs(1.0 / s - conf) > 1e-12)
            q.put(bad)
    finally:
        dist.destroy_process_group()


def test_vocab_parallel_merge_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_vocab_parallel_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(120)
        assert p.exitcode == 0
    assert q.get(timeout=5) == 0


def _aggregate_worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench

        t, n = bench.aggregate_over_ranks(10.0 + 5 * rank, 100 + rank, dist, "cpu")
        q.put((rank, t, n))
    finally:
        dist.destroy_process_group()


def test_bench_aggregation_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_aggregate_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    assert got == [(0, 15.0, 201.0), (1, 15.0, 201.0)]
