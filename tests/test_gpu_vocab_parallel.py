"""The vocabulary-parallel split through the library (bd_lmhead_partials on
each head shard, bd_merge_commit on the gathered partials) against the float64
oracle on the whole head, and against the single-call commit step.

Shards run as separate calls on the one GPU; the two-rank case exchanges the
library's partials between two gloo processes (copied to host memory), each
rank holding half of the head on the same device. No kernel of one rank waits
for another's.
"""

import os
import socket

import numpy as np
import pytest
import torch

from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B256X8X64_E4M3, B8X2X32_BF16, generate, scaled

pytestmark = pytest.mark.gpu

bdc = pytest.importorskip("paper_2609_33887_gb300")
B = bdc.bdcommit


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield


def shard_bounds(V, cuts):
    edges = [0] + list(cuts) + [V]
    return list(zip(edges[:-1], edges[1:]))


def run_split(wl, bounds):
    cfg = wl.cfg
    g = wl.to("cuda")
    parts = []
    for lo, hi in bounds:
        scale = None if g.weight_scale is None else g.weight_scale[lo:hi]
        parts.append(bdc.lmhead_partials(g.hidden, g.weight[lo:hi], lo, g.pos_masked, g.block_flags, cfg.n_seq,
                                         cfg.n_slots, cfg.block_len, shard_scale=scale,
                                         mask_token_id=cfg.mask_token_id))
    pm = torch.stack([p[0] for p in parts]).contiguous()
    ps = torch.stack([p[1] for p in parts]).contiguous()
    pa = torch.stack([p[2] for p in parts]).contiguous()
    tokens, conf, commit, counts = bdc.merge_commit(pm, ps, pa, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots,
                                                    cfg.block_len, wl.tau, counts=True)
    torch.cuda.synchronize()
    st = bdc.bd_get_device_status()
    assert st == 0, bdc.bd_status_string(st)
    out = {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
           "commit": commit.cpu().numpy().view(np.uint32), "counts": counts.cpu().numpy()}
    return out, (pm.cpu(), ps.cpu(), pa.cpu())


CASES = {
    # two uneven bf16 shards, the mask token in the second, inside a ragged v-tile
    "bf16_2": (scaled(B8X2X32_BF16, n_seq=4, n_slots=2, d=192, V=3000, mask_token_id=2100), [1111]),
    # four shards, one of them narrower than a v-tile
    "bf16_4": (scaled(B8X2X32_BF16, n_seq=4, n_slots=2, d=256, V=3000), [700, 900, 2000]),
    # E4M3 shards with their row scales (the 8-bit path), three shards
    "e4m3_3": (scaled(B256X8X64_E4M3, n_seq=3, n_slots=2, d=256, V=4000, mask_token_id=0), [1024, 2900]),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_split_matches_the_oracle_on_the_whole_head(name):
    cfg, cuts = CASES[name]
    wl = generate(cfg)
    out, (pm, ps, pa) = run_split(wl, shard_bounds(cfg.V, cuts))
    ref = oracle_on_workload(wl)
    rep = compare(out, ref, wl.tau, cfg.weight_dtype, cfg.block_len, cfg.n_slots)
    assert rep.ok(), rep.failures
    assert rep.n_live > 0
    # positions without a prediction carry the empty partial in every shard
    live = ref["tokens"] >= 0
    assert torch.all(pm[:, ~torch.from_numpy(live)] == -np.inf)
    assert torch.all(pa[:, ~torch.from_numpy(live)] == -1)
    assert torch.all(ps[:, ~torch.from_numpy(live)] == 0)
    # every shard's argmax lies in its own rows
    for g, (lo, hi) in enumerate(shard_bounds(cfg.V, cuts)):
        a = pa[g, torch.from_numpy(live)]
        assert torch.all((a >= lo) & (a < hi))


@pytest.mark.parametrize("name", sorted(CASES))
def test_split_agrees_with_the_single_call(name):
    cfg, cuts = CASES[name]
    wl = generate(cfg)
    out, _ = run_split(wl, shard_bounds(cfg.V, cuts))
    g = wl.to("cuda")
    tokens, conf, commit, _ = bdc.commit_step(g.hidden, g.weight, g.pos_masked, g.block_flags, cfg.n_seq,
                                              cfg.n_slots, cfg.block_len, wl.tau, weight_scale=g.weight_scale,
                                              mask_token_id=cfg.mask_token_id)
    torch.cuda.synchronize()
    # the same per-part arithmetic, merged in another grouping: tokens equal,
    # confidences equal up to the order of the fp32 sums
    assert np.array_equal(out["tokens"], tokens.cpu().numpy())
    assert np.abs(out["conf"] - conf.cpu().numpy()).max() < 1e-5


@pytest.mark.parametrize("share", ["0", "1"])
@pytest.mark.parametrize("name", ["bf16_4", "e4m3_3"])
def test_split_with_spill_pairs(name, share, monkeypatch):
    # each shard's LM head on clusters of two pairs (sharing head tiles or
    # token rows) plus the spill launch
    monkeypatch.setenv("BD_PAIR_MC", "2")
    monkeypatch.setenv("BD_PAIR_SPILL", "1")
    monkeypatch.setenv("BD_SPILL_PCT", "50")
    monkeypatch.setenv("BD_PAIR_SHARE", share)
    cfg, cuts = CASES[name]
    wl = generate(cfg)
    out, _ = run_split(wl, shard_bounds(cfg.V, cuts))
    rep = compare(out, oracle_on_workload(wl), wl.tau, cfg.weight_dtype, cfg.block_len, cfg.n_slots)
    assert rep.ok(), rep.failures
    assert rep.n_live > 0


def test_argument_errors():
    cfg, cuts = CASES["bf16_2"]
    wl = generate(cfg).to("cuda")
    P = cfg.P
    m = torch.empty(P, device="cuda")
    s_ = torch.empty(P, device="cuda")
    a = torch.empty(P, dtype=torch.int32, device="cuda")
    args = (wl.hidden, wl.weight[:100], None, 0, wl.pos_masked, wl.block_flags, cfg.n_seq, cfg.n_slots,
            cfg.block_len, -1, m, s_, a)
    assert B.bd_lmhead_partials(*args) == B.BD_OK
    bad = list(args)
    bad[3] = -1
    assert B.bd_lmhead_partials(*bad) == B.BD_ERR_ARG
    tok = torch.empty(P, dtype=torch.int32, device="cuda")
    conf = torch.empty(P, device="cuda")
    com = torch.empty(P, dtype=torch.int32, device="cuda")
    margs = [m, s_, a, 1, wl.pos_masked, wl.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len, wl.tau, tok, conf, com]
    assert B.bd_merge_commit(*margs) == B.BD_OK
    for k, v in ((3, 0), (3, 5000)):
        b2 = list(margs)
        b2[k] = v
        assert B.bd_merge_commit(*b2) == B.BD_ERR_ARG
    b2 = list(margs)
    b2[9] = ()
    assert B.bd_merge_commit(*b2) == B.BD_ERR_TAU
    torch.cuda.synchronize()
    assert bdc.bd_get_device_status() == 0


# ------------------------------------------------------------ two gloo ranks --

def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import paper_2609_33887_gb300 as lib

        torch.cuda.set_device(0)
        cfg, _ = CASES["bf16_2"]
        wl = generate(cfg)
        g = wl.to("cuda")
        V = cfg.V
        lo, hi = rank * V // world, (rank + 1) * V // world
        # this rank's shard of the head, on its device (the same GPU here)
        m, s_, a = lib.lmhead_partials(g.hidden, g.weight[lo:hi].clone(), lo, g.pos_masked, g.block_flags,
                                       cfg.n_seq, cfg.n_slots, cfg.block_len, mask_token_id=cfg.mask_token_id)
        torch.cuda.synchronize()
        assert lib.bd_get_device_status() == 0
        # the one exchange: 12 bytes per position and rank, through host memory
        mine = torch.stack([m.cpu(), s_.cpu(), a.cpu().view(torch.float32)])
        gathered = [torch.empty_like(mine) for _ in range(world)]
        dist.all_gather(gathered, mine)
        pm = torch.stack([t[0] for t in gathered]).contiguous().cuda()
        ps = torch.stack([t[1] for t in gathered]).contiguous().cuda()
        pa = torch.stack([t[2].view(torch.int32) for t in gathered]).contiguous().cuda()
        tokens, conf, commit, _ = lib.merge_commit(pm, ps, pa, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots,
                                                   cfg.block_len, wl.tau)
        torch.cuda.synchronize()
        out = {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
               "commit": commit.cpu().numpy().view(np.uint32)}
        ref = oracle_on_workload(wl)
        rep = compare(out, ref, wl.tau, cfg.weight_dtype, cfg.block_len, cfg.n_slots)
        q.put((rank, rep.failures, rep.n_live))
    except Exception as exc:  # noqa: BLE001 - reported to the parent
        q.put((rank, [repr(exc)], 0))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_exchange_the_library_partials():
    import torch.multiprocessing as mp

    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = [q.get(timeout=300) for _ in ps]
    for p in ps:
        p.join(timeout=60)
    for rank, failures, n_live in res:
        assert not failures, (rank, failures)
        assert n_live > 0
