"""Host logic of the partitioned step (paper_2606_30634_gb300.shard): the
pieces tile the set exactly once with aligned, near-equal ranges, and two
gloo ranks (CPU) that each step their shard with the oracle, exchanging only
the squared gradient norm through ``dpo.allreduce_sqnorm``, reproduce the
oracle over the whole set with global clipping (App. E.1)."""
from __future__ import annotations

import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2606_30634_gb300 import dpo, shard

NUMELS = [3000, 517, 4096, 1, 0, 2222]


@pytest.mark.parametrize("world", [1, 2, 3, 7, 64])
def test_pieces_tile_the_set(world):
    numels = NUMELS
    cover = [np.zeros(n, np.int32) for n in numels]
    total = sum(numels)
    sizes = []
    for r in range(world):
        lo, hi = shard.bounds(total, world, r)
        sizes.append(hi - lo)
        if r < world - 1:
            assert hi % dpo.ALIGN_ELEMS == 0
        pieces = shard.partition(numels, world, r)
        assert sum(b - a for _, a, b in pieces) == hi - lo
        assert [i for i, _, _ in pieces] == sorted({i for i, _, _ in pieces})
        for i, a, b in pieces:
            assert 0 <= a < b <= numels[i]
            cover[i][a:b] += 1
    assert all((c == 1).all() for c in cover)
    assert sum(sizes) == total
    assert max(sizes) - min(sizes) <= 2 * dpo.ALIGN_ELEMS   # each cut moves down < ALIGN


def test_bounds_rejects_bad_ranks():
    with pytest.raises(ValueError):
        shard.bounds(10, 2, 2)
    with pytest.raises(ValueError):
        shard.bounds(10, 0, 0)
    assert shard.bounds(0, 4, 3) == (0, 0)
    assert shard.partition([0, 0], 2, 1) == []


@pytest.mark.parametrize("world,rank", [(1, 0), (2, 1), (3, 0), (3, 2)])
def test_shard_optimizer_seeds_each_piece(monkeypatch, world, rank):
    """A fill function (start, out) seeds the shard's master exactly as the
    full flat weights would: each piece reads its own global range, into its
    own offset of the shard's arena layout; flags follow their tensors."""
    import torch
    got = []

    class Capture:   # stands in for the device context (no GPU here)
        def __init__(self, numels, **kw):
            got.append((list(numels), kw))

    monkeypatch.setattr(shard, "DelayedAdamW", Capture)
    full = torch.arange(sum(NUMELS), dtype=torch.float32) * 0.5 - 7.0
    calls = []

    def fill(start, out):
        calls.append((start, out.numel()))
        out.copy_(full[start:start + out.numel()])

    wd = [True, False, True, True, False, True]
    _, pieces = shard.shard_optimizer(NUMELS, world, rank, x0=fill, device="cpu", wd_on=wd)
    _, pieces2 = shard.shard_optimizer(NUMELS, world, rank, x0=full, wd_on=wd)
    assert pieces == pieces2
    starts = np.concatenate([[0], np.cumsum(NUMELS)])
    assert calls == [(int(starts[i]) + a, b - a) for i, a, b in pieces]
    (n1, kw1), (n2, kw2) = got
    assert n1 == n2 == [b - a for _, a, b in pieces]
    assert torch.equal(kw1["x0"], kw2["x0"])
    assert kw1["wd_on"] == [wd[i] for i, _, _ in pieces]


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _oracle_setup(seed=0x5A4D, sigma_x=0.02):
    import oracle
    from paper_2606_30634_gb300 import synth
    total = sum(NUMELS)
    x0 = synth.host_normal(seed, synth.STREAM_INIT, 0, 0, total, sigma_x).astype(np.float64)
    hp = oracle.HParams(ef_lambda=1.0, max_grad_norm=0.02).as_f32()
    return x0, hp


def _grad(k, seed=0x5A4D, sigma=1e-3):
    from paper_2606_30634_gb300 import synth
    g = synth.host_normal(seed, synth.STREAM_GRAD, k, 0, sum(NUMELS), sigma, synth.BF16)
    return synth.bf16_bits_to_f32(g).astype(np.float64)


def _rank(rank, world, port, steps, q):
    import torch
    import torch.distributed as dist
    import oracle
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        x0, hp = _oracle_setup()
        starts = np.concatenate([[0], np.cumsum(NUMELS)])
        pieces = shard.partition(NUMELS, world, rank)
        idx = np.concatenate([np.arange(starts[i] + a, starts[i] + b) for i, a, b in pieces])
        wd = np.array([i % 2 == 0 for i in range(len(NUMELS))])
        t_of = np.searchsorted(starts, idx, side="right") - 1
        ref = oracle.DelayedOptimizer([x0[idx]], hp, ef=True, x_store=oracle.F32,
                                      stash_store=oracle.BF16, param_store=oracle.BF16)
        ref.mask = wd[t_of].astype(np.uint8)
        local = []
        for k in range(1, steps + 1):
            g = _grad(k)[idx]
            acc = torch.tensor([oracle.sqnorm(g)], dtype=torch.float64)
            local.append(float(acc.item()))
            dpo.allreduce_sqnorm(acc)
            ref.step(g, sq=float(acc.item()))
        q.put((rank, idx, ref.x.copy(), ref.m.copy(), ref.last_clip, local))
    finally:
        dist.destroy_process_group()


def test_two_ranks_step_as_one_gloo():
    import oracle
    world, steps = 2, 4
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, steps, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=180) for _ in procs), key=lambda r: r[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0

    x0, hp = _oracle_setup()
    starts = np.concatenate([[0], np.cumsum(NUMELS)])
    wd = [i % 2 == 0 for i in range(len(NUMELS))]
    full = oracle.DelayedOptimizer(np.split(x0, starts[1:-1]), hp, ef=True, x_store=oracle.F32,
                                   stash_store=oracle.BF16, param_store=oracle.BF16, wd_on=wd)
    for k in range(1, steps + 1):
        full.step(_grad(k))
    assert full.last_clip < 0.5   # clipping is active (the norm is about 0.1)
    for rank, idx, x, m, clip, local in res:
        assert local[-1] < full.last_sqnorm
        assert clip == pytest.approx(full.last_clip, rel=1e-12)
        # the two norms differ only in fp64 summation order, so the fp32-stored
        # state agrees but for a rare one-ulp rounding flip
        np.testing.assert_allclose(x, full.x[idx], rtol=0, atol=1e-8)
        np.testing.assert_allclose(m, full.m[idx], rtol=1e-6, atol=0)
    got = np.sort(np.concatenate([r[1] for r in res]))
    assert (got == np.arange(sum(NUMELS))).all()
