"""The partitioned step as it runs under a launcher: two ranks, each its own
process with its own CUDA context and its own shard of the set (ZeRO-1
style), clipping from one global norm (App. E.1). Every step each rank adds
its shard's squared gradient norm (dpo_grad_sqnorm), the ranks sum the fp64
scalar with a torch.distributed all-reduce (gloo), and each rank's fused step
clips from the total (dpo_set_clip_source). The whole set then equals the
oracle over all parameters.

The test runs on the one GPU this suite has: both processes use device 0.
The exchange happens on the host between two launches of each rank, so no
kernel of one rank waits on a kernel of the other; the processes share the
GPU the way two jobs would.
"""
from __future__ import annotations

import os
import queue
import socket
from datetime import timedelta

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import oracle
from paper_2606_30634_gb300 import dpo, shard, synth
from parity_util import TOL_ONE_STEP, TOL_RUN, rel_err

pytestmark = pytest.mark.gpu

NUMELS = [3000, 517, 4096, 1, 2222, 9001]
WD_ON = [True, False, True, False, True, True]
SEED, SIGMA_X, SIGMA_G = 0x5A4E, 0.02, 1e-3
CLIP = 0.02          # below these gradients' norm (about 0.14): clipping is active
STEPS = 5
WORLD = 2


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, port: int, out) -> None:
    """One rank: its shard through the library, the norm summed over gloo.
    Sends (rank, step, per-piece arrays, clip coefficient) after each step,
    or (rank, "error", message)."""
    try:
        import torch.distributed as dist
        os.environ["MASTER_ADDR"] = "127.0.0.1"
        os.environ["MASTER_PORT"] = str(port)
        dist.init_process_group("gloo", rank=rank, world_size=WORLD,
                                timeout=timedelta(seconds=120))
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        starts = np.concatenate([[0], np.cumsum(NUMELS)])

        def fill(start, buf):   # this rank's start weights only
            synth.dev_normal(SEED, synth.STREAM_INIT, 0, int(start), buf, SIGMA_X)

        opt, pieces = shard.shard_optimizer(NUMELS, WORLD, rank, wd_on=WD_ON, x0=fill, ef=True,
                                            stash_dtype=dpo.DPO_BF16, max_grad_norm=CLIP,
                                            device=dev)
        acc = torch.zeros(1, dtype=torch.float64, device=dev)
        opt.set_clip_source(acc)
        try:
            for k in range(1, STEPS + 1):
                for j, (i, a, _) in enumerate(pieces):
                    synth.dev_normal(SEED, synth.STREAM_GRAD, k, int(starts[i]) + a,
                                     opt.grads(j), SIGMA_G)
                dpo.global_sqnorm([opt], acc)   # own share, then the all-reduce
                opt.step()
                torch.cuda.synchronize(dev)
                arrays = [(i, a, b, opt.view(opt.master, j).cpu().numpy(),
                           opt.view(opt.m, j).cpu().numpy(), opt.view(opt.v, j).cpu().numpy())
                          for j, (i, a, b) in enumerate(pieces)]
                out.put((rank, k, arrays, dpo.dpo_get_flags(opt.ctx)[2], acc.item()))
        finally:
            opt.close()
        dist.barrier()
        dist.destroy_process_group()
    except Exception as e:   # reported to the test, which fails with it
        out.put((rank, "error", repr(e)))


def test_two_rank_processes_step_one_set(cuda_device):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, port, out)) for r in range(WORLD)]
    for p in procs:
        p.start()
    got = {}
    try:
        while len(got) < WORLD * STEPS:
            try:
                msg = out.get(timeout=300)
            except queue.Empty:
                pytest.fail("a rank sent nothing for 300 s")
            if msg[1] == "error":
                pytest.fail(f"rank {msg[0]}: {msg[2]}")
            got[(msg[0], msg[1])] = msg[2:]
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0, p.exitcode
    finally:
        for p in procs:
            if p.is_alive():
                p.terminate()
                p.join(timeout=30)

    total = sum(NUMELS)
    starts = np.concatenate([[0], np.cumsum(NUMELS)])
    x0 = synth.host_normal(SEED, synth.STREAM_INIT, 0, 0, total, SIGMA_X).astype(np.float64)
    hp = oracle.HParams(ef_lambda=1.0, max_grad_norm=CLIP).as_f32()
    ref = oracle.DelayedOptimizer(np.split(x0, starts[1:-1]), hp, ef=True, x_store=oracle.F32,
                                  stash_store=oracle.BF16, param_store=oracle.BF16, wd_on=WD_ON)
    for k in range(1, STEPS + 1):
        g = synth.bf16_bits_to_f32(synth.host_normal(SEED, synth.STREAM_GRAD, k, 0, total,
                                                     SIGMA_G, synth.BF16)).astype(np.float64)
        ref.step(g, tag=ref.read_weights("stale")[1])
        assert ref.last_clip < 0.5
        master, m, v = np.full(total, np.nan), np.full(total, np.nan), np.full(total, np.nan)
        for r in range(WORLD):
            arrays, clip, sq = got[(r, k)]
            # the all-reduced scalar is the squared norm over the whole set
            assert sq == pytest.approx(oracle.sqnorm(g), rel=1e-6)
            assert clip == pytest.approx(ref.last_clip, rel=1e-6)
            for i, a, b, xm, xmm, xv in arrays:
                lo = int(starts[i])
                master[lo + a:lo + b] = xm
                m[lo + a:lo + b] = xmm
                v[lo + a:lo + b] = xv
        assert not np.isnan(master).any()   # the ranks' pieces cover the set
        tol = TOL_ONE_STEP if k == 1 else TOL_RUN
        assert rel_err(master, ref.x) <= tol
        assert rel_err(m, ref.m) <= tol
        assert rel_err(v, ref.v) <= tol
