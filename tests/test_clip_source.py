"""GPU parity of global clipping across contexts (App. E.1: one norm over all
parameters): an AdamW context and a delayed-Muon context clipping from one
shared sum of squares, and a parameter set partitioned into two shards
(``paper_2606_30634_gb300.shard``) stepping as one. Through the C ABI
(dpo_grad_sqnorm, dpo_set_clip_source and their dpo_muon twins), against
the oracle, which clips from the squared norm over every gradient."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_2606_30634_gb300 import dpo, shard, synth
from parity_util import TOL_ONE_STEP, TOL_RUN, Case, Run, rel_err
from test_muon_parity import Pair, _flat

pytestmark = pytest.mark.gpu

B = dpo.DPO_BF16
CLIP = 0.04   # well below the norm of these gradients (about 0.6): clipping is active


def test_shared_clip_adamw_and_muon(cuda_device):
    run = Run(Case(numels=[4096, 1000, 77, 0, 300], ef=True, stash_dtype=B, max_grad_norm=CLIP,
                   seed=0x5C1), cuda_device)
    pair = Pair([(256, 512), (300, 700)], cuda_device, ns_steps=1, max_grad_norm=CLIP)
    acc = torch.zeros(1, dtype=torch.float64, device=cuda_device)
    run.gpu.set_clip_source(acc)
    pair.gpu.set_clip_source(acc)
    try:
        for k in range(1, 5):
            own = k == 4   # the last call goes back to each context's own norm
            if own:
                run.gpu.set_clip_source(None)
                pair.gpu.set_clip_source(None)
            g = run.draw(k)
            gs = pair.draw(k)
            if not own:
                dpo.global_sqnorm([run.gpu, pair.gpu], acc)
            run.gpu.step()
            pair.gpu.step()
            sq_a = oracle.sqnorm(g)
            sq_m = sum(oracle.sqnorm(x) for x in gs)
            run.ref.step(g, tag=run.ref.read_weights("stale")[1],
                         sq=sq_a if own else sq_a + sq_m)
            pair.ref.step(gs, sq=sq_m if own else sq_a + sq_m)
            run.k = pair.k = k
            torch.cuda.synchronize()
            if not own:
                assert acc.item() == pytest.approx(sq_a + sq_m, rel=1e-6)
                assert pair.ref.last_clip == run.ref.last_clip < 0.2
            _, norm, clip = dpo.dpo_get_flags(run.gpu.ctx)
            assert norm == pytest.approx(np.sqrt(sq_a if own else sq_a + sq_m), rel=1e-6)
            assert clip == pytest.approx(run.ref.last_clip, rel=1e-6)
            tol = TOL_ONE_STEP if k == 1 else TOL_RUN
            run.assert_close(tol)
            assert rel_err(pair.cat(pair.gpu.mom), _flat(pair.ref.mom)) <= tol
    finally:
        run.close()
        pair.close()


def test_partitioned_set_steps_as_one(cuda_device):
    """Two shards of one set (ragged tensors split across the boundary), each
    its own context, clipping from the summed norm, equal the oracle over the
    whole set."""
    numels = [3000, 517, 4096, 1, 2222]
    wd_on = [True, False, True, False, True]
    seed, sigma_x, sigma_g = 0x5A4D, 0.02, 1e-3
    total = sum(numels)
    x0 = torch.empty(total, dtype=torch.float32, device=cuda_device)
    synth.dev_normal(seed, synth.STREAM_INIT, 0, 0, x0, sigma_x)
    opts = [shard.shard_optimizer(numels, 2, r, wd_on=wd_on, x0=x0, ef=True, stash_dtype=B,
                                  max_grad_norm=0.02, device=cuda_device) for r in range(2)]
    acc = torch.zeros(1, dtype=torch.float64, device=cuda_device)
    for o, _ in opts:
        o.set_clip_source(acc)
    starts = np.concatenate([[0], np.cumsum(numels)])
    x0_h = synth.host_normal(seed, synth.STREAM_INIT, 0, 0, total, sigma_x).astype(np.float64)
    hp = oracle.HParams(ef_lambda=1.0, max_grad_norm=0.02).as_f32()
    ref = oracle.DelayedOptimizer(np.split(x0_h, starts[1:-1]), hp, ef=True,
                                  x_store=oracle.F32, stash_store=oracle.BF16,
                                  param_store=oracle.BF16, wd_on=wd_on)
    try:
        for k in range(1, 6):
            for o, pieces in opts:
                for j, (i, a, b) in enumerate(pieces):
                    synth.dev_normal(seed, synth.STREAM_GRAD, k, int(starts[i]) + a,
                                     o.grads(j), sigma_g)
            dpo.global_sqnorm([o for o, _ in opts], acc)
            for o, _ in opts:
                o.step()
            g = synth.bf16_bits_to_f32(synth.host_normal(seed, synth.STREAM_GRAD, k, 0, total,
                                                         sigma_g, synth.BF16))
            ref.step(g.astype(np.float64), tag=ref.read_weights("stale")[1])
            assert ref.last_clip < 0.5
            torch.cuda.synchronize()
            master = np.empty(total)
            m = np.empty(total)
            for o, pieces in opts:
                for j, (i, a, b) in enumerate(pieces):
                    lo = int(starts[i])
                    master[lo + a:lo + b] = o.view(o.master, j).cpu().numpy()
                    m[lo + a:lo + b] = o.view(o.m, j).cpu().numpy()
            tol = TOL_ONE_STEP if k == 1 else TOL_RUN
            assert rel_err(master, ref.x) <= tol
            assert rel_err(m, ref.m) <= tol
            for o, _ in opts:
                assert dpo.dpo_get_flags(o.ctx)[2] == pytest.approx(ref.last_clip, rel=1e-6)
    finally:
        for o, _ in opts:
            o.close()
