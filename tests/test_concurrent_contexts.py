"""Independent contexts stepping at once on two CUDA streams, as a framework
with several parameter groups (or an AdamW context beside a Muon one) runs
them: the launches of the two contexts interleave with no synchronization
between them, and each context still equals its own oracle (Alg. 1 with EF
and clipping; Alg. 2 with EF). The library keeps every scratch buffer in
its context, so nothing is shared between them."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from oracle.muon import DelayedMuon as OracleMuon, MuonHParams
from paper_2606_30634_gb300 import dpo, muon, synth
from parity_util import TOL_RUN, bf16_raw_ulps_above_floor, rel_err
from test_muon_parity import _flat, close_with_flips, inputs

pytestmark = pytest.mark.gpu

B = dpo.DPO_BF16
STEPS = 5


def _adamw(numels, seed, clip, device):
    """A clipped EF context on bf16 weights, gradients and stash, and its oracle."""
    total = sum(numels)
    offs = np.concatenate([[0], np.cumsum(numels)])
    opt = dpo.DelayedAdamW(numels, param_dtype=B, stash_dtype=B, grad_dtype=B, ef=True,
                           max_grad_norm=clip, device=device)
    for i in range(len(numels)):   # x_0 into each tensor's slice of the padded arena
        synth.dev_normal(seed, synth.STREAM_INIT, 0, int(offs[i]), opt.view(opt.master, i), 0.02)
    dpo.dpo_stash(opt.ctx)         # stash and bf16 weights := x_0
    x0h = synth.host_normal(seed, synth.STREAM_INIT, 0, 0, total, 0.02).astype(np.float64)
    hp = oracle.HParams(ef_lambda=1.0, max_grad_norm=clip).as_f32()
    ref = oracle.DelayedOptimizer(np.split(x0h, offs[1:-1]), hp, ef=True, x_store=oracle.F32,
                                  stash_store=oracle.BF16, param_store=oracle.BF16)
    return opt, ref, offs


def test_two_adamw_contexts_on_two_streams(cuda_device):
    sets = [([70_001, 13, 4099], 0xA1, 0.02), ([50_000, 777], 0xB2, 0.05)]
    runs = [_adamw(n, seed, clip, cuda_device) for n, seed, clip in sets]
    streams = [torch.cuda.Stream(cuda_device) for _ in runs]
    torch.cuda.synchronize()
    try:
        for k in range(1, STEPS + 1):
            for (opt, _, offs), (_, seed, _), s in zip(runs, sets, streams):
                with torch.cuda.stream(s):
                    for i in range(len(offs) - 1):
                        synth.dev_normal(seed, synth.STREAM_GRAD, k, int(offs[i]), opt.grads(i),
                                         1e-3)
                    opt.step(stream=s)
        torch.cuda.synchronize()
        for (opt, ref, offs), (numels, seed, _) in zip(runs, sets):
            total = sum(numels)
            for k in range(1, STEPS + 1):
                g = synth.bf16_bits_to_f32(synth.host_normal(seed, synth.STREAM_GRAD, k, 0, total,
                                                             1e-3, synth.BF16))
                ref.step(g.astype(np.float64), tag=ref.read_weights("stale")[1])
            assert ref.last_clip < 0.5   # clipping active in every context
            master = torch.cat([opt.view(opt.master, i) for i in range(len(numels))])
            assert rel_err(master.cpu().numpy().astype(np.float64), ref.x) <= TOL_RUN
            assert dpo.dpo_get_flags(opt.ctx)[2] == pytest.approx(ref.last_clip, rel=1e-6)
            latest = torch.cat([opt.view(opt.param, i) for i in range(len(numels))])
            bits = latest.view(torch.int16).cpu().numpy().view(np.uint16)
            assert bf16_raw_ulps_above_floor(bits, ref.read_weights("latest")[0])[0] <= 1
    finally:
        for opt, _, _ in runs:
            opt.close()


def test_two_muon_contexts_on_two_streams(cuda_device):
    """Each context's Newton-Schulz GEMMs are persistent launches over every
    SM; the two streams' launches queue behind one another's CTAs on the
    device, with no wait between them."""
    sets = [([(256, 768), (768, 256)], 0xC3), ([(300, 700)], 0xD4)]
    lr, ns = 2e-3, 1
    pairs = []
    for shapes, seed in sets:
        xs, _ = inputs(shapes, seed, 1)
        gpu = muon.DelayedMuon(shapes, lr=lr, ef=True, ns_steps=ns, device=cuda_device,
                               x0=[torch.from_numpy(x) for x in xs])
        hp = MuonHParams(lr=lr, ef_lambda=1.0, ns_steps=ns, ns_store=oracle.BF16).as_f32()
        ref = OracleMuon([x.astype(np.float64) for x in xs], hp, ef=True, x_store=oracle.F32,
                         stash_store=oracle.BF16, param_store=oracle.BF16)
        pairs.append((gpu, ref))
    streams = [torch.cuda.Stream(cuda_device) for _ in pairs]
    torch.cuda.synchronize()
    try:
        for k in range(STEPS):
            for (gpu, _), (shapes, seed), s in zip(pairs, sets, streams):
                _, gs = inputs(shapes, seed, k + 1)
                with torch.cuda.stream(s):
                    for i, g in enumerate(gs):
                        gpu.grads(i).copy_(torch.from_numpy(g.view(np.int16))
                                           .view(torch.bfloat16).reshape(g.shape),
                                           non_blocking=False)
                    gpu.step(stream=s)
        torch.cuda.synchronize()
        for (gpu, ref), (shapes, seed) in zip(pairs, sets):
            for k in range(STEPS):
                _, gs = inputs(shapes, seed, k + 1)
                ref.step([synth.bf16_bits_to_f32(g).astype(np.float64) for g in gs])
            assert gpu.status() == 0
            mom = np.concatenate([gpu.view(gpu.mom, i).cpu().numpy().ravel()
                                  for i in range(len(shapes))])
            master = np.concatenate([gpu.view(gpu.master, i).cpu().numpy().ravel()
                                     for i in range(len(shapes))])
            assert rel_err(mom.astype(np.float64), _flat(ref.mom)) <= TOL_RUN
            du = lr * 0.2 * np.sqrt(max(max(sh) for sh in shapes)) * 2.0 ** -7
            close_with_flips(master, _flat(ref.x), TOL_RUN, STEPS * du, 1e-3)
    finally:
        for gpu, _ in pairs:
            gpu.close()
