"""dpo_grad_norm_noalloc, the gradient-norm entry point that allocates no
device memory, checked against the norm the clipped dpo_step computes and
against the oracle's fp64 sum of squares of the same values.

Some callers cannot call cudaMalloc: a framework whose caching allocator has
already reserved the GPU's memory, or a latency-critical loop that cannot take
the implicit device synchronization of cudaMalloc/cudaFree. For them the
library computes the global gradient norm and clip coefficient with its
scratch in a fixed device array. The results must equal what the existing
path (dpo_step with clipping, read back with dpo_get_flags) computes, and the
norm must match the plain fp64 sum to the norm bar of the parity tests
(1e-6 relative).

This file is named to be collected last, so a run that stops at its first
failure has run every other test before reaching it.
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
from paper_2606_30634_gb300 import dpo, synth

# ragged sizes; the largest spans several of the entry point's chunks
NUMELS = [4095, 8, 300_001, 0, 17, (1 << 21) + 5]
NORM_REL = 1e-6


def _call(L, grad, numel, grad_dtype, max_norm, norm, clip):
    stream = torch.cuda.current_stream().cuda_stream
    rc = L.dpo_grad_norm_noalloc(grad.data_ptr() if grad is not None else None, numel,
                                 grad_dtype, max_norm, norm.data_ptr(), clip.data_ptr(), stream)
    assert rc == dpo.DPO_OK
    torch.cuda.synchronize()
    return norm.item(), clip.item()


def _host_draw(n, grad_dtype, step, sigma=1e-3):
    """(device buffer, the oracle's fp64 sum of squares of its values)."""
    if grad_dtype == dpo.DPO_BF16:
        bits = synth.host_normal(91, synth.STREAM_GRAD, step, 0, n, sigma, synth.BF16)
        dev = torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
        return dev, oracle.sqnorm_bf16(bits)
    vals = synth.host_normal(91, synth.STREAM_GRAD, step, 0, n, sigma, synth.F32)
    return torch.from_numpy(vals).cuda(), oracle.sqnorm_f32(vals)


@pytest.mark.gpu
@pytest.mark.parametrize("grad_dtype", [dpo.DPO_BF16, dpo.DPO_F32])
def test_noalloc_norm_matches_clipped_step_on_two_calls(cuda_device, grad_dtype):
    L = dpo.load()
    opt = dpo.DelayedAdamW(NUMELS, grad_dtype=grad_dtype, ef=True, max_grad_norm=0.5,
                           device=cuda_device)
    norm = torch.zeros(1, dtype=torch.float64, device=cuda_device)
    clip = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    stream = torch.cuda.current_stream().cuda_stream
    offs = np.concatenate([[0], np.cumsum(NUMELS)])
    try:
        for k in (1, 2):   # two calls in a row, each on a fresh gradient
            for i, n in enumerate(NUMELS):
                if n:
                    synth.dev_normal(77, synth.STREAM_GRAD, k, int(offs[i]), opt.grads(i), 1e-3)
            # the whole zero-padded gradient arena: padding adds nothing to the norm
            rc = L.dpo_grad_norm_noalloc(opt.grad.data_ptr(), opt.grad.numel(), grad_dtype,
                                         0.5, norm.data_ptr(), clip.data_ptr(), stream)
            assert rc == dpo.DPO_OK
            opt.step()
            _, ref_norm, ref_clip = dpo.dpo_get_flags(opt.ctx)
            torch.cuda.synchronize()
            assert 0.0 < ref_clip < 1.0
            assert norm.item() == pytest.approx(ref_norm, rel=NORM_REL)
            assert clip.item() == pytest.approx(ref_clip, rel=NORM_REL)
    finally:
        opt.close()


@pytest.mark.gpu
@pytest.mark.parametrize("grad_dtype", [dpo.DPO_BF16, dpo.DPO_F32])
def test_noalloc_norm_matches_the_oracle_across_chunk_counts(cuda_device, grad_dtype):
    """Against the oracle's fp64 sum of the same values, over calls in a row
    whose chunk counts differ (3 chunks, then 1, then hundreds, then 1
    again): each call starts its arrival count from zero, whatever the last
    call left in the shared scratch."""
    L = dpo.load()
    norm = torch.zeros(1, dtype=torch.float64, device=cuda_device)
    clip = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    for step, n in enumerate([3 * 8192 - 5, 100, 4_194_311, 7, 20_000_003], start=1):
        g, sq = _host_draw(n, grad_dtype, step)
        got_norm, got_clip = _call(L, g, n, grad_dtype, 0.25, norm, clip)
        assert got_norm == pytest.approx(math.sqrt(sq), rel=NORM_REL), n
        assert got_clip == pytest.approx(oracle.clip_coef(sq, 0.25), rel=NORM_REL), n


@pytest.mark.gpu
def test_noalloc_degenerate_cases(cuda_device):
    """numel == 0 gives norm 0 and coefficient 1; max_grad_norm <= 0 gives 1
    (no clipping); a NaN in the gradient gives a NaN norm and coefficient, as
    the clipped dpo_step does."""
    L = dpo.load()
    norm = torch.full((1,), 7.0, dtype=torch.float64, device=cuda_device)
    clip = torch.full((1,), 7.0, dtype=torch.float32, device=cuda_device)
    assert _call(L, None, 0, dpo.DPO_BF16, 1.0, norm, clip) == (0.0, 1.0)

    g, sq = _host_draw(50_000, dpo.DPO_BF16, 1, sigma=1.0)   # norm ~ 224: would clip
    for max_norm in (0.0, -1.0):
        got_norm, got_clip = _call(L, g, 50_000, dpo.DPO_BF16, max_norm, norm, clip)
        assert got_norm == pytest.approx(math.sqrt(sq), rel=NORM_REL)
        assert got_clip == 1.0

    bad = g.clone()
    bad.view(torch.int16)[12_345] = 0x7FC0   # bf16 quiet NaN
    got_norm, got_clip = _call(L, bad, 50_000, dpo.DPO_BF16, 1.0, norm, clip)
    assert math.isnan(got_norm) and math.isnan(got_clip)
    assert math.isnan(oracle.clip_coef(float("nan"), 1.0))   # the oracle's reading
    # the next call is unaffected by the NaN one
    got_norm, _ = _call(L, g, 50_000, dpo.DPO_BF16, 1.0, norm, clip)
    assert got_norm == pytest.approx(math.sqrt(sq), rel=NORM_REL)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    L = dpo.load()
    fake = 1 << 40   # never dereferenced: the argument checks come first
    rc = L.dpo_grad_norm_noalloc(fake, dpo.DPO_NOALLOC_MAX_NUMEL + 1, dpo.DPO_BF16, 1.0,
                                 fake, fake, None)
    assert rc == dpo.DPO_EINVAL
    rc = L.dpo_grad_norm_noalloc(fake + 16, 100, dpo.DPO_BF16, 1.0, fake, fake, None)
    assert rc == dpo.DPO_EALIGN
    rc = L.dpo_grad_norm_noalloc(fake, 100, 5, 1.0, fake, fake, None)
    assert rc == dpo.DPO_EDTYPE
    for bad in (float("inf"), float("nan")):   # as dpo_init's hyperparameters
        rc = L.dpo_grad_norm_noalloc(fake, 100, dpo.DPO_BF16, bad, fake, fake, None)
        assert rc == dpo.DPO_EINVAL
