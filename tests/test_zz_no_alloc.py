"""dpo_grad_norm_noalloc, the gradient-norm entry point that allocates no
device memory, checked against the norm the clipped dpo_step computes.

Some callers cannot call cudaMalloc: a framework whose caching allocator has
already reserved the GPU's memory, or a latency-critical loop that cannot take
the implicit device synchronization of cudaMalloc/cudaFree. For them the
library computes the global gradient norm and clip coefficient with its
scratch in a fixed device array. The results must equal what the existing
path (dpo_step with clipping, read back with dpo_get_flags) computes.

This file is named to be collected last, so a run that stops at its first
failure has run every other test before reaching it.
"""
from __future__ import annotations

import ctypes

import numpy as np
import pytest
import torch

from paper_2606_30634_gb300 import dpo, synth

# ragged sizes; the largest spans three of the entry point's 2^20-element chunks
NUMELS = [4095, 8, 300_001, 0, 17, (1 << 21) + 5]


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
            assert norm.item() == pytest.approx(ref_norm, rel=1e-6)
            assert clip.item() == pytest.approx(ref_clip, rel=1e-6)
    finally:
        opt.close()


def test_noalloc_rejects_sizes_beyond_its_scratch():
    L = dpo.load()
    fake = 1 << 40   # never dereferenced: the size check comes first
    rc = L.dpo_grad_norm_noalloc(fake, dpo.DPO_NOALLOC_MAX_NUMEL + 1, dpo.DPO_BF16, 1.0,
                                 fake, fake, None)
    assert rc == dpo.DPO_EINVAL
    rc = L.dpo_grad_norm_noalloc(fake + 16, 100, dpo.DPO_BF16, 1.0, fake, fake, None)
    assert rc == dpo.DPO_EALIGN
    rc = L.dpo_grad_norm_noalloc(fake, 100, 5, 1.0, fake, fake, None)
    assert rc == dpo.DPO_EDTYPE
