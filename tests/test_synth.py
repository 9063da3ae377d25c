"""Seeded input generator: known answers, distribution, host/device identity."""
from __future__ import annotations

import os

import numpy as np
import pytest
import torch

from paper_2606_30634_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def test_philox_known_answers():
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        assert synth.philox(v[0:4], v[4:6]) == v[6:10]


def test_normal_moments_and_support():
    x = synth.host_normal(123, synth.STREAM_GRAD, 1, 0, 2_000_000, 1e-3).astype(np.float64)
    assert abs(x.mean()) < 3e-6
    assert x.std() == pytest.approx(1e-3, rel=3e-3)
    assert np.abs(x).max() <= 4 * np.sqrt(1.5) * 1e-3 * (1 + 1e-6)
    # excess kurtosis of Irwin-Hall(8) is -6/40
    k = np.mean((x / x.std()) ** 4) - 3
    assert k == pytest.approx(-0.15, abs=0.02)


def test_streams_steps_and_indices_are_independent():
    a = synth.host_normal(1, 1, 1, 0, 1000, 1.0)
    assert not np.array_equal(a, synth.host_normal(1, 1, 2, 0, 1000, 1.0))
    assert not np.array_equal(a, synth.host_normal(1, 2, 1, 0, 1000, 1.0))
    assert not np.array_equal(a, synth.host_normal(2, 1, 1, 0, 1000, 1.0))
    # a value depends only on its global index
    b = synth.host_normal(1, 1, 1, 400, 600, 1.0)
    np.testing.assert_array_equal(a[400:], b)
    idx = np.array([999, 0, 401, 5_000_000_000])
    at = synth.host_normal_at(1, 1, 1, idx, 1.0)
    np.testing.assert_array_equal(at[:3], a[[999, 0, 401]])
    assert at[3] == synth.host_normal(1, 1, 1, 5_000_000_000, 1, 1.0)[0]


def test_bf16_draws_are_rne_of_fp32_draws():
    f = synth.host_normal(9, 1, 3, 0, 100_000, 1e-3)
    b = synth.host_normal(9, 1, 3, 0, 100_000, 1e-3, dtype=synth.BF16)
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(b, ref)


def test_uniform_range():
    u = synth.host_uniform(5, synth.STREAM_CURV, 0, 0, 100_000)
    assert u.min() >= 0.0 and u.max() < 1.0
    assert u.mean() == pytest.approx(0.5, abs=0.01)
    a = synth.curvature_from_uniform(u)
    assert a.min() >= np.float32(1e-3) * (1 - 1e-6) and a.max() <= 1.0


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_device_fill_equals_host_fill(cuda_device, dtype):
    n, off = 1_000_003, 7_777
    out = torch.empty(n, dtype=dtype, device=cuda_device)
    synth.dev_normal(0xD0D0, synth.STREAM_GRAD, 4, off, out, 1e-3)
    torch.cuda.synchronize()
    if dtype == torch.float32:
        ref = synth.host_normal(0xD0D0, synth.STREAM_GRAD, 4, off, n, 1e-3)
        np.testing.assert_array_equal(out.cpu().numpy(), ref)
    else:
        ref = synth.host_normal(0xD0D0, synth.STREAM_GRAD, 4, off, n, 1e-3, dtype=synth.BF16)
        np.testing.assert_array_equal(out.cpu().view(torch.int16).numpy().view(np.uint16), ref)
