"""GPU parity on the five workloads at full size, in the launch configuration
the benchmark times.

flat 1M and the 16M quadratic are compared on every element (the quadratic's
loss trajectory too, every step, for the full 1000 steps). The three model-
shaped sets (124M, 1.24B, 6.74B parameters) are compared on a sample: ~1e6
random elements plus the first and last elements of every tensor; the step is
elementwise, so the oracle regenerates the seeded inputs of just those
elements. The clipped 1.24B set needs the whole gradient's norm each step,
which the oracle computes from a full host-side draw; it runs all of its 50
steps.

The quadratic loop's EF buffer is held to the normwise bound (see
parity_util): the delayed EF loop amplifies per-step rounding differences.
Its elementwise figure is still computed at every comparison and printed in
the session's parity summary.
"""
from __future__ import annotations

import gc

import numpy as np
import pytest
import torch

import oracle
from paper_2606_30634_gb300 import dpo, synth
from paper_2606_30634_gb300.synth import workloads as W
from parity_util import TOL_ONE_STEP, TOL_RUN, Case, Run, rel_err, sample_indices

pytestmark = pytest.mark.gpu


def _case(w: W.Workload, ef: bool, correction: int = dpo.DPO_CORR_EF,
          stash_mode: int = None) -> Case:
    """The workload as the benchmark runs it: the ping-pong stash where the
    layout allows it (bf16 param and stash, the standard rule or EF)."""
    if stash_mode is None:
        pp = (w.param_dtype == W.BF16 and w.stash_dtype == W.BF16
              and correction == dpo.DPO_CORR_EF)
        stash_mode = dpo.DPO_STASH_PINGPONG if pp else dpo.DPO_STASH_COPY
    return Case(w.numels, param_dtype=w.param_dtype, stash_dtype=w.stash_dtype,
                grad_dtype=w.grad_dtype, ef=ef, max_grad_norm=w.max_grad_norm, lr=w.lr,
                weight_decay=w.weight_decay, seed=w.seed, grad_sigma=W.GRAD_SIGMA,
                init_sigma=W.INIT_SIGMA, correction=correction, stash_mode=stash_mode)


def _free():
    gc.collect()
    torch.cuda.empty_cache()


def _run_steps(run: Run, steps: int, check_every: int = 1):
    worst = {}
    for k in range(1, steps + 1):
        run.step()
        if k == 1 or k % check_every == 0 or k == steps:
            e = run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
            for key, v in e.items():
                worst[key] = max(worst.get(key, 0), v)
    return worst


@pytest.mark.parametrize("ef", [False, True])
def test_flat_1m_fp32(cuda_device, ef):
    w = W.FLAT
    run = Run(_case(w, ef), cuda_device)
    try:
        _run_steps(run, w.steps)
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("ef", [True, False])
def test_quadratic_16m_1000_steps(cuda_device, ef):
    """Emulated delayed training on the noisy diagonal quadratic: each step
    evaluates the gradient and the loss at the stash (the weights a delayed
    forward/backward reads), then steps. Loss trajectory and final state
    against the oracle running the same loop on the host."""
    w = W.QUADRATIC
    N = w.n_params
    case = _case(w, ef)
    run = Run(case, cuda_device)
    try:
        u = synth.host_uniform(w.seed, synth.STREAM_CURV, 0, 0, N)
        a_host = synth.curvature_from_uniform(u)
        a = torch.from_numpy(a_host).to(cuda_device)
        wstar = torch.empty(N, dtype=torch.float32, device=cuda_device)
        synth.dev_normal(w.seed, synth.STREAM_TARGET, 0, 0, wstar, 1.0)
        wstar_host = synth.host_normal(w.seed, synth.STREAM_TARGET, 0, 0, N, 1.0)
        a64, ws64 = a_host.astype(np.float64), wstar_host.astype(np.float64)
        partials = torch.empty(1024, dtype=torch.float64, device=cuda_device)
        gpu_loss, ref_loss = [], []
        for k in range(1, w.steps + 1):
            synth.dev_quadratic(w.seed, k, a, wstar, run.gpu.stale(0), W.QUAD_NOISE_SIGMA,
                                run.gpu.grads(0), partials)
            run.gpu.step()
            gpu_loss.append(0.5 * float(partials.sum().item()))
            stale, tag = run.ref.read_weights("stale")
            noise = synth.host_normal(w.seed, synth.STREAM_NOISE, k, 0, N, W.QUAD_NOISE_SIGMA)
            g, loss = oracle.quadratic(a64, ws64, stale, noise, oracle.F32)
            ref_loss.append(loss)
            run.ref.step(g, tag=tag)
            run.k = k
            if k == 1:
                run.assert_close(TOL_ONE_STEP)
            elif k % 250 == 0:
                run.assert_close(TOL_RUN, normwise=("ef",))
        gl, rl = np.array(gpu_loss), np.array(ref_loss)
        assert np.max(np.abs(gl - rl) / np.abs(rl)) <= TOL_RUN
        assert rl[-1] < 0.9 * rl[0]   # the emulated training makes progress
        run.assert_close(TOL_RUN, normwise=("ef",))
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("ef", [False, True])
def test_gpt2_small_124m(cuda_device, ef):
    w = W.GPT2_SMALL
    run = Run(_case(w, ef), cuda_device, sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=10)
    finally:
        run.close()
        _free()


def test_llama_1b_clipped(cuda_device):
    """Global-norm clipping at 1.0 over all 146 tensors (the gradient norm of
    N(0, 1e-3^2) draws over 1.24e9 elements is about 35, so every step clips);
    EF on; all 50 steps. The GPU's norm matches the oracle's full fp64 norm
    each step."""
    w = W.LLAMA_1B
    assert w.steps == 50
    run = Run(_case(w, True), cuda_device, sample=sample_indices(w.numels, 1_000_000))
    try:
        for k in range(1, w.steps + 1):
            run.step()
            e = run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
            _, norm, coef = dpo.dpo_get_flags(run.gpu.ctx)
            assert norm ** 2 == pytest.approx(run.ref.last_sqnorm, rel=1e-6)
            assert coef == pytest.approx(run.ref.last_clip, rel=1e-6)
            assert coef < 0.05
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("ef,stash", [(True, None), (False, None),
                                      (True, dpo.DPO_STASH_COPY)])
def test_llama_7b(cuda_device, ef, stash):
    """The 6.74e9-parameter set: bf16 params, stash and grads, fp32
    master/m/v (and EF buffer): ~148 GB resident with EF. As the benchmark
    runs it (the ping-pong stash), and with the copying stash."""
    w = W.LLAMA_7B
    run = Run(_case(w, ef, stash_mode=stash), cuda_device,
              sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=5)
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("corr", [dpo.DPO_CORR_SAPIPE_SAME, dpo.DPO_CORR_SAPIPE_UPDATED])
def test_gpt2_small_sapipe(cuda_device, corr):
    """SAPipe-WP prediction (App. B.1) on the 124M set, 100 steps."""
    w = W.GPT2_SMALL
    run = Run(_case(w, True, corr), cuda_device, sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=10)
    finally:
        run.close()
        _free()


def test_llama_7b_sapipe_updated(cuda_device):
    w = W.LLAMA_7B
    run = Run(_case(w, True, dpo.DPO_CORR_SAPIPE_UPDATED), cuda_device,
              sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=5)
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("rule,kw", [
    ("nadam", dict(optimizer=dpo.DPO_OPT_NADAM)),
    ("lion", dict(optimizer=dpo.DPO_OPT_LION, beta1=0.9, beta2=0.99, lr=5e-4, weight_decay=0.5)),
    ("adan", dict(optimizer=dpo.DPO_OPT_ADAN, beta1=0.98, beta2=0.92, beta3=0.99)),
])
def test_gpt2_small_other_rules_ef(cuda_device, rule, kw):
    """NAdam, Lion and Adan with EF on the 124M set, 100 steps (Tab. ef_360m
    compares these under EF)."""
    w = W.GPT2_SMALL
    case = _case(w, True)
    for key, val in kw.items():
        setattr(case, key, val)
    run = Run(case, cuda_device, sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=10)
    finally:
        run.close()
        _free()


@pytest.mark.parametrize("rule,kw", [
    ("nadam", dict(optimizer=dpo.DPO_OPT_NADAM)),
    ("lion", dict(optimizer=dpo.DPO_OPT_LION, beta1=0.9, beta2=0.99, lr=5e-4, weight_decay=0.5)),
    ("adan", dict(optimizer=dpo.DPO_OPT_ADAN, beta1=0.98, beta2=0.92, beta3=0.99)),
])
def test_gpt2_small_other_rules_sapipe_updated(cuda_device, rule, kw):
    """SAPipe-WP with the updated state (App. B.1) for NAdam, Lion and Adan
    on the 124M set, 100 steps: each rule's own step at k + 1 predicts the
    point the next gradient is taken at."""
    w = W.GPT2_SMALL
    case = _case(w, True, dpo.DPO_CORR_SAPIPE_UPDATED)
    for key, val in kw.items():
        setattr(case, key, val)
    run = Run(case, cuda_device, sample=sample_indices(w.numels, 1_000_000))
    try:
        _run_steps(run, w.steps, check_every=10)
    finally:
        run.close()
        _free()
