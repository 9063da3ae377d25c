"""GPU parity: the CUDA path through the C ABI against the oracle, element by
element, on small seeded tables spanning many CTAs, ragged tails and empty
tensors, in every supported dtype / mode combination."""
from __future__ import annotations

import ctypes

import numpy as np
import pytest
import torch

from paper_2606_30634_gb300 import dpo, synth
import oracle
from parity_util import TOL_ONE_STEP, TOL_RUN, Case, Run, bf16_ord, bf16_ulps, rel_err

pytestmark = pytest.mark.gpu

# many CTA ranges, 8-element packets with partial tails, an empty tensor
RAGGED = [1, 7, 8, 9, 4095, 4096, 65537, 0, 3, 300_001, 33]

F, B = dpo.DPO_F32, dpo.DPO_BF16

COMBOS = [
    # param, stash, grad, ef, clip, delay
    (B, F, B, False, 0.0, 1),   # GPT-2 / Llama-1B-like layout
    (B, F, B, True, 0.0, 1),
    (B, F, B, True, 0.3, 1),    # clipped (the norm of this table is ~0.6)
    (B, B, B, True, 0.0, 1),    # Llama-7B layout
    (B, B, B, False, 0.0, 1),
    (F, F, F, False, 0.0, 1),   # flat fp32
    (F, F, F, True, 0.0, 1),
    (F, B, F, True, 0.05, 1),
    (B, F, F, False, 0.0, 0),   # synchronous AdamW
    (F, F, B, False, 0.02, 0),
]


@pytest.mark.parametrize("pdt,sdt,gdt,ef,clip,delay", COMBOS)
def test_ragged_table_parity(cuda_device, pdt, sdt, gdt, ef, clip, delay):
    case = Case(RAGGED, param_dtype=pdt, stash_dtype=sdt, grad_dtype=gdt, ef=ef,
                max_grad_norm=clip, delay=delay)
    run = Run(case, cuda_device)
    try:
        errs = []
        for k in range(1, 7):
            run.step()
            errs.append(run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN))
            if clip > 0:
                _, norm, coef = dpo.dpo_get_flags(run.gpu.ctx)
                assert norm ** 2 == pytest.approx(run.ref.last_sqnorm, rel=1e-6)
                assert coef == pytest.approx(run.ref.last_clip, rel=1e-6)
                assert coef < 1.0   # the threshold is below the gradient norm
    finally:
        run.close()


@pytest.mark.parametrize("lam", [0.0, 0.5, 2.0])
def test_ef_lambda_sweep(cuda_device, lam):
    """App. A.4: lambda-scaled correction, lambda in {0, 0.5, 2}."""
    run = Run(Case(RAGGED, ef=True, ef_lambda=lam), cuda_device)
    try:
        for k in range(1, 5):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


def test_changing_lr_and_weight_decay_mask(cuda_device):
    """Learning rate changing every call (the schedule is host-side), decay
    on every other tensor. The fp32 update x - u carries an absolute error of
    a few ulps of u, so the one-step bar, set for lr = 3e-4, scales with lr."""
    wd_on = [i % 2 == 0 for i in range(len(RAGGED))]
    run = Run(Case(RAGGED, ef=True, wd_on=wd_on, weight_decay=0.5), cuda_device)
    try:
        for k, lr in enumerate([1e-3, 5e-4, 2e-3, 0.0, 1e-4], start=1):
            run.step(lr)
            run.assert_close(TOL_ONE_STEP * lr / 3e-4 if k == 1 else TOL_RUN)
    finally:
        run.close()


def test_ef_lambda_zero_is_standard_bitwise(cuda_device):
    a = Run(Case(RAGGED, ef=False), cuda_device)
    b = Run(Case(RAGGED, ef=True, ef_lambda=0.0), cuda_device)
    try:
        for _ in range(4):
            a.step()
            b.step()
        torch.cuda.synchronize()
        assert torch.equal(a.gpu.master, b.gpu.master)
        assert torch.equal(a.gpu.param, b.gpu.param)
    finally:
        a.close()
        b.close()


def test_stash_is_previous_latest_bitwise(cuda_device):
    """After every step the stash (bf16) equals the previous step's bf16
    latest weights: the next gradient is evaluated one version behind."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True), cuda_device)
    try:
        prev = run.gpu.param.clone()
        for _ in range(4):
            run.step()
            torch.cuda.synchronize()
            for i, n in enumerate(RAGGED):
                assert torch.equal(run.gpu.view(run.gpu.stash, i), run.gpu.view(prev, i))
            prev = run.gpu.param.clone()
        for i in range(len(RAGGED)):
            if RAGGED[i] == 0:
                continue   # torch gives empty views a null data_ptr
            p, dt = dpo.dpo_read_weights(run.gpu.ctx, dpo.DPO_STALE, i)
            assert dt == B and p == run.gpu.view(run.gpu.stash, i).data_ptr()
            p, dt = dpo.dpo_read_weights(run.gpu.ctx, dpo.DPO_LATEST, i)
            assert dt == B and p == run.gpu.view(run.gpu.param, i).data_ptr()
    finally:
        run.close()


def test_padding_between_tensors_untouched(cuda_device):
    """Guard values in the alignment padding of every arena survive steps."""
    run = Run(Case(RAGGED, ef=True), cuda_device)
    try:
        lay = run.gpu.layout
        pad = torch.ones(lay.total, dtype=torch.bool, device=cuda_device)
        for o, n in zip(lay.offsets, lay.numels):
            pad[o:o + n] = False
        arenas = [run.gpu.master, run.gpu.m, run.gpu.v, run.gpu.param, run.gpu.stash, run.gpu.ef]
        for a in arenas:
            a[pad] = -3.5   # exact in bf16 and fp32
        for _ in range(3):
            run.step()
        torch.cuda.synchronize()
        for a in arenas:
            assert bool((a[pad].float() == -3.5).all())
        run.assert_close(TOL_RUN)
    finally:
        run.close()


def test_deterministic(cuda_device):
    outs = []
    for _ in range(2):
        run = Run(Case(RAGGED, ef=True, max_grad_norm=1e-3), cuda_device)
        for _ in range(3):
            run.step()
        torch.cuda.synchronize()
        outs.append((run.gpu.master.clone(), dpo.dpo_get_flags(run.gpu.ctx)))
        run.close()
    assert torch.equal(outs[0][0], outs[1][0])
    assert outs[0][1] == outs[1][1]


def test_checkpoint_resume_bitwise(cuda_device):
    """5 steps, save, restore into a new context (INIT_RESUME), 5 more steps:
    bitwise equal to 10 straight steps."""
    case = Case(RAGGED, stash_dtype=B, ef=True, max_grad_norm=0.05)
    straight = Run(case, cuda_device)
    split = Run(case, cuda_device)
    try:
        for _ in range(10):
            straight.step()
        for _ in range(5):
            split.step()
        sd = split.gpu.state_dict()
        split.gpu.close()
        fresh = dpo.DelayedAdamW(case.numels, param_dtype=case.param_dtype,
                                 stash_dtype=case.stash_dtype, grad_dtype=case.grad_dtype,
                                 ef=True, max_grad_norm=case.max_grad_norm,
                                 device=cuda_device, init_mode=dpo.DPO_INIT_RESUME)
        fresh.load_state(sd)
        split.gpu = fresh
        assert dpo.dpo_get_step(fresh.ctx) == 5
        for _ in range(5):
            split.step()
        torch.cuda.synchronize()
        for name in ("master", "m", "v", "param", "stash", "ef"):
            assert torch.equal(getattr(straight.gpu, name), getattr(split.gpu, name)), name
    finally:
        straight.close()
        split.close()


def test_checkpoint_resume_after_synchronous_start(cuda_device):
    """Synchronous start of 3 calls (odd), delayed training with EF and the
    ping-pong stash, a checkpoint after call 5, restored into a new
    context, 3 more calls: bitwise equal to 8 straight calls. The restored
    phase start keeps Alg. 1's t = k - k0, which decides both where EF
    starts and which of the two weight buffers holds which version."""
    case = Case(RAGGED, stash_dtype=B, ef=True, stash_mode=dpo.DPO_STASH_PINGPONG,
                schedule={1: 0, 4: 1})
    straight = Run(case, cuda_device)
    split = Run(case, cuda_device)
    try:
        for _ in range(8):
            straight.step()
        for _ in range(5):
            split.step()
        sd = split.gpu.state_dict()
        assert sd["phase_start"] == 3 and sd["k"] == 5 and sd["delay"] == 1
        split.gpu.close()
        fresh = dpo.DelayedAdamW(case.numels, param_dtype=case.param_dtype,
                                 stash_dtype=case.stash_dtype, grad_dtype=case.grad_dtype,
                                 ef=True, device=cuda_device, init_mode=dpo.DPO_INIT_RESUME,
                                 keep_stash=True, stash_mode=dpo.DPO_STASH_PINGPONG)
        fresh.load_state(sd)
        split.gpu = fresh
        for _ in range(3):
            split.step()
        torch.cuda.synchronize()
        for name in ("master", "m", "v", "ef"):
            assert torch.equal(getattr(straight.gpu, name), getattr(split.gpu, name)), name
        for a, b in zip(straight.gpu.role_arenas(), split.gpu.role_arenas()):
            assert torch.equal(a, b)
    finally:
        straight.close()
        split.close()


def test_host_io_switch_keeps_the_delayed_phase(cuda_device):
    """use_host_io rebuilds the context: the step counter and the start of
    the delayed phase carry over. Switching right after entering delayed
    training (synchronous start of two calls) leaves the next call Alg. 1's
    first delayed iteration: standard rule, EF from the call after."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True, schedule={1: 0}), cuda_device)
    try:
        for _ in range(2):
            run.step()
        run.gpu.set_delay(1)
        run.ref.set_delay(1)
        run.gpu.use_host_io()
        assert run.gpu.k == 2 and dpo.dpo_get_phase_start(run.gpu.ctx) == 2
        for _ in range(4):
            run.step()
            run.assert_close(TOL_RUN)
    finally:
        run.close()


def test_lion_zero_gradient_moves_only_by_decay(cuda_device):
    """Lion's sign(0) = 0 on the GPU as in the oracle: a zero gradient from
    the zero start state leaves the update at the decay term alone, so every
    weight matches the oracle's x (1 - lr wd) path, decayed and undecayed
    tensors alike."""
    case = Case([4096, 77, 300_001], optimizer=dpo.DPO_OPT_LION, stash_dtype=B,
                wd_on=[True, False, True])
    run = Run(case, cuda_device)
    try:
        x0 = run.gather(run.gpu.master).astype(np.float64)
        run.gpu.grad.zero_()
        run.gpu.step()
        run.ref.step(np.zeros(run.idx.size), tag=run.ref.read_weights("stale")[1])
        torch.cuda.synchronize()
        run.assert_close(TOL_ONE_STEP)
        got = run.gather(run.gpu.master).astype(np.float64)
        moved = got != x0
        assert not moved[4096:4096 + 77].any()        # no decay: untouched
        assert moved[:4096].mean() > 0.99             # decay: x (1 - lr wd)
    finally:
        run.close()


def test_nonfinite_gradient_flag(cuda_device):
    run = Run(Case([1000, 17], max_grad_norm=1.0), cuda_device)
    try:
        run.step()
        flags, norm, _ = dpo.dpo_get_flags(run.gpu.ctx)
        assert flags == 0 and np.isfinite(norm)
        synth.dev_normal(1, synth.STREAM_GRAD, 9, 0, run.gpu.grads(0), 1e-3)
        run.gpu.grads(1)[3] = float("nan")
        run.gpu.step()
        flags, norm, coef = dpo.dpo_get_flags(run.gpu.ctx)
        assert flags & dpo.DPO_FLAG_NONFINITE and np.isnan(norm) and np.isnan(coef)
        assert bool(torch.isnan(run.gpu.master[:1000]).all())   # NaN reaches every element
        flags, _, _ = dpo.dpo_get_flags(run.gpu.ctx)
        assert flags == 0   # reading cleared the flag
    finally:
        run.close()


def test_dpo_stash_resets_stale_copy(cuda_device):
    run = Run(Case(RAGGED, stash_dtype=F), cuda_device)
    try:
        run.step()
        run.step()
        dpo.dpo_stash(run.gpu.ctx)
        torch.cuda.synchronize()
        assert torch.equal(run.gpu.stash, run.gpu.master)
    finally:
        run.close()


def test_misaligned_device_pointer_rejected(cuda_device):
    buf = torch.zeros(1 << 12, dtype=torch.float32, device=cuda_device)
    p = buf.data_ptr()
    t = dpo.dpo_tensor(param=None, master=p + 4, m=p + 8192, v=p + 4096, stash=p + 12288,
                       ef=None, grad=p + 2048, numel=10, flags=1)
    with pytest.raises(dpo.DpoError) as e:
        dpo.dpo_init([t], F, F, F, dpo.dpo_hparams(0.9, 0.95, 1e-8, 0.1, 0.0, 0.0, 1))
    assert e.value.code == dpo.DPO_EALIGN


def test_host_pointer_rejected(cuda_device):
    host = np.zeros(1 << 12, np.float32)
    p = host.ctypes.data
    p += (-p) % 32
    t = dpo.dpo_tensor(param=None, master=p, m=p + 4096, v=p + 8192, stash=p + 12288, ef=None,
                       grad=p + 13824, numel=10, flags=1)
    with pytest.raises(dpo.DpoError) as e:
        dpo.dpo_init([t], F, F, F, dpo.dpo_hparams(0.9, 0.95, 1e-8, 0.1, 0.0, 0.0, 1))
    assert e.value.code == dpo.DPO_EINVAL


def test_launch_geometry_is_persistent(cuda_device):
    run = Run(Case([50_000_000]), cuda_device)
    try:
        steps, norms, threads = dpo.dpo_launch_config(run.gpu.ctx)
        sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
        assert threads == 128 and steps == 4 * sms and norms % sms == 0   # standard rule: 4 CTAs/SM
        sb, nb = dpo.dpo_algorithmic_bytes(run.gpu.ctx)
        assert sb == 50_000_000 * (12 + 2 + 12 + 4 + 2) and nb == 0
    finally:
        run.close()


@pytest.mark.parametrize("stash_mode,per_sm", [(dpo.DPO_STASH_PINGPONG, 5), (dpo.DPO_STASH_COPY, 3)])
def test_launch_geometry_lion_with_history(cuda_device, stash_mode, per_sm):
    """The measured grid table: Lion with an update history takes five CTAs
    per SM under the ping-pong stash, three with the copying stash."""
    run = Run(Case([5_000_000, 123], stash_dtype=B, ef=True, optimizer=dpo.DPO_OPT_LION,
                   stash_mode=stash_mode), cuda_device)
    try:
        steps, _, _ = dpo.dpo_launch_config(run.gpu.ctx)
        sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
        assert steps == per_sm * sms
    finally:
        run.close()


@pytest.mark.parametrize("host_grad,host_param,stash_mode", [
    (True, True, dpo.DPO_STASH_COPY), (True, False, dpo.DPO_STASH_COPY),
    (False, True, dpo.DPO_STASH_COPY), (True, False, dpo.DPO_STASH_PINGPONG)])
def test_host_io_parity(cuda_device, host_grad, host_param, stash_mode):
    """Gradients read from and/or bf16 weights written to pinned host memory
    by the fused kernel itself (no staging copy): same results. Gradients in
    host memory also with the ping-pong stash (the end-to-end benchmark's
    configuration: the weights stay on the device)."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True, max_grad_norm=0.3, host_grad=host_grad,
                   host_param=host_param, stash_mode=stash_mode), cuda_device)
    try:
        assert run.gpu.grad.is_cuda != host_grad and run.gpu.param.is_cuda != host_param
        for k in range(1, 5):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
        p, _ = dpo.dpo_read_weights(run.gpu.ctx, dpo.DPO_LATEST, 0)
        assert p == run.gpu.view(run.gpu.param, 0).data_ptr()
    finally:
        run.close()


def test_switch_to_host_io_continues_bitwise(cuda_device):
    """use_host_io() mid-run rebuilds the context over host arenas (RESUME,
    same step counter): the run continues exactly as the device-only one."""
    case = Case(RAGGED, stash_dtype=B, ef=True)
    a, b = Run(case, cuda_device), Run(case, cuda_device)
    try:
        for _ in range(3):
            a.step()
            b.step()
        b.gpu.use_host_io()
        assert not b.gpu.grad.is_cuda and not b.gpu.param.is_cuda
        for _ in range(3):
            a.step()
            b.step()
        torch.cuda.synchronize()
        assert torch.equal(a.gpu.master, b.gpu.master)
        assert torch.equal(a.gpu.param.cpu(), b.gpu.param)
        assert dpo.dpo_get_step(b.gpu.ctx) == 6
    finally:
        a.close()
        b.close()


SP_SAME, SP_UPD = dpo.DPO_CORR_SAPIPE_SAME, dpo.DPO_CORR_SAPIPE_UPDATED


@pytest.mark.parametrize("corr", [SP_SAME, SP_UPD])
@pytest.mark.parametrize("pdt,sdt,gdt,clip", [(B, B, B, 0.0), (B, F, B, 0.3), (F, F, F, 0.0)])
def test_sapipe_parity(cuda_device, corr, pdt, sdt, gdt, clip):
    """App. B.1 SAPipe-WP prediction (same / updated optimizer state): the
    stash receives the prediction point, the weights the standard rule."""
    run = Run(Case(RAGGED, param_dtype=pdt, stash_dtype=sdt, grad_dtype=gdt, ef=True,
                   correction=corr, max_grad_norm=clip), cuda_device)
    try:
        for k in range(1, 7):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


def test_sapipe_same_weights_equal_standard_rule_bitwise(cuda_device):
    a = Run(Case(RAGGED, ef=False), cuda_device)
    b = Run(Case(RAGGED, ef=True, correction=SP_SAME), cuda_device)
    try:
        for _ in range(4):
            a.step()
            b.step()
        torch.cuda.synchronize()
        assert torch.equal(a.gpu.master, b.gpu.master)
        assert not torch.equal(a.gpu.stash, b.gpu.stash)   # prediction points differ
    finally:
        a.close()
        b.close()


HALF = [i >= len(RAGGED) // 2 for i in range(len(RAGGED))]   # WPipe: second half synchronous


@pytest.mark.parametrize("ef,corr", [(False, dpo.DPO_CORR_EF), (True, dpo.DPO_CORR_EF),
                                     (True, SP_SAME), (True, SP_UPD)])
def test_wpipe_half_synchronous_parity(cuda_device, ef, corr):
    """App. B.2 WPipe: the second half of the model trains synchronously (no
    stash, no correction), the first half one-step delayed."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=ef, correction=corr, sync=HALF,
                   max_grad_norm=0.3), cuda_device)
    try:
        for k in range(1, 7):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
        for i, sy in enumerate(HALF):
            if RAGGED[i] == 0:
                continue
            p, _ = dpo.dpo_read_weights(run.gpu.ctx, dpo.DPO_STALE, i)
            ref = run.gpu.view(run.gpu.param if sy else run.gpu.stash, i)
            assert p == ref.data_ptr()
    finally:
        run.close()


def test_synchronous_lm_head_parity(cuda_device):
    """App. A.9: the last tensor (the LM head) synchronous, the rest delayed with EF."""
    sync = [False] * (len(RAGGED) - 1) + [True]
    run = Run(Case(RAGGED, ef=True, sync=sync), cuda_device)
    try:
        for k in range(1, 6):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("ef,corr", [(True, dpo.DPO_CORR_EF), (True, SP_UPD), (False, 0)])
def test_synchronous_start_then_delayed(cuda_device, ef, corr):
    """Sec. 3.1 synchronous start: calls 1-3 synchronous, then delayed; Alg. 1
    restarts at the switch (standard rule at its first delayed call)."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=ef, correction=corr, delay=0, schedule={4: 1}),
              cuda_device)
    try:
        for k in range(1, 9):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
            assert run.gpu.delay == (1 if k >= 4 else 0)
    finally:
        run.close()


# ---------------- ping-pong stash (PipeDream-2BW's two weight versions)

PP = dpo.DPO_STASH_PINGPONG


@pytest.mark.parametrize("ef,sync", [(True, False), (False, False), (True, True)])
def test_pingpong_stash_parity(cuda_device, ef, sync):
    """The bf16 param and stash buffers swap roles instead of the stash being
    written: the latest and stale views, and all state, match the oracle over
    odd and even calls (and with every other tensor trained synchronously)."""
    sync_l = [i % 2 == 1 for i in range(len(RAGGED))] if sync else None
    run = Run(Case(RAGGED, stash_dtype=B, ef=ef, sync=sync_l, stash_mode=PP), cuda_device)
    try:
        for k in range(1, 7):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


def test_pingpong_stash_switches(cuda_device):
    """Synchronous start, delayed calls 3-5 (odd: the latest weights end in
    the stash buffer), cooldown, and delayed again: the roles follow the
    delayed phase and the synchronous calls find the latest weights."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True, delay=0, schedule={3: 1, 6: 0, 8: 1},
                   stash_mode=PP), cuda_device)
    try:
        for k in range(1, 11):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("corr", [dpo.DPO_CORR_EF, SP_SAME])
def test_reentering_delayed_training_parity(cuda_device, corr):
    """Delayed calls 1-2, synchronous 3-4, delayed again from 5: the device
    restarts Alg. 1 there as the oracle does (history zeroed, so SAPipe's
    first prediction is x itself, EF from the second call)."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True, correction=corr, schedule={3: 0, 5: 1}),
              cuda_device)
    try:
        for k in range(1, 9):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("rule", ["nadam", "adan"])
def test_rules_across_mode_switches_parity(cuda_device, rule):
    """NAdam's and Adan's statistics continue across a synchronous start, a
    cooldown and a re-entry (Adan's zero first difference only at the run's
    first gradient), on the device as in the oracle."""
    run = Run(Case(RAGGED, stash_dtype=B, ef=True, schedule={1: 0, 3: 1, 6: 0, 8: 1},
                   **RULES[rule]), cuda_device)
    try:
        for k in range(1, 11):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("dc", [0.0, 1e4])
def test_pingpong_equals_copy_stash_bitwise(cuda_device, dc):
    """Same seeded run with the copying and the ping-pong stash: master, m, v,
    EF buffer and the latest / stale weights bitwise equal after every call,
    DC-ASGD included (it reads the stale buffer the new weights then overwrite)."""
    runs = [Run(Case(RAGGED, stash_dtype=B, ef=True, dc_lambda=dc, stash_mode=m), cuda_device)
            for m in (dpo.DPO_STASH_COPY, PP)]
    try:
        for k in range(1, 6):
            for r in runs:
                r.step()
            torch.cuda.synchronize()
            a, b = runs[0].gpu, runs[1].gpu
            for name in ("master", "m", "v", "ef"):
                assert torch.equal(getattr(a, name), getattr(b, name)), (k, name)
            for ra, rb in zip(a.role_arenas(), b.role_arenas()):
                assert torch.equal(ra.view(torch.int16), rb.view(torch.int16)), k
            la, _ = dpo.dpo_read_weights(b.ctx, dpo.DPO_LATEST, 6)
            assert la == (b.table[6].stash if k % 2 else b.table[6].param)
    finally:
        for r in runs:
            r.close()


def test_synchronous_cooldown(cuda_device):
    """App. A.10: delayed with EF for 5 calls, then synchronous."""
    run = Run(Case(RAGGED, ef=True, schedule={6: 0}), cuda_device)
    try:
        for k in range(1, 10):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


def test_set_delay_needs_stash_buffers(cuda_device):
    opt = dpo.DelayedAdamW([1000, 24], delay=0, keep_stash=False, device=cuda_device)
    try:
        with pytest.raises(dpo.DpoError) as e:
            opt.set_delay(1)
        assert e.value.code == dpo.DPO_ESTATE
    finally:
        opt.close()


# ---------------- other elementwise optimizers under delay (Tab. main_results)
# with the paper's settings where it gives them (Lion: lr 5e-4, wd 0.5, App. E.1)

RULES = {
    "nadam": dict(optimizer=dpo.DPO_OPT_NADAM, momentum_decay=0.004),
    "lion": dict(optimizer=dpo.DPO_OPT_LION, beta1=0.9, beta2=0.99, lr=5e-4, weight_decay=0.5),
    "adan": dict(optimizer=dpo.DPO_OPT_ADAN, beta1=0.98, beta2=0.92, beta3=0.99),
}


@pytest.mark.parametrize("rule", sorted(RULES))
@pytest.mark.parametrize("ef,corr", [(False, dpo.DPO_CORR_EF), (True, dpo.DPO_CORR_EF),
                                     (True, SP_SAME), (True, SP_UPD)])
@pytest.mark.parametrize("pdt,sdt,gdt", [(B, B, B), (B, F, B), (F, F, F)])
def test_rule_parity(cuda_device, rule, ef, corr, pdt, sdt, gdt):
    """NAdam, Lion and Adan under the standard rule, EF and both SAPipe-WP
    predictions (the updated state: each rule's own step at k + 1), with
    clipping, in every layout."""
    run = Run(Case(RAGGED, param_dtype=pdt, stash_dtype=sdt, grad_dtype=gdt, ef=ef,
                   correction=corr, max_grad_norm=0.3, **RULES[rule]), cuda_device)
    try:
        for k in range(1, 7):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("clip", [0.0, 0.3])
def test_dc_asgd_parity_multistep(cuda_device, clip):
    """DC-ASGD's Taylor compensation (Sec. 3.1) with EF over six steps, at
    lambda = 1e4 with an fp32 stash, with and without clipping (the
    compensation then corrects the clipped gradient). The term multiplies
    x_t - stash by lambda g^2, so at larger lambda (the paper sweeps up to
    1e8) a one-rounding difference between the two sides' master or stash,
    allowed by the fp32 and bf16 bars, is amplified into the gradient: there
    the step is checked on identical inputs instead (next test)."""
    run = Run(Case(RAGGED, stash_dtype=F, ef=True, dc_lambda=1e4, max_grad_norm=clip),
              cuda_device)
    try:
        for k in range(1, 7):
            run.step()
            run.assert_close(TOL_ONE_STEP if k == 1 else TOL_RUN)
    finally:
        run.close()


@pytest.mark.parametrize("dc", [1e4, 1e6, 1e8])
@pytest.mark.parametrize("sdt", [B, F])
def test_dc_asgd_step_on_identical_inputs(cuda_device, dc, sdt):
    """One DC-ASGD + EF step from a state both sides hold bit for bit, k = 1
    done. The stash x_s ~ N(0, 0.02^2) is held in the stash dtype, the master
    is x_s + sign(g)|N(0, (3e-4)^2)| in fp32, so the compensation term
    lambda g^2 (x - x_s) has the sign of g and g + lambda g^2 (x - x_s) never
    cancels: where it cancels the compensated gradient keeps only the digits
    fp32 leaves and the Adam step near g~ = 0 amplifies them, which no fp32
    implementation matches to the one-step bar. Every buffer within that bar."""
    numels, seed = RAGGED, 0xDC
    N = sum(numels)
    gb = synth.host_normal(seed, synth.STREAM_GRAD, 2, 0, N, 1e-3, synth.BF16)
    g = synth.bf16_bits_to_f32(gb).astype(np.float64)
    xs = synth.host_normal(seed, synth.STREAM_INIT, 0, 0, N, 0.02).astype(np.float32)
    if sdt == B:
        xs = torch.from_numpy(xs).to(torch.bfloat16).float().numpy()
    off = np.abs(synth.host_normal(seed, 7, 0, 0, N, 3e-4)).astype(np.float32)
    x = (xs + np.sign(g).astype(np.float32) * off).astype(np.float32)
    # the construction holds after fp32 rounding: no offset opposes its gradient
    assert np.all(np.sign(x.astype(np.float64) - xs) * np.sign(g) >= 0)
    opt = dpo.DelayedAdamW(numels, stash_dtype=sdt, ef=True, dc_lambda=dc, device=cuda_device,
                           init_mode=dpo.DPO_INIT_RESUME)
    try:
        offs = np.concatenate([[0], np.cumsum(numels)])
        for i, n in enumerate(numels):
            if n:
                sl = slice(int(offs[i]), int(offs[i + 1]))
                opt.view(opt.master, i).copy_(torch.from_numpy(x[sl]))
                opt.view(opt.stash, i).copy_(torch.from_numpy(xs[sl]))
                opt.grads(i).copy_(torch.from_numpy(gb[sl].view(np.int16)).view(torch.bfloat16))
        dpo.dpo_set_step(opt.ctx, 1)
        opt.step()
        hp = oracle.HParams(lr=3e-4, ef_lambda=1.0, dc_lambda=dc).as_f32()
        ref = oracle.DelayedOptimizer([x.astype(np.float64)], hp, ef=True, x_store=oracle.F32,
                                      stash_store=oracle.BF16 if sdt == B else oracle.F32,
                                      param_store=oracle.BF16)
        ref.stash[:] = xs
        ref.k, ref.t = 1, 1
        ref.step(synth.bf16_bits_to_f32(gb).astype(np.float64))
        torch.cuda.synchronize()
        cat = lambda a: torch.cat([opt.view(a, i) for i in range(len(numels))])
        assert rel_err(cat(opt.master).cpu().numpy(), ref.x) <= TOL_ONE_STEP
        assert rel_err(cat(opt.m).cpu().numpy(), ref.m) <= TOL_ONE_STEP
        assert rel_err(cat(opt.v).cpu().numpy(), ref.v) <= TOL_ONE_STEP
        assert rel_err(cat(opt.ef).cpu().numpy(), ref.u_prev) <= TOL_ONE_STEP
        p = cat(opt.param).view(torch.int16).cpu().numpy().view(np.uint16)
        assert bf16_ulps(p, ref.param) <= 1.0
        # the compensation mattered: it moved the first moment away from (1 - beta1) g
        assert np.max(np.abs(ref.m - 0.1 * g)) > 1e-3 * np.max(np.abs(0.1 * g))
    finally:
        opt.close()


@pytest.mark.parametrize("name,case,n_sync", [
    ("adamw_ef_pingpong", Case(RAGGED, stash_dtype=B, ef=True,
                               stash_mode=dpo.DPO_STASH_PINGPONG), 0),
    ("nadam_ef_after_sync_start", Case(RAGGED, ef=True, optimizer=dpo.DPO_OPT_NADAM), 3),
    ("adan_clipped", Case(RAGGED, optimizer=dpo.DPO_OPT_ADAN, max_grad_norm=0.05), 0),
    ("nadam_sapipe_updated", Case(RAGGED, ef=True, optimizer=dpo.DPO_OPT_NADAM,
                                  correction=dpo.DPO_CORR_SAPIPE_UPDATED), 0),
    ("adan_sapipe_updated", Case(RAGGED, ef=True, optimizer=dpo.DPO_OPT_ADAN,
                                 correction=dpo.DPO_CORR_SAPIPE_UPDATED), 2),
])
def test_capturable_step_replays_in_a_cuda_graph(cuda_device, name, case, n_sync):
    """One dpo_step captured in a CUDA graph (capturable mode) and replayed
    six times with fresh gradients and a learning rate written to device
    memory between replays, beside an eager run: the device-formed scalars
    follow k (bias corrections, NAdam's products, Adan's first step), t = k -
    k0 (EF from t = 2, the ping-pong roles) and the schedule, so both runs
    agree at every call (fp32 state to 1e-6, bf16 weights to one ulp)."""
    eager, cap = Run(case, cuda_device), Run(case, cuda_device)
    lrs = [None] + [3e-4 * (1.0 - 0.07 * i) for i in range(1, 1 + n_sync + 6)]
    lr_t = torch.empty(1, dtype=torch.float32, device=cuda_device)
    try:
        k = 0
        if n_sync:
            for r in (eager, cap):
                r.gpu.set_delay(0)
        for _ in range(n_sync):
            k += 1
            for r in (eager, cap):
                r.draw(k)
                r.gpu.step(lrs[k])
        if n_sync:
            for r in (eager, cap):
                r.gpu.set_delay(1)
        cap.gpu.set_capturable(True, lr_source=lr_t)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            cap.gpu.step()
        for _ in range(6):
            k += 1
            eager.draw(k)
            cap.draw(k)
            lr_t.fill_(lrs[k])
            eager.gpu.step(lrs[k])
            graph.replay()
            torch.cuda.synchronize()
            for buf in ("master", "m", "v", "n", "grad_prev", "ef"):
                a, b = getattr(eager.gpu, buf), getattr(cap.gpu, buf)
                if a is not None:
                    assert rel_err(b.cpu().numpy(), a.cpu().numpy().astype(np.float64)) <= 1e-6, \
                        (name, k, buf)
            la, _ = eager.gpu.role_arenas()
            lb, _ = cap.gpu.role_arenas()
            if la is not None:
                d = bf16_ord(lb.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.int64) - \
                    bf16_ord(la.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.int64)
                assert np.max(np.abs(d)) <= 1, (name, k)
        assert cap.gpu.k == eager.gpu.k == k
        cap.gpu.set_capturable(False)
        assert cap.gpu.k == k
    finally:
        eager.close()
        cap.close()


def test_start_weights_in_every_form(cuda_device):
    """x_0 given per tensor, as the tensors' plain concatenation, or in the
    arena layout gives the same start state; any other length is refused."""
    numels = [1000, 3, 517]
    x = torch.randn(sum(numels), dtype=torch.float32, device=cuda_device)
    parts = list(torch.split(x, numels))
    built = [dpo.DelayedAdamW(numels, ef=True, stash_dtype=B, device=cuda_device, x0=x0)
             for x0 in (parts, x)]
    arena = built[1].master.clone()
    built.append(dpo.DelayedAdamW(numels, ef=True, stash_dtype=B, device=cuda_device, x0=arena))
    try:
        for o in built:
            for i in range(len(numels)):
                assert torch.equal(o.view(o.master, i), parts[i])
                assert torch.equal(o.view(o.param, i), parts[i].to(torch.bfloat16))
        with pytest.raises(ValueError):
            dpo.DelayedAdamW(numels, device=cuda_device, x0=x[:-1])
    finally:
        for o in built:
            o.close()
