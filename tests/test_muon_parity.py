"""GPU parity of delayed Muon (Alg. 2): momentum, Newton-Schulz on the
tcgen05 tensor cores, the delayed / EF update, stash and weights, through the
C ABI (include/dpo_muon.h), against the oracle (oracle/muon.py).

Newton-Schulz in bf16 is sensitive to its own rounding decisions: a product
that lands within an fp32 accumulation error of a bf16 rounding boundary
rounds the other way, and from the third step on such flips cascade. The
oracle accumulates exactly and rounds every iterate to bf16 once; the kernels
accumulate in fp32. The bars below come from running the two arithmetics side
by side on the CPU (an fp32-accumulation emulation against the oracle, same
inputs), with about 3x margin:
  steps 0: identical except rare one-ulp flips of X_0
  steps 1 / 2: normwise <= 2e-4 / 5e-4, differing elements <= 0.2% / 1%
  steps 5: normwise <= 1.5e-2 (measured 4.7e-3 to 5.8e-3), singular values
           within 5e-3 (measured <= 1.3e-3)
The momentum does not depend on Newton-Schulz and is held to the one-step
bar of the elementwise path.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from oracle.muon import DelayedMuon as OracleMuon, MuonHParams
from paper_2606_30634_gb300 import dpo, muon, synth
from parity_util import TOL_ONE_STEP, TOL_RUN, bf16_ulps, rel_err

pytestmark = pytest.mark.gpu

F, B = dpo.DPO_F32, dpo.DPO_BF16
# wide, tall, ragged (padded to 256 inside), several tiles, tiny, empty, and
# a shape whose 96 output tiles outnumber the CTA pairs (each pair then walks
# several tiles, reading operands other pairs' tiles are being written next to)
SHAPES = [(256, 512), (512, 256), (300, 700), (64, 96), (1, 7), (0, 5), (768, 2304),
          (1024, 3072), (3072, 1024)]
NS_BARS = {1: (2e-4, 2e-3), 2: (5e-4, 1e-2)}


def inputs(shapes, seed, k, gdt=None):
    """x_0 ~ N(0, 0.02^2) (fp32) and the k-th gradient ~ N(0, 1e-3^2) (bf16
    bits, or fp32 with gdt = synth.F32), per matrix, from the seeded
    generator."""
    xs, gs, off = [], [], 0
    for r, c in shapes:
        n = r * c
        xs.append(synth.host_normal(seed, synth.STREAM_INIT, 0, off, n, 0.02).reshape(r, c))
        gs.append(synth.host_normal(seed, synth.STREAM_GRAD, k, off, n, 1e-3,
                                    synth.BF16 if gdt is None else gdt).reshape(r, c))
        off += n
    return xs, gs


def bf16_to_f64(bits):
    return synth.bf16_bits_to_f32(np.asarray(bits)).astype(np.float64)


class Pair:
    """The GPU context and the oracle on the same seeded inputs."""

    def __init__(self, shapes, device, seed=0x3A0, ns_steps=5, ef=True, delay=1, sdt=B,
                 lr=2e-3, momentum=0.95, wd=0.1, max_grad_norm=0.0, rms_scale=0.2, sync=None,
                 schedule=None, correction=0, gdt=B, wd_on=None):
        self.shapes, self.seed, self.lr = shapes, seed, lr
        self.schedule = schedule or {}
        xs, _ = inputs(shapes, seed, 1)
        self.gdt = gdt
        self.gpu = muon.DelayedMuon(shapes, stash_dtype=sdt, grad_dtype=gdt, lr=lr,
                                    momentum=momentum, weight_decay=wd, ef=ef,
                                    max_grad_norm=max_grad_norm, rms_scale=rms_scale,
                                    ns_steps=ns_steps, delay=delay, device=device,
                                    x0=[torch.from_numpy(x) for x in xs], sync=sync,
                                    keep_stash=True, correction=correction, wd_on=wd_on)
        hp = MuonHParams(lr=lr, momentum=momentum, weight_decay=wd, ef_lambda=1.0,
                         ns_steps=ns_steps, rms_scale=rms_scale, ns_store=oracle.BF16,
                         max_grad_norm=max_grad_norm, delay=delay,
                         correction=correction).as_f32()
        self.ref = OracleMuon([x.astype(np.float64) for x in xs], hp, ef=ef, x_store=oracle.F32,
                              stash_store=oracle.BF16 if sdt == B else oracle.F32,
                              param_store=oracle.BF16,
                              delayed=None if sync is None else [not q for q in sync],
                              wd_on=wd_on)
        self.sync = sync or [False] * len(shapes)
        self.k = 0

    def draw(self, k: int):
        """Gradient k (the seeded draw numbered k + 1) into the GPU's grad
        arena; returned as fp64 matrices for the oracle."""
        if self.gdt == F:
            _, gs = inputs(self.shapes, self.seed, k + 1, synth.F32)
            for i, g in enumerate(gs):
                if g.size:
                    self.gpu.grads(i).copy_(torch.from_numpy(g))
            return [g.astype(np.float64) for g in gs]
        _, gs = inputs(self.shapes, self.seed, k + 1)
        for i, g in enumerate(gs):
            if g.size:
                self.gpu.grads(i).copy_(torch.from_numpy(g.view(np.int16)).view(torch.bfloat16)
                                        .reshape(g.shape))
        return [bf16_to_f64(g) for g in gs]

    def step(self, sq=None, before=None):
        """One call on both sides; ``sq`` and ``before`` as in Run.step."""
        if self.k + 1 in self.schedule:
            self.gpu.set_delay(self.schedule[self.k + 1])
            self.ref.set_delay(self.schedule[self.k + 1])
        self.k += 1
        gs = self.draw(self.k)
        if before is not None:
            before(gs)
        self.gpu.step()
        self.ref.step(gs, sq=sq)
        torch.cuda.synchronize()

    def cat(self, arena):
        return np.concatenate([self.gpu.view(arena, i).float().cpu().numpy().ravel()
                               for i in range(len(self.shapes))])

    def o_pairs(self):
        got = [self.gpu.last_update(i).float().cpu().numpy().astype(np.float64)
               for i in range(len(self.shapes))]
        return got, list(self.ref.o)

    def close(self):
        assert self.gpu.status() == 0, "a tensor-core pipeline wait gave up"
        self.gpu.close()


def _flat(a):
    return np.concatenate([x.ravel() for x in a]) if a else np.zeros(0)


def _ulp(v):
    return np.exp2(np.floor(np.log2(np.maximum(np.abs(v), 2.0 ** -126))) - 7)


@pytest.mark.parametrize("steps", [0, 1, 2, 5])
def test_newton_schulz_parity(cuda_device, steps):
    p = Pair(SHAPES, cuda_device, ns_steps=steps)
    try:
        p.step()
        got, ref = p.o_pairs()
        g, r = _flat(got), _flat(ref)
        d = np.abs(g - r)
        norm = np.linalg.norm(g - r) / np.linalg.norm(r)
        frac = float(np.mean(d > 0))
        print(f"steps {steps}: normwise {norm:.3e}, differing {frac:.4%}, "
              f"max {d.max() / np.abs(r).max():.3e}")
        if steps == 0:
            assert frac <= 1e-3
            assert np.all(d <= _ulp(r))
        elif steps in NS_BARS:
            assert norm <= NS_BARS[steps][0] and frac <= NS_BARS[steps][1]
        else:
            assert norm <= 1.5e-2
            for gi, ri in zip(got, ref):
                if gi.size:
                    sg = np.linalg.svd(gi, compute_uv=False)
                    sr = np.linalg.svd(ri, compute_uv=False)
                    assert np.max(np.abs(sg - sr)) <= 5e-3
        # the padding of every matrix stays out of the result: O has the
        # matrix's shape and the momentum is the same as the oracle's
        assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= TOL_ONE_STEP
    finally:
        p.close()


def test_newton_schulz_parity_past_one_band(cuda_device):
    """A matrix with more block rows (18, ragged) than one band of the full
    product's tile walk (16) and more block columns (19) than rows: one
    Newton-Schulz step against the oracle at the one-step bars, and every
    256 x 256 output tile on its own, so a tile the walk skipped or visited
    twice would stand out."""
    shape = (4353, 4700)
    p = Pair([shape], cuda_device, ns_steps=1, seed=0xB4D)
    try:
        p.step()
        (g,), (r,) = p.o_pairs()
        d = np.abs(g - r)
        norm = np.linalg.norm(g - r) / np.linalg.norm(r)
        frac = float(np.mean(d > 0))
        print(f"{shape}: normwise {norm:.3e}, differing {frac:.4%}")
        assert norm <= NS_BARS[1][0] and frac <= NS_BARS[1][1]
        worst = max(np.linalg.norm(d[i:i + 256, j:j + 256]) /
                    np.linalg.norm(r[i:i + 256, j:j + 256])
                    for i in range(0, shape[0], 256) for j in range(0, shape[1], 256))
        assert worst <= 10 * NS_BARS[1][0], f"tile normwise {worst:.3e}"
    finally:
        p.close()

def close_with_flips(gpu, ref, tol, flip, max_frac):
    """Elementwise at the floored bar ``tol`` except where a flipped bf16
    rounding of O moved an element: at most ``max_frac`` of the elements may
    miss the bar, and none by more than ``flip`` (absolute)."""
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    d = np.abs(gpu - ref)
    den = np.maximum(np.abs(ref), 1e-2 * np.sqrt(np.mean(ref * ref)))
    bad = d > tol * den
    assert np.mean(bad) <= max_frac, f"{np.mean(bad):.2e} of the elements off the bar"
    assert np.all(d[bad] <= flip + tol * den[bad]), f"max miss {d[bad].max():.3e} > {flip:.3e}"


@pytest.mark.parametrize("steps,sdt,ef,delay,gdt", [(0, B, True, 1, B), (1, F, True, 1, B),
                                                    (1, B, False, 1, B), (0, B, False, 0, B),
                                                    (1, F, True, 1, F)])
def test_muon_step_parity(cuda_device, steps, sdt, ef, delay, gdt):
    """Four calls of Alg. 2 (EF from the second), every buffer checked after
    each. The momentum does not depend on O: one-step bar, then the run bar
    (the EMA rounds twice where the oracle rounds once). The weights, stash,
    bf16 weights and update history are held elementwise to the run / one-ulp
    bars except where a bf16 rounding of O flipped (see the module note):
    such a flip moves U by at most lr r ulp(O) <= lr r 2^-7 (|O| < 2), and
    the weights by that much per call so far."""
    p = Pair(SHAPES, cuda_device, ns_steps=steps, ef=ef, delay=delay, sdt=sdt, gdt=gdt)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    try:
        for k in range(4):
            p.step()
            assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= (TOL_ONE_STEP if k == 0
                                                                    else TOL_RUN)
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            vals = lambda a: p.cat(a).astype(np.float64)
            ref_p = _flat(p.ref.param)
            close_with_flips(vals(p.gpu.param), ref_p, 2.0 ** -7, (k + 1) * du, 1e-3)
            if delay == 1:
                close_with_flips(vals(p.gpu.stash), _flat(p.ref.stash),
                                 2.0 ** -7 if sdt == B else TOL_RUN, k * du, 1e-3)
            if ef and delay == 1:
                close_with_flips(p.cat(p.gpu.ef), _flat(p.ref.u_prev), 1e-5, du, 2e-3)
    finally:
        p.close()


@pytest.mark.parametrize("sync,schedule", [(True, None), (False, {1: 0, 3: 1, 5: 0}),
                                           (True, {1: 0, 2: 1})])
def test_muon_sync_matrices_and_mode_switches(cuda_device, sync, schedule):
    """Per-matrix synchronous training (every other matrix) and synchronous
    start / cooldown: Alg. 1 restarts at each switch into delayed training.
    One Newton-Schulz step, so O agrees up to rare flips (module note)."""
    sync_l = [i % 2 == 1 for i in range(len(SHAPES))] if sync else None
    p = Pair(SHAPES, cuda_device, ns_steps=1, ef=True, sync=sync_l, schedule=schedule,
             delay=0 if schedule else 1)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    try:
        for k in range(6):
            p.step()
            assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= (TOL_ONE_STEP if k == 0
                                                                    else TOL_RUN)
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            u, ur = p.cat(p.gpu.ef), _flat(p.ref.u_prev)
            close_with_flips(u, ur, 1e-5, du, 2e-3)
            if p.gpu.delay == 1:
                keep = np.concatenate([np.full(r * c, not p.sync[i]) for i, (r, c)
                                       in enumerate(SHAPES)])
                st = p.cat(p.gpu.stash).astype(np.float64)[keep]
                close_with_flips(st, _flat(p.ref.stash)[keep], 2.0 ** -7, k * du, 1e-3)
    finally:
        p.close()


def test_muon_sapipe_same_state(cuda_device):
    """SAPipe-WP with the same state (App. B.1): the stash receives the
    prediction point X_t - U_prev, the weights take the standard rule."""
    p = Pair(SHAPES, cuda_device, ns_steps=1, ef=True, correction=1)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    try:
        for k in range(5):
            p.step()
            assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= (TOL_ONE_STEP if k == 0
                                                                    else TOL_RUN)
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            close_with_flips(p.cat(p.gpu.ef), _flat(p.ref.u_prev), 1e-5, du, 2e-3)
            close_with_flips(p.cat(p.gpu.stash).astype(np.float64), _flat(p.ref.stash), 2.0 ** -7,
                             (k + 1) * du, 1e-3)
    finally:
        p.close()


@pytest.mark.parametrize("sync,clip,ns_steps", [(None, 0.0, 1), ([i % 3 == 1 for i in range(9)], 0.5, 1),
                                           (None, 0.0, 5)])
def test_muon_sapipe_updated_state(cuda_device, sync, clip, ns_steps):
    """SAPipe-WP with the updated state (App. B.1): the history holds the
    prediction update U' = lr (r NS(mu M + (1 - mu) G^) + wd X_{t+1}) from a
    second Newton-Schulz chain, the stash X_t - U'_prev, the weights the
    standard rule; a synchronous matrix (every third) keeps a zero history
    and no stash; with clipping, the prediction consumes the clipped
    gradient. U' carries the flip bound of one Newton-Schulz output (module
    note) and the stash that of the previous call's U' and weights; with 5
    Newton-Schulz steps, where the two bf16 iterations decorrelate, U' is
    held to the 5-step output bar, normwise (Frobenius, over the delayed
    matrices), as test_newton_schulz_parity holds O."""
    p = Pair(SHAPES, cuda_device, ns_steps=ns_steps, ef=True, correction=2, sync=sync,
             max_grad_norm=clip)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    keep = np.concatenate([np.full(r * c, not p.sync[i]) for i, (r, c) in enumerate(SHAPES)])
    try:
        for k in range(5):
            p.step()
            assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= (TOL_ONE_STEP if k == 0
                                                                    else TOL_RUN)
            u, ur = p.cat(p.gpu.ef), _flat(p.ref.u_prev)
            assert np.all(u[~keep] == 0.0)
            if ns_steps == 1:
                close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
                close_with_flips(u[keep], ur[keep], 1e-5, du, 2e-3)
                close_with_flips(p.cat(p.gpu.stash).astype(np.float64)[keep],
                                 _flat(p.ref.stash)[keep], 2.0 ** -7, (k + 1) * du, 1e-3)
            else:
                norm = np.linalg.norm(u[keep] - ur[keep]) / np.linalg.norm(ur[keep])
                print(f"call {k + 1}: U' normwise {norm:.3e}")
                assert norm <= 1.5e-2, (k, norm)
    finally:
        p.close()


def test_muon_clipping(cuda_device):
    """Global clipping over all matrices scales the gradient before the
    momentum (the norm of these gradients is ~1.3)."""
    p = Pair(SHAPES, cuda_device, ns_steps=1, max_grad_norm=0.5)
    try:
        p.step()
        assert p.ref.last_clip < 0.5
        assert rel_err(p.cat(p.gpu.mom), _flat(p.ref.mom)) <= TOL_ONE_STEP
    finally:
        p.close()


def test_muon_without_rms_scaling(cuda_device):
    """rms_scale = 0: Alg. 2 as printed, U = lr (O + wd X_t), no
    0.2 sqrt(max(r, c)) factor; two calls against the oracle."""
    p = Pair(SHAPES, cuda_device, ns_steps=1, ef=True, rms_scale=0.0)
    du = p.lr * 2.0 ** -7
    try:
        for k in range(2):
            p.step()
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            close_with_flips(p.cat(p.gpu.ef), _flat(p.ref.u_prev), 1e-5, du, 2e-3)
    finally:
        p.close()


def test_muon_flops_and_workspace(cuda_device):
    shapes = [(256, 512), (512, 256), (300, 700)]
    m = muon.DelayedMuon(shapes, ns_steps=5, device=cuda_device)
    try:
        want = sum(5 * (a * (a + 1) * b + a * (a + 1) * a + 2 * a * a * b)
                   for a, b in ((min(r, c), max(r, c)) for r, c in shapes))
        assert m.flops() == pytest.approx(want, rel=1e-12)
        # (256, 512) and (512, 256) share the 256 x 512 group; (300, 700) pads to 512 x 768;
        # per matrix X twice, X^T, A and B
        ws = 2 * ((2 * (256 * 512 * 3 + 256 * 256 * 2)) + (512 * 768 * 3 + 512 * 512 * 2))
        assert m.workspace_bytes() == ws
    finally:
        m.close()


def test_muon_full_size_shapes(cuda_device):
    """The Llama-7B matrix shapes (4096 x 4096, 11008 x 4096 tall, 4096 x
    11008 wide): one call, then properties that hold at any size. The
    momentum equals (1 - mu) g on sampled elements; O's singular values
    follow the scalar quintic applied to those of M / ||M||_F (numpy-free:
    torch.linalg.svdvals on the GPU in fp32) within 2e-2."""
    shapes = [(4096, 4096), (11008, 4096), (4096, 11008)]
    gpu = muon.DelayedMuon(shapes, ns_steps=5, ef=True, device=cuda_device)
    try:
        off = 0
        for i, (r, c) in enumerate(shapes):
            synth.dev_normal(0x7B, synth.STREAM_GRAD, 1, off, gpu.grads(i).view(-1), 1e-3)
            off += r * c
        gpu.step()
        torch.cuda.synchronize()
        assert gpu.status() == 0
        a, b_, c_ = muon.NS_COEFFS
        for i, (r, c) in enumerate(shapes):
            m = gpu.view(gpu.mom, i)
            g = gpu.grads(i).float()
            idx = torch.randint(0, r * c, (4096,), generator=torch.Generator().manual_seed(i))
            mg = m.reshape(-1)[idx.to(m.device)].double()
            want = (g.reshape(-1)[idx.to(m.device)].double() *
                    float(np.float32(1.0) - np.float32(0.95)))
            assert torch.max(torch.abs(mg - want) / torch.abs(want).clamp_min(1e-12)) <= 1e-6
            s = torch.linalg.svdvals(m.double() if r * c <= (1 << 24) else m).double()
            x = s / (torch.linalg.norm(s) + 1e-7)
            for _ in range(5):
                x = a * x + b_ * x ** 3 + c_ * x ** 5
            so = torch.linalg.svdvals(gpu.last_update(i).float()).double()
            err = torch.max(torch.abs(torch.sort(so).values - torch.sort(x).values)).item()
            print(f"{r}x{c}: singular values within {err:.3e}")
            assert err <= 2e-2
    finally:
        gpu.close()


def test_gemm_wait_timeout_reports_status(cuda_device):
    """The failure path of the tensor-core pipeline, without a GPU fault: one
    GEMM launch whose MMA lane waits on a phase nothing completes gives up
    after its one-second limit, every role leaves through its own bounded
    wait, the step returns and the status says which waits gave up
    (4: accumulator hand-off, 2: free stage; not 1 or 8, since every TMA
    stage issued has landed). After clearing, the context and the GPU work
    on: the next call reports nothing, and a fresh context holds parity."""
    import time
    shapes = [(256, 512), (512, 768)]
    m = muon.DelayedMuon(shapes, ns_steps=1, device=cuda_device)
    try:
        off = 0
        for i, (r, c) in enumerate(shapes):
            synth.dev_normal(0x57A1, synth.STREAM_GRAD, 1, off, m.grads(i).view(-1), 1e-3)
            off += r * c
        m.step()
        torch.cuda.synchronize()
        assert m.status() == 0
        m.test_stall(1)
        t0 = time.monotonic()
        m.step()
        torch.cuda.synchronize()
        took = time.monotonic() - t0
        bits = m.status()
        assert bits & 4 and bits & ~(2 | 4) == 0, bits
        assert 0.9 < took < 10.0, took
        m.clear_status()
        m.step()
        torch.cuda.synchronize()
        assert m.status() == 0
    finally:
        m.close()
    p = Pair([(256, 512), (300, 700)], cuda_device, ns_steps=1)
    try:
        p.step()
        got, ref = p.o_pairs()
        g, r = _flat(got), _flat(ref)
        assert np.linalg.norm(g - r) / np.linalg.norm(r) <= NS_BARS[1][0]
    finally:
        p.close()


def test_muon_checkpoint_resume_after_synchronous_start(cuda_device):
    """Synchronous start of 3 calls, delayed training with EF from call 4,
    a checkpoint after call 5 restored into a new context (INIT_RESUME), 3
    more calls: bitwise equal to 8 straight calls (k and the phase start
    restored, so EF starts at the same call)."""
    shapes = [(256, 512), (300, 700)]
    kw = dict(ns_steps=1, ef=True, keep_stash=True, device=cuda_device)

    def grads(m, k):
        off = 0
        for i, (r, c) in enumerate(shapes):
            synth.dev_normal(0xC4E, synth.STREAM_GRAD, k, off, m.grads(i).view(-1), 1e-3)
            off += r * c

    x0 = [torch.from_numpy(x) for x in inputs(shapes, 0xC4E, 1)[0]]
    straight = muon.DelayedMuon(shapes, x0=x0, **kw)
    split = muon.DelayedMuon(shapes, x0=x0, **kw)
    fresh = None
    try:
        for m in (straight, split):
            m.set_delay(0)
        for k in range(1, 9):
            if k == 4:
                straight.set_delay(1)
            grads(straight, k)
            straight.step()
        for k in range(1, 6):
            if k == 4:
                split.set_delay(1)
            grads(split, k)
            split.step()
        sd = split.state_dict()
        assert sd["phase_start"] == 3 and sd["k"] == 5 and sd["delay"] == 1
        fresh = muon.DelayedMuon(shapes, init_mode=dpo.DPO_INIT_RESUME, **kw)
        fresh.load_state(sd)
        for k in range(6, 9):
            grads(fresh, k)
            fresh.step()
        torch.cuda.synchronize()
        for name in muon.DelayedMuon.STATE:
            assert torch.equal(getattr(straight, name), getattr(fresh, name)), name
        assert straight.status() == 0 and fresh.status() == 0
    finally:
        for m in (straight, split, fresh):
            if m is not None:
                m.close()


def test_muon_capturable_step_replays_in_a_cuda_graph(cuda_device):
    """Capturable mode: after a 2-call synchronous start, one dpo_muon_step
    (clipped, EF) captured in a CUDA graph and replayed five times with fresh
    gradients and a learning rate written between replays equals an eager
    run bitwise at every call (the device forms the same lr, lr wd and EF
    start as the host; the Newton-Schulz chain is deterministic)."""
    shapes = [(256, 512), (300, 700)]
    kw = dict(ns_steps=1, ef=True, keep_stash=True, max_grad_norm=0.5, device=cuda_device)
    x0 = [torch.from_numpy(x) for x in inputs(shapes, 0x6A, 1)[0]]
    eager, cap = muon.DelayedMuon(shapes, x0=x0, **kw), muon.DelayedMuon(shapes, x0=x0, **kw)
    lr_t = torch.empty(1, dtype=torch.float32, device=cuda_device)
    lrs = [None] + [2e-3 * (1.0 - 0.05 * i) for i in range(1, 8)]

    def grads(m, k):
        off = 0
        for i, (r, c) in enumerate(shapes):
            synth.dev_normal(0x6A, synth.STREAM_GRAD, k, off, m.grads(i).view(-1), 1e-3)
            off += r * c

    try:
        for m in (eager, cap):
            m.set_delay(0)
        for k in (1, 2):
            for m in (eager, cap):
                grads(m, k)
                m.step(lrs[k])
        for m in (eager, cap):
            m.set_delay(1)
        cap.set_capturable(True, lr_source=lr_t)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            cap.step()
        for k in range(3, 8):
            grads(eager, k)
            grads(cap, k)
            lr_t.fill_(lrs[k])
            eager.step(lrs[k])
            graph.replay()
            torch.cuda.synchronize()
            for name in muon.DelayedMuon.STATE:
                assert torch.equal(getattr(eager, name), getattr(cap, name)), (k, name)
        assert cap.k == eager.k == 7 and cap.phase_start == 2
        cap.set_capturable(False)
        assert cap.k == 7
        assert eager.status() == 0 and cap.status() == 0
    finally:
        eager.close()
        cap.close()


def test_muon_weight_decay_mask_parity(cuda_device):
    """Per-matrix decay (DPO_WD_ON): matrices without it take U = lr r O
    only; three calls against the oracle with the same mask."""
    wd_on = [i % 2 == 0 for i in range(len(SHAPES))]
    p = Pair(SHAPES, cuda_device, ns_steps=1, ef=True, wd_on=wd_on)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    try:
        for k in range(3):
            p.step()
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            close_with_flips(p.cat(p.gpu.ef), _flat(p.ref.u_prev), 1e-5, du, 2e-3)
    finally:
        p.close()


@pytest.mark.parametrize("correction", [0, 1])
def test_muon_reentering_delayed_training_parity(cuda_device, correction):
    """Delayed calls 1-2, synchronous 3-4, delayed again from 5 (EF or SAPipe
    same state): Alg. 1 restarts at the re-entry on the device as in the
    oracle."""
    p = Pair(SHAPES, cuda_device, ns_steps=1, ef=True, schedule={3: 0, 5: 1},
             correction=correction)
    r_max = 0.2 * np.sqrt(max(max(sh) for sh in SHAPES))
    du = p.lr * r_max * 2.0 ** -7
    try:
        for k in range(7):
            p.step()
            close_with_flips(p.cat(p.gpu.master), _flat(p.ref.x), TOL_RUN, (k + 1) * du, 1e-3)
            if p.gpu.delay == 1:
                close_with_flips(p.cat(p.gpu.stash).astype(np.float64), _flat(p.ref.stash),
                                 2.0 ** -7, (k + 1) * du, 1e-3)
    finally:
        p.close()
