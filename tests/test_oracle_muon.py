"""Pins of the delayed-Muon oracle (Alg. 2) against facts outside it.

* Newton-Schulz is a matrix polynomial in M M^T times M, so on M = U S V^T
  it acts on each singular value alone: O = U p^s(S / (||M||_F + eps)) V^T
  with p(x) = a x + b x^3 + c x^5 iterated s times. The singular vectors come
  from numpy's SVD (a library routine); the scalar recursion is one line.
* On a diagonal matrix every iterate stays diagonal, so the bf16 iteration
  is a scalar recursion with one bf16 rounding per formed quantity.
* The Muon step is checked by hand on small cases: the update scale, the
  momentum's weighting, decay on the current weights, and Alg. 2's EF line
  X_{t+1} = X_t - 2 U_{t-1} + U_{t-2}.
"""
from __future__ import annotations

import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import muon
from oracle.muon import NS_COEFFS, DelayedMuon, MuonHParams, newton_schulz

F64, F32, BF16 = oracle.F64, oracle.F32, oracle.BF16
A_, B_, C_ = NS_COEFFS


@pytest.fixture(scope="module")
def lib():
    path = os.environ.get("DPO_ORACLE_LIB")
    return oracle.load(path) if path else oracle.load()


def p_iter(x, steps):
    for _ in range(steps):
        x = A_ * x + B_ * x ** 3 + C_ * x ** 5
    return x


def with_singular_values(rng, rows, cols, s):
    u, _ = np.linalg.qr(rng.normal(size=(rows, rows)))
    v, _ = np.linalg.qr(rng.normal(size=(cols, cols)))
    r = min(rows, cols)
    return u[:, :r] @ np.diag(s) @ v[:, :r].T, u[:, :r], v[:, :r]


@pytest.mark.parametrize("rows,cols", [(5, 9), (9, 5), (7, 7), (1, 6), (6, 1)])
@pytest.mark.parametrize("steps", [1, 2, 5])
def test_ns_acts_on_singular_values(lib, rows, cols, steps):
    rng = np.random.default_rng(rows * 100 + cols + steps)
    s = np.sort(rng.uniform(0.05, 3.0, min(rows, cols)))[::-1]
    M, u, v = with_singular_values(rng, rows, cols, s)
    eps = 1e-7
    expect = u @ np.diag(p_iter(s / (np.linalg.norm(s) + eps), steps)) @ v.T
    O = newton_schulz(M, steps=steps, store=F64, eps=eps, lib=lib)
    assert O.shape == (rows, cols)
    assert np.max(np.abs(O - expect)) < 1e-12


def test_ns_rank_one(lib):
    """M = 4 u v^T: normalised, its one singular value is 4 / (4 + eps)."""
    u = np.array([3.0, 4.0]) / 5.0
    v = np.array([1.0, 2.0, 2.0]) / 3.0
    M = 4.0 * np.outer(u, v)
    O = newton_schulz(M, steps=5, store=F64, eps=1e-7, lib=lib)
    np.testing.assert_allclose(O, p_iter(4.0 / (4.0 + 1e-7), 5) * np.outer(u, v), rtol=1e-13)


def test_ns_zero_steps_is_normalisation(lib):
    M = np.arange(12.0).reshape(3, 4) - 5.0
    O = newton_schulz(M, steps=0, store=F64, eps=1e-7, lib=lib)
    np.testing.assert_allclose(O, M / (math.sqrt(np.sum(M * M)) + 1e-7), rtol=1e-15)


@pytest.mark.parametrize("store", [F64, BF16])
def test_ns_transpose(lib, store):
    """NS(M^T) = NS(M)^T exactly: both run on the same wide orientation."""
    M = np.random.default_rng(3).normal(size=(6, 11))
    O = newton_schulz(M, store=store, lib=lib)
    Ot = newton_schulz(M.T.copy(), store=store, lib=lib)
    assert np.array_equal(Ot, O.T)


@pytest.mark.parametrize("rows,cols", [(4, 4), (4, 7), (7, 4)])
def test_ns_bf16_on_diagonal(lib, rows, cols):
    """A diagonal M stays diagonal: each entry follows x0 = bf(d / (||d|| +
    eps)), then A = bf(x^2), B = bf(b A + c A^2), x = bf(a x + B x)."""
    d = np.array([1.7, -0.3, 0.021, 0.9])
    M = np.zeros((rows, cols))
    for i in range(4):
        M[i, i] = d[i]
    bf = lambda z: oracle.round_to(np.asarray(z, np.float64), BF16, lib)
    x = bf(d / (math.sqrt(np.sum(d * d)) + 1e-7))
    for _ in range(5):
        a = bf(x * x)
        b = bf(B_ * a + C_ * (a * a))
        x = bf(A_ * x + b * x)
    O = newton_schulz(M, steps=5, store=BF16, eps=1e-7, lib=lib)
    expect = np.zeros((rows, cols))
    for i in range(4):
        expect[i, i] = x[i]
    assert np.array_equal(O, expect)
    # and the result differs from the exact iteration (rounding happened)
    assert not np.array_equal(O, newton_schulz(M, steps=5, store=F64, eps=1e-7, lib=lib))


def test_ns_bf16_iterates_are_bf16(lib):
    M = np.random.default_rng(4).normal(size=(8, 20))
    O = newton_schulz(M, store=BF16, lib=lib)
    assert np.array_equal(O, oracle.round_to(O, BF16, lib))


# ----------------------------------------------------------------- step ----

def _hp(**kw):
    base = dict(lr=0.01, momentum=0.95, weight_decay=0.1, ns_store=F64, delay=1)
    base.update(kw)
    return MuonHParams(**base)


def test_muon_first_step_by_hand(lib):
    """First call: M = (1 - mu) g, whose normalisation removes (1 - mu) (up
    to eps); U = lr (0.2 sqrt(max(rows, cols)) O + wd X_0); standard rule."""
    rng = np.random.default_rng(5)
    x0 = rng.normal(size=(4, 9))
    s = np.array([2.0, 1.0, 0.5, 0.1])
    g, u, v = with_singular_values(rng, 4, 9, s)
    hp = _hp(ns_eps=0.0)
    opt = DelayedMuon([x0], hp, ef=True, x_store=F64, stash_store=F64, param_store=F64, lib=lib)
    opt.step([g])
    O = u @ np.diag(p_iter(s / np.linalg.norm(s), 5)) @ v.T
    U = 0.01 * (0.2 * 3.0 * O + 0.1 * x0)
    np.testing.assert_allclose(opt.mom[0], 0.05 * g, rtol=1e-14, atol=1e-16)
    np.testing.assert_allclose(opt.x[0], x0 - U, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(opt.u_prev[0], U, rtol=1e-12, atol=1e-14)
    assert np.array_equal(opt.stash[0], x0)
    assert np.array_equal(opt.param[0], opt.x[0])


def test_muon_scale_uses_the_larger_dimension(lib):
    """Zero decay: U = lr * 0.2 sqrt(max(rows, cols)) O, for both shapes."""
    for shape in [(4, 25), (25, 4)]:
        rng = np.random.default_rng(6)
        g = rng.normal(size=shape)
        opt = DelayedMuon([np.zeros(shape)], _hp(weight_decay=0.0), x_store=F64,
                          stash_store=F64, lib=lib)
        opt.step([g])
        O = newton_schulz(0.05 * g, store=F64, lib=lib)
        np.testing.assert_allclose(-opt.x[0], 0.01 * 0.2 * 5.0 * O, rtol=1e-13, atol=1e-16)


def test_muon_momentum_weights_the_history(lib):
    """With no Newton-Schulz steps O = M / ||M||: after gradients g1, g2 the
    direction is that of mu g1 + g2 (Sec. 2.2's EMA), not (1 - mu) g1 + g2."""
    rng = np.random.default_rng(7)
    g1, g2 = rng.normal(size=(3, 5)), rng.normal(size=(3, 5))
    opt = DelayedMuon([np.zeros((3, 5))], _hp(weight_decay=0.0, ns_steps=0, ns_eps=0.0,
                                              rms_scale=0.0), x_store=F64, stash_store=F64,
                      lib=lib)
    opt.step([g1])
    x1 = opt.x[0].copy()
    opt.step([g2])
    d = 0.95 * g1 + g2
    np.testing.assert_allclose(x1 - opt.x[0], 0.01 * d / np.linalg.norm(d), rtol=1e-12)


def test_muon_decay_acts_on_current_weights(lib):
    """Zero gradients give O = 0, so each call scales X_t by (1 - lr wd);
    under delay the stash lags one version and is not what decays."""
    x0 = np.random.default_rng(8).normal(size=(3, 4))
    opt = DelayedMuon([x0], _hp(lr=0.1, weight_decay=0.5), x_store=F64, stash_store=F64,
                      lib=lib)
    for k in range(1, 5):
        opt.step([np.zeros((3, 4))])
        np.testing.assert_allclose(opt.x[0], (1 - 0.05) ** k * x0, rtol=1e-14)


def test_muon_ef_is_algorithm_2(lib):
    """EF with lambda = 1: X_2 = X_1 - U_0 (standard rule at t = 1), then
    X_{t+1} = X_t - 2 U_{t-1} + U_{t-2}, with U_{t-1} = lr (s O + wd X_t)
    rebuilt from the Newton-Schulz outputs; the stash holds X_t."""
    rng = np.random.default_rng(9)
    x0 = rng.normal(size=(5, 3))
    opt = DelayedMuon([x0], _hp(ef_lambda=1.0), ef=True, x_store=F64, stash_store=F64, lib=lib)
    xs, us = [x0.copy()], []
    for k in range(5):
        xt = opt.x[0].copy()
        opt.step([rng.normal(size=(5, 3))])
        us.append(0.01 * (0.2 * math.sqrt(5) * opt.o[0] + 0.1 * xt))
        assert np.array_equal(opt.stash[0], xt)
        if k == 0:
            np.testing.assert_allclose(opt.x[0], xt - us[0], rtol=1e-14)
        else:
            np.testing.assert_allclose(opt.x[0], xt - 2 * us[k] + us[k - 1], rtol=1e-13)
        xs.append(opt.x[0].copy())


def test_muon_empty_and_clip(lib):
    """A 0 x n matrix is a no-op; clipping scales the gradient before the
    momentum (global norm over all matrices)."""
    opt = DelayedMuon([np.zeros((0, 4)), np.ones((2, 2))],
                      _hp(max_grad_norm=1.0, ns_steps=0, ns_eps=0.0, rms_scale=0.0,
                          weight_decay=0.0), x_store=F64, stash_store=F64, lib=lib)
    g = np.full((2, 2), 3.0)   # norm 6
    opt.step([np.zeros((0, 4)), g])
    assert opt.last_clip == pytest.approx(1.0 / (6.0 + 1e-6), rel=1e-15)
    np.testing.assert_allclose(opt.mom[1], 0.05 * g * opt.last_clip, rtol=1e-15)


def test_muon_per_matrix_delay_is_independent(lib):
    """A table mixing a delayed and a synchronous matrix gives, matrix by
    matrix, bitwise the runs of each matrix alone in its mode; the
    synchronous one never writes its stash or history."""
    rng = np.random.default_rng(10)
    x0 = [rng.normal(size=(4, 6)), rng.normal(size=(7, 3))]
    grads = [[rng.normal(size=(4, 6)), rng.normal(size=(7, 3))] for _ in range(4)]
    mixed = DelayedMuon(x0, _hp(ef_lambda=1.0), ef=True, x_store=F64, stash_store=F64,
                        delayed=[True, False], lib=lib)
    alone = [DelayedMuon([x0[0]], _hp(ef_lambda=1.0), ef=True, x_store=F64, stash_store=F64,
                         lib=lib),
             DelayedMuon([x0[1]], _hp(ef_lambda=1.0, delay=0), ef=True, x_store=F64,
                         stash_store=F64, lib=lib)]
    for g in grads:
        mixed.step(g)
        alone[0].step([g[0]])
        alone[1].step([g[1]])
    assert np.array_equal(mixed.x[0], alone[0].x[0])
    assert np.array_equal(mixed.x[1], alone[1].x[0])
    assert np.array_equal(mixed.stash[1], x0[1]) and not np.any(mixed.u_prev[1])


def test_muon_synchronous_start_restarts_alg1(lib):
    """Two synchronous calls, then delayed: the switch stashes the current
    weights and zeroes the history; the first delayed call takes the
    standard rule, the next ones Alg. 2's EF line; the stash lags by one."""
    rng = np.random.default_rng(11)
    x0 = rng.normal(size=(5, 8))
    opt = DelayedMuon([x0], _hp(ef_lambda=1.0, delay=0), ef=True, x_store=F64,
                      stash_store=F64, lib=lib)
    scale = 0.2 * math.sqrt(8)
    for _ in range(2):
        xt = opt.x[0].copy()
        opt.step([rng.normal(size=(5, 8))])
        np.testing.assert_allclose(opt.x[0], xt - 0.01 * (scale * opt.o[0] + 0.1 * xt),
                                   rtol=1e-13)
    assert not np.any(opt.u_prev[0])
    opt.set_delay(1)
    assert np.array_equal(opt.stash[0], opt.x[0])
    us = []
    for k in range(3):
        xt = opt.x[0].copy()
        opt.step([rng.normal(size=(5, 8))])
        us.append(0.01 * (scale * opt.o[0] + 0.1 * xt))
        assert np.array_equal(opt.stash[0], xt)
        want = xt - us[0] if k == 0 else xt - 2 * us[k] + us[k - 1]
        np.testing.assert_allclose(opt.x[0], want, rtol=1e-13)
    # cooldown: the standard rule again, stash and history left as they were
    opt.set_delay(0)
    stash, hist = opt.stash[0].copy(), opt.u_prev[0].copy()
    xt = opt.x[0].copy()
    opt.step([rng.normal(size=(5, 8))])
    np.testing.assert_allclose(opt.x[0], xt - 0.01 * (scale * opt.o[0] + 0.1 * xt), rtol=1e-13)
    assert np.array_equal(opt.stash[0], stash) and np.array_equal(opt.u_prev[0], hist)


def test_muon_sapipe_same_state(lib):
    """SAPipe-WP with the same state (App. B.1): the weights are bitwise the
    standard rule's; the stash holds the prediction point X_t - U_prev, so
    consecutive prediction points move by Eq. (1)'s displacement -2U + U_prev,
    which an independent EF run's weights show (zero decay: the updates of
    the two runs are the same)."""
    rng = np.random.default_rng(12)
    x0 = rng.normal(size=(4, 6))
    grads = [rng.normal(size=(4, 6)) for _ in range(6)]
    sp = DelayedMuon([x0], _hp(weight_decay=0.0, correction=oracle.CORR_SAPIPE_SAME), ef=True,
                     x_store=F64, stash_store=F64, lib=lib)
    std = DelayedMuon([x0], _hp(weight_decay=0.0), x_store=F64, stash_store=F64, lib=lib)
    ef = DelayedMuon([x0], _hp(weight_decay=0.0, ef_lambda=1.0), ef=True, x_store=F64,
                     stash_store=F64, lib=lib)
    stash, efx = [], [x0.copy()]
    for g in grads:
        xt = sp.x[0].copy()
        hist = sp.u_prev[0].copy()
        for o in (sp, std, ef):
            o.step([g])
        assert np.array_equal(sp.x[0], std.x[0])
        assert np.array_equal(sp.stash[0], xt - hist)
        stash.append(sp.stash[0].copy())
        efx.append(ef.x[0].copy())
    # stash after call k+1 minus after call k == EF weights after call k minus after call k-1
    for k in range(2, len(grads)):
        np.testing.assert_allclose(stash[k] - stash[k - 1], efx[k] - efx[k - 1],
                                   rtol=1e-9, atol=1e-15)


@pytest.mark.parametrize("x_store,ns_store", [(F64, F64), (F32, BF16)])
def test_muon_sapipe_updated_is_the_next_step_on_a_repeated_gradient(lib, x_store, ns_store):
    """SAPipe-WP with the updated state (App. B.1) for Muon: the prediction
    update stored after call k is, bitwise, the update that call k + 1 of a
    run whose gradient k + 1 repeats gradient k stores (EF at lambda = 0:
    the standard rule, keeping each update in its history): the same momentum
    formed once more, the same Newton-Schulz, decay on X_{t+1}. Also with
    fp32 state and bf16 Newton-Schulz iterates. The weights follow the
    standard rule and the stash holds X_t - U_prev with U_prev the previous
    prediction update."""
    rng = np.random.default_rng(14)
    x0 = rng.normal(size=(5, 8))
    grads = [rng.normal(size=(5, 8)) for _ in range(5)]
    kw = dict(x_store=x_store, stash_store=x_store, lib=lib)
    sp = DelayedMuon([x0], _hp(correction=oracle.CORR_SAPIPE_UPDATED, ns_store=ns_store),
                     ef=True, **kw)
    std = DelayedMuon([x0], _hp(ns_store=ns_store), **kw)
    for k in range(1, len(grads) + 1):
        xt, hist = sp.x[0].copy(), sp.u_prev[0].copy()
        sp.step([grads[k - 1]])
        std.step([grads[k - 1]])
        assert np.array_equal(sp.x[0], std.x[0])
        assert np.array_equal(sp.stash[0], oracle.round_to(xt - hist, x_store, lib))
        rep = DelayedMuon([x0], _hp(ef_lambda=0.0, ns_store=ns_store), ef=True, **kw)
        for g in grads[:k] + [grads[k - 1]]:
            rep.step([g])
        assert np.array_equal(sp.u_prev[0], rep.u_prev[0])


def test_muon_sapipe_updated_by_hand(lib):
    """1 x 2 matrix, mu = 0.5, lr = 0.1, wd = 0, no RMS scaling, no
    Newton-Schulz steps (O = M / ||M||), eps 0; gradients (3, 4), (4, -3).
    Call 1: M = (1.5, 2), U = 0.1 (0.6, 0.8); prediction M' = (2.25, 3), the
    same direction. Call 2: M = (2.75, -0.5), U = 0.1 M / sqrt(7.8125);
    prediction M' = 0.5 M + 0.5 (4, -3) = (3.375, -1.75), so
    U' = 0.1 M' / sqrt(14.453125), a direction the same state would miss.
    Call 2 reads the stash X_1 - U'_1 = (0.88, 0.84)."""
    hp = _hp(lr=0.1, momentum=0.5, weight_decay=0.0, rms_scale=0.0, ns_steps=0, ns_eps=0.0,
             correction=oracle.CORR_SAPIPE_UPDATED)
    o = DelayedMuon([np.array([[1.0, 1.0]])], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    o.step([np.array([[3.0, 4.0]])])
    np.testing.assert_allclose(o.x[0], [[0.94, 0.92]], rtol=1e-15)
    np.testing.assert_allclose(o.u_prev[0], [[0.06, 0.08]], rtol=1e-15)
    o.step([np.array([[4.0, -3.0]])])
    np.testing.assert_allclose(o.stash[0], [[0.88, 0.84]], rtol=1e-15)
    u2 = 0.1 * np.array([2.75, -0.5]) / math.sqrt(7.8125)
    np.testing.assert_allclose(o.x[0], [[0.94 - u2[0], 0.92 - u2[1]]], rtol=1e-15)
    np.testing.assert_allclose(o.u_prev[0], [0.1 * np.array([3.375, -1.75]) /
                                             math.sqrt(14.453125)], rtol=1e-15)


def test_muon_ef_lambda_scales_the_correction(lib):
    """Eq. (1) for Muon's update: X_{t+1} = X_t - U - lambda (U - U_prev).
    At lambda = 0 the EF run is bitwise the standard one; at lambda = 1/2 the
    weights sit halfway between the standard and lambda = 1 runs (the same
    U_t in all three while no correction has changed X_t: first two calls)."""
    rng = np.random.default_rng(23)
    x0 = rng.normal(size=(4, 6))
    grads = [rng.normal(size=(4, 6)) for _ in range(4)]
    runs = {}
    for lam in (None, 0.0, 0.5, 1.0):
        opt = DelayedMuon([x0], _hp(ef_lambda=lam or 0.0), ef=lam is not None, x_store=F64,
                          stash_store=F64, lib=lib)
        xs = []
        for g in grads:
            opt.step([g])
            xs.append(opt.x[0].copy())
        runs[lam] = xs
    for a, b in zip(runs[None], runs[0.0]):
        assert np.array_equal(a, b)
    # second call: the first EF correction, on identical X_2 and U
    half = 0.5 * (runs[None][1] + runs[1.0][1])
    assert np.max(np.abs(runs[0.5][1] - half)) < 1e-14
    assert np.max(np.abs(runs[1.0][1] - runs[None][1])) > 1e-6


def test_muon_sapipe_prediction_rounds_through_the_master(lib):
    """As for the elementwise rules: the SAPipe-WP stash is X_t - U_prev in
    the master's format (fp32), then the stash's (bf16); 1 + 2^-8 - (-2^-30)
    lands on the bf16 tie and rounds to even, 1.0."""
    x0 = np.full((2, 2), 1.0 + 2.0 ** -8)
    opt = DelayedMuon([x0], _hp(lr=0.0, weight_decay=0.0, correction=1), ef=True,
                      x_store=F32, stash_store=BF16, lib=lib)
    opt.u_prev[0][...] = -(2.0 ** -30)
    opt.step([np.ones((2, 2))])
    assert np.all(opt.stash[0] == 1.0)



def test_muon_clip_from_a_supplied_norm(lib):
    """Global clipping (App. E.1) across contexts: two Muon oracles, one per
    matrix, each given the squared norm over both gradients, take torch's
    clip_grad_norm_ coefficient over the pair and step exactly as one oracle
    over both matrices, bitwise."""
    rng = np.random.default_rng(37)
    xs = [rng.normal(size=(4, 6)), rng.normal(size=(5, 3))]
    hp = _hp(max_grad_norm=1.0, ef_lambda=1.0)
    both = DelayedMuon(xs, hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    one = [DelayedMuon([x], hp, ef=True, x_store=F64, stash_store=F64, lib=lib) for x in xs]
    for _ in range(3):
        gs = [rng.normal(0, 0.5, x.shape) for x in xs]
        params = [torch.nn.Parameter(torch.zeros(x.shape, dtype=torch.float64)) for x in xs]
        for p_, g in zip(params, gs):
            p_.grad = torch.tensor(g)
        torch.nn.utils.clip_grad_norm_(params, 1.0)
        coef = float(params[0].grad[0, 0] / gs[0][0, 0])
        assert coef < 0.5   # clipping is active
        sq = sum(oracle.sqnorm(g, lib=lib) for g in gs)
        both.step(gs)
        for o, g in zip(one, gs):
            o.step([g], sq=sq)
        for o in [both] + one:
            assert o.last_clip == pytest.approx(coef, rel=1e-13)
        for i in range(2):
            assert np.array_equal(one[i].x[0], both.x[i])

def test_muon_weight_decay_mask(lib):
    """A matrix without decay is the same run as a context whose decay is
    zero, bitwise; the decayed matrix beside it is unchanged by the mask."""
    rng = np.random.default_rng(31)
    xa, xb = rng.normal(size=(4, 6)), rng.normal(size=(5, 3))
    grads = [[rng.normal(size=(4, 6)), rng.normal(size=(5, 3))] for _ in range(3)]
    mixed = DelayedMuon([xa, xb], _hp(), ef=True, x_store=F64, stash_store=F64, lib=lib,
                        wd_on=[True, False])
    decayed = DelayedMuon([xa], _hp(), ef=True, x_store=F64, stash_store=F64, lib=lib)
    plain = DelayedMuon([xb], _hp(weight_decay=0.0), ef=True, x_store=F64, stash_store=F64,
                        lib=lib)
    for ga, gb in grads:
        mixed.step([ga, gb])
        decayed.step([ga])
        plain.step([gb])
    assert np.array_equal(mixed.x[0], decayed.x[0])
    assert np.array_equal(mixed.x[1], plain.x[0])



def test_muon_initial_state_is_x0_in_its_storage_formats(lib):
    """The start state holds each matrix's X_0 as the device stores it: the
    master cast to fp32, the stash and the weights that value cast to bf16
    (torch's casts), before any call."""
    rng = np.random.default_rng(45)
    xs = [rng.normal(0, 0.02, (6, 10)), rng.normal(0, 0.02, (3, 4))]
    opt = DelayedMuon(xs, _hp(ef_lambda=1.0), ef=True, x_store=F32, stash_store=BF16,
                      param_store=BF16, lib=lib)
    for i, x in enumerate(xs):
        x32 = torch.tensor(x).float()
        np.testing.assert_array_equal(opt.x[i], x32.double().numpy())
        np.testing.assert_array_equal(opt.stash[i], x32.bfloat16().double().numpy())
        np.testing.assert_array_equal(opt.param[i], x32.bfloat16().double().numpy())

def test_muon_stored_state_is_in_its_storage_format(lib):
    """Muon's buffers hold values of their storage formats after each call:
    master, momentum and the EF history in fp32, stash and weights in
    bf16."""
    rng = np.random.default_rng(43)
    x0 = rng.normal(0, 0.02, (6, 10))
    opt = DelayedMuon([x0], _hp(ef_lambda=1.0, ns_store=BF16), ef=True, x_store=F32,
                      stash_store=BF16, param_store=BF16, lib=lib)
    f32 = lambda a: np.array_equal(np.asarray(a).astype(np.float32).astype(np.float64), a)
    bf16 = lambda a: f32(a) and not np.any(np.asarray(a, np.float32).view(np.uint32) & 0xFFFF)
    for _ in range(3):
        opt.step([rng.normal(0, 1e-3, (6, 10))])
        assert f32(opt.x[0]) and f32(opt.mom[0]) and f32(opt.u_prev[0])
        assert bf16(opt.stash[0]) and bf16(opt.param[0])


def test_muon_weights_round_the_stored_master(lib):
    """As for the elementwise rules: a 1 x 1 matrix, no Newton-Schulz steps
    and eps 0 give O = sign(M) = -1, so with lr = 2^-30, no decay and no RMS
    scaling X_1 = 1 + 2^-8 + 2^-30, stored in fp32 as the bf16 tie 1 + 2^-8;
    the bf16 weights are then 1.0, not 1 + 2^-7."""
    opt = DelayedMuon([np.array([[1.0 + 2.0 ** -8]])],
                      _hp(lr=2.0 ** -30, weight_decay=0.0, rms_scale=0.0, ns_steps=0,
                          ns_eps=0.0, ns_store=F64), x_store=F32, stash_store=F32,
                      param_store=BF16, lib=lib)
    opt.step([np.array([[-1.0]])])
    assert opt.x[0][0, 0] == 1.0 + 2.0 ** -8
    assert opt.param[0][0, 0] == 1.0


@pytest.mark.parametrize("steps", [1, 2, 3])
@pytest.mark.parametrize("tall", [False, True])
def test_newton_schulz_bf16_restated_exactly(lib, steps, tall):
    """An independent restatement of the bf16 iteration (numpy products,
    torch's bf16 rounding) on inputs where every fp64 operation is exact: a
    2 x 8 matrix of +-1 entries (||M||_F = 4, X_0 = M / 4 exact with eps 0,
    each product a sum of few short-mantissa terms). The iteration runs on
    the orientation with the smaller Gram matrix (2 x 2), for the matrix and
    for its 8 x 2 transpose; the oracle must agree bitwise."""
    import torch
    rng = np.random.default_rng(61)
    Mw = rng.choice([-1.0, 1.0], size=(2, 8))
    M = Mw.T.copy() if tall else Mw
    bf = lambda x: torch.tensor(x, dtype=torch.float64).to(torch.bfloat16).double().numpy()
    a, b, c = NS_COEFFS
    X = bf(Mw / 4.0)
    for _ in range(steps):
        A = bf(X @ X.T)
        B = bf(b * A + c * (A @ A))
        X = bf(a * X + B @ X)
    want = X.T if tall else X
    got = newton_schulz(M, steps=steps, store=BF16, eps=0.0, lib=lib)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("correction", [0, 1])
def test_muon_reentering_delayed_training_restarts(lib, correction):
    """Delayed, synchronous, delayed again: from the re-entry on, the run is a
    fresh Alg. 1 run (stash at X, history zero, standard rule first, then EF
    or SAPipe's prediction) started at the weights and momentum reached
    there."""
    rng = np.random.default_rng(73)
    x0 = rng.normal(size=(4, 6))
    grads = [rng.normal(size=(4, 6)) for _ in range(10)]
    hp = _hp(ef_lambda=1.0, correction=correction)
    o = DelayedMuon([x0], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    for k, g in enumerate(grads[:7], start=1):
        if k == 4:
            o.set_delay(0)
        o.step([g])
    o.set_delay(1)
    fresh = DelayedMuon([o.x[0].copy()], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    fresh.mom[0][...] = o.mom[0]
    for g in grads[7:]:
        o.step([g])
        fresh.step([g])
        assert np.array_equal(o.x[0], fresh.x[0])
        assert np.array_equal(o.stash[0], fresh.stash[0])


def test_muon_momentum_depends_only_on_consumed_gradients(lib):
    """Muon's momentum takes each consumed gradient whatever the delay mode:
    a run with a synchronous start, a cooldown and a re-entry holds the same
    momentum as a run delayed throughout, given the same gradients."""
    rng = np.random.default_rng(83)
    x0 = rng.normal(size=(3, 5))
    grads = [rng.normal(size=(3, 5)) for _ in range(8)]
    runs = []
    for schedule in ({}, {1: 0, 3: 1, 5: 0, 7: 1}):
        o = DelayedMuon([x0], _hp(ef_lambda=1.0), ef=True, x_store=F64, stash_store=F64, lib=lib)
        for c, g in enumerate(grads, start=1):
            if c in schedule:
                o.set_delay(schedule[c])
            o.step([g])
        runs.append(o.mom[0].copy())
    assert np.array_equal(runs[0], runs[1])
