"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these compares the oracle with itself: each expected value comes from
a library routine (torch.optim.AdamW, torch's bf16 cast), exact rational
arithmetic on a worked example, a closed-form trajectory, or an invariant that
the update rule implies. ``test_oracle_mutants.py`` plants single mistakes in
a copy of the oracle and checks that these pins catch each one.

Paper passages (arXiv 2606.30634): Alg. 1 (delayed update, standard rule for
t <= 1), Eq. (1) of Sec. 3.2 (Error Feedback), App. A.4 (lambda-scaled EF),
App. B.1 (SAPipe weight prediction has EF's displacement), Alg. 2 (decay on
X_t), Sec. 2.1 / App. E.1 (AdamW beta = (0.9, 0.95), wd 0.1, clip 1.0).
"""
from __future__ import annotations

import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import BF16, F32, F64, HParams

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


@pytest.fixture
def lib():
    """The oracle under test: the default build, or (when DPO_ORACLE_LIB
    names one) a build with a planted mistake from test_oracle_mutants."""
    path = os.environ.get("DPO_ORACLE_LIB")
    return oracle.load(path) if path else oracle.load()


# ---------------------------------------------------------------- P1 ------
# Delay-free application of the AdamW rule equals torch.optim.AdamW.

def _torch_adamw_run(x0s, grads, hp: HParams, lrs, max_norm=0.0):
    ps = [torch.nn.Parameter(torch.tensor(x, dtype=torch.float64)) for x in x0s]
    opt = torch.optim.AdamW(ps, lr=lrs[0], betas=(hp.beta1, hp.beta2),
                            eps=hp.eps, weight_decay=hp.weight_decay,
                            foreach=False, fused=False)
    traj = []
    for gs, lr in zip(grads, lrs):
        for p, g in zip(ps, gs):
            p.grad = torch.tensor(g, dtype=torch.float64)
        if max_norm > 0:
            torch.nn.utils.clip_grad_norm_(ps, max_norm)
        for group in opt.param_groups:
            group["lr"] = lr
        opt.step()
        traj.append(np.concatenate([p.detach().numpy().ravel() for p in ps]))
    return traj


def _oracle_run(lib, x0s, grads, hp: HParams, lrs, ef=False):
    o = oracle.DelayedOptimizer(x0s, hp, ef=ef, x_store=F64, stash_store=F64,
                                lib=lib)
    traj = []
    for gs, lr in zip(grads, lrs):
        o.step(np.concatenate([np.ravel(g) for g in gs]), lr=lr)
        traj.append(o.x.copy())
    return traj, o


def _rel(a, b):
    return np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-300))


@pytest.mark.parametrize("delay", [0, 1])
@pytest.mark.parametrize("max_norm", [0.0, 1.0])
def test_p1_matches_torch_adamw(lib, delay, max_norm):
    """Applying the given gradient sequence, the oracle's weights equal
    torch.optim.AdamW's (delay changes only where gradients are evaluated,
    not the arithmetic of the update). Includes clipping at 1.0 against
    torch.nn.utils.clip_grad_norm_ and a changing learning rate."""
    rng = np.random.default_rng(7)
    shapes = [(5, 3), (7,), (1,)]
    x0s = [rng.normal(0, 0.5, s) for s in shapes]
    grads = [[rng.normal(0, 0.7, s) for s in shapes] for _ in range(12)]
    lrs = [1e-2 * (1 + 0.1 * i) for i in range(12)]
    hp = HParams(lr=lrs[0], beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1,
                 max_grad_norm=max_norm, delay=delay)
    ref = _torch_adamw_run(x0s, grads, hp, lrs, max_norm)
    got, _ = _oracle_run(lib, x0s, grads, hp, lrs)
    for r, g in zip(ref, got):
        assert _rel(g, r) < 1e-12


def test_p1_other_betas_and_eps(lib):
    """Same pin away from the paper's constants, so a swapped beta or a
    misplaced eps cannot hide behind them."""
    rng = np.random.default_rng(11)
    x0s = [rng.normal(0, 1, (9,))]
    grads = [[rng.normal(0, 1e-3, (9,))] for _ in range(6)]
    hp = HParams(lr=0.05, beta1=0.5, beta2=0.7, eps=1e-3, weight_decay=0.3,
                 delay=0)
    lrs = [0.05] * 6
    ref = _torch_adamw_run(x0s, grads, hp, lrs)
    got, _ = _oracle_run(lib, x0s, grads, hp, lrs)
    for r, g in zip(ref, got):
        assert _rel(g, r) < 1e-12


# ---------------------------------------------------------------- P2 ------
# Hand-worked example: scalar x0 = 1, beta = (0.9, 0.95), lr = 0.1, stale
# gradients 2, 1, -0.5. By hand:
#   k=1: m = 0.2,   v = 0.2,    1-b1^k = 0.1,   1-b2^k = 0.05     -> m_hat = 2, v_hat = 4
#   k=2: m = 0.28,  v = 0.24,   1-b1^k = 0.19,  1-b2^k = 0.0975
#   k=3: m = 0.202, v = 0.2405, 1-b1^k = 0.271, 1-b2^k = 0.142625
# Alg. 1 uses the standard rule at the first update in both modes; EF then
# applies x - 2u + u_prev (Eq. (1)).

_HAND_MV = [(0.2, 0.2, 0.1, 0.05), (0.28, 0.24, 0.19, 0.0975),
            (0.202, 0.2405, 0.271, 0.142625)]


@pytest.mark.parametrize("ef", [False, True])
def test_p2_hand_steps_no_decay(lib, ef):
    """eps = 0, wd = 0: u1 = lr sign(g) = 0.1 (Adam's first step)."""
    u1 = 0.1
    u2 = 0.1 * (0.28 / 0.19) / math.sqrt(0.24 / 0.0975)
    u3 = 0.1 * (0.202 / 0.271) / math.sqrt(0.2405 / 0.142625)
    if ef:
        x = [1 - u1, 1 - u1 - 2 * u2 + u1]
        x.append(x[1] - 2 * u3 + u2)
    else:
        x = [1 - u1, 1 - u1 - u2, 1 - u1 - u2 - u3]
    assert abs(u2 - 0.0939293068293407) < 1e-15   # worked by hand
    hp = HParams(lr=0.1, beta1=0.9, beta2=0.95, eps=0.0, weight_decay=0.0,
                 ef_lambda=1.0 if ef else 0.0)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, ef=ef, x_store=F64,
                                stash_store=F64, lib=lib)
    for k, (g, u) in enumerate(zip([2.0, 1.0, -0.5], [u1, u2, u3])):
        w, tag = o.read_weights("stale")
        o.step(np.array([g]), tag=tag)
        mk, vk, _, _ = _HAND_MV[k]
        assert o.m[0] == pytest.approx(mk, rel=1e-15)
        assert o.v[0] == pytest.approx(vk, rel=1e-15)
        assert o.x[0] == pytest.approx(x[k], rel=1e-14)
        if ef:
            assert o.u_prev[0] == pytest.approx(u, rel=1e-14)


@pytest.mark.parametrize("ef", [False, True])
def test_p2_hand_steps_with_decay(lib, ef):
    """wd = 0.1, eps = 1e-8: the decay term acts on the current master x_t
    (Alg. 2), not on the stale copy the gradient was evaluated at."""
    x1 = 1.0 - 0.1 * (2.0 / (2.0 + 1e-8) + 0.1 * 1.0)
    u1 = 1.0 - x1
    u2 = 0.1 * ((0.28 / 0.19) / (math.sqrt(0.24 / 0.0975) + 1e-8) + 0.1 * x1)
    x2 = x1 - 2 * u2 + u1 if ef else x1 - u2
    u3 = 0.1 * ((0.202 / 0.271) / (math.sqrt(0.2405 / 0.142625) + 1e-8) + 0.1 * x2)
    x3 = x2 - 2 * u3 + u2 if ef else x2 - u3
    hp = HParams(lr=0.1, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1,
                 ef_lambda=1.0 if ef else 0.0)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, ef=ef, x_store=F64,
                                stash_store=F64, lib=lib)
    for g, xk in zip([2.0, 1.0, -0.5], [x1, x2, x3]):
        o.step(np.array([g]), tag=o.read_weights()[1])
        assert o.x[0] == pytest.approx(xk, rel=1e-14)


# ---------------------------------------------------------------- P3 ------

@pytest.mark.parametrize("ef", [False, True])
@pytest.mark.parametrize("c", [0.3, -2.0, 3e-9])
def test_p3_constant_gradient_no_decay(lib, ef, c):
    """Constant gradient c, wd = 0: m_hat = c and v_hat = c^2 at every step,
    so u = lr c / (|c| + eps) and x_n = x_0 - n u in both modes (EF is the
    identity for a constant update: -2u + u = -u)."""
    lr, eps, n = 1e-2, 1e-8, 40
    hp = HParams(lr=lr, eps=eps, weight_decay=0.0, ef_lambda=1.0 if ef else 0.0)
    o = oracle.DelayedOptimizer([np.array([0.7])], hp, ef=ef, x_store=F64,
                                stash_store=F64, lib=lib)
    u = lr * c / (abs(c) + eps)
    for i in range(1, n + 1):
        o.step(np.array([c]))
        assert o.x[0] == pytest.approx(0.7 - i * u, rel=1e-12, abs=1e-14)


def _linear_recurrence_closed_form(coeffs, init, n):
    """Closed form of e_{j+1} = sum_i coeffs[i] e_{j-i} from the roots of its
    characteristic polynomial (distinct roots), fitted to ``init``."""
    order = len(coeffs)
    poly = np.concatenate([[1.0], -np.asarray(coeffs, dtype=float)])
    roots = np.roots(poly)
    V = np.array([[r ** j for r in roots] for j in range(order)], dtype=complex)
    amp = np.linalg.solve(V, np.asarray(init[:order], dtype=complex))
    return np.array([np.real(np.sum(amp * roots ** j)) for j in range(n)])


@pytest.mark.parametrize("ef", [False, True])
def test_p3_constant_gradient_with_decay(lib, ef):
    """Constant c, wd > 0, a = lr wd, s = c/(|c|+eps), fixed point
    x* = -s/wd. Standard: e_{n+1} = (1-a) e_n. EF: e_1 = (1-a) e_0 (first
    update is standard), then e_{n+1} = (1-2a) e_n + a e_{n-1}; its closed
    form comes from the roots of r^2 - (1-2a) r - a."""
    lr, wd, eps, c, x0, n = 0.05, 0.4, 1e-8, 0.8, 1.5, 60
    a = lr * wd
    s = c / (abs(c) + eps)
    xstar = -s / wd
    e0 = x0 - xstar
    if ef:
        e = _linear_recurrence_closed_form([1 - 2 * a, a], [e0, (1 - a) * e0], n + 1)
    else:
        e = np.array([e0 * (1 - a) ** j for j in range(n + 1)])
    hp = HParams(lr=lr, eps=eps, weight_decay=wd, ef_lambda=1.0 if ef else 0.0)
    o = oracle.DelayedOptimizer([np.array([x0])], hp, ef=ef, x_store=F64,
                                stash_store=F64, lib=lib)
    for j in range(1, n + 1):
        o.step(np.array([c]))
        assert o.x[0] - xstar == pytest.approx(e[j], rel=1e-10, abs=1e-12)


def test_p3_sign_regime_switch_is_one_call_late(lib):
    """beta1 = beta2 = 0, eps = 0, wd = 0: u = lr sign(g). On the quadratic
    a/2 (x - x*)^2 started above x*, x_n = x_0 - n lr while the gradient is
    positive. The gradient is evaluated at the stash, one version behind, so
    the first upward step comes exactly one call later than without delay."""
    lr, x0, xstar, a = 0.1, 1.0, 0.53, 2.0

    def run(delay):
        hp = HParams(lr=lr, beta1=0.0, beta2=0.0, eps=0.0, weight_decay=0.0,
                     delay=delay)
        o = oracle.DelayedOptimizer([np.array([x0])], hp, x_store=F64,
                                    stash_store=F64, lib=lib)
        xs = [x0]
        for _ in range(12):
            w, tag = o.read_weights("stale")
            g, _ = oracle.quadratic([a], [xstar], w, None, F64, lib=lib)
            o.step(g, tag=tag)
            xs.append(o.x[0])
        return np.array(xs)

    sync, delayed = run(0), run(1)
    flip = lambda xs: int(np.argmax(np.diff(xs) > 0)) + 1
    # Without delay the gradient at x_{n-1} turns negative once x_{n-1} < x*.
    k_sync = next(k for k in range(1, 20) if x0 - (k - 1) * lr < xstar)
    assert flip(sync) == k_sync
    assert flip(delayed) == k_sync + 1
    for xs, kf in ((sync, k_sync), (delayed, k_sync + 1)):
        np.testing.assert_allclose(xs[:kf], x0 - lr * np.arange(kf), rtol=0, atol=1e-14)


@pytest.mark.parametrize("ef", [False, True])
def test_p3_sgd_driver_closed_form(lib, ef):
    """Alg. 1 driver with the test-only rule u = eta g on f = a/2 x^2, so
    g_{t-1} = a x_{t-1}. Standard: x_{t+1} = x_t - eta a x_{t-1}, roots of
    r^2 - r + eta a. EF: x_{t+1} = x_t - 2 eta a x_{t-1} + eta a x_{t-2},
    roots of r^3 - r^2 + 2 eta a r - eta a. Initial values x_0 = x_1 and
    x_2 = (1 - eta a) x_0 (the first update is standard)."""
    eta, a, x0, n = 0.3, 0.25, 1.0, 50
    q = eta * a
    if ef:
        e = _linear_recurrence_closed_form([1.0, -2 * q, q], [x0, x0, (1 - q) * x0], n + 2)
    else:
        e = _linear_recurrence_closed_form([1.0, -q], [x0, x0], n + 2)
    hp = HParams(lr=eta, weight_decay=0.0, rule=oracle.RULE_SGD,
                 ef_lambda=1.0 if ef else 0.0)
    o = oracle.DelayedOptimizer([np.array([x0])], hp, ef=ef, x_store=F64,
                                stash_store=F64, lib=lib)
    for t in range(1, n + 1):
        w, tag = o.read_weights("stale")
        g, _ = oracle.quadratic([a], [0.0], w, None, F64, lib=lib)
        o.step(g, tag=tag)
        # after call t the master holds x_{t+1}
        assert o.x[0] == pytest.approx(e[t + 1], rel=1e-11, abs=1e-13)


# ---------------------------------------------------------------- P4 ------

def _random_run(lib, ef, lam, steps, store, n=257, seed=3, wd_on=None,
                shapes=None, perm=None, stash_store=None):
    rng = np.random.default_rng(seed)
    shapes = shapes or [n]
    x0 = rng.normal(0, 0.02, sum(shapes))
    grads = [rng.normal(0, 1e-3, sum(shapes)) for _ in range(steps)]
    if store == F32:
        x0 = x0.astype(np.float32).astype(np.float64)
        grads = [g.astype(np.float32).astype(np.float64) for g in grads]
    if perm is not None:
        x0 = x0[perm]
        grads = [g[perm] for g in grads]
    parts = np.split(x0, np.cumsum(shapes)[:-1])
    hp = HParams(lr=3e-4, ef_lambda=lam)
    o = oracle.DelayedOptimizer(parts, hp, ef=ef, x_store=store,
                                stash_store=stash_store or store,
                                param_store=BF16 if store == F32 else None,
                                wd_on=wd_on, lib=lib)
    hist = []
    for g in grads:
        o.step(g, tag=o.read_weights()[1])
        hist.append(dict(x=o.x.copy(), u=None if o.u_prev is None else o.u_prev.copy(),
                         stash=o.stash.copy(),
                         param=None if o.param is None else o.param.copy()))
    return o, hist


def test_p4a_ef_lambda_zero_is_standard_bitwise(lib):
    """App. A.4: lambda = 0 recovers standard delayed training."""
    _, h_std = _random_run(lib, ef=False, lam=0.0, steps=8, store=F32)
    _, h_ef0 = _random_run(lib, ef=True, lam=0.0, steps=8, store=F32)
    for a, b in zip(h_std, h_ef0):
        assert np.array_equal(a["x"], b["x"])
        assert np.array_equal(a["param"], b["param"])


@pytest.mark.parametrize("lam", [1.0, 0.5, 2.0])
def test_p4b_sapipe_restatement(lib, lam):
    """App. B.1: with p_t = x_t + lambda u_{t-2}, EF is the standard
    recursion p_{t+1} = p_t - u_{t-1}, and x_{t+1} = p_t - (1+lambda) u_{t-1}
    (for lambda = 1 these are SAPipe-WP's prediction points, whose
    displacement is Eq. (1)'s). Holds from the second update on."""
    o, hist = _random_run(lib, ef=True, lam=lam, steps=10, store=F64)
    # hist[j] is the state after call k = j + 1: x_{k+1} and u_{k-1}.
    for t in range(1, len(hist)):
        p_t = hist[t - 1]["x"] + lam * hist[t - 1]["u"]
        u = hist[t]["u"]
        p_next = hist[t]["x"] + lam * u
        np.testing.assert_allclose(p_next, p_t - u, rtol=1e-12, atol=1e-17)
        np.testing.assert_allclose(hist[t]["x"], p_t - (1 + lam) * u,
                                   rtol=1e-12, atol=1e-17)


def test_p4c_version_lag(lib):
    """Sec. 2 / Alg. 1: the gradient consumed at call k was evaluated at
    x_{k-1}, the stash; the stash after each call is the previous master
    (bitwise the previous bf16 weights when the stash is bf16)."""
    o, hist = _random_run(lib, ef=True, lam=1.0, steps=6, store=F32,
                          stash_store=BF16)
    for t in range(1, len(hist)):
        assert np.array_equal(hist[t]["stash"], hist[t - 1]["param"])
    o2, hist2 = _random_run(lib, ef=False, lam=0.0, steps=6, store=F32)
    for t in range(1, len(hist2)):
        assert np.array_equal(hist2[t]["stash"], hist2[t - 1]["x"])
    # evaluating the gradient at the latest weights instead is rejected
    latest_tag = o.read_weights("latest")[1]
    with pytest.raises(oracle.StaleVersionError):
        o.step(np.zeros(o.x.size), tag=latest_tag)
    assert o.read_weights("stale")[1] == o.k and latest_tag == o.k + 1


@pytest.mark.parametrize("lam", [0.0, 1.0, 3.0])
def test_p4d_displacement_bound(lib, lam):
    """|x_{t+1} - x_t| <= (1 + 2|lambda|) max(|u_{t-1}|, |u_{t-2}|) per
    element (the step-size bound used in App. D's proofs, for tau = 1)."""
    o, hist = _random_run(lib, ef=True, lam=lam, steps=8, store=F64)
    for t in range(1, len(hist)):
        d = np.abs(hist[t]["x"] - hist[t - 1]["x"])
        bound = (1 + 2 * abs(lam)) * np.maximum(np.abs(hist[t]["u"]), np.abs(hist[t - 1]["u"]))
        assert np.all(d <= bound * (1 + 1e-12) + 1e-300)


def test_p4e_permutation_and_split_invariance(lib):
    """The step is elementwise: permuting elements or splitting them into
    tensors differently leaves every value unchanged (clipping off)."""
    n = 300
    perm = np.random.default_rng(0).permutation(n)
    _, h_a = _random_run(lib, ef=True, lam=1.0, steps=5, store=F32, n=n)
    _, h_b = _random_run(lib, ef=True, lam=1.0, steps=5, store=F32, n=n,
                         perm=perm)
    _, h_c = _random_run(lib, ef=True, lam=1.0, steps=5, store=F32,
                         shapes=[1, 150, 7, 142])
    for a, b, c in zip(h_a, h_b, h_c):
        assert np.array_equal(a["x"][perm], b["x"])
        assert np.array_equal(a["x"], c["x"])


def test_weight_decay_mask(lib):
    """A tensor with decay switched off takes the wd = 0 update."""
    rng = np.random.default_rng(5)
    x0 = [rng.normal(0, 1, 4), rng.normal(0, 1, 3)]
    g = rng.normal(0, 1, 7)
    hp = HParams(lr=0.01, weight_decay=0.5)
    o = oracle.DelayedOptimizer(x0, hp, x_store=F64, stash_store=F64,
                                wd_on=[True, False], lib=lib)
    o.step(g)
    ref_on = _torch_adamw_run([x0[0]], [[g[:4]]], hp, [0.01])[0]
    ref_off = _torch_adamw_run([x0[1]], [[g[4:]]],
                               HParams(lr=0.01, weight_decay=0.0), [0.01])[0]
    assert _rel(o.x[:4], ref_on) < 1e-13
    assert _rel(o.x[4:], ref_off) < 1e-13


# ------------------------------------------------------------- storage ----

def test_bf16_rounding_matches_torch(lib):
    """The oracle's own bf16 rounding equals torch's fp32 -> bf16 cast
    (round to nearest even) on ties, subnormals, overflow and random values."""
    rng = np.random.default_rng(1)
    vals = [rng.normal(0, s, 4000).astype(np.float32) for s in (1e-3, 1.0, 1e30)]
    bits = np.arange(0, 1 << 16, 7, dtype=np.uint32)
    ties = ((bits << 16) | 0x8000).view(np.float32)      # exactly halfway
    near = ((bits << 16) | 0x7FFF).view(np.float32)
    tiny = (np.arange(1, 3000, dtype=np.uint32)).view(np.float32)  # subnormals
    big = np.array([3.3895e38, 3.39e38, -3.4028235e38, 65504.0], np.float32)
    x = np.concatenate(vals + [ties, near, tiny, big])
    x = x[np.isfinite(x)]
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = oracle.round_to(x.astype(np.float64), BF16, lib=lib)
    np.testing.assert_array_equal(got, ref)


def test_f32_rounding_matches_numpy(lib):
    x = np.random.default_rng(2).normal(0, 1, 1000) * 10.0 ** np.random.default_rng(3).integers(-40, 38, 1000)
    np.testing.assert_array_equal(oracle.round_to(x, F32, lib=lib),
                                  x.astype(np.float32).astype(np.float64))


def test_sqnorm_and_clip(lib):
    rng = np.random.default_rng(4)
    g = rng.normal(0, 1, 200_001)
    ref = math.fsum(v * v for v in g)
    assert oracle.sqnorm(g, lib=lib) == pytest.approx(ref, rel=1e-13)
    g32 = g.astype(np.float32)
    assert oracle.sqnorm_f32(g32, lib=lib) == pytest.approx(
        math.fsum(float(v) ** 2 for v in g32), rel=1e-13)
    gb = torch.from_numpy(g32).to(torch.bfloat16)
    bits = gb.view(torch.int16).numpy().view(np.uint16)
    assert oracle.sqnorm_bf16(bits, lib=lib) == pytest.approx(
        math.fsum(float(v) ** 2 for v in gb.double().numpy()), rel=1e-13)
    assert oracle.clip_coef(4.0, 1.0, lib=lib) == pytest.approx(1.0 / (2.0 + 1e-6), rel=1e-15)
    assert oracle.clip_coef(0.25, 1.0, lib=lib) == 1.0
    assert oracle.clip_coef(4.0, 0.0, lib=lib) == 1.0


def test_clip_nonfinite_norm_like_torch(lib):
    """A NaN gradient makes every clipped element NaN and an infinite norm
    zeroes the finite ones, as torch.nn.utils.clip_grad_norm_ does."""
    for bad in (float("nan"), float("inf")):
        g = np.array([0.5, bad, -2.0])
        p = torch.nn.Parameter(torch.zeros(3, dtype=torch.float64))
        p.grad = torch.tensor(g)
        torch.nn.utils.clip_grad_norm_([p], 1.0)
        coef = oracle.clip_coef(oracle.sqnorm(g, lib=lib), 1.0, lib=lib)
        with np.errstate(invalid="ignore"):   # 0 * inf is NaN on purpose
            np.testing.assert_array_equal(coef * g, p.grad.numpy())



def test_clip_from_a_supplied_norm(lib):
    """Global clipping (App. E.1): two oracles over the halves of a set, each
    given the squared norm over the whole gradient, take torch's
    clip_grad_norm_ coefficient over the whole set and step exactly as one
    oracle over the set, bitwise."""
    rng = np.random.default_rng(12)
    x0 = [rng.normal(0, 1, 300), rng.normal(0, 1, 217)]
    hp = HParams(lr=0.01, weight_decay=0.1, max_grad_norm=1.0, ef_lambda=1.0)
    full = oracle.DelayedOptimizer(x0, hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    halves = [oracle.DelayedOptimizer([x], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
              for x in x0]
    for _ in range(4):
        g = rng.normal(0, 0.2, 517)
        params = [torch.nn.Parameter(torch.zeros(n, dtype=torch.float64)) for n in (300, 217)]
        params[0].grad, params[1].grad = torch.tensor(g[:300]), torch.tensor(g[300:])
        torch.nn.utils.clip_grad_norm_(params, 1.0)
        coef = float(params[0].grad[0] / g[0])
        assert coef < 0.5   # clipping is active
        sq = oracle.sqnorm(g, lib=lib)
        full.step(g)
        halves[0].step(g[:300], sq=sq)
        halves[1].step(g[300:], sq=sq)
        for o in [full] + halves:
            assert o.last_clip == pytest.approx(coef, rel=1e-13)
        assert np.array_equal(np.concatenate([h.x for h in halves]), full.x)

def test_quadratic_gradient_is_loss_derivative(lib):
    """grad = d loss / dw (central differences) when the noise is zero."""
    rng = np.random.default_rng(6)
    n = 20
    a = np.exp(rng.uniform(np.log(1e-3), 0, n))
    ws, w = rng.normal(0, 1, n), rng.normal(0, 1, n)
    g, loss = oracle.quadratic(a, ws, w, None, F64, lib=lib)
    h = 1e-6
    for i in range(n):
        e = np.zeros(n)
        e[i] = h
        lp = oracle.quadratic(a, ws, w + e, None, F64, lib=lib)[1]
        lm = oracle.quadratic(a, ws, w - e, None, F64, lib=lib)[1]
        assert g[i] == pytest.approx((lp - lm) / (2 * h), rel=1e-6, abs=1e-9)
    assert loss == pytest.approx(0.5 * np.sum(a * (w - ws) ** 2), rel=1e-14)


def test_quadratic_noise_enters_the_gradient(lib):
    """With a noise sample, the harness's gradient is the loss derivative
    (central differences, the noise is not part of the loss) plus that
    sample: the stale-gradient noise of the quadratic workload."""
    rng = np.random.default_rng(16)
    n = 12
    a = np.exp(rng.uniform(np.log(1e-3), 0, n))
    ws, w, noise = rng.normal(0, 1, n), rng.normal(0, 1, n), rng.normal(0, 1e-2, n)
    g, _ = oracle.quadratic(a, ws, w, noise, F64, lib=lib)
    h = 1e-6
    for i in range(n):
        e = np.zeros(n)
        e[i] = h
        lp = oracle.quadratic(a, ws, w + e, None, F64, lib=lib)[1]
        lm = oracle.quadratic(a, ws, w - e, None, F64, lib=lib)[1]
        assert g[i] - (lp - lm) / (2 * h) == pytest.approx(noise[i], abs=1e-8)


@pytest.mark.parametrize("store", [F32, BF16])
def test_quadratic_gradient_in_its_storage_format(lib, store):
    """The harness's gradient is delivered in the gradient's storage format
    (the dtype the step consumes)."""
    rng = np.random.default_rng(17)
    n = 200
    a = np.exp(rng.uniform(np.log(1e-3), 0, n))
    g, _ = oracle.quadratic(a, rng.normal(0, 1, n), rng.normal(0, 1, n),
                            rng.normal(0, 1e-2, n), store, lib=lib)
    assert _fp32_exact(g)
    if store == BF16:
        assert _bf16_exact(g)


# ------------------------------------------------------- SAPipe-WP (App. B.1)

def _fixed_grad_run(lib, correction, steps=8, wd=0.1, ef=True, lam=1.0, beta=(0.9, 0.95),
                    eps=1e-8, n=64, seed=21, max_norm=0.0):
    rng = np.random.default_rng(seed)
    x0 = rng.normal(0, 0.5, n)
    grads = [rng.normal(0, 1.0, n) for _ in range(steps)]
    hp = HParams(lr=0.01, beta1=beta[0], beta2=beta[1], eps=eps, weight_decay=wd,
                 ef_lambda=lam, correction=correction, max_grad_norm=max_norm)
    o = oracle.DelayedOptimizer([x0], hp, ef=ef, x_store=F64, stash_store=F64, lib=lib)
    hist = []
    for g in grads:
        o.step(g, tag=o.read_weights()[1])
        hist.append(dict(x=o.x.copy(), stash=o.stash.copy(), u=o.u_prev.copy() if ef else None,
                         m=o.m.copy(), v=o.v.copy()))
    return hist, grads, x0, hp


def test_sapipe_same_weights_follow_the_standard_rule(lib):
    """SAPipe-WP changes only where the next gradient is evaluated: the
    weights take the standard delayed update, bitwise."""
    h_sp, _, _, _ = _fixed_grad_run(lib, oracle.CORR_SAPIPE_SAME)
    h_std, _, _, _ = _fixed_grad_run(lib, oracle.CORR_EF, ef=False)
    for a, b in zip(h_sp, h_std):
        assert np.array_equal(a["x"], b["x"])


def test_sapipe_same_prediction_points_move_like_ef(lib):
    """App. B.1: the displacement between consecutive SAPipe prediction points
    is -2 u(g_{t-1}) + u(g_{t-2}), Eq. (1)'s. Checked against the identity and
    against an EF run's weight displacement on the same gradient sequence
    (wd = 0, so both runs form the same updates)."""
    h_sp, _, _, _ = _fixed_grad_run(lib, oracle.CORR_SAPIPE_SAME, wd=0.0)
    h_ef, _, _, _ = _fixed_grad_run(lib, oracle.CORR_EF, wd=0.0)
    for j in range(1, len(h_sp)):
        u_prev = h_sp[j - 1]["u"]
        u_prev2 = h_sp[j - 2]["u"] if j >= 2 else 0.0
        d_stash = h_sp[j]["stash"] - h_sp[j - 1]["stash"]
        np.testing.assert_allclose(d_stash, -2 * u_prev + u_prev2, rtol=1e-11, atol=1e-15)
        if j >= 2:   # the EF weights take the same displacement one call earlier
            d_ef = h_ef[j - 1]["x"] - h_ef[j - 2]["x"]
            np.testing.assert_allclose(d_stash, d_ef, rtol=1e-11, atol=1e-15)


@pytest.mark.parametrize("max_norm", [0.0, 3.0])
def test_sapipe_updated_prediction_is_adamw_stepped_again(lib, max_norm):
    """The updated-state prediction update is what torch.optim.AdamW applies
    when stepped once more on the same gradient from the state its real step
    left (then discarded); with clipping (norms about 8 against 3), on the
    same clipped gradient the real step consumed."""
    hist, grads, x0, hp = _fixed_grad_run(lib, oracle.CORR_SAPIPE_UPDATED, max_norm=max_norm)
    clip = lambda g: g * (min(1.0, max_norm / (np.sqrt(np.sum(g * g)) + 1e-6))
                          if max_norm > 0 else 1.0)
    grads = [clip(g) for g in grads]
    p = torch.nn.Parameter(torch.tensor(x0))
    opt = torch.optim.AdamW([p], lr=hp.lr, betas=(hp.beta1, hp.beta2), eps=hp.eps,
                            weight_decay=hp.weight_decay, foreach=False, fused=False)
    for k, g in enumerate(grads):
        p.grad = torch.tensor(g)
        opt.step()
        np.testing.assert_allclose(p.detach().numpy(), hist[k]["x"], rtol=1e-12)
        # prediction: one more step on the same gradient from a copy of the state
        q = torch.nn.Parameter(p.detach().clone())
        opt2 = torch.optim.AdamW([q], lr=hp.lr, betas=(hp.beta1, hp.beta2), eps=hp.eps,
                                 weight_decay=hp.weight_decay, foreach=False, fused=False)
        st = opt.state[p]
        opt2.state[q] = {"step": st["step"].clone(), "exp_avg": st["exp_avg"].clone(),
                         "exp_avg_sq": st["exp_avg_sq"].clone()}
        q.grad = torch.tensor(g)
        opt2.step()
        u_pred = p.detach().numpy() - q.detach().numpy()
        np.testing.assert_allclose(hist[k]["u"], u_pred, rtol=1e-10, atol=1e-16)
        # the next forward reads the previous prediction point
        if k >= 1:
            np.testing.assert_allclose(hist[k]["stash"], hist[k - 1]["x"] - hist[k - 1]["u"],
                                       rtol=1e-13)


def test_sapipe_updated_equals_same_when_adam_is_memoryless(lib):
    """beta1 = beta2 = 0, eps = 0, wd = 0: every Adam update is lr sign(g),
    so recomputing it from the updated state changes nothing."""
    kw = dict(wd=0.0, beta=(0.0, 0.0), eps=0.0)
    h_u, _, _, _ = _fixed_grad_run(lib, oracle.CORR_SAPIPE_UPDATED, **kw)
    h_s, _, _, _ = _fixed_grad_run(lib, oracle.CORR_SAPIPE_SAME, **kw)
    for a, b in zip(h_u, h_s):
        for key in ("x", "stash", "u"):
            assert np.array_equal(a[key], b[key])


def test_sapipe_updated_hand_steps(lib):
    """x0 = 1, beta = (0.9, 0.95), eps = 0, wd = 0, lr = 0.1, gradients 2, 1.
    Call 1: m = 0.2, v = 0.2, u = 0.1; prediction from m' = 0.38, v' = 0.39
    at k = 2 (1 - b1^2 = 0.19, 1 - b2^2 = 0.0975): m_hat = 2, v_hat = 4, so 0.1.
    Call 2: stash = x_2 - 0.1 = 0.8; u = 0.1 (0.28/0.19) / sqrt(0.24/0.0975);
    prediction from m' = 0.352, v' = 0.278 at k = 3 (0.271, 0.142625)."""
    hp = HParams(lr=0.1, beta1=0.9, beta2=0.95, eps=0.0, weight_decay=0.0,
                 correction=oracle.CORR_SAPIPE_UPDATED)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, ef=True, x_store=F64, stash_store=F64,
                                lib=lib)
    o.step(np.array([2.0]), tag=o.read_weights()[1])
    assert o.stash[0] == 1.0 and o.x[0] == pytest.approx(0.9, rel=1e-15)
    assert o.u_prev[0] == pytest.approx(0.1, rel=1e-15)
    o.step(np.array([1.0]), tag=o.read_weights()[1])
    assert o.stash[0] == pytest.approx(0.8, rel=1e-15)
    u2 = 0.1 * (0.28 / 0.19) / math.sqrt(0.24 / 0.0975)
    assert o.x[0] == pytest.approx(0.9 - u2, rel=1e-14)
    assert o.u_prev[0] == pytest.approx(0.1 * (0.352 / 0.271) / math.sqrt(0.278 / 0.142625),
                                        rel=1e-14)


def _rule_run(lib, rule, correction, grads, x0, ef=True, max_norm=0.0, store=F64, **kw):
    hp = HParams(lr=kw.pop("lr", 0.01), weight_decay=kw.pop("wd", 0.1), rule=rule,
                 correction=correction, max_grad_norm=max_norm, **kw)
    o = oracle.DelayedOptimizer([x0], hp, ef=ef, x_store=store, stash_store=store, lib=lib)
    hist = []
    for g in grads:
        o.step(g, tag=o.read_weights()[1])
        hist.append(dict(x=o.x.copy(), stash=o.stash.copy(),
                         u=o.u_prev.copy() if ef else None))
    return hist


RULE_KW = {oracle.RULE_ADAMW: {}, oracle.RULE_NADAM: dict(momentum_decay=0.004),
           oracle.RULE_LION: dict(beta1=0.9, beta2=0.99),
           oracle.RULE_ADAN: dict(beta1=0.98, beta2=0.92, beta3=0.99),
           oracle.RULE_SGD: {}}


@pytest.mark.parametrize("rule", sorted(RULE_KW))
@pytest.mark.parametrize("max_norm,store", [(0.0, F64), (3.0, F64), (0.0, F32)])
def test_sapipe_updated_prediction_is_the_next_step_on_a_repeated_gradient(lib, rule, max_norm,
                                                                          store):
    """App. B.1's updated-state prediction is the optimizer's own step taken
    once more on the same gradient from the state the real step left: for
    every rule, the prediction update stored after call k equals, bitwise,
    the update stored by call k + 1 of a run whose gradient k + 1 repeats
    gradient k. That run is EF at lambda = 0, which is the standard rule
    bitwise and keeps each update in its history buffer; the SAPipe run's
    weights follow the standard rule too, so both runs start call k + 1 from
    the same stored state. With clipping (norms about 8 against 3) the
    repeated gradient takes the same coefficient; with fp32 storage the
    prediction reads the statistics as stored."""
    rng = np.random.default_rng(31)
    n, steps = 48, 6
    x0 = rng.normal(0, 0.5, n)
    grads = [rng.normal(0, 1.0, n) for _ in range(steps)]
    sp = _rule_run(lib, rule, oracle.CORR_SAPIPE_UPDATED, grads, x0, max_norm=max_norm,
                   store=store, **RULE_KW[rule])
    for k in range(1, steps + 1):
        rep = _rule_run(lib, rule, oracle.CORR_EF, grads[:k] + [grads[k - 1]], x0,
                        max_norm=max_norm, store=store, ef_lambda=0.0, **RULE_KW[rule])
        np.testing.assert_array_equal(sp[k - 1]["x"], rep[k - 1]["x"])
        np.testing.assert_array_equal(sp[k - 1]["u"], rep[k]["u"])


@pytest.mark.parametrize("max_norm", [0.0, 1.5])
def test_sapipe_updated_nadam_is_torch_nadam_stepped_again(lib, f64_default, max_norm):
    """NAdam's prediction update is what torch.optim.NAdam (decoupled decay)
    applies when stepped once more on the same (clipped) gradient from a copy
    of the state its real step left: moments, step count and the running
    product of its momentum schedule."""
    rng = np.random.default_rng(33)
    x0 = rng.normal(0, 0.5, 40)
    grads = [rng.normal(0, 0.7, 40) for _ in range(7)]
    hist = _rule_run(lib, oracle.RULE_NADAM, oracle.CORR_SAPIPE_UPDATED, grads, x0,
                     max_norm=max_norm, lr=2e-2, momentum_decay=0.004)
    kw = dict(lr=2e-2, betas=(0.9, 0.95), eps=1e-8, weight_decay=0.1, momentum_decay=0.004,
              decoupled_weight_decay=True, foreach=False)
    p = torch.nn.Parameter(torch.tensor(x0))
    opt = torch.optim.NAdam([p], **kw)
    for k, g in enumerate(grads):
        p.grad = torch.tensor(g)
        if max_norm > 0:
            torch.nn.utils.clip_grad_norm_([p], max_norm)
        gc = p.grad.clone()
        opt.step()
        np.testing.assert_allclose(p.detach().numpy(), hist[k]["x"], rtol=1e-12)
        q = torch.nn.Parameter(p.detach().clone())
        opt2 = torch.optim.NAdam([q], **kw)
        opt2.state[q] = {key: val.clone() for key, val in opt.state[p].items()}
        q.grad = gc
        opt2.step()
        np.testing.assert_allclose(hist[k]["u"], p.detach().numpy() - q.detach().numpy(),
                                   rtol=1e-10, atol=1e-16)


def test_sapipe_updated_lion_hand_steps(lib):
    """Lion, beta = (0.5, 0.5), lr = 0.1, wd = 0, x0 = 1, gradients -2, 0.5, 0.5.
    Call 1: c = -1 (u = -0.1, x = 1.1), m = -1; prediction c' = 0.5(-1) +
    0.5(-2) = -1.5, so -0.1. Call 2: c = -0.25 (u = -0.1, x = 1.2), m = -0.25;
    prediction c' = -0.125 + 0.25 = 0.125, so +0.1: the updated state flips
    the sign the same state would keep. Call 3 reads the stash
    x_3 - u'_2 = 1.2 - 0.1 = 1.1 (same state: 1.3)."""
    hist = _rule_run(lib, oracle.RULE_LION, oracle.CORR_SAPIPE_UPDATED,
                     [np.array([-2.0]), np.array([0.5]), np.array([0.5])], np.array([1.0]),
                     lr=0.1, wd=0.0, beta1=0.5, beta2=0.5)
    assert [h["x"][0] for h in hist[:2]] == pytest.approx([1.1, 1.2], abs=1e-15)
    assert [h["u"][0] for h in hist[:2]] == pytest.approx([-0.1, 0.1], abs=1e-15)
    assert hist[1]["stash"][0] == pytest.approx(1.2, abs=1e-15)
    assert hist[2]["stash"][0] == pytest.approx(1.1, abs=1e-15)


def test_sapipe_updated_adan_hand_steps(lib):
    """Adan, beta = (0.98, 0.92, 0.99), lr = 0.1, eps = 0, wd = 0, x0 = 1,
    gradients 2, then 1. Call 1: m = 0.04, v = 0 (no difference yet),
    n = 0.04, u = 0.1; the prediction at k = 2 (difference 0: the stored
    previous gradient is 2 itself) from m' = 0.0792, v' = 0, n' = 0.0796 is
    0.1 (0.0792/0.0396) / sqrt(0.0796/0.0199) = 0.1. Call 2: diff = -1,
    m = 0.0592, v = -0.08, n = 0.039664; prediction at k = 3 from
    m' = 0.078016, v' = 0.92(-0.08) = -0.0736, n' = 0.04926736 with
    1 - beta^3 = 0.058808, 0.221312, 0.029701."""
    hist = _rule_run(lib, oracle.RULE_ADAN, oracle.CORR_SAPIPE_UPDATED,
                     [np.array([2.0]), np.array([1.0])], np.array([1.0]), lr=0.1, wd=0.0,
                     eps=0.0, beta1=0.98, beta2=0.92, beta3=0.99)
    assert hist[0]["u"][0] == pytest.approx(0.1, rel=1e-14)
    pred2 = 0.1 * ((0.078016 / 0.058808 + 0.92 * -0.0736 / 0.221312) /
                   math.sqrt(0.04926736 / 0.029701))
    assert hist[1]["u"][0] == pytest.approx(pred2, rel=1e-12)
    # the real second update, for contrast (1 - beta^2 = 0.0396, 0.1536, 0.0199)
    u2 = 0.1 * ((0.0592 / 0.0396 + 0.92 * -0.08 / 0.1536) / math.sqrt(0.039664 / 0.0199))
    assert hist[1]["x"][0] == pytest.approx(0.9 - u2, rel=1e-13)


# ------------------------------- per-tensor delay and mode switches (Sec. 3.1,
# App. A.9 synchronous LM head, App. B.2 WPipe)

def _sgd_quadratic_run(lib, a, x0, steps, ef=False, delayed=None, schedule=None, eta=0.3):
    """Alg. 1 driver, SGD rule, on f = sum a_i/2 x_i^2; ``schedule[c]`` is the
    delay mode to switch to before call c (1-based)."""
    hp = HParams(lr=eta, weight_decay=0.0, rule=oracle.RULE_SGD, ef_lambda=1.0 if ef else 0.0,
                 delay=(schedule or {}).get(0, 1))
    o = oracle.DelayedOptimizer([np.array([v]) for v in x0], hp, ef=ef, x_store=F64,
                                stash_store=F64, delayed=delayed, lib=lib)
    xs = [o.x.copy()]
    for c in range(1, steps + 1):
        if schedule and c in schedule:
            o.set_delay(schedule[c])
        w, tag = o.read_weights("stale")
        g, _ = oracle.quadratic(a, [0.0] * len(a), w, None, F64, lib=lib)
        o.step(g, tag=tag)
        xs.append(o.x.copy())
    return np.array(xs)


def _alg1_closed_form(q, x_start, n, ef):
    """Alg. 1 from x_0 = x_1 = x_start with u = eta g on a/2 x^2 (q = eta a):
    element j of the result is x_j."""
    if ef:
        return _linear_recurrence_closed_form([1.0, -2 * q, q],
                                              [x_start, x_start, (1 - q) * x_start], n)
    return _linear_recurrence_closed_form([1.0, -q], [x_start, x_start], n)


def test_per_tensor_delay_sync_and_delayed_side_by_side(lib):
    """One run, two tensors: the synchronous one decays geometrically,
    x_{t+1} = (1 - q) x_t, the delayed one follows Alg. 1's recurrence."""
    a, x0, n, eta = [0.25, 0.5], [1.0, -2.0], 30, 0.3
    xs = _sgd_quadratic_run(lib, a, x0, n, delayed=[True, False], eta=eta)
    q0, q1 = eta * a[0], eta * a[1]
    e0 = _alg1_closed_form(q0, x0[0], n + 2, ef=False)
    for c in range(1, n + 1):
        assert xs[c][0] == pytest.approx(e0[c + 1], rel=1e-11, abs=1e-13)
        assert xs[c][1] == pytest.approx(x0[1] * (1 - q1) ** c, rel=1e-11, abs=1e-13)


@pytest.mark.parametrize("ef", [False, True])
def test_synchronous_start_then_delay(lib, ef):
    """S synchronous steps, then delayed training (Sec. 3.1): geometric
    decay, then Alg. 1 restarted from the switch point (its first delayed
    call uses the standard rule even under EF)."""
    a, x0, S, n, eta = [0.25], [1.0], 5, 25, 0.3
    q = eta * a[0]
    xs = _sgd_quadratic_run(lib, a, x0, S + n, ef=ef, schedule={0: 0, S + 1: 1}, eta=eta)
    for c in range(1, S + 1):
        assert xs[c][0] == pytest.approx((1 - q) ** c, rel=1e-12)
    xS = (1 - q) ** S
    e = _alg1_closed_form(q, xS, n + 2, ef)
    for j in range(1, n + 1):   # call S + j leaves x_{j+1} of the restarted run
        assert xs[S + j][0] == pytest.approx(e[j + 1], rel=1e-10, abs=1e-13)


@pytest.mark.parametrize("ef", [False, True])
def test_synchronous_cooldown(lib, ef):
    """Delayed training, then synchronous from call D + 1 (App. A.10): Alg. 1,
    then geometric decay from the weights reached."""
    a, x0, D, n, eta = [0.25], [1.0], 12, 10, 0.3
    q = eta * a[0]
    xs = _sgd_quadratic_run(lib, a, x0, D + n, ef=ef, schedule={D + 1: 0}, eta=eta)
    e = _alg1_closed_form(q, x0[0], D + 2, ef)
    for c in range(1, D + 1):
        assert xs[c][0] == pytest.approx(e[c + 1], rel=1e-10, abs=1e-13)
    for j in range(1, n + 1):
        assert xs[D + j][0] == pytest.approx(xs[D][0] * (1 - q) ** j, rel=1e-11, abs=1e-14)


def test_per_tensor_delay_is_elementwise(lib):
    """With fixed gradients, a mixed table equals, tensor by tensor, an
    all-delayed run and an all-synchronous run (bitwise)."""
    rng = np.random.default_rng(8)
    sizes = [13, 7, 21]
    x0 = [rng.normal(0, 0.5, s) for s in sizes]
    grads = [rng.normal(0, 1.0, sum(sizes)) for _ in range(6)]

    def run(delayed, delay):
        hp = HParams(lr=0.01, ef_lambda=1.0, delay=delay)
        o = oracle.DelayedOptimizer(x0, hp, ef=True, x_store=F32, stash_store=F32,
                                    delayed=delayed, lib=lib)
        for g in grads:
            o.step(g)
        return o

    mixed = run([True, False, True], 1)
    all_d, all_s = run(None, 1), run(None, 0)
    for i, ref in ((0, all_d), (1, all_s), (2, all_d)):
        for name in ("x", "m", "v"):
            assert np.array_equal(mixed.tensor(name, i), ref.tensor(name, i))
    assert np.array_equal(mixed.tensor("stash", 0), all_d.tensor("stash", 0))
    assert np.array_equal(mixed.tensor("u_prev", 2), all_d.tensor("u_prev", 2))
    assert np.array_equal(mixed.tensor("u_prev", 1), np.zeros(7))   # history untouched


# ------------------- other elementwise optimizers under delay (Tab. main_results)

@pytest.fixture
def f64_default():
    """torch keeps NAdam's running product of mu in the default scalar dtype:
    make it fp64 for the duration of a test."""
    prev = torch.get_default_dtype()
    torch.set_default_dtype(torch.float64)
    try:
        yield
    finally:
        torch.set_default_dtype(prev)


@pytest.mark.parametrize("delay", [0, 1])
@pytest.mark.parametrize("psi,max_norm", [(0.004, 0.0), (0.02, 0.0), (0.004, 1.5)])
def test_nadam_matches_torch(lib, f64_default, delay, psi, max_norm):
    """NAdam = torch.optim.NAdam with decoupled weight decay, including its
    momentum schedule mu_k = beta1 (1 - 0.5 * 0.96^(k psi)), changing lr."""
    rng = np.random.default_rng(12)
    shapes = [(4, 3), (5,)]
    x0s = [rng.normal(0, 0.5, s) for s in shapes]
    grads = [[rng.normal(0, 0.7, s) for s in shapes] for _ in range(10)]
    lrs = [2e-2 * (1 + 0.05 * i) for i in range(10)]
    ps = [torch.nn.Parameter(torch.tensor(x)) for x in x0s]
    opt = torch.optim.NAdam(ps, lr=lrs[0], betas=(0.9, 0.95), eps=1e-8, weight_decay=0.1,
                            momentum_decay=psi, decoupled_weight_decay=True, foreach=False)
    hp = HParams(lr=lrs[0], weight_decay=0.1, delay=delay, rule=oracle.RULE_NADAM,
                 momentum_decay=psi, max_grad_norm=max_norm)
    o = oracle.DelayedOptimizer(x0s, hp, x_store=F64, stash_store=F64, lib=lib)
    for gs, lr in zip(grads, lrs):
        for p, g in zip(ps, gs):
            p.grad = torch.tensor(g)
        if max_norm > 0:   # the clipped gradient enters every term
            torch.nn.utils.clip_grad_norm_(ps, max_norm)
        for group in opt.param_groups:
            group["lr"] = lr
        opt.step()
        o.step(np.concatenate([g.ravel() for g in gs]), lr=lr)
        ref = np.concatenate([p.detach().numpy().ravel() for p in ps])
        assert _rel(o.x, ref) < 1e-12


def test_lion_hand_steps(lib):
    """Lion, beta = (0.9, 0.99), lr = 0.1, wd = 0, gradients 2, -1, 0.05:
    c1 = 0.1*2 = 0.2 (+), m1 = 0.01*2 = 0.02;
    c2 = 0.9*0.02 + 0.1*(-1) = -0.082 (-), m2 = 0.99*0.02 + 0.01*(-1) = 0.0098;
    c3 = 0.9*0.0098 + 0.1*0.05 = 0.01382 (+). With the coefficients' roles
    swapped the second step would move up, not down."""
    hp = HParams(lr=0.1, beta1=0.9, beta2=0.99, weight_decay=0.0, rule=oracle.RULE_LION)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    xs = []
    for g in (2.0, -1.0, 0.05):
        o.step(np.array([g]), tag=o.read_weights()[1])
        xs.append(o.x[0])
    assert xs == pytest.approx([0.9, 1.0, 0.9], abs=1e-15)
    assert o.m[0] == pytest.approx(0.99 * 0.0098 + 0.01 * 0.05, rel=1e-14)


def test_lion_moves_every_weight_by_exactly_lr(lib):
    """A sign update: |x_{t+1} - (1 - lr wd) x_t| = lr for every element
    whose interpolation c is non-zero, whatever the gradient scale."""
    rng = np.random.default_rng(13)
    x0 = rng.normal(0, 1, 200)
    hp = HParams(lr=3e-3, beta1=0.9, beta2=0.99, weight_decay=0.5, rule=oracle.RULE_LION)
    o = oracle.DelayedOptimizer([x0], hp, x_store=F64, stash_store=F64, lib=lib)
    for s in (1e-6, 1.0, 1e3):
        x = o.x.copy()
        o.step(rng.normal(0, s, 200))
        np.testing.assert_allclose(np.abs(o.x - (1 - 3e-3 * 0.5) * x), 3e-3, rtol=1e-12)


def test_adan_first_step_is_adams(lib):
    """At the first gradient diff = 0 and the bias-corrected moments are g and
    g^2: Adan's update is Adam's first step lr (g / (|g| + eps) + wd x)."""
    rng = np.random.default_rng(14)
    x0, g = rng.normal(0, 1, 50), rng.normal(0, 1, 50)
    hp = HParams(lr=0.01, beta1=0.98, beta2=0.92, beta3=0.99, eps=1e-8, weight_decay=0.1,
                 rule=oracle.RULE_ADAN)
    o = oracle.DelayedOptimizer([x0], hp, x_store=F64, stash_store=F64, lib=lib)
    o.step(g)
    np.testing.assert_allclose(o.x, x0 - 0.01 * (g / (np.abs(g) + 1e-8) + 0.1 * x0), rtol=1e-13)


def test_adan_constant_gradient_closed_form(lib):
    """Constant gradient c: diff = 0, so u = lr (c / (|c| + eps) + wd x) and
    x_n - x* = (x_0 - x*) (1 - lr wd)^n with x* = -c / ((|c| + eps) wd)."""
    lr, wd, eps, c, x0 = 0.05, 0.4, 1e-8, -0.7, 1.5
    xstar = -(c / (abs(c) + eps)) / wd
    hp = HParams(lr=lr, beta1=0.98, beta2=0.92, beta3=0.99, eps=eps, weight_decay=wd,
                 rule=oracle.RULE_ADAN)
    o = oracle.DelayedOptimizer([np.array([x0])], hp, x_store=F64, stash_store=F64, lib=lib)
    for j in range(1, 40):
        o.step(np.array([c]))
        assert o.x[0] - xstar == pytest.approx((x0 - xstar) * (1 - lr * wd) ** j, rel=1e-10)


def test_adan_hand_steps(lib):
    """beta = (0.98, 0.92, 0.99), eps = 0, wd = 0, lr = 0.1, gradients 2, 1.
    Step 1: u = 0.1 (Adam's first step). Step 2: diff = -1, m = 0.0592,
    v = -0.08, w = 1 - 0.92 = 0.08, n = 0.99*0.04 + 0.01*0.0064 = 0.039664;
    u = 0.1 (0.0592/0.0396 - 0.92*0.08/0.1536) / sqrt(0.039664/0.0199)."""
    hp = HParams(lr=0.1, beta1=0.98, beta2=0.92, beta3=0.99, eps=0.0, weight_decay=0.0,
                 rule=oracle.RULE_ADAN)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    o.step(np.array([2.0]), tag=o.read_weights()[1])
    assert o.x[0] == pytest.approx(0.9, rel=1e-14)
    o.step(np.array([1.0]), tag=o.read_weights()[1])
    u2 = 0.1 * (0.0592 / 0.0396 - 0.92 * 0.08 / 0.1536) / math.sqrt(0.039664 / 0.0199)
    assert o.x[0] == pytest.approx(0.9 - u2, rel=1e-13)
    assert o.v[0] == pytest.approx(-0.08, rel=1e-14)
    assert o.n3[0] == pytest.approx(0.039664, rel=1e-14)


def test_dc_asgd_compensation(lib):
    """DC-ASGD (Sec. 3.1): g~ = g + lambda g^2 (x_t - x_stale), the stale
    weights being the stash the gradient came from. With beta1 = 0 the first
    moment is exactly g~. At the first call the stash equals x_t (no
    correction); lambda = 0 is the plain rule bitwise."""
    lam = 50.0
    hp = HParams(lr=0.1, beta1=0.0, beta2=0.95, eps=1e-8, weight_decay=0.0, dc_lambda=lam)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    o.step(np.array([2.0]), tag=o.read_weights()[1])
    assert o.m[0] == 2.0
    x2, x1 = o.x[0], o.stash[0]
    o.step(np.array([1.0]), tag=o.read_weights()[1])
    assert o.m[0] == pytest.approx(1.0 + lam * 1.0 * (x2 - x1), rel=1e-14)
    assert x1 == 1.0 and x2 < 1.0
    # a gradient of magnitude other than 1, and negative: the term is g^2,
    # not |g| or g |g|
    x3, x2s = o.x[0], o.stash[0]
    o.step(np.array([-3.0]), tag=o.read_weights()[1])
    assert o.m[0] == pytest.approx(-3.0 + lam * 9.0 * (x3 - x2s), rel=1e-14)
    assert x3 != x2s
    # lambda = 0: identical to the plain rule
    rng = np.random.default_rng(15)
    x0, grads = rng.normal(0, 1, 30), [rng.normal(0, 1, 30) for _ in range(5)]
    runs = []
    for dl in (0.0, None):
        o = oracle.DelayedOptimizer([x0], HParams(lr=0.01, dc_lambda=dl or 0.0), x_store=F32,
                                    stash_store=F32, lib=lib)
        for g in grads:
            o.step(g)
        runs.append(o.x.copy())
    assert np.array_equal(runs[0], runs[1])


def test_dc_asgd_leaves_synchronous_tensors_alone(lib):
    """DC-ASGD compensates for the staleness of a delayed tensor's gradient
    (Sec. 3.1). A tensor trained synchronously (WPipe, App. B.2) has a fresh
    gradient and no stash, so in a mixed table it follows the plain
    synchronous rule bitwise, whatever lambda_dc."""
    rng = np.random.default_rng(21)
    xa, xb = rng.normal(0, 1, 9), rng.normal(0, 1, 6)
    grads = [rng.normal(0, 1, 15) for _ in range(5)]
    hp = HParams(lr=0.05, dc_lambda=30.0)
    mixed = oracle.DelayedOptimizer([xa, xb], hp, x_store=F32, stash_store=F32,
                                    delayed=[True, False], lib=lib)
    plain = oracle.DelayedOptimizer([xb], HParams(lr=0.05, delay=0), x_store=F32,
                                    stash_store=F32, lib=lib)
    for g in grads:
        mixed.step(g)
        plain.step(g[9:])
    assert np.array_equal(mixed.x[9:], plain.x)
    # the delayed tensor is compensated: it differs from the lambda_dc = 0 run
    nodc = oracle.DelayedOptimizer([xa, xb], HParams(lr=0.05), x_store=F32, stash_store=F32,
                                   delayed=[True, False], lib=lib)
    for g in grads:
        nodc.step(g)
    assert np.max(np.abs(mixed.x[:9] - nodc.x[:9])) > 1e-6


def test_lion_sign_of_zero_is_zero(lib):
    """Lion's update is the sign of the interpolation c, and sign(0) = 0: a
    zero gradient from the zero start state moves no weight without decay,
    and only by the decay lr wd x_t with it."""
    for wd in (0.0, 0.1):
        hp = HParams(lr=0.1, beta1=0.9, beta2=0.99, weight_decay=wd, rule=oracle.RULE_LION)
        o = oracle.DelayedOptimizer([np.array([1.0, -2.0])], hp, x_store=F64, stash_store=F64,
                                    lib=lib)
        o.step(np.zeros(2), tag=o.read_weights()[1])
        assert o.x.tolist() == pytest.approx([1.0 - 0.1 * wd, -2.0 * (1.0 - 0.1 * wd)],
                                             abs=1e-16)


def test_sapipe_prediction_is_a_master_weight_rounded_to_the_stash(lib):
    """SAPipe-WP's stash (App. B.1) is the predicted weight x_t - u_prev, a
    weight in the master's format (fp32) then stored in the stash's (bf16):
    two roundings. x_t = 1 + 2^-8 and u_prev = -2^-30 give 1 + 2^-8 + 2^-30,
    which fp32 rounds to the bf16 tie 1 + 2^-8 and bf16 then rounds to even,
    1.0; rounded once it would be 1 + 2^-7."""
    hp = HParams(lr=0.0, weight_decay=0.0, correction=oracle.CORR_SAPIPE_SAME)
    o = oracle.DelayedOptimizer([np.array([1.0 + 2.0 ** -8])], hp, ef=True, x_store=F32,
                                stash_store=BF16, lib=lib)
    o.u_prev[:] = -(2.0 ** -30)
    o.step(np.array([0.5]), tag=o.read_weights()[1])
    assert o.stash[0] == 1.0
    assert o.x[0] == 1.0 + 2.0 ** -8


def _fp32_exact(a):
    a = np.asarray(a, dtype=np.float64)
    return np.array_equal(a.astype(np.float32).astype(np.float64), a)


def _bf16_exact(a):
    a = np.asarray(a, dtype=np.float64)
    bits = a.astype(np.float32).view(np.uint32)
    return _fp32_exact(a) and not np.any(bits & 0xFFFF)


def test_stored_state_is_in_its_storage_format(lib):
    """Every buffer holds values of its own storage format after each call
    (the oracle rounds each stored quantity once, as the device stores it):
    master, m, v and the EF history in fp32, the stash and the bf16 weights
    in bf16."""
    rng = np.random.default_rng(41)
    x0 = rng.normal(0, 0.02, 300)
    o = oracle.DelayedOptimizer([x0], HParams(lr=1e-3, ef_lambda=1.0).as_f32(), ef=True,
                                x_store=F32, stash_store=BF16, param_store=BF16, lib=lib)
    for _ in range(4):
        o.step(rng.normal(0, 1e-3, 300), tag=o.read_weights()[1])
        assert _fp32_exact(o.x) and _fp32_exact(o.m) and _fp32_exact(o.v)
        assert _fp32_exact(o.u_prev)
        assert _bf16_exact(o.stash) and _bf16_exact(o.param)



def test_initial_state_is_x0_in_its_storage_formats(lib):
    """Alg. 1's start state holds x_0 as the device stores it: the master is
    x_0 cast to fp32, the stash and the weights that fp32 value cast to bf16
    (torch's casts, round to nearest even), before any call."""
    rng = np.random.default_rng(44)
    x0 = rng.normal(0, 0.02, 513)
    o = oracle.DelayedOptimizer([x0[:300], x0[300:]], HParams(ef_lambda=1.0), ef=True,
                                x_store=F32, stash_store=BF16, param_store=BF16, lib=lib)
    x32 = torch.tensor(x0).float()
    np.testing.assert_array_equal(o.x, x32.double().numpy())
    xb = x32.bfloat16().double().numpy()
    np.testing.assert_array_equal(o.stash, xb)
    np.testing.assert_array_equal(o.param, xb)


def test_fp32_settings_are_torch_casts():
    """HParams.as_f32 (and the Muon twin) hand the oracle the numbers a
    device given fp32 settings computes with: every real is torch's fp32 cast
    of the setting, every integer setting unchanged."""
    from oracle.muon import MuonHParams
    hp = HParams(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1, ef_lambda=0.7,
                 max_grad_norm=1.3, delay=1, rule=oracle.RULE_ADAN, correction=0,
                 beta3=0.99, momentum_decay=4e-3, dc_lambda=0.04)
    mh = MuonHParams(lr=2e-3, momentum=0.95, weight_decay=0.1, ef_lambda=0.7, ns_eps=1e-7,
                     rms_scale=0.2, max_grad_norm=1.3)
    for src in (hp, mh):
        got = src.as_f32()
        for name, v in vars(src).items():
            w = getattr(got, name)
            if isinstance(v, float):
                assert w == torch.tensor(v, dtype=torch.float32).item(), name
            else:
                assert w == v, name

def test_bf16_weights_round_the_stored_master(lib):
    """The bf16 weights are the stored fp32 master rounded to bf16 (a5): two
    roundings from the update's exact result. x_0 = 1 + 2^-8, SGD rule with
    u = -2^-30: x_1 = 1 + 2^-8 + 2^-30, stored in fp32 as 1 + 2^-8 (a bf16
    tie), so the bf16 copy is 1.0; rounding the exact result once would give
    1 + 2^-7."""
    hp = HParams(lr=1.0, weight_decay=0.0, rule=oracle.RULE_SGD, delay=0)
    o = oracle.DelayedOptimizer([np.array([1.0 + 2.0 ** -8])], hp, x_store=F32,
                                stash_store=F32, param_store=BF16, lib=lib)
    o.step(np.array([-(2.0 ** -30)]), tag=o.read_weights()[1])
    assert o.x[0] == 1.0 + 2.0 ** -8
    assert o.param[0] == 1.0


def test_dc_asgd_compensates_the_clipped_gradient(lib):
    """Reading 20: the clip coefficient scales the gradient that arrived and
    the compensation corrects the consumed one, so g~ = s g + lambda (s g)^2
    (x_t - stash). beta1 = 0 makes the first moment exactly g~."""
    lam = 50.0
    hp = HParams(lr=0.1, beta1=0.0, beta2=0.95, eps=1e-8, weight_decay=0.0, dc_lambda=lam,
                 max_grad_norm=1.0)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    o.step(np.array([2.0]), tag=o.read_weights()[1])
    x2, x1 = o.x[0], o.stash[0]
    o.step(np.array([3.0]), tag=o.read_weights()[1])
    gh = 3.0 / (3.0 + 1e-6)
    assert o.m[0] == pytest.approx(gh + lam * gh * gh * (x2 - x1), rel=1e-13)


def test_adan_previous_gradient_is_the_consumed_one(lib):
    """Reading 19: Adan's stored previous gradient is the one consumed,
    clipped; its difference at the next call is taken between consumed
    gradients."""
    hp = HParams(lr=0.01, rule=oracle.RULE_ADAN, max_grad_norm=1.0)
    g = np.array([3.0, -4.0])
    o = oracle.DelayedOptimizer([np.array([0.5, 0.25])], hp, x_store=F64, stash_store=F64,
                                lib=lib)
    o.step(g, tag=o.read_weights()[1])
    np.testing.assert_allclose(o.g_prev, g * (1.0 / (5.0 + 1e-6)), rtol=1e-15)


def test_lion_blends_the_clipped_gradient(lib):
    """Lion's sign takes the interpolation of m and the consumed (clipped)
    gradient. beta = (0.99, 0.5), clip at 1, gradients 1 then -100: the
    clipped second gradient is -1, so c = 0.99 * 0.5 - 0.01 > 0 and the
    weight keeps moving down (1 -> 0.9 -> 0.8); the raw -100 would flip the
    sign and move it back up."""
    hp = HParams(lr=0.1, beta1=0.99, beta2=0.5, weight_decay=0.0, rule=oracle.RULE_LION,
                 max_grad_norm=1.0)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    xs = []
    for g in (1.0, -100.0):
        o.step(np.array([g]), tag=o.read_weights()[1])
        xs.append(o.x[0])
    assert xs == pytest.approx([0.9, 0.8], abs=1e-15)


def test_lion_sign_before_the_momentum_update(lib):
    """Lion takes the sign of beta1 m_{t-1} + (1 - beta1) g before m moves to
    its beta2 average. beta = (0.5, 0): after g = 1 (m = 1), g = -0.5 gives
    c = 0.5 - 0.25 > 0 (down again, 0.9 -> 0.8); the updated m (-0.5) would
    give c < 0."""
    hp = HParams(lr=0.1, beta1=0.5, beta2=0.0, weight_decay=0.0, rule=oracle.RULE_LION)
    o = oracle.DelayedOptimizer([np.array([1.0])], hp, x_store=F64, stash_store=F64, lib=lib)
    xs = []
    for g in (1.0, -0.5):
        o.step(np.array([g]), tag=o.read_weights()[1])
        xs.append(o.x[0])
    assert xs == pytest.approx([0.9, 0.8], abs=1e-15)


def test_synchronous_tensor_stash_untouched(lib):
    """A tensor trained synchronously (App. B.2) has no stale version: its
    stash is never written while the delayed tensor beside it rotates."""
    rng = np.random.default_rng(51)
    xa, xb = rng.normal(0, 1, 5), rng.normal(0, 1, 4)
    o = oracle.DelayedOptimizer([xa, xb], HParams(lr=0.05, ef_lambda=1.0), ef=True,
                                x_store=F64, stash_store=F64, delayed=[True, False], lib=lib)
    s0 = o.stash.copy()
    for _ in range(3):
        o.step(rng.normal(0, 1, 9))
    assert np.array_equal(o.stash[5:], s0[5:])
    assert not np.array_equal(o.stash[:5], s0[:5])


@pytest.mark.parametrize("corr", [oracle.CORR_EF, oracle.CORR_SAPIPE_SAME])
def test_reentering_delayed_training_restarts_alg1(lib, corr):
    """Delayed, synchronous, then delayed again (Sec. 3.1, App. A.10): from the
    re-entry on, the run is a fresh Alg. 1 run started at the weights reached
    there (SGD rule: no optimizer state besides the stash and the history):
    the stash restarts at x, the history at zero, the first call takes the
    standard rule and EF (or SAPipe's prediction) starts from there."""
    rng = np.random.default_rng(71)
    a = np.exp(rng.uniform(np.log(0.05), 0, 6))
    x0 = rng.normal(0, 1, 6)
    hp = HParams(lr=0.3, weight_decay=0.0, rule=oracle.RULE_SGD, ef_lambda=1.0, correction=corr)

    def drive(o, n, switch=None):
        xs = []
        for c in range(1, n + 1):
            if switch and c in switch:
                o.set_delay(switch[c])
            w, tag = o.read_weights("stale")
            g, _ = oracle.quadratic(a, np.zeros(6), w, None, F64, lib=lib)
            o.step(g, tag=tag)
            xs.append(o.x.copy())
        return xs

    o = oracle.DelayedOptimizer([x0], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    xs = drive(o, 11, {5: 0, 8: 1})      # delayed 1-4, synchronous 5-7, delayed 8-11
    fresh = oracle.DelayedOptimizer([xs[6]], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
    ys = drive(fresh, 4)
    for got, want in zip(xs[7:], ys):
        assert np.array_equal(got, want)


@pytest.mark.parametrize("rule", [oracle.RULE_ADAMW, oracle.RULE_NADAM, oracle.RULE_ADAN])
def test_statistics_depend_only_on_consumed_gradients(lib, rule):
    """The optimizer statistics (m, v; Adan's n and previous gradient) are
    updated with the gradient each call consumes (Alg. 1), whatever the
    delay mode: with the same gradient sequence, a run with a synchronous
    start, a cooldown and a re-entry holds the same statistics as a run
    delayed throughout. (Adan's first-step rule, a zero difference, belongs
    to the first gradient of the run, not of a delayed phase.)"""
    rng = np.random.default_rng(81)
    x0 = rng.normal(0, 0.5, 20)
    grads = [rng.normal(0, 1, 20) for _ in range(9)]
    hp = HParams(lr=0.01, ef_lambda=1.0, rule=rule)
    runs = []
    for schedule in ({}, {1: 0, 3: 1, 6: 0, 8: 1}):
        o = oracle.DelayedOptimizer([x0], hp, ef=True, x_store=F64, stash_store=F64, lib=lib)
        for c, g in enumerate(grads, start=1):
            if c in schedule:
                o.set_delay(schedule[c])
            o.step(g)
        runs.append(o)
    a, b = runs
    for name in ("m", "v", "n3", "g_prev"):
        if getattr(a, name) is not None:
            assert np.array_equal(getattr(a, name), getattr(b, name)), name
