"""CPU oracle of the one-step-delayed AdamW step with Error Feedback.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` import this
package. The product package ``paper_2606_30634_gb300`` never imports it, and
the oracle imports nothing from the product package.

The arithmetic lives in ``dpo_oracle.c`` (plain C, double precision, one
element at a time). This module marshals numpy arrays to it and implements the
driver of Alg. 1 (Delayed Gradient Update) around it: the iteration counter,
the weight-version stash and the version tags that check which weights each
gradient was evaluated at.

Paper: arXiv 2606.30634. Passages followed:
  * Alg. 1 (Sec. 2): delayed update x_{t+1} = x_t - u_{t-1}(g_{t-1}); the
    standard rule for t <= 1; g_{-1} = 0, u_{-1} = 0, so iteration t = 0 only
    copies x_1 = x_0.
  * Eq. (1) (Sec. 3.2) and App. A.4: Error Feedback,
    x_{t+1} = x_t - u_{t-1} - lambda (u_{t-1} - u_{t-2}).
  * Sec. 2: PipeDream-2BW keeps one stashed weight version, which is what
    the next forward/backward reads.
  * Sec. 2.1 / 2.2 / App. E.1: AdamW with beta = (0.9, 0.95), EMA moments,
    weight decay 0.1, global clipping at 1.0. Alg. 2: decay acts on x_t.

Readings where the paper is silent (each pinned by a test in
``tests/test_oracle_pins.py``): AdamW follows the decoupled form with bias
correction and eps outside the square root; clipping scales the consumed
(stale) gradient by min(1, max_norm / (||g|| + 1e-6)); the stash holds the
pre-update x_t; bf16 copies are round-to-nearest-even from the fp32 master.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

from . import build as _build

F64, F32, BF16 = 0, 1, 2
RULE_ADAMW, RULE_SGD, RULE_NADAM, RULE_LION, RULE_ADAN = 0, 1, 2, 3, 4
CORR_EF, CORR_SAPIPE_SAME, CORR_SAPIPE_UPDATED = 0, 1, 2
STORE_NAMES = {"f64": F64, "f32": F32, "bf16": BF16}

_lib = None


class _HParams(ctypes.Structure):
    _fields_ = [
        ("lr", ctypes.c_double),
        ("beta1", ctypes.c_double),
        ("beta2", ctypes.c_double),
        ("eps", ctypes.c_double),
        ("weight_decay", ctypes.c_double),
        ("ef_lambda", ctypes.c_double),
        ("beta3", ctypes.c_double),
        ("momentum_decay", ctypes.c_double),
        ("dc_lambda", ctypes.c_double),
        ("delay", ctypes.c_int),
        ("rule", ctypes.c_int),
        ("correction", ctypes.c_int),
        ("x_store", ctypes.c_int),
        ("stash_store", ctypes.c_int),
        ("param_store", ctypes.c_int),
    ]


_dp = ctypes.POINTER(ctypes.c_double)


def load(path: Optional[str] = None):
    """Load (building if needed) the oracle library; ``path`` selects another
    build of the same source (tests use it for planted-mistake variants)."""
    global _lib
    default = path is None
    if default:
        if _lib is not None:
            return _lib
        path = _build.build()
    lib = ctypes.CDLL(path)
    lib.oracle_step.restype = ctypes.c_int
    lib.oracle_step.argtypes = [
        ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.POINTER(_HParams), _dp,
        ctypes.c_double, ctypes.POINTER(ctypes.c_uint8), ctypes.POINTER(ctypes.c_uint8),
        _dp, _dp, _dp, _dp, _dp, _dp, _dp, _dp]
    lib.oracle_sqnorm.restype = ctypes.c_double
    lib.oracle_sqnorm.argtypes = [ctypes.c_int64, _dp]
    lib.oracle_sqnorm_f32.restype = ctypes.c_double
    lib.oracle_sqnorm_f32.argtypes = [ctypes.c_int64, ctypes.POINTER(ctypes.c_float)]
    lib.oracle_sqnorm_bf16.restype = ctypes.c_double
    lib.oracle_sqnorm_bf16.argtypes = [ctypes.c_int64, ctypes.POINTER(ctypes.c_uint16)]
    lib.oracle_clip_coef.restype = ctypes.c_double
    lib.oracle_clip_coef.argtypes = [ctypes.c_double, ctypes.c_double]
    lib.oracle_round.restype = ctypes.c_double
    lib.oracle_round.argtypes = [ctypes.c_double, ctypes.c_int]
    lib.oracle_round_n.restype = None
    lib.oracle_round_n.argtypes = [ctypes.c_int64, _dp, _dp, ctypes.c_int]
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_num_threads.argtypes = []
    lib.oracle_set_num_threads.restype = None
    lib.oracle_set_num_threads.argtypes = [ctypes.c_int]
    lib.oracle_quadratic.restype = ctypes.c_double
    lib.oracle_quadratic.argtypes = [ctypes.c_int64, _dp, _dp, _dp, _dp,
                                     ctypes.c_int, _dp]
    lib.oracle_newton_schulz.restype = ctypes.c_int
    lib.oracle_newton_schulz.argtypes = [ctypes.c_int64, ctypes.c_int64, _dp, ctypes.c_double,
                                         ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                         ctypes.c_int, ctypes.c_int, _dp]
    lib.oracle_muon_step.restype = ctypes.c_int
    lib.oracle_muon_step.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                     ctypes.c_void_p, _dp, ctypes.c_double, _dp, _dp, _dp, _dp,
                                     _dp, _dp]
    if default:
        _lib = lib
    return lib


def _ptr(a: Optional[np.ndarray], ctype=ctypes.c_double):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def num_threads(lib=None) -> int:
    return int((lib or load()).oracle_num_threads())


def set_num_threads(n: int, lib=None) -> None:
    (lib or load()).oracle_set_num_threads(int(n))


def round_to(x, store: int, lib=None) -> np.ndarray:
    """Round every value to a storage format (F64, F32 or BF16)."""
    lib = lib or load()
    x = _f64(x)
    out = np.empty_like(x)
    lib.oracle_round_n(x.size, _ptr(x), _ptr(out), store)
    return out


def sqnorm(g, lib=None) -> float:
    """sum g_i^2 in double, fixed order."""
    lib = lib or load()
    g = _f64(g)
    return float(lib.oracle_sqnorm(g.size, _ptr(g)))


def sqnorm_f32(g: np.ndarray, lib=None) -> float:
    lib = lib or load()
    g = np.ascontiguousarray(g, dtype=np.float32)
    return float(lib.oracle_sqnorm_f32(g.size, _ptr(g, ctypes.c_float)))


def sqnorm_bf16(bits: np.ndarray, lib=None) -> float:
    """sum g_i^2 for a gradient given as bf16 bit patterns (uint16)."""
    lib = lib or load()
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return float(lib.oracle_sqnorm_bf16(bits.size, _ptr(bits, ctypes.c_uint16)))


def clip_coef(sq: float, max_norm: float, lib=None) -> float:
    return float((lib or load()).oracle_clip_coef(sq, max_norm))


def quadratic(a, wstar, w, noise, store: int, lib=None):
    """Noisy diagonal quadratic 1/2 sum a (w - w*)^2: returns (grad, loss)
    with grad = a (w - w*) + noise rounded to ``store``, loss at ``w``."""
    lib = lib or load()
    a, wstar, w = _f64(a), _f64(wstar), _f64(w)
    noise = None if noise is None else _f64(noise)
    g = np.empty_like(w)
    loss = lib.oracle_quadratic(w.size, _ptr(a), _ptr(wstar), _ptr(w),
                                _ptr(noise), store, _ptr(g))
    return g, float(loss)


@dataclass
class HParams:
    """Hyperparameters of the step (values as the real numbers the oracle
    uses; pass fp32-representable values to compare with an fp32 device)."""
    lr: float = 3e-4
    beta1: float = 0.9
    beta2: float = 0.95
    eps: float = 1e-8
    weight_decay: float = 0.1
    ef_lambda: float = 0.0
    max_grad_norm: float = 0.0
    delay: int = 1
    rule: int = RULE_ADAMW
    correction: int = CORR_EF
    beta3: float = 0.99
    momentum_decay: float = 0.004
    dc_lambda: float = 0.0

    def as_f32(self) -> "HParams":
        """The same settings with every real rounded to fp32: the exact
        numbers a device receiving fp32 hyperparameters computes with."""
        r = lambda v: float(np.float32(v))
        return HParams(r(self.lr), r(self.beta1), r(self.beta2), r(self.eps),
                       r(self.weight_decay), r(self.ef_lambda),
                       r(self.max_grad_norm), self.delay, self.rule, self.correction,
                       r(self.beta3), r(self.momentum_decay), r(self.dc_lambda))


class StaleVersionError(AssertionError):
    """A gradient was evaluated at weights other than Alg. 1 prescribes."""


@dataclass
class DelayedOptimizer:
    """Alg. 1 with AdamW (or the test-only SGD rule) over a set of tensors.

    The tensors are kept concatenated (the step is elementwise; only the clip
    norm spans them). Version tags follow Alg. 1's iterate index: with delay
    from the start, after construction the stash holds x_0 (tag 0) and the
    master holds x_1 = x_0 (tag 1, iteration t = 0 applies u_{-1} = 0); after
    call k the master holds x_{k+1} and the stash x_k. With delay = 1 the
    gradient consumed by a call must be evaluated at the stale view (the
    stash, or the latest weights for tensors trained synchronously); with
    delay = 0 at the latest weights.

    ``delayed`` marks per tensor whether it takes delayed updates (default
    all): WPipe (App. B.2) delays half the model, the LM-head ablation
    (App. A.9) keeps the head synchronous. ``set_delay`` switches the whole
    run between synchronous and delayed training (synchronous start and
    cooldown, Sec. 3.1): entering delayed training stashes the current
    weights and restarts Alg. 1 (u_{-1} = 0, standard rule at its first call).
    """
    x0: Sequence[np.ndarray]
    hp: HParams = field(default_factory=HParams)
    ef: bool = False
    x_store: int = F32
    stash_store: int = F32
    param_store: Optional[int] = None
    grad_store: int = F32
    wd_on: Optional[Sequence[bool]] = None
    lib: object = None
    delayed: Optional[Sequence[bool]] = None

    def __post_init__(self):
        self.lib = self.lib or load()
        self.sizes = [int(np.asarray(t).size) for t in self.x0]
        self.offsets = np.concatenate([[0], np.cumsum(self.sizes)]).astype(np.int64)
        n = int(self.offsets[-1])
        flat = (np.concatenate([_f64(t).ravel() for t in self.x0])
                if self.x0 else np.zeros(0))
        self.x = round_to(flat, self.x_store, self.lib)
        self.m = np.zeros(n)
        self.v = np.zeros(n)
        adan = self.hp.rule == RULE_ADAN
        self.n3 = np.zeros(n) if adan else None
        self.g_prev = np.zeros(n) if adan else None
        self.u_prev = np.zeros(n) if self.ef else None
        self.stash = round_to(self.x, self.stash_store, self.lib)
        self.param = (round_to(self.x, self.param_store, self.lib)
                      if self.param_store is not None else None)
        self.mask = self._tensor_mask(self.wd_on, n)
        self.delay_mask = self._tensor_mask(self.delayed, n)
        self.delay = self.hp.delay
        self.k = 0
        self.t = 0   # Alg. 1 iteration within the current delayed phase
        self.latest_tag = 1 if self.delay == 1 else 0
        self.stash_tag = 0
        self.last_clip = 1.0
        self.last_sqnorm = 0.0

    def _tensor_mask(self, flags, n):
        if flags is None:
            return None
        if not n:
            return np.zeros(0, np.uint8)
        return np.concatenate([np.full(s, 1 if on else 0, np.uint8)
                               for s, on in zip(self.sizes, flags)])

    def read_weights(self, which: str = "stale"):
        """(weights, tag): the stale view (what the next forward/backward
        reads under delay = 1: the stash, with the latest weights for
        synchronously trained tensors) or the latest weights."""
        latest = self.param if self.param is not None else self.x
        if which == "stale" and self.delay == 1:
            if self.delay_mask is None:
                return self.stash, self.stash_tag
            return np.where(self.delay_mask == 1, self.stash, latest), self.stash_tag
        return latest, self.latest_tag

    def set_delay(self, delay: int) -> None:
        """Switch between synchronous (0) and one-step-delayed (1) training.
        Entering delayed training stashes the current weights and zeroes the
        update history: Alg. 1 restarts there."""
        if delay == self.delay:
            return
        if delay == 1:
            self.stash = round_to(self.x, self.stash_store, self.lib)
            if self.u_prev is not None:
                self.u_prev[:] = 0.0
            self.t = 0
            self.stash_tag = self.latest_tag
        self.delay = delay

    def step(self, g, tag: Optional[int] = None, lr: Optional[float] = None,
             sq: Optional[float] = None) -> None:
        """One call of Alg. 1. ``g``: the gradient (flat, all tensors);
        ``tag``: version tag of the weights it was evaluated at (checked when
        given); ``sq``: the gradient's squared norm when ``g`` covers only a
        sample of the elements (clipping needs the full norm)."""
        g = _f64(g).ravel()
        expected = self.stash_tag if self.delay == 1 else self.latest_tag
        if tag is not None and tag != expected:
            raise StaleVersionError(
                f"gradient from version {tag}, Alg. 1 needs version {expected}")
        self.k += 1
        if self.delay == 1:
            self.t += 1
        if sq is None:
            sq = float(self.lib.oracle_sqnorm(g.size, _ptr(g)))
        self.last_sqnorm = sq
        clip = self.lib.oracle_clip_coef(sq, self.hp.max_grad_norm)
        self.last_clip = clip
        hp = _HParams(lr if lr is not None else self.hp.lr, self.hp.beta1,
                      self.hp.beta2, self.hp.eps, self.hp.weight_decay,
                      self.hp.ef_lambda, self.hp.beta3, self.hp.momentum_decay,
                      self.hp.dc_lambda, self.delay, self.hp.rule, self.hp.correction,
                      self.x_store, self.stash_store,
                      self.param_store if self.param_store is not None else F64)
        rc = self.lib.oracle_step(
            g.size, self.k, max(self.t, 1), ctypes.byref(hp), _ptr(g), clip,
            _ptr(self.mask, ctypes.c_uint8), _ptr(self.delay_mask, ctypes.c_uint8),
            _ptr(self.x), _ptr(self.m), _ptr(self.v), _ptr(self.u_prev), _ptr(self.stash),
            _ptr(self.param), _ptr(self.n3), _ptr(self.g_prev))
        if rc != 0:
            raise ValueError("oracle_step rejected its arguments")
        if self.delay == 1:
            self.stash_tag = self.latest_tag
        self.latest_tag += 1

    def tensor(self, name: str, i: int) -> np.ndarray:
        """Slice of state buffer ``name`` for tensor ``i``."""
        buf = getattr(self, name)
        return buf[self.offsets[i]:self.offsets[i + 1]]
