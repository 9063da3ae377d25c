"""CPU oracle of delayed Muon (Alg. 2, Sec. 4): driver around
``oracle_newton_schulz`` and ``oracle_muon_step`` in ``dpo_oracle.c``.

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs import it.

Passages followed:
  * Alg. 2: momentum of the stale gradient, Newton-Schulz orthogonalisation,
    U_{t-1} = eta (O_{t-1} + lambda X_t), and the standard or EF update
    X_{t+1} = X_t - 2 U_{t-1} + U_{t-2} (the EF form of Eq. (1) at lambda = 1).
  * Sec. 2.1: Muon at momentum 0.95 with update RMS 0.2.
  * Sec. 2.2: the momentum decay mu weighs the previous momentum (an EMA);
    Alg. 2 prints the two weights swapped.
Readings (pinned in ``tests/test_oracle_muon.py``): the quintic iteration
and its coefficients are those of Jordan et al. 2024, 5 steps, eps 1e-7 on
the Frobenius norm, applied to the wide orientation; the RMS scaling is
0.2 sqrt(max(rows, cols)) (Liu et al. 2025); Newton-Schulz in bf16 rounds
each iterate once when it is formed.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

from . import BF16, F32, F64, _f64, _ptr, load, round_to

NS_COEFFS = (3.4445, -4.7750, 2.0315)


class _MuonHParams(ctypes.Structure):
    _fields_ = [
        ("lr", ctypes.c_double),
        ("momentum", ctypes.c_double),
        ("weight_decay", ctypes.c_double),
        ("ef_lambda", ctypes.c_double),
        ("ns_a", ctypes.c_double),
        ("ns_b", ctypes.c_double),
        ("ns_c", ctypes.c_double),
        ("ns_steps", ctypes.c_int),
        ("ns_eps", ctypes.c_double),
        ("rms_scale", ctypes.c_double),
        ("ns_store", ctypes.c_int),
        ("delay", ctypes.c_int),
        ("correction", ctypes.c_int),
        ("x_store", ctypes.c_int),
        ("stash_store", ctypes.c_int),
        ("param_store", ctypes.c_int),
    ]


@dataclass
class MuonHParams:
    lr: float = 2e-3
    momentum: float = 0.95
    weight_decay: float = 0.1
    ef_lambda: float = 0.0
    ns_a: float = NS_COEFFS[0]
    ns_b: float = NS_COEFFS[1]
    ns_c: float = NS_COEFFS[2]
    ns_steps: int = 5
    ns_eps: float = 1e-7
    rms_scale: float = 0.2
    ns_store: int = BF16
    max_grad_norm: float = 0.0
    delay: int = 1
    correction: int = 0   # CORR_EF, CORR_SAPIPE_SAME or CORR_SAPIPE_UPDATED (App. B.1)

    def as_f32(self) -> "MuonHParams":
        """Every real rounded to fp32, as a device taking fp32 settings sees them."""
        r = lambda v: float(np.float32(v))
        return MuonHParams(r(self.lr), r(self.momentum), r(self.weight_decay),
                           r(self.ef_lambda), r(self.ns_a), r(self.ns_b), r(self.ns_c),
                           self.ns_steps, r(self.ns_eps), r(self.rms_scale), self.ns_store,
                           r(self.max_grad_norm), self.delay, self.correction)


def newton_schulz(M, steps: int = 5, store: int = F64, eps: float = 1e-7,
                  coeffs=NS_COEFFS, lib=None) -> np.ndarray:
    """Newton-Schulz orthogonalisation of a 2-D array (see dpo_oracle.h)."""
    lib = lib or load()
    M = _f64(M)
    rows, cols = M.shape
    O = np.empty_like(M)
    rc = lib.oracle_newton_schulz(rows, cols, _ptr(M), eps, coeffs[0], coeffs[1], coeffs[2],
                                  steps, store, _ptr(O))
    if rc != 0:
        raise ValueError("oracle_newton_schulz rejected its arguments")
    return O


@dataclass
class DelayedMuon:
    """Alg. 2 over a set of weight matrices (each its own Newton-Schulz).

    Versions follow Alg. 1 as in DelayedOptimizer: after construction the
    stash holds X_0 and the master X_1 = X_0; with delay = 1 call k consumes
    the gradient evaluated at the stash and leaves the stash at X_k. Clipping
    takes the global norm over all matrices.

    ``wd_on`` marks per matrix whether its update decays X_t (default all;
    embeddings and norms commonly go without). ``delayed`` marks per matrix
    whether it takes delayed updates (default
    all; a synchronous matrix has no stash write and no correction, as WPipe
    and the synchronous LM head train part of the model). ``set_delay``
    switches the whole run between synchronous and delayed training
    (synchronous start and cooldown, Sec. 3.1): entering delayed training
    stashes the current weights and restarts Alg. 1.
    """
    x0: Sequence[np.ndarray]
    hp: MuonHParams = field(default_factory=MuonHParams)
    ef: bool = False
    x_store: int = F32
    stash_store: int = F32
    param_store: Optional[int] = None
    lib: object = None
    delayed: Optional[Sequence[bool]] = None
    wd_on: Optional[Sequence[bool]] = None

    def __post_init__(self):
        self.lib = self.lib or load()
        self.shapes = [tuple(np.asarray(t).shape) for t in self.x0]
        assert all(len(s) == 2 for s in self.shapes), "Muon takes 2-D matrices"
        self.x = [round_to(_f64(t), self.x_store, self.lib).reshape(s)
                  for t, s in zip(self.x0, self.shapes)]
        self.mom = [np.zeros(s) for s in self.shapes]
        self.u_prev = [np.zeros(s) for s in self.shapes] if self.ef else None
        self.stash = [round_to(x, self.stash_store, self.lib).reshape(x.shape) for x in self.x]
        self.param = ([round_to(x, self.param_store, self.lib).reshape(x.shape) for x in self.x]
                      if self.param_store is not None else None)
        self.o = [np.zeros(s) for s in self.shapes]
        self.delay = self.hp.delay
        self.k = 0
        self.t = 0   # Alg. 1 iteration within the current delayed phase
        self.last_clip = 1.0

    def set_delay(self, delay: int) -> None:
        """Switch between synchronous (0) and delayed (1) training; entering
        delayed training stashes the current weights and zeroes the update
        history (Alg. 1 restarts)."""
        if delay == self.delay:
            return
        if delay == 1:
            self.stash = [round_to(x, self.stash_store, self.lib).reshape(x.shape)
                          for x in self.x]
            if self.u_prev is not None:
                for u in self.u_prev:
                    u[...] = 0.0
            self.t = 0
        self.delay = delay

    def step(self, grads: Sequence[np.ndarray], lr: Optional[float] = None,
             sq: Optional[float] = None) -> None:
        grads = [_f64(g).reshape(s) for g, s in zip(grads, self.shapes)]
        self.k += 1
        if self.delay == 1:
            self.t += 1
        if sq is None:
            sq = sum(float(self.lib.oracle_sqnorm(g.size, _ptr(g))) for g in grads)
        clip = self.lib.oracle_clip_coef(sq, self.hp.max_grad_norm)
        self.last_clip = clip
        h = self.hp
        for i, (rows, cols) in enumerate(self.shapes):
            dly = self.delay if self.delayed is None or self.delayed[i] else 0
            wd = h.weight_decay if self.wd_on is None or self.wd_on[i] else 0.0
            hp = _MuonHParams(lr if lr is not None else h.lr, h.momentum, wd,
                              h.ef_lambda, h.ns_a, h.ns_b, h.ns_c, h.ns_steps, h.ns_eps,
                              h.rms_scale, h.ns_store, dly, h.correction, self.x_store,
                              self.stash_store,
                              self.param_store if self.param_store is not None else F64)
            rc = self.lib.oracle_muon_step(
                rows, cols, max(self.t, 1), ctypes.byref(hp), _ptr(grads[i]), clip,
                _ptr(self.x[i]), _ptr(self.mom[i]),
                _ptr(self.u_prev[i]) if self.u_prev is not None else None,
                _ptr(self.stash[i]), _ptr(self.param[i]) if self.param is not None else None,
                _ptr(self.o[i]))
            if rc != 0:
                raise ValueError("oracle_muon_step rejected its arguments")
