"""ctypes binding of include/dpo_muon.h: one-step-delayed Muon (Alg. 2).

Argument marshalling only: every step of the path runs in libdpo.so's
kernels (momentum, normalisation, the tcgen05 Newton-Schulz GEMMs, the
update). Like ``dpo``, it raises when the library cannot be built or loaded;
there is no other implementation.
"""
from __future__ import annotations

import ctypes
from typing import List, Optional, Sequence, Tuple

from .dpo import (DPO_BF16, DPO_F32, DPO_INIT_FRESH, DPO_OK, DPO_SYNC, DPO_WD_ON, ALIGN_ELEMS,
                  DpoError, _stream, load)

NS_COEFFS = (3.4445, -4.7750, 2.0315)


class dpo_matrix(ctypes.Structure):
    _fields_ = [("param", ctypes.c_void_p), ("master", ctypes.c_void_p),
                ("mom", ctypes.c_void_p), ("stash", ctypes.c_void_p), ("ef", ctypes.c_void_p),
                ("grad", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("flags", ctypes.c_uint32)]


class dpo_muon_hparams(ctypes.Structure):
    _fields_ = [("momentum", ctypes.c_float), ("weight_decay", ctypes.c_float),
                ("ef_lambda", ctypes.c_float), ("max_grad_norm", ctypes.c_float),
                ("ns_a", ctypes.c_float), ("ns_b", ctypes.c_float), ("ns_c", ctypes.c_float),
                ("ns_eps", ctypes.c_float), ("rms_scale", ctypes.c_float),
                ("ns_steps", ctypes.c_int), ("delay", ctypes.c_int),
                ("correction", ctypes.c_int)]


EXPORTS = ("dpo_muon_init", "dpo_muon_step", "dpo_muon_set_delay", "dpo_muon_last_update",
           "dpo_muon_copy_update",
           "dpo_muon_get_status",
           "dpo_muon_get_step", "dpo_muon_set_step", "dpo_muon_flops",
           "dpo_muon_set_timing", "dpo_muon_get_gemm_time",
           "dpo_muon_workspace_bytes", "dpo_muon_last_error", "dpo_muon_destroy",
           "dpo_muon_grad_sqnorm", "dpo_muon_set_clip_source", "dpo_muon_clear_status",
           "dpo_muon_test_stall", "dpo_muon_get_phase_start", "dpo_muon_set_phase_start",
           "dpo_muon_set_capturable")

_typed = False


def lib() -> ctypes.CDLL:
    global _typed
    L = load()
    if not _typed:
        P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
        sig = {
            "dpo_muon_init": (I, [ctypes.POINTER(P), ctypes.POINTER(dpo_matrix), I, I, I,
                                  ctypes.POINTER(dpo_muon_hparams), I, P]),
            "dpo_muon_step": (I, [P, F, P]),
            "dpo_muon_set_delay": (I, [P, I, P]),
            "dpo_muon_last_update": (I, [P, I, ctypes.POINTER(P),
                                         ctypes.POINTER(ctypes.c_int64)]),
            "dpo_muon_copy_update": (I, [P, I, P, P]),
            "dpo_muon_get_status": (I, [P, ctypes.POINTER(ctypes.c_uint32)]),
            "dpo_muon_get_step": (I, [P, ctypes.POINTER(ctypes.c_int64)]),
            "dpo_muon_set_step": (I, [P, ctypes.c_int64]),
            "dpo_muon_flops": (I, [P, ctypes.POINTER(ctypes.c_double)]),
            "dpo_muon_set_timing": (I, [P, I]),
            "dpo_muon_get_gemm_time": (I, [P, ctypes.POINTER(ctypes.c_double),
                                           ctypes.POINTER(ctypes.c_int64)]),
            "dpo_muon_workspace_bytes": (I, [P, ctypes.POINTER(ctypes.c_int64)]),
            "dpo_muon_last_error": (ctypes.c_char_p, [P]),
            "dpo_muon_destroy": (None, [P]),
            "dpo_muon_grad_sqnorm": (I, [P, P, P]),
            "dpo_muon_set_clip_source": (I, [P, P]),
            "dpo_muon_clear_status": (I, [P, P]),
            "dpo_muon_test_stall": (I, [P, I]),
            "dpo_muon_get_phase_start": (I, [P, ctypes.POINTER(ctypes.c_int64)]),
            "dpo_muon_set_phase_start": (I, [P, ctypes.c_int64]),
            "dpo_muon_set_capturable": (I, [P, I, P, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _typed = True
    return L


def _check(rc: int, ctx) -> None:
    if rc != DPO_OK:
        raise DpoError(rc, lib().dpo_muon_last_error(ctx).decode())


def hparams(momentum=0.95, weight_decay=0.1, ef_lambda=1.0, max_grad_norm=0.0,
            coeffs=NS_COEFFS, ns_eps=1e-7, rms_scale=0.2, ns_steps=5,
            delay=1, correction=0) -> dpo_muon_hparams:
    return dpo_muon_hparams(momentum, weight_decay, ef_lambda, max_grad_norm, coeffs[0],
                            coeffs[1], coeffs[2], ns_eps, rms_scale, ns_steps, delay,
                            correction)


class DelayedMuon:
    """Owns the state of delayed Muon for a set of matrices and drives the C
    ABI. Arenas (torch, on the device): master, mom, ef (fp32), grad (grad
    dtype), param (bf16), stash (stash dtype, delay 1); each matrix sits at
    the same element offset in every arena, 256-byte aligned."""

    def __init__(self, shapes: Sequence[Tuple[int, int]], *, stash_dtype=DPO_BF16,
                 grad_dtype=DPO_BF16, lr=2e-3, momentum=0.95, weight_decay=0.1, ef=False,
                 ef_lambda=1.0, max_grad_norm=0.0, coeffs=NS_COEFFS, ns_eps=1e-7,
                 rms_scale=0.2, ns_steps=5, delay=1, wd_on: Optional[Sequence[bool]] = None,
                 device=None, x0=None, init_mode=DPO_INIT_FRESH, stream=None,
                 sync: Optional[Sequence[bool]] = None, keep_stash: Optional[bool] = None,
                 correction: int = 0):
        import torch
        self.torch = torch
        self.device = torch.device(device or "cuda")
        self.shapes = [(int(r), int(c)) for r, c in shapes]
        self.numels = [r * c for r, c in self.shapes]
        self.offsets, o = [], 0
        for n in self.numels:
            self.offsets.append(o)
            o += -(-n // ALIGN_ELEMS) * ALIGN_ELEMS
        total = max(o, ALIGN_ELEMS)
        tdt = {DPO_F32: torch.float32, DPO_BF16: torch.bfloat16}
        alloc = lambda dt: torch.zeros(total, dtype=dt, device=self.device)
        self.master = alloc(torch.float32)
        self.mom = alloc(torch.float32)
        self.ef = alloc(torch.float32) if ef else None
        self.grad = alloc(tdt[grad_dtype])
        self.param = alloc(torch.bfloat16)
        keep_stash = delay == 1 if keep_stash is None else keep_stash
        self.stash = alloc(tdt[stash_dtype]) if keep_stash else None
        self.lr, self.delay = lr, delay
        if isinstance(x0, (list, tuple)):   # one array per matrix
            for i, xi in enumerate(x0):
                self.view(self.master, i).copy_(torch.as_tensor(xi).reshape(self.shapes[i]))
        elif x0 is not None:
            self.master.copy_(x0)
        self.stash_dtype, self.grad_dtype = stash_dtype, grad_dtype
        self.hp = hparams(momentum, weight_decay, ef_lambda if ef else 0.0, max_grad_norm,
                          coeffs, ns_eps, rms_scale, ns_steps, delay, correction)
        wd_on = list(wd_on) if wd_on is not None else [True] * len(self.shapes)
        self.sync = list(sync) if sync is not None else [False] * len(self.shapes)
        ptr = lambda t, off: (t.data_ptr() + off * t.element_size()) if t is not None else None
        mats = []
        for (r, c), off, wd, sy in zip(self.shapes, self.offsets, wd_on, self.sync):
            mats.append(dpo_matrix(ptr(self.param, off), ptr(self.master, off),
                                   ptr(self.mom, off), ptr(self.stash, off), ptr(self.ef, off),
                                   ptr(self.grad, off), r, c,
                                   (DPO_WD_ON if wd else 0) | (DPO_SYNC if sy else 0)))
        self.table = mats
        L = lib()
        arr = (dpo_matrix * len(mats))(*mats)
        out = ctypes.c_void_p()
        _check(L.dpo_muon_init(ctypes.byref(out), arr, len(mats), stash_dtype, grad_dtype,
                               ctypes.byref(self.hp), init_mode, _stream(stream)), None)
        self.ctx = out.value

    def view(self, arena, i: int):
        off, (r, c) = self.offsets[i], self.shapes[i]
        return arena[off:off + r * c].view(r, c)

    def grads(self, i: int):
        return self.view(self.grad, i)

    def stale(self, i: int):
        """What the next forward/backward reads for matrix i."""
        return self.view(self.stash if self.delay == 1 and not self.sync[i] else self.param, i)

    def set_delay(self, delay: int, stream=None) -> None:
        """Switch between synchronous and delayed training (dpo_muon_set_delay)."""
        _check(lib().dpo_muon_set_delay(self.ctx, delay, _stream(stream)), self.ctx)
        self.delay = delay
        self.hp.delay = delay

    def step(self, lr: Optional[float] = None, stream=None) -> None:
        _check(lib().dpo_muon_step(self.ctx, self.lr if lr is None else lr, _stream(stream)),
               self.ctx)

    def last_update(self, i: int):
        """The Newton-Schulz output O of the last step for matrix i (bf16,
        rows x cols), copied out of the workspace."""
        torch = self.torch
        r, c = self.shapes[i]
        if r * c == 0:
            return torch.zeros((r, c), dtype=torch.bfloat16, device=self.device)
        out = torch.empty((r, c), dtype=torch.bfloat16, device=self.device)
        _check(lib().dpo_muon_copy_update(self.ctx, i, out.data_ptr(), _stream(None)), self.ctx)
        return out

    def status(self) -> int:
        v = ctypes.c_uint32()
        _check(lib().dpo_muon_get_status(self.ctx, ctypes.byref(v)), self.ctx)
        return int(v.value)

    def set_capturable(self, on: bool = True, lr_source=None, stream=None) -> None:
        """Capturable mode (dpo_muon_set_capturable); ``lr_source`` a
        one-element float32 device tensor, kept alive here, or None."""
        _check(lib().dpo_muon_set_capturable(self.ctx, 1 if on else 0,
                                             lr_source.data_ptr() if lr_source is not None
                                             else None, _stream(stream)), self.ctx)
        self._lr_src = lr_source if on else None

    def clear_status(self, stream=None) -> None:
        _check(lib().dpo_muon_clear_status(self.ctx, _stream(stream)), self.ctx)

    def test_stall(self, launches: int) -> None:
        """Make the next ``launches`` GEMM launches give up a wait (include/dpo_muon.h)."""
        _check(lib().dpo_muon_test_stall(self.ctx, launches), self.ctx)

    @property
    def k(self) -> int:
        v = ctypes.c_int64()
        _check(lib().dpo_muon_get_step(self.ctx, ctypes.byref(v)), self.ctx)
        return int(v.value)

    def set_step(self, k: int) -> None:
        _check(lib().dpo_muon_set_step(self.ctx, k), self.ctx)

    @property
    def phase_start(self) -> int:
        v = ctypes.c_int64()
        _check(lib().dpo_muon_get_phase_start(self.ctx, ctypes.byref(v)), self.ctx)
        return int(v.value)

    STATE = ("master", "mom", "ef", "param", "stash")

    def state_dict(self) -> dict:
        """Every arena, k, the start of the current delayed phase and the
        delay mode."""
        return {"k": self.k, "phase_start": self.phase_start, "delay": self.delay,
                **{n: getattr(self, n).clone() for n in self.STATE
                   if getattr(self, n) is not None}}

    def load_state(self, sd: dict) -> None:
        """Restore a state_dict into a context built with init_mode
        DPO_INIT_RESUME, the same shapes and the same delay mode."""
        if int(sd["delay"]) != self.delay:
            raise ValueError(f"checkpoint taken with delay {sd['delay']}, context has {self.delay}")
        for n in self.STATE:
            if getattr(self, n) is not None:
                getattr(self, n).copy_(sd[n])
        self.set_step(int(sd["k"]))
        _check(lib().dpo_muon_set_phase_start(self.ctx, int(sd["phase_start"])), self.ctx)

    def flops(self) -> float:
        v = ctypes.c_double()
        _check(lib().dpo_muon_flops(self.ctx, ctypes.byref(v)), self.ctx)
        return float(v.value)

    def set_timing(self, on: bool = True) -> None:
        _check(lib().dpo_muon_set_timing(self.ctx, 1 if on else 0), self.ctx)

    def gemm_time(self):
        """(milliseconds, launches) of the Newton-Schulz GEMM chains since the
        last call (needs set_timing)."""
        ms, n = ctypes.c_double(), ctypes.c_int64()
        _check(lib().dpo_muon_get_gemm_time(self.ctx, ctypes.byref(ms), ctypes.byref(n)),
               self.ctx)
        return float(ms.value), int(n.value)

    def grad_sqnorm(self, acc, stream=None) -> None:
        """Add the sum of G^2 over all matrices to ``acc`` (a float64 device
        scalar; dpo_muon_grad_sqnorm)."""
        _check(lib().dpo_muon_grad_sqnorm(self.ctx, acc.data_ptr(), _stream(stream)), self.ctx)

    def set_clip_source(self, acc=None) -> None:
        """Clip from the sum of squares in ``acc`` (kept alive here), or from
        this context's own norm when None."""
        _check(lib().dpo_muon_set_clip_source(self.ctx, acc.data_ptr() if acc is not None
                                              else None), self.ctx)
        self._clip_src = acc

    def workspace_bytes(self) -> int:
        v = ctypes.c_int64()
        _check(lib().dpo_muon_workspace_bytes(self.ctx, ctypes.byref(v)), self.ctx)
        return int(v.value)

    def close(self) -> None:
        if getattr(self, "ctx", None):
            lib().dpo_muon_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
