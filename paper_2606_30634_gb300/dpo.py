"""Python binding of the C ABI in include/dpo.h (argument marshalling only).

Every function here has the name and meaning of the C entry point it wraps;
each step of the optimizer runs in ``libdpo.so``'s CUDA kernels. PyTorch only
provides device memory and streams: buffers are passed as raw device
pointers, streams as ``cudaStream_t`` handles.

``DelayedAdamW`` is a convenience owner of the state buffers for a list of
parameter shapes: it lays every state kind out as one flat, 256-byte-aligned
device arena (the layout the kernels stream through) and builds the tensor
table from it.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import List, Optional, Sequence

from . import build as _build

DPO_OK, DPO_EINVAL, DPO_EALIGN, DPO_EDTYPE, DPO_ECUDA, DPO_ESTATE, DPO_ENOMEM = 0, -1, -2, -3, -4, -5, -6
DPO_F32, DPO_BF16 = 0, 1
DPO_WD_ON = 1
DPO_SYNC = 2
DPO_STALE, DPO_LATEST = 0, 1
DPO_INIT_FRESH, DPO_INIT_RESUME = 0, 1
DPO_FLAG_NONFINITE = 1
DPO_CORR_EF, DPO_CORR_SAPIPE_SAME, DPO_CORR_SAPIPE_UPDATED = 0, 1, 2
DPO_OPT_ADAMW, DPO_OPT_NADAM, DPO_OPT_LION, DPO_OPT_ADAN = 0, 1, 2, 3
DPO_STASH_COPY, DPO_STASH_PINGPONG = 0, 1

EXPORTS = ("dpo_init", "dpo_stash", "dpo_step", "dpo_read_weights", "dpo_get_step",
           "dpo_set_step", "dpo_get_flags", "dpo_algorithmic_bytes", "dpo_launch_config",
           "dpo_last_error", "dpo_destroy", "dpo_grad_norm_noalloc", "dpo_set_delay",
           "dpo_grad_sqnorm", "dpo_set_clip_source", "dpo_test_fail_allocs",
           "dpo_get_phase_start", "dpo_set_phase_start", "dpo_set_capturable",
           "dpo_set_timing", "dpo_get_timing")

DPO_NOALLOC_CHUNK_ELEMS = 1 << 20
DPO_NOALLOC_MAX_CHUNKS = 16384
DPO_NOALLOC_MAX_NUMEL = DPO_NOALLOC_MAX_CHUNKS * DPO_NOALLOC_CHUNK_ELEMS


class DpoError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"[{code}] {msg}")
        self.code = code


class dpo_hparams(ctypes.Structure):
    _fields_ = [("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
                ("weight_decay", ctypes.c_float), ("ef_lambda", ctypes.c_float),
                ("max_grad_norm", ctypes.c_float), ("delay", ctypes.c_int),
                ("correction", ctypes.c_int), ("optimizer", ctypes.c_int),
                ("beta3", ctypes.c_float), ("momentum_decay", ctypes.c_float),
                ("dc_lambda", ctypes.c_float), ("stash_mode", ctypes.c_int)]


class dpo_tensor(ctypes.Structure):
    _fields_ = [("param", ctypes.c_void_p), ("master", ctypes.c_void_p), ("m", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("stash", ctypes.c_void_p), ("ef", ctypes.c_void_p),
                ("grad", ctypes.c_void_p), ("n", ctypes.c_void_p), ("grad_prev", ctypes.c_void_p),
                ("numel", ctypes.c_int64), ("flags", ctypes.c_uint32)]


_lib = None


def lib_path() -> str:
    return os.path.join(_build.OUT, "libdpo.so")


def load() -> ctypes.CDLL:
    """Load libdpo.so (building it first if it is missing or stale; the
    DPO_LIBRARY environment variable names another build of it). Raises if
    it cannot be built: there is no other implementation to fall back to."""
    global _lib
    if _lib is not None:
        return _lib
    path = os.environ.get("DPO_LIBRARY") or _build.build()["libdpo.so"]
    if not os.path.exists(path):
        raise RuntimeError(f"libdpo.so is missing at {path}")
    L = ctypes.CDLL(path)
    P, I, F, V = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, None
    sig = {
        "dpo_init": (I, [ctypes.POINTER(P), ctypes.POINTER(dpo_tensor), I, I, I, I,
                         ctypes.POINTER(dpo_hparams), I, P]),
        "dpo_stash": (I, [P, P]),
        "dpo_set_delay": (I, [P, I, P]),
        "dpo_step": (I, [P, F, P]),
        "dpo_read_weights": (I, [P, I, I, ctypes.POINTER(P), ctypes.POINTER(I)]),
        "dpo_get_step": (I, [P, ctypes.POINTER(ctypes.c_int64)]),
        "dpo_set_step": (I, [P, ctypes.c_int64]),
        "dpo_get_flags": (I, [P, ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_double),
                              ctypes.POINTER(F), P]),
        "dpo_algorithmic_bytes": (I, [P, ctypes.POINTER(ctypes.c_int64),
                                      ctypes.POINTER(ctypes.c_int64)]),
        "dpo_launch_config": (I, [P, ctypes.POINTER(I), ctypes.POINTER(I), ctypes.POINTER(I)]),
        "dpo_last_error": (ctypes.c_char_p, [P]),
        "dpo_destroy": (V, [P]),
        "dpo_grad_norm_noalloc": (I, [P, ctypes.c_int64, I, F, P, P, P]),
        "dpo_grad_sqnorm": (I, [P, P, P]),
        "dpo_set_clip_source": (I, [P, P]),
        "dpo_test_fail_allocs": (I, [I, I]),
        "dpo_get_phase_start": (I, [P, ctypes.POINTER(ctypes.c_int64)]),
        "dpo_set_phase_start": (I, [P, ctypes.c_int64]),
        "dpo_set_capturable": (I, [P, I, P, P]),
        "dpo_set_timing": (I, [P, I]),
        "dpo_get_timing": (I, [P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                               ctypes.POINTER(ctypes.c_int64)]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(rc: int, ctx) -> None:
    if rc != DPO_OK:
        raise DpoError(rc, dpo_last_error(ctx))


def dpo_last_error(ctx) -> str:
    return load().dpo_last_error(ctx).decode()


def dpo_init(table: Sequence[dpo_tensor], param_dtype: int, stash_dtype: int, grad_dtype: int,
             hp: dpo_hparams, init_mode: int = DPO_INIT_FRESH, stream=None):
    """Returns the context handle (an int). Raises DpoError on failure."""
    L = load()
    arr = (dpo_tensor * len(table))(*table)
    out = ctypes.c_void_p()
    rc = L.dpo_init(ctypes.byref(out), arr, len(table), param_dtype, stash_dtype, grad_dtype,
                    ctypes.byref(hp), init_mode, _stream(stream))
    _check(rc, None)
    return out.value


def dpo_stash(ctx, stream=None) -> None:
    _check(load().dpo_stash(ctx, _stream(stream)), ctx)


def dpo_set_delay(ctx, delay: int, stream=None) -> None:
    _check(load().dpo_set_delay(ctx, delay, _stream(stream)), ctx)


def dpo_step(ctx, lr: float, stream=None) -> None:
    _check(load().dpo_step(ctx, lr, _stream(stream)), ctx)


def _dptr(t) -> Optional[int]:
    return t if isinstance(t, int) or t is None else t.data_ptr()


def dpo_grad_sqnorm(ctx, acc, stream=None) -> None:
    """Add the context's sum of g^2 to ``acc`` (a float64 device scalar)."""
    _check(load().dpo_grad_sqnorm(ctx, _dptr(acc), _stream(stream)), ctx)


def dpo_set_clip_source(ctx, acc) -> None:
    """Clip later steps from the sum of squares in ``acc`` (None: own norm)."""
    _check(load().dpo_set_clip_source(ctx, _dptr(acc)), ctx)


def dpo_test_fail_allocs(after: int, count: int) -> None:
    """Make the library's device allocations after the next ``after`` fail,
    ``count`` of them (include/dpo.h); (0, 0) turns the hook off."""
    _check(load().dpo_test_fail_allocs(after, count), None)


def allreduce_sqnorm(acc, group=None) -> None:
    """Sum ``acc`` over the ranks of ``group`` (torch.distributed), each rank
    holding one shard of the parameter set: the one exchange of a
    partitioned step. Nothing to do without an initialised process group."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(acc, op=dist.ReduceOp.SUM, group=group)


def global_sqnorm(optimizers, acc, stream=None, group=None) -> None:
    """||g||^2 over every parameter that ``optimizers`` (DelayedAdamW,
    DelayedMuon) hold, into ``acc`` (a one-element float64 device tensor):
    zeroed, each context's share added in list order on ``stream``, then
    summed over ``group``'s ranks. Optimizers whose clip source is ``acc``
    then clip from the norm over all of them (App. E.1): step them on the
    same stream (the default, torch's current one) or after an event on it,
    since the step reads ``acc`` on the device when it runs."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream(acc.device)
    with torch.cuda.stream(s):
        acc.zero_()
        for o in optimizers:
            o.grad_sqnorm(acc, s)
        allreduce_sqnorm(acc, group)


def dpo_set_timing(ctx, on: bool) -> None:
    _check(load().dpo_set_timing(ctx, 1 if on else 0), ctx)


def dpo_get_timing(ctx):
    """(norm-pass ms, fused-step ms, calls) since the last read."""
    tn, ts, n = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check(load().dpo_get_timing(ctx, ctypes.byref(tn), ctypes.byref(ts), ctypes.byref(n)), ctx)
    return tn.value, ts.value, n.value


def dpo_read_weights(ctx, which: int, tensor: int):
    ptr, dt = ctypes.c_void_p(), ctypes.c_int()
    _check(load().dpo_read_weights(ctx, which, tensor, ctypes.byref(ptr), ctypes.byref(dt)), ctx)
    return ptr.value, dt.value


def dpo_get_step(ctx) -> int:
    k = ctypes.c_int64()
    _check(load().dpo_get_step(ctx, ctypes.byref(k)), ctx)
    return k.value


def dpo_set_step(ctx, k: int) -> None:
    _check(load().dpo_set_step(ctx, k), ctx)


def dpo_set_capturable(ctx, on: bool, lr_source=None, stream=None) -> None:
    """Capturable mode (include/dpo.h): step counters on the device."""
    _check(load().dpo_set_capturable(ctx, 1 if on else 0, _dptr(lr_source), _stream(stream)), ctx)


def dpo_get_phase_start(ctx) -> int:
    k0 = ctypes.c_int64()
    _check(load().dpo_get_phase_start(ctx, ctypes.byref(k0)), ctx)
    return k0.value


def dpo_set_phase_start(ctx, k0: int) -> None:
    _check(load().dpo_set_phase_start(ctx, k0), ctx)


def dpo_get_flags(ctx, stream=None):
    f, n, c = ctypes.c_uint32(), ctypes.c_double(), ctypes.c_float()
    _check(load().dpo_get_flags(ctx, ctypes.byref(f), ctypes.byref(n), ctypes.byref(c),
                                _stream(stream)), ctx)
    return f.value, n.value, c.value


def dpo_algorithmic_bytes(ctx):
    s, n = ctypes.c_int64(), ctypes.c_int64()
    _check(load().dpo_algorithmic_bytes(ctx, ctypes.byref(s), ctypes.byref(n)), ctx)
    return s.value, n.value


def dpo_launch_config(ctx):
    a, b, t = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(load().dpo_launch_config(ctx, ctypes.byref(a), ctypes.byref(b), ctypes.byref(t)), ctx)
    return a.value, b.value, t.value


def dpo_destroy(ctx) -> None:
    if ctx:
        load().dpo_destroy(ctx)


def dpo_grad_norm_noalloc(grad, numel: int, grad_dtype: int, max_grad_norm: float, norm_out,
                          clip_out, stream=None) -> None:
    """Norm and clip coefficient of one contiguous device gradient buffer,
    with no device allocation (scratch in a fixed device array; see
    include/dpo.h for its limit and sharing rules). ``grad``, ``norm_out``
    (float64) and ``clip_out`` (float32) are device pointers or tensors."""
    ptr = lambda t: t if isinstance(t, int) or t is None else t.data_ptr()
    rc = load().dpo_grad_norm_noalloc(ptr(grad), numel, grad_dtype, max_grad_norm,
                                      ptr(norm_out), ptr(clip_out), _stream(stream))
    if rc != DPO_OK:
        raise DpoError(rc, "dpo_grad_norm_noalloc rejected its arguments or failed")


# ------------------------------------------------------------------ owner --

ALIGN_ELEMS = 128   # 256-byte alignment of every tensor in every arena (bf16 or fp32)
STATE_BUFFERS = ("master", "m", "v", "n", "grad_prev", "param", "stash", "ef")


@dataclass
class Layout:
    numels: List[int]
    offsets: List[int]   # element offset of each tensor in every arena
    total: int           # arena length in elements (padded)

    @staticmethod
    def of(numels: Sequence[int]) -> "Layout":
        offs, o = [], 0
        for n in numels:
            offs.append(o)
            o += -(-int(n) // ALIGN_ELEMS) * ALIGN_ELEMS
        return Layout([int(n) for n in numels], offs, max(o, ALIGN_ELEMS))


class DelayedAdamW:
    """Owns the state of a one-step-delayed optimizer step (AdamW by default;
    ``optimizer`` selects NAdam, Lion or Adan) for a set of parameter tensors
    and drives the C ABI.

    Arenas (torch tensors on the device): master, m, v (fp32), grad (grad
    dtype), param (bf16, only with param_dtype BF16), stash (stash dtype,
    delay 1), ef (fp32, when ``ef`` is set). Each tensor occupies a slice of
    every arena (``layout.offsets``), padded to a multiple of ALIGN_ELEMS.
    ``x0``, the fp32 start weights, fills the master before dpo_init(FRESH):
    a sequence with one tensor per parameter tensor, their plain
    concatenation (``sum(numels)`` elements), or a tensor in the arena layout
    (``layout.total`` elements). Pass ``init_mode=DPO_INIT_RESUME`` to start from arenas
    restored by ``load_state``. ``ef`` allocates the update-history buffer the
    staleness ``correction`` (DPO_CORR_*) uses. With ``host_grad`` / ``host_param`` the grad /
    param arenas are pinned host memory instead, which the fused kernel reads
    and writes across the host link (see include/dpo.h).
    """

    def __init__(self, numels: Sequence[int], *, param_dtype=DPO_BF16, stash_dtype=DPO_F32,
                 grad_dtype=DPO_BF16, lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8,
                 weight_decay=0.1, ef=False, ef_lambda=1.0, max_grad_norm=0.0, delay=1,
                 wd_on: Optional[Sequence[bool]] = None, device=None, x0=None,
                 init_mode=DPO_INIT_FRESH, stream=None, host_grad=False, host_param=False,
                 correction=DPO_CORR_EF, sync: Optional[Sequence[bool]] = None,
                 keep_stash: Optional[bool] = None, optimizer=DPO_OPT_ADAMW, beta3=0.99,
                 momentum_decay=0.004, dc_lambda=0.0, stash_mode=DPO_STASH_COPY):
        import torch
        self.torch = torch
        self.device = torch.device(device or "cuda")
        self.layout = Layout.of(numels)
        self.param_dtype, self.stash_dtype, self.grad_dtype = param_dtype, stash_dtype, grad_dtype
        self.delay = delay
        self.lr = lr
        tdt = {DPO_F32: torch.float32, DPO_BF16: torch.bfloat16}
        n = self.layout.total
        # zero-filled, so the alignment padding between tensors is defined
        alloc = lambda dt: torch.zeros(n, dtype=dt, device=self.device)
        host_alloc = lambda dt: torch.zeros(n, dtype=dt, pin_memory=True)
        self.master = alloc(torch.float32)
        self.m = alloc(torch.float32)
        self.v = alloc(torch.float32) if optimizer != DPO_OPT_LION else None
        self.n = alloc(torch.float32) if optimizer == DPO_OPT_ADAN else None
        self.grad_prev = alloc(torch.float32) if optimizer == DPO_OPT_ADAN else None
        self.grad = (host_alloc if host_grad else alloc)(tdt[grad_dtype])
        self.param = ((host_alloc if host_param else alloc)(torch.bfloat16)
                      if param_dtype == DPO_BF16 else None)
        keep_stash = delay == 1 if keep_stash is None else keep_stash
        self.stash = alloc(tdt[stash_dtype]) if keep_stash else None
        self.ef = alloc(torch.float32) if ef else None
        if x0 is not None:
            self._fill_master(x0)
        self.hp = dpo_hparams(beta1, beta2, eps, weight_decay, ef_lambda if ef else 0.0,
                              max_grad_norm, delay, correction, optimizer, beta3,
                              momentum_decay, dc_lambda, stash_mode)
        self.wd_on = list(wd_on) if wd_on is not None else [True] * len(numels)
        self.sync = list(sync) if sync is not None else [False] * len(numels)
        self.ctx = None
        self._clip_src = None
        self._capturable = False
        self._lr_src = None
        self._init(init_mode, stream)

    def _init(self, init_mode, stream) -> None:
        table = []
        for i, (cnt, off) in enumerate(zip(self.layout.numels, self.layout.offsets)):
            ptr = lambda t: (t.data_ptr() + off * t.element_size()) if t is not None else None
            flags = (DPO_WD_ON if self.wd_on[i] else 0) | (DPO_SYNC if self.sync[i] else 0)
            table.append(dpo_tensor(ptr(self.param), ptr(self.master), ptr(self.m), ptr(self.v),
                                    ptr(self.stash), ptr(self.ef), ptr(self.grad), ptr(self.n),
                                    ptr(self.grad_prev), cnt, flags))
        self.table = table
        self.ctx = dpo_init(table, self.param_dtype, self.stash_dtype, self.grad_dtype, self.hp,
                            init_mode, stream)
        if self._clip_src is not None:
            dpo_set_clip_source(self.ctx, self._clip_src)
        if self._capturable:   # a rebuilt context (use_host_io) keeps the mode
            dpo_set_capturable(self.ctx, True, self._lr_src, stream)

    def use_host_io(self, grad: bool = True, param: bool = True, stream=None) -> None:
        """Move the grad and/or bf16 param arenas to pinned host memory (their
        contents copied) and rebuild the context over them, keeping the step
        counter and all device state: from then on each step reads its
        gradients from and writes its new weights to host memory directly."""
        torch = self.torch
        k, k0 = self.k, dpo_get_phase_start(self.ctx)
        torch.cuda.synchronize(self.device)
        if param and self.hp.stash_mode == DPO_STASH_PINGPONG:
            # host weights take the copying stash: put both versions in their
            # buffers' own roles first
            latest, stale = self.role_arenas()
            if latest is not self.param:
                self.param.copy_(latest)
                self.stash.copy_(stale)
            self.hp.stash_mode = DPO_STASH_COPY
        dpo_destroy(self.ctx)
        self.ctx = None
        to_host = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True).copy_(t)
        if grad and self.grad.is_cuda:
            self.grad = to_host(self.grad)
        if param and self.param is not None and self.param.is_cuda:
            self.param = to_host(self.param)
        self._init(DPO_INIT_RESUME, stream)
        dpo_set_step(self.ctx, k)
        dpo_set_phase_start(self.ctx, k0)

    def view(self, arena, i: int):
        off, cnt = self.layout.offsets[i], self.layout.numels[i]
        return arena[off:off + cnt]

    def _fill_master(self, x0) -> None:
        """Copy start weights into the master arena (see the class notes for
        the forms ``x0`` may take)."""
        lay = self.layout
        if isinstance(x0, (list, tuple)):
            if len(x0) != len(lay.numels):
                raise ValueError(f"x0 has {len(x0)} tensors for {len(lay.numels)}")
            for i, t in enumerate(x0):
                self.view(self.master, i).copy_(t.reshape(-1))
            return
        flat = x0.reshape(-1)
        if flat.numel() == lay.total:
            self.master.copy_(flat)
        elif flat.numel() == sum(lay.numels):
            start = 0
            for i, n in enumerate(lay.numels):
                self.view(self.master, i).copy_(flat[start:start + n])
                start += n
        else:
            raise ValueError(f"x0 has {flat.numel()} elements: expected {sum(lay.numels)} "
                             f"(the tensors one after another) or {lay.total} (arena layout)")

    def grads(self, i: int):
        return self.view(self.grad, i)

    def _swapped(self, i: int) -> bool:
        """Ping-pong stash: tensor i's param and stash buffers hold each
        other's role (include/dpo.h, DPO_STASH_PINGPONG)."""
        if self.hp.stash_mode != DPO_STASH_PINGPONG or self.delay != 1 or self.sync[i]:
            return False
        p, _ = dpo_read_weights(self.ctx, DPO_LATEST, i)
        return p != self.table[i].param

    def stale(self, i: int):
        """What the next forward/backward reads (dpo_read_weights(DPO_STALE))."""
        if self.delay == 1 and not self.sync[i]:
            return self.view(self.param if self._swapped(i) else self.stash, i)
        return self.latest(i)

    def role_arenas(self):
        """(latest, stale) arenas, each tensor in its role: the param and stash
        arenas, or (ping-pong stash, odd calls) copies with the delayed
        tensors' slices exchanged."""
        if self.stash is None or not any(self._swapped(i) for i in range(len(self.sync))):
            return self.param, self.stash
        latest, stale = self.param.clone(), self.stash.clone()
        for i in range(len(self.sync)):
            if self._swapped(i):
                self.view(latest, i).copy_(self.view(self.stash, i))
                self.view(stale, i).copy_(self.view(self.param, i))
        return latest, stale

    def set_delay(self, delay: int, stream=None) -> None:
        """Switch between synchronous and delayed training (dpo_set_delay)."""
        dpo_set_delay(self.ctx, delay, stream)
        self.delay = delay
        self.hp.delay = delay

    def latest(self, i: int):
        if self.param is None:
            return self.view(self.master, i)
        return self.view(self.stash if self._swapped(i) else self.param, i)

    def step(self, lr: Optional[float] = None, stream=None) -> None:
        dpo_step(self.ctx, self.lr if lr is None else lr, stream)

    def set_capturable(self, on: bool = True, lr_source=None, stream=None) -> None:
        """Capturable mode (dpo_set_capturable): the step counters live on
        the device, so a step captured in a CUDA graph can be replayed.
        ``lr_source``: a one-element float32 device tensor read at every
        step (kept alive here), or None for the lr passed to step()."""
        dpo_set_capturable(self.ctx, on, lr_source, stream)
        self._capturable = bool(on)
        self._lr_src = lr_source if on else None

    def set_timing(self, on: bool = True) -> None:
        """Record CUDA events around the norm pass and the fused step of
        every step (dpo_set_timing); read them with kernel_times()."""
        dpo_set_timing(self.ctx, on)

    def kernel_times(self):
        """(norm-pass ms, fused-step ms, calls) summed over the steps timed
        since the last read (dpo_get_timing); waits for those steps."""
        return dpo_get_timing(self.ctx)

    def grad_sqnorm(self, acc, stream=None) -> None:
        """Add this context's sum of g^2 to ``acc`` (dpo_grad_sqnorm)."""
        dpo_grad_sqnorm(self.ctx, acc, stream)

    def set_clip_source(self, acc=None) -> None:
        """Clip from the sum of squares in ``acc`` (a float64 device tensor
        kept alive here), or from this context's own norm when None."""
        dpo_set_clip_source(self.ctx, acc)
        self._clip_src = acc

    def restash(self, stream=None) -> None:
        dpo_stash(self.ctx, stream)

    @property
    def k(self) -> int:
        return dpo_get_step(self.ctx)

    def state_dict(self) -> dict:
        """Every state arena, the step counter k, the start of the current
        delayed phase (Alg. 1's t = k - k0) and the delay mode."""
        bufs = {n: getattr(self, n) for n in STATE_BUFFERS}
        return {"k": self.k, "phase_start": dpo_get_phase_start(self.ctx), "delay": self.delay,
                **{n: b.clone() for n, b in bufs.items() if b is not None}}

    def load_state(self, sd: dict) -> None:
        """Restore a state_dict into a context built with init_mode
        DPO_INIT_RESUME and the same delay mode."""
        if "delay" in sd and int(sd["delay"]) != self.delay:
            raise ValueError(f"checkpoint taken with delay {sd['delay']}, context has {self.delay}")
        for n in STATE_BUFFERS:
            if getattr(self, n) is not None:
                getattr(self, n).copy_(sd[n])
        dpo_set_step(self.ctx, int(sd["k"]))
        dpo_set_phase_start(self.ctx, int(sd.get("phase_start", 0)))

    def close(self) -> None:
        if getattr(self, "ctx", None):
            dpo_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
