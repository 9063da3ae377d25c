"""Parity harness: the CUDA path (through the C ABI) and the oracle, run on the
same seeded inputs and compared element by element.

Tolerances (the error metric below):
  fp32 state   err = max_i |gpu_i - ref_i| / max(|ref_i|, 1e-2 rms(ref))
               <= 1e-6 after one step, <= 1e-4 after any number of steps;
               except for buffers named in ``normwise`` (the EF buffer of the
               1000-step quadratic loop), held to the normwise relative max
               error max_i |gpu_i - ref_i| / max_i |ref_i| <= 1e-4: there the
               delayed EF feedback loop amplifies any per-step rounding
               difference (the oracle itself, started one ulp away, drifts
               by 7.5e-5 elementwise), so the elementwise figure measures the
               loop's conditioning rather than the implementation;
  bf16 copies  within 1 bf16 ulp of the oracle's bf16 value, the ulp taken at
               the same floored scale max(|ref_i|, 1e-2 rms(ref)): where
               x_{t+1} = x_t - u cancels to a value far below the tensor's
               scale, fp32 rounding differences of the master (allowed by
               the fp32 metric) are many ulps of the tiny bf16 value;
               and, on every element with |ref_i| >= 1e-2 rms(ref), within
               1 bf16 code point unfloored (the ordered-integer distance of
               the two bit patterns). The number of elements under the floor
               is reported beside it.

DPO_PARITY_LOG=<file> appends every comparison's errors as a JSON line; the
worst figure of every buffer per test is also kept in WORST, which the test
session prints at its end (tests/conftest.py).
"""
from __future__ import annotations

import json
import os

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

import oracle
from paper_2606_30634_gb300 import dpo, synth

TOL_ONE_STEP = 1e-6
TOL_RUN = 1e-4

# test id -> {buffer metric: worst value over the test's comparisons}
WORST: dict = {}


def record(test: str, errors: dict) -> None:
    """Keep the worst value of every metric of one comparison (elementwise
    figures of normwise-held buffers and the under-floor counts included)."""
    w = WORST.setdefault(test or "?", {})
    for key, val in errors.items():
        w[key] = max(w.get(key, 0), val)

STORE = {dpo.DPO_F32: oracle.F32, dpo.DPO_BF16: oracle.BF16}
RULE = {dpo.DPO_OPT_ADAMW: oracle.RULE_ADAMW, dpo.DPO_OPT_NADAM: oracle.RULE_NADAM,
        dpo.DPO_OPT_LION: oracle.RULE_LION, dpo.DPO_OPT_ADAN: oracle.RULE_ADAN}


def rel_err(gpu: np.ndarray, ref: np.ndarray) -> float:
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    if not np.array_equal(np.isfinite(gpu), np.isfinite(ref)):
        return float("inf")
    fin = np.isfinite(ref)
    gpu, ref = gpu[fin], ref[fin]
    if ref.size == 0:
        return 0.0
    floor = 1e-2 * np.sqrt(np.mean(ref * ref))
    den = np.maximum(np.abs(ref), floor if floor > 0 else np.finfo(np.float64).tiny)
    return float(np.max(np.abs(gpu - ref) / den))


def norm_err(gpu: np.ndarray, ref: np.ndarray) -> float:
    """max_i |gpu_i - ref_i| / max_i |ref_i| over the finite elements."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    if not np.array_equal(np.isfinite(gpu), np.isfinite(ref)):
        return float("inf")
    fin = np.isfinite(ref)
    scale = np.max(np.abs(ref[fin])) if fin.any() else 0.0
    if scale == 0.0:
        return float(np.max(np.abs(gpu[fin] - ref[fin]))) if fin.any() else 0.0
    return float(np.max(np.abs(gpu[fin] - ref[fin])) / scale)


def bf16_ord(bits: np.ndarray) -> np.ndarray:
    b = np.asarray(bits, np.uint16).astype(np.int32)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def bf16_bits_of(values: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of values that are exactly bf16 (the oracle's)."""
    f = np.asarray(values, np.float64).astype(np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def bf16_ulps(gpu_bits: np.ndarray, ref_values: np.ndarray) -> float:
    """max_i |gpu_i - ref_i| in bf16 ulps of max(|ref_i|, 1e-2 rms(ref))."""
    if len(gpu_bits) == 0:
        return 0.0
    ref = np.asarray(ref_values, np.float64)
    gpu = (np.asarray(gpu_bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    if not np.array_equal(np.isfinite(gpu), np.isfinite(ref)):
        return float("inf")
    fin = np.isfinite(ref)
    gpu, ref = gpu[fin], ref[fin]
    if ref.size == 0:
        return 0.0
    floor = 1e-2 * np.sqrt(np.mean(ref * ref))
    scale = np.maximum(np.abs(ref), floor if floor > 0 else 2.0 ** -126)
    ulp = np.exp2(np.floor(np.log2(scale)) - 7)   # bf16: 8 significant bits
    return float(np.max(np.abs(gpu - ref) / ulp))


def bf16_raw_ulps(gpu_bits: np.ndarray, ref_values: np.ndarray) -> int:
    """Unfloored distance in bf16 code points over all elements (reported)."""
    if len(gpu_bits) == 0:
        return 0
    return int(np.max(np.abs(bf16_ord(gpu_bits) - bf16_ord(bf16_bits_of(ref_values)))))


def bf16_raw_ulps_above_floor(gpu_bits: np.ndarray, ref_values: np.ndarray):
    """(distance in bf16 code points over the elements with |ref_i| >=
    1e-2 rms(ref), the number of elements under that floor). Above the floor
    the fp32 masters agree to 1e-4 of |ref_i|, far inside one bf16 spacing
    (2^-8 relative), so their round-to-nearest-even images are at most one
    code point apart."""
    if len(gpu_bits) == 0:
        return 0, 0
    ref = np.asarray(ref_values, np.float64)
    fin = np.isfinite(ref)
    floor = 1e-2 * np.sqrt(np.mean(ref[fin] * ref[fin])) if fin.any() else 0.0
    above = fin & (np.abs(ref) >= floor)
    under = int(np.count_nonzero(fin & ~above))
    if not above.any():
        return 0, under
    d = np.abs(bf16_ord(np.asarray(gpu_bits)[above]) - bf16_ord(bf16_bits_of(ref[above])))
    return int(np.max(d)), under


@dataclass
class Case:
    numels: Sequence[int]
    param_dtype: int = dpo.DPO_BF16
    stash_dtype: int = dpo.DPO_F32
    grad_dtype: int = dpo.DPO_BF16
    ef: bool = False
    ef_lambda: float = 1.0
    max_grad_norm: float = 0.0
    delay: int = 1
    lr: float = 3e-4
    weight_decay: float = 0.1
    wd_on: Optional[Sequence[bool]] = None
    seed: int = 0xD0D0
    grad_sigma: float = 1e-3
    init_sigma: float = 0.02
    correction: int = dpo.DPO_CORR_EF   # with ef: EF, SAPipe same / updated state
    optimizer: int = dpo.DPO_OPT_ADAMW
    beta1: float = 0.9
    beta2: float = 0.95
    beta3: float = 0.99
    momentum_decay: float = 0.004
    dc_lambda: float = 0.0
    sync: Optional[Sequence[bool]] = None      # per tensor: trained synchronously
    schedule: Optional[dict] = None            # call k -> delay mode switched to before it
    host_grad: bool = False     # grad arena in pinned host memory
    host_param: bool = False    # bf16 param arena in pinned host memory
    stash_mode: int = dpo.DPO_STASH_COPY   # or DPO_STASH_PINGPONG (bf16 param and stash)


class Run:
    """A GPU optimizer and an oracle over the same seeded set."""

    def __init__(self, case: Case, device, sample: Optional[np.ndarray] = None):
        import torch
        self.torch = torch
        self.c = case
        self.N = int(sum(case.numels))
        self.offs = np.concatenate([[0], np.cumsum(case.numels)]).astype(np.int64)
        self.gpu = dpo.DelayedAdamW(
            case.numels, param_dtype=case.param_dtype, stash_dtype=case.stash_dtype,
            grad_dtype=case.grad_dtype, lr=case.lr, weight_decay=case.weight_decay,
            ef=case.ef, ef_lambda=case.ef_lambda, max_grad_norm=case.max_grad_norm,
            delay=case.delay, wd_on=case.wd_on, device=device,
            x0=self._dev_x0(device), init_mode=dpo.DPO_INIT_FRESH,
            host_grad=case.host_grad, host_param=case.host_param, correction=case.correction,
            sync=case.sync, keep_stash=True, optimizer=case.optimizer, beta1=case.beta1,
            beta2=case.beta2, beta3=case.beta3, momentum_decay=case.momentum_decay,
            dc_lambda=case.dc_lambda, stash_mode=case.stash_mode)
        # the oracle tracks every element, or only ``sample`` (global indices)
        self.sample = sample
        idx = np.arange(self.N) if sample is None else np.asarray(sample, np.int64)
        self.idx = idx
        x0 = synth.host_normal_at(case.seed, synth.STREAM_INIT, 0, idx, case.init_sigma)
        hp = oracle.HParams(lr=case.lr, beta1=case.beta1, beta2=case.beta2,
                            weight_decay=case.weight_decay,
                            ef_lambda=case.ef_lambda if case.ef else 0.0,
                            max_grad_norm=case.max_grad_norm, delay=case.delay,
                            correction=case.correction, rule=RULE[case.optimizer],
                            beta3=case.beta3, momentum_decay=case.momentum_decay,
                            dc_lambda=case.dc_lambda).as_f32()
        if sample is None:
            parts = np.split(x0.astype(np.float64), self.offs[1:-1])
            wd = case.wd_on
        else:
            parts = [x0.astype(np.float64)]
            wd = None if case.wd_on is None else [True]
            self._mask = None
            if case.wd_on is not None:
                t_of = np.searchsorted(self.offs, idx, side="right") - 1
                self._mask = np.array(case.wd_on, bool)[t_of]
        delayed = None if case.sync is None else [not s_ for s_ in case.sync]
        if sample is not None and delayed is not None:
            delayed = [True]
        self.ref = oracle.DelayedOptimizer(
            parts, hp, ef=case.ef, x_store=oracle.F32, stash_store=STORE[case.stash_dtype],
            param_store=oracle.BF16 if case.param_dtype == dpo.DPO_BF16 else None, wd_on=wd,
            delayed=delayed)
        if sample is not None and case.wd_on is not None:
            self.ref.mask = self._mask.astype(np.uint8)
        t_of_s = np.searchsorted(self.offs, idx, side="right") - 1
        self.sync_mask = (np.zeros(idx.size, bool) if case.sync is None
                          else np.array(case.sync, bool)[t_of_s])
        if sample is not None and case.sync is not None:
            self.ref.delay_mask = (~self.sync_mask).astype(np.uint8)
        # arena index of every tracked element
        t_of = np.searchsorted(self.offs, idx, side="right") - 1
        self._t_of = t_of
        arena_off = np.asarray(self.gpu.layout.offsets, np.int64)
        self.arena_idx = arena_off[t_of] + (idx - self.offs[t_of])
        self._arena_idx_cpu = torch.from_numpy(self.arena_idx)
        self._arena_idx_dev = self._arena_idx_cpu.to(device)
        self.k = 0

    def _dev_x0(self, device):
        import torch
        x0 = torch.zeros(dpo.Layout.of(self.c.numels).total, dtype=torch.float32, device=device)
        lay = dpo.Layout.of(self.c.numels)
        for i, (o, n) in enumerate(zip(lay.offsets, lay.numels)):
            if n:
                synth.dev_normal(self.c.seed, synth.STREAM_INIT, 0, int(self.offs[i]),
                                 x0[o:o + n], self.c.init_sigma)
        return x0

    def draw(self, k: int) -> np.ndarray:
        """Gradient k on both sides: drawn into the GPU's grad arena, and
        returned (tracked elements, fp64) for the oracle."""
        c = self.c
        for i, n in enumerate(c.numels):
            if n:
                synth.dev_normal(c.seed, synth.STREAM_GRAD, k, int(self.offs[i]),
                                 self.gpu.grads(i), c.grad_sigma)
        gdt = synth.BF16 if c.grad_dtype == dpo.DPO_BF16 else synth.F32
        g = synth.host_normal_at(c.seed, synth.STREAM_GRAD, k, self.idx, c.grad_sigma, gdt)
        g = synth.bf16_bits_to_f32(g) if gdt == synth.BF16 else g
        return g.astype(np.float64)

    def step(self, lr: Optional[float] = None, sq: Optional[float] = None, before=None):
        """Draw gradient k+1 on both sides and take one step on each. ``sq``:
        the squared norm the oracle clips from (default: its own gradient's);
        ``before``: called after the draw, before the GPU step."""
        c = self.c
        k = self.k + 1
        if c.schedule and k in c.schedule:
            self.gpu.set_delay(c.schedule[k])
            self.ref.set_delay(c.schedule[k])
        g = self.draw(k)
        if before is not None:
            before(g)
        self.gpu.step(lr)
        if sq is None and c.max_grad_norm > 0 and self.sample is not None:
            sq = self.full_sqnorm(k)
        lr32 = None if lr is None else float(np.float32(lr))
        self.ref.step(g, tag=self.ref.read_weights("stale")[1], lr=lr32, sq=sq)
        self.k = k

    def full_sqnorm(self, k: int) -> float:
        """The oracle's squared norm of the whole k-th gradient (drawn on the
        host in chunks)."""
        c = self.c
        gdt = synth.BF16 if c.grad_dtype == dpo.DPO_BF16 else synth.F32
        total, chunk = 0.0, 1 << 24
        for lo in range(0, self.N, chunk):
            n = min(chunk, self.N - lo)
            g = synth.host_normal(c.seed, synth.STREAM_GRAD, k, lo, n, c.grad_sigma, gdt)
            total += oracle.sqnorm_bf16(g) if gdt == synth.BF16 else oracle.sqnorm_f32(g)
        return total

    def gather(self, arena) -> np.ndarray:
        t = arena.index_select(0, self._arena_idx_dev if arena.is_cuda else self._arena_idx_cpu)
        if t.dtype == self.torch.bfloat16:
            return t.view(self.torch.int16).cpu().numpy().view(np.uint16)
        return t.cpu().numpy()

    def role_values(self):
        """(latest, stale) weights of the tracked elements, each tensor's two
        weight buffers read in their roles (the ping-pong stash swaps them on
        odd calls; include/dpo.h, DPO_STASH_PINGPONG)."""
        g = self.gpu
        p = self.gather(g.param) if g.param is not None else None
        st = self.gather(g.stash) if g.stash is not None else None
        if p is None or st is None or self.c.stash_mode != dpo.DPO_STASH_PINGPONG:
            return p, st
        swapped = np.array([g._swapped(i) for i in range(len(self.c.numels))], bool)
        m = swapped[self._t_of]
        return np.where(m, st, p), np.where(m, p, st)

    def input_mismatch(self) -> np.ndarray:
        """Tracked elements whose master or stash differ bitwise between the
        GPU and the oracle (inputs of the next step)."""
        self.torch.cuda.synchronize()
        bad = self.gather(self.gpu.master).astype(np.float64) != self.ref.x
        _, stale = self.role_values()
        if stale is not None:
            s = stale
            if self.c.stash_dtype == dpo.DPO_BF16:
                s = synth.bf16_bits_to_f32(s)
            bad |= s.astype(np.float64) != self.ref.stash
        return bad

    def compare(self, mask: Optional[np.ndarray] = None) -> dict:
        """Errors of every state buffer against the oracle (over the tracked
        elements, or those ``mask`` selects)."""
        self.torch.cuda.synchronize()
        g, r = self.gpu, self.ref
        sel = np.ones(self.idx.size, bool) if mask is None else mask
        out = {"master": rel_err(self.gather(g.master)[sel], r.x[sel]),
               "m": rel_err(self.gather(g.m)[sel], r.m[sel])}
        if g.v is not None:
            out["v"] = rel_err(self.gather(g.v)[sel], r.v[sel])
        if g.n is not None:
            out["n"] = rel_err(self.gather(g.n)[sel], r.n3[sel])
            out["grad_prev"] = rel_err(self.gather(g.grad_prev)[sel], r.g_prev[sel])
        if g.ef is not None:
            # the update history of a synchronously trained tensor stays
            # untouched (zero on both sides); the metric's floor is taken over
            # the delayed tensors' history, where it carries values
            e = self.gather(g.ef)
            keep = ~self.sync_mask & sel
            out["ef"] = rel_err(e[keep], r.u_prev[keep])
            out["ef_norm"] = norm_err(e[keep], r.u_prev[keep])
            sync_sel = self.sync_mask & sel
            if sync_sel.any():
                out["ef_sync_absdiff"] = float(np.max(np.abs(e[sync_sel] - r.u_prev[sync_sel])))
        # the weight buffers in their roles (the ping-pong stash swaps them);
        # under delay 0 the stale view is the latest weights and the stash
        # buffer is not read (the ping-pong stash refreshes it on leaving
        # delayed training, the copying stash leaves it as it was)
        latest, stale = self.role_values()
        if stale is not None and (g.delay == 1 or self.c.stash_mode == dpo.DPO_STASH_COPY):
            # the stash of a synchronously trained tensor is never read
            keep = ~self.sync_mask & sel
            s, rs = stale[keep], r.stash[keep]
            if self.c.stash_dtype == dpo.DPO_BF16:
                out["stash_ulp"] = bf16_ulps(s, rs)
                out["stash_raw_ulp"], out["stash_under_floor"] = bf16_raw_ulps_above_floor(s, rs)
                out["stash_raw_ulp_all"] = bf16_raw_ulps(s, rs)
            else:
                out["stash"] = rel_err(s, rs)
        if latest is not None:
            p = latest[sel]
            out["param_ulp"] = bf16_ulps(p, r.param[sel])
            out["param_raw_ulp"], out["param_under_floor"] = bf16_raw_ulps_above_floor(
                p, r.param[sel])
            out["param_raw_ulp_all"] = bf16_raw_ulps(p, r.param[sel])
        return out

    def assert_close(self, tol: float, normwise: Sequence[str] = (),
                     mask: Optional[np.ndarray] = None) -> dict:
        e = self.compare(mask)
        test = os.environ.get("PYTEST_CURRENT_TEST", "").rsplit(" (", 1)[0]
        log = os.environ.get("DPO_PARITY_LOG")
        if log:
            with open(log, "a") as f:
                f.write(json.dumps({"test": test, "k": self.k, "tol": tol, **e}) + "\n")
        record(test, e)
        for key, val in e.items():
            if key.endswith("_raw_ulp_all") or key.endswith("_under_floor") or key.endswith("_norm"):
                continue
            if key in normwise:
                assert e[key + "_norm"] <= tol, (key, e)
            elif key.endswith("_absdiff"):
                assert val == 0.0, (key, e)
            elif key.endswith("_ulp"):
                assert val <= 1.0, (key, e)
            else:
                assert val <= tol, (key, e)
        return e

    def close(self):
        self.gpu.close()


def sample_indices(numels: Sequence[int], n_random: int, seed: int = 1, edge: int = 9) -> np.ndarray:
    """Random global indices plus the first and last ``edge`` elements of
    every tensor (tensor boundaries and partial packets)."""
    offs = np.concatenate([[0], np.cumsum(numels)]).astype(np.int64)
    N = int(offs[-1])
    rng = np.random.default_rng(seed)
    parts = [rng.integers(0, N, n_random)]
    for i, n in enumerate(numels):
        if n:
            lo, hi = offs[i], offs[i + 1]
            parts.append(np.arange(lo, min(hi, lo + edge)))
            parts.append(np.arange(max(lo, hi - edge), hi))
    return np.unique(np.concatenate(parts))
