"""Seeded synthetic inputs (binding of include/dpo_synth.h).

Test and benchmark infrastructure, shared by the CUDA side and the oracle
side: it draws the inputs (initial weights, gradients, the quadratic's
curvature, minimiser and noise) and holds none of the optimizer's arithmetic.
Values depend only on (seed, stream, step, global element index), so the
device fill of a whole 6.7e9-element set and the host fill of a sample of its
indices agree bit for bit.

Workload recipe (parameter sets shaped like the paper's models, App. E.2):
  seed      0xD0D0 + workload number
  x_0       N(0, 0.02^2), stream INIT, step 0
  gradients N(0, 1e-3^2) per step, stream GRAD, step = call index k (1-based)
  quadratic a = exp(ln(1e-3) (1 - U)) (log-uniform in [1e-3, 1]), w* ~ N(0, 1),
            noise N(0, 1e-2^2) per step.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

STREAM_INIT, STREAM_GRAD, STREAM_NOISE, STREAM_CURV, STREAM_TARGET = 0, 1, 2, 3, 4
F32, BF16 = 0, 1

_lib = None


def load():
    global _lib
    if _lib is not None:
        return _lib
    from .. import build as _build
    path = _build.build()["libdpo_synth.so"]
    L = ctypes.CDLL(path)
    u64, u32, i64, P = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int64, ctypes.c_void_p
    L.synth_philox.restype = None
    L.synth_philox.argtypes = [ctypes.POINTER(u32), ctypes.POINTER(u32), ctypes.POINTER(u32)]
    L.synth_normal_scale.restype = ctypes.c_float
    L.synth_normal_scale.argtypes = [ctypes.c_double]
    for name in ("synth_host_normal", "synth_dev_normal"):
        getattr(L, name).restype = ctypes.c_int
    L.synth_host_normal.argtypes = [u64, u32, u32, i64, i64, ctypes.c_float, ctypes.c_int, P]
    L.synth_host_normal_at.restype = ctypes.c_int
    L.synth_host_normal_at.argtypes = [u64, u32, u32, P, i64, ctypes.c_float, ctypes.c_int, P]
    L.synth_host_uniform.restype = ctypes.c_int
    L.synth_host_uniform.argtypes = [u64, u32, u32, i64, i64, P]
    L.synth_host_uniform_at.restype = ctypes.c_int
    L.synth_host_uniform_at.argtypes = [u64, u32, u32, P, i64, P]
    L.synth_dev_normal.argtypes = [u64, u32, u32, i64, i64, ctypes.c_float, ctypes.c_int, P, P]
    L.synth_dev_quadratic.restype = ctypes.c_int
    L.synth_dev_quadratic.argtypes = [u64, u32, i64, P, P, P, ctypes.c_float, P, P, ctypes.c_int, P]
    _lib = L
    return L


def philox(ctr, key):
    L = load()
    c = (ctypes.c_uint32 * 4)(*ctr)
    k = (ctypes.c_uint32 * 2)(*key)
    o = (ctypes.c_uint32 * 4)()
    L.synth_philox(c, k, o)
    return list(o)


def normal_scale(sigma: float) -> float:
    return float(load().synth_normal_scale(sigma))


def _rc(rc):
    if rc != 0:
        raise RuntimeError(f"synth call failed ({rc})")


def host_normal(seed, stream, step, offset, n, sigma, dtype=F32) -> np.ndarray:
    """fp32 values (dtype F32) or bf16 bit patterns as uint16 (dtype BF16)."""
    out = np.empty(n, np.float32 if dtype == F32 else np.uint16)
    _rc(load().synth_host_normal(seed, stream, step, offset, n, normal_scale(sigma), dtype,
                                 out.ctypes.data))
    return out


def host_normal_at(seed, stream, step, idx, sigma, dtype=F32) -> np.ndarray:
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    out = np.empty(idx.size, np.float32 if dtype == F32 else np.uint16)
    _rc(load().synth_host_normal_at(seed, stream, step, idx.ctypes.data, idx.size,
                                    normal_scale(sigma), dtype, out.ctypes.data))
    return out


def host_uniform(seed, stream, step, offset, n) -> np.ndarray:
    out = np.empty(n, np.float32)
    _rc(load().synth_host_uniform(seed, stream, step, offset, n, out.ctypes.data))
    return out


def host_uniform_at(seed, stream, step, idx) -> np.ndarray:
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    out = np.empty(idx.size, np.float32)
    _rc(load().synth_host_uniform_at(seed, stream, step, idx.ctypes.data, idx.size,
                                     out.ctypes.data))
    return out


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def curvature_from_uniform(u: np.ndarray) -> np.ndarray:
    """a = exp(ln(1e-3) (1 - u)): log-uniform in [1e-3, 1], as fp32."""
    return np.exp(np.log(1e-3) * (1.0 - u.astype(np.float64))).astype(np.float32)


def dev_normal(seed, stream, step, offset, out, sigma, cuda_stream=None) -> None:
    """Fill the torch tensor ``out`` (fp32 or bf16, contiguous, on the device)
    with draws for indices offset .. offset + out.numel() - 1."""
    import torch
    dtype = F32 if out.dtype == torch.float32 else BF16
    assert out.dtype in (torch.float32, torch.bfloat16) and out.is_contiguous()
    s = cuda_stream if cuda_stream is not None else torch.cuda.current_stream().cuda_stream
    _rc(load().synth_dev_normal(seed, stream, step, offset, out.numel(), normal_scale(sigma),
                                dtype, out.data_ptr(), s))


def dev_quadratic(seed, step, a, wstar, w, noise_sigma, grad, partials, cuda_stream=None) -> None:
    import torch
    s = cuda_stream if cuda_stream is not None else torch.cuda.current_stream().cuda_stream
    _rc(load().synth_dev_quadratic(seed, step, w.numel(), a.data_ptr(), wstar.data_ptr(),
                                   w.data_ptr(), normal_scale(noise_sigma), grad.data_ptr(),
                                   partials.data_ptr(), partials.numel(), s))
