"""The C-ABI libraries load and export what include/*.h declares, and the
host-side argument checks of dpo_init reject bad tables before touching the
GPU (no compute call is made here; runs without a GPU)."""
from __future__ import annotations

import ctypes
import glob
import os
import re

import pytest

from paper_2606_30634_gb300 import build as pkg_build
from paper_2606_30634_gb300 import dpo, muon

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

HEADER_LIB = {"dpo.h": "libdpo.so", "dpo_muon.h": "libdpo.so", "dpo_synth.h": "libdpo_synth.so"}


def declared_functions(header: str):
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = "\n".join(l for l in text.splitlines() if not l.lstrip().startswith("#"))
    names = []
    for stmt in text.split(";"):
        stmt = stmt.strip()
        if "(" not in stmt or stmt.startswith("typedef") or "{" in stmt.split("(")[0]:
            continue
        m = re.search(r"(\w+)\s*\($", stmt.split("(")[0] + "(")
        if m and m.group(1) not in ("extern",):
            names.append(m.group(1))
    return names


def test_every_header_is_mapped_to_a_library():
    headers = {os.path.basename(h) for h in glob.glob(os.path.join(ROOT, "include", "*.h"))}
    assert headers == set(HEADER_LIB)


@pytest.mark.parametrize("header", sorted(HEADER_LIB))
def test_library_exports_every_declared_symbol(header):
    libs = pkg_build.build()
    lib = ctypes.CDLL(libs[HEADER_LIB[header]])
    names = declared_functions(os.path.join(ROOT, "include", header))
    assert len(names) >= 5
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_python_binding_wraps_every_dpo_entry_point():
    names = declared_functions(os.path.join(ROOT, "include", "dpo.h"))
    assert set(names) == set(dpo.EXPORTS)
    for n in names:
        assert callable(getattr(dpo, n))


def test_python_binding_types_every_muon_entry_point():
    names = declared_functions(os.path.join(ROOT, "include", "dpo_muon.h"))
    assert set(names) == set(muon.EXPORTS)
    L = muon.lib()
    for n in names:
        assert getattr(L, n).argtypes is not None


# ---- dpo_muon_init host-side validation (returns before any CUDA call) ----

def _m(i, rows=64, cols=96, **kw):
    step = 1 << 20
    b = BASE + (64 + i) * 16 * step
    d = dict(param=b, master=b + step, mom=b + 2 * step, stash=b + 3 * step, ef=None,
             grad=b + 4 * step, rows=rows, cols=cols, flags=dpo.DPO_WD_ON)
    d.update(kw)
    return muon.dpo_matrix(**d)


def _muon_init(mats, hp=None, sdt=dpo.DPO_BF16, gdt=dpo.DPO_BF16, mode=0):
    L = muon.lib()
    arr = (muon.dpo_matrix * max(1, len(mats)))(*mats)
    out = ctypes.c_void_p(123)
    rc = L.dpo_muon_init(ctypes.byref(out), arr, len(mats), sdt, gdt,
                         ctypes.byref(hp or muon.hparams()), mode, None)
    return rc, out.value, L.dpo_muon_last_error(None).decode()


@pytest.mark.parametrize("case,code", [
    ("bad_dtype", dpo.DPO_EDTYPE), ("momentum_one", dpo.DPO_EINVAL),
    ("ns_steps", dpo.DPO_EINVAL), ("negative_shape", dpo.DPO_EINVAL),
    ("no_stash", dpo.DPO_EINVAL), ("ef_mismatch", dpo.DPO_EINVAL),
    ("misaligned", dpo.DPO_EALIGN), ("no_master", dpo.DPO_EINVAL), ("bad_mode", dpo.DPO_EINVAL),
    ("bad_correction", dpo.DPO_EINVAL)])
def test_muon_init_rejects(case, code):
    mats, hp, kw = [_m(0), _m(1, rows=300, cols=20)], muon.hparams(), {}
    if case == "bad_dtype":
        kw["gdt"] = 7
    elif case == "momentum_one":
        hp = muon.hparams(momentum=1.0)
    elif case == "ns_steps":
        hp = muon.hparams(ns_steps=17)
    elif case == "negative_shape":
        mats[1] = _m(1, rows=-1)
    elif case == "no_stash":
        mats[0] = _m(0, stash=None)
    elif case == "ef_mismatch":
        mats[0] = _m(0, ef=BASE + (1 << 30))
    elif case == "misaligned":
        mats[1] = _m(1, master=BASE + (1 << 31) + 16)
    elif case == "no_master":
        mats[1] = _m(1, master=None)
    elif case == "bad_mode":
        kw["mode"] = 5
    elif case == "bad_correction":
        hp = muon.hparams(correction=3)
    rc, out, msg = _muon_init(mats, hp, **kw)
    assert rc == code and out is None and msg


# ---- host-side validation (returns before any CUDA call) -----------------

def _hp(**kw):
    d = dict(beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1, ef_lambda=0.0,
             max_grad_norm=0.0, delay=1)
    d.update(kw)
    return dpo.dpo_hparams(**d)


BASE = 1 << 40   # fake, never dereferenced: validation fails before any use


def _t(i, numel=100, **kw):
    step = 1 << 20
    b = BASE + i * 16 * step
    d = dict(param=b, master=b + step, m=b + 2 * step, v=b + 3 * step, stash=b + 4 * step,
             ef=None, grad=b + 5 * step, numel=numel, flags=dpo.DPO_WD_ON)
    d.update(kw)
    return dpo.dpo_tensor(**d)


def _init(table, hp=None, pdt=dpo.DPO_BF16, sdt=dpo.DPO_F32, gdt=dpo.DPO_BF16, mode=0):
    L = dpo.load()
    arr = (dpo.dpo_tensor * max(1, len(table)))(*table)
    out = ctypes.c_void_p(123)
    rc = L.dpo_init(ctypes.byref(out), arr if table else None, len(table), pdt, sdt, gdt,
                    ctypes.byref(hp or _hp()), mode, None)
    return rc, out.value, L.dpo_last_error(None).decode()


@pytest.mark.parametrize("case,expect", [
    ("misaligned_master", dpo.DPO_EALIGN),
    ("misaligned_grad", dpo.DPO_EALIGN),
    ("overlap", dpo.DPO_EINVAL),
    ("negative_numel", dpo.DPO_EINVAL),
    ("null_master", dpo.DPO_EINVAL),
    ("missing_stash", dpo.DPO_EINVAL),
    ("ef_mixed", dpo.DPO_EINVAL),
    ("lambda_without_ef", dpo.DPO_EINVAL),
    ("bad_dtype", dpo.DPO_EDTYPE),
    ("bad_beta", dpo.DPO_EINVAL),
    ("nan_eps", dpo.DPO_EINVAL),
    ("bad_delay", dpo.DPO_EINVAL),
    ("fp32_param_buffer", dpo.DPO_EINVAL),
    ("bf16_no_param", dpo.DPO_EINVAL),
    ("empty_table", dpo.DPO_EINVAL),
    ("bad_flags", dpo.DPO_EINVAL),
    ("bad_mode", dpo.DPO_EINVAL),
    ("bad_stash_mode", dpo.DPO_EINVAL),
    ("pingpong_fp32_stash", dpo.DPO_EDTYPE),
    ("pingpong_sapipe", dpo.DPO_EINVAL),
])
def test_init_rejects(case, expect):
    tbl = [_t(0), _t(1, numel=7)]
    hp, kw = None, {}
    if case == "misaligned_master":
        tbl[1] = _t(1, master=tbl[1].master + 4)
    elif case == "misaligned_grad":
        tbl[0] = _t(0, grad=tbl[0].grad + 2)
    elif case == "overlap":
        tbl[1] = _t(1, m=tbl[0].v + 32)
    elif case == "negative_numel":
        tbl[1] = _t(1, numel=-1)
    elif case == "null_master":
        tbl[0] = _t(0, master=None)
    elif case == "missing_stash":
        tbl[1] = _t(1, stash=None)
    elif case == "ef_mixed":
        tbl[0] = _t(0, ef=BASE + (1 << 30))
    elif case == "lambda_without_ef":
        hp = _hp(ef_lambda=1.0)
    elif case == "bad_dtype":
        kw = dict(gdt=7)
    elif case == "bad_beta":
        hp = _hp(beta2=1.0)
    elif case == "nan_eps":
        hp = _hp(eps=float("nan"))
    elif case == "bad_delay":
        hp = _hp(delay=2)
    elif case == "fp32_param_buffer":
        kw = dict(pdt=dpo.DPO_F32)
    elif case == "bf16_no_param":
        tbl[0] = _t(0, param=None)
    elif case == "empty_table":
        tbl = []
    elif case == "bad_flags":
        tbl[0] = _t(0, flags=8)
    elif case == "bad_mode":
        kw = dict(mode=5)
    elif case == "bad_stash_mode":
        hp = _hp(stash_mode=2)
    elif case == "pingpong_fp32_stash":
        hp = _hp(stash_mode=dpo.DPO_STASH_PINGPONG)   # the helper's stash is fp32
    elif case == "pingpong_sapipe":
        hp = _hp(stash_mode=dpo.DPO_STASH_PINGPONG, correction=dpo.DPO_CORR_SAPIPE_SAME)
        kw = dict(sdt=dpo.DPO_BF16)
    rc, out, msg = _init(tbl, hp, **kw)
    assert rc == expect, msg
    assert out is None
    assert msg


def test_zero_length_tensor_is_not_validated():
    """numel == 0 entries are skipped entirely (their pointers are unused)."""
    tbl = [_t(0, numel=0, master=None, grad=3), _t(1, master=BASE + 8)]
    rc, _, msg = _init(tbl)
    assert rc == dpo.DPO_EALIGN and "tensor 1" in msg


def test_calls_on_null_context():
    L = dpo.load()
    assert L.dpo_step(None, 1e-3, None) == dpo.DPO_EINVAL
    assert L.dpo_stash(None, None) == dpo.DPO_EINVAL
    k = ctypes.c_int64()
    assert L.dpo_get_step(None, ctypes.byref(k)) == dpo.DPO_EINVAL
    assert L.dpo_set_step(None, 3) == dpo.DPO_EINVAL
    L.dpo_destroy(None)


@pytest.mark.parametrize("program", ["consumer", "muon_consumer"])
def test_headers_serve_a_plain_c_program(program, tmp_path):
    """include/dpo.h and include/dpo_muon.h compile as C11 (no C++), and a C
    program using them links against libdpo.so: the GPU tests run the same
    programs (tests/test_c_consumer.py)."""
    import shutil
    import subprocess
    cc = os.environ.get("CC", "gcc")
    nvcc = shutil.which("nvcc")
    if shutil.which(cc) is None or nvcc is None:
        pytest.skip("no C compiler or CUDA toolkit")
    cuda = os.path.dirname(os.path.dirname(nvcc))
    here = os.path.dirname(os.path.abspath(__file__))
    lib = pkg_build.build()["libdpo.so"]
    exe = str(tmp_path / program)
    r = subprocess.run([cc, "-std=c11", "-O2", "-Wall", "-Wextra", "-Werror", "-pedantic",
                        "-I", os.path.join(os.path.dirname(here), "include"),
                        "-I", os.path.join(cuda, "include"),
                        os.path.join(here, "c_abi", program + ".c"), "-o", exe, lib,
                        "-L", os.path.join(cuda, "lib64"), "-lcudart"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    assert os.path.getsize(exe) > 0
