"""The C ABI from plain C. Small C programs (tests/c_abi/), built with the
host C compiler against include/dpo.h and include/dpo_muon.h and linked to
libdpo.so, with no Python or PyTorch in them, own their buffers (CUDA runtime
allocations) and write their results, which equal the oracle's on the same
seeded inputs:
- consumer.c: one-step-delayed AdamW with Error Feedback and global-norm
  clipping (Alg. 1, Eq. (1), App. E.1) through dpo_init / dpo_step /
  dpo_read_weights / dpo_get_flags / dpo_get_step;
- muon_consumer.c: delayed Muon with Error Feedback (Alg. 2) on a wide, a
  tall and a padded matrix through dpo_muon_init / dpo_muon_step /
  dpo_muon_get_status / dpo_muon_get_step."""
from __future__ import annotations

import os
import shutil
import struct
import subprocess

import numpy as np
import pytest

import oracle
from paper_2606_30634_gb300 import dpo, synth
from oracle.muon import DelayedMuon as OracleMuon, MuonHParams
from parity_util import (TOL_RUN, bf16_raw_ulps_above_floor, bf16_ulps, rel_err)
from test_muon_parity import _flat, close_with_flips

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
NUMELS = [1000, 37, 4099, 8]       # ragged: packet tails of 0, 5, 3 and 0 elements
STEPS = 4
SEED = 0xC0DE
LR, CLIP = 3e-4, 0.02              # below these gradients' norm (about 0.1): clipping is on


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home:
        return home
    nvcc = shutil.which("nvcc")
    return os.path.dirname(os.path.dirname(nvcc)) if nvcc else "/usr/local/cuda"


def _build_consumer(out_dir: str, name: str = "consumer") -> str:
    lib = dpo.lib_path()
    dpo.load()   # builds libdpo.so when it is missing or stale
    cuda = _cuda_home()
    exe = os.path.join(out_dir, name)
    cmd = [os.environ.get("CC", "gcc"), "-std=c11", "-O2", "-Wall", "-Werror",
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
           os.path.join(HERE, "c_abi", name + ".c"), "-o", exe, lib,
           "-L", os.path.join(cuda, "lib64"), "-lcudart",
           f"-Wl,-rpath,{os.path.dirname(lib)}:{os.path.join(cuda, 'lib64')}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, f"building the C consumer failed:\n{r.stdout}\n{r.stderr}"
    return exe


def test_plain_c_consumer_matches_the_oracle(tmp_path):
    exe = _build_consumer(str(tmp_path))
    total = sum(NUMELS)
    x0 = synth.host_normal(SEED, synth.STREAM_INIT, 0, 0, total, 0.02)
    grads = [synth.host_normal(SEED, synth.STREAM_GRAD, k, 0, total, 1e-3, synth.BF16)
             for k in range(1, STEPS + 1)]
    inp, outp = tmp_path / "in.bin", tmp_path / "out.bin"
    with open(inp, "wb") as f:
        f.write(struct.pack("<ii", len(NUMELS), STEPS))
        f.write(np.asarray(NUMELS, np.int64).tobytes())
        f.write(struct.pack("<ff", LR, CLIP))
        f.write(x0.astype(np.float32).tobytes())
        for g in grads:
            f.write(g.astype(np.uint16).tobytes())
    r = subprocess.run([exe, str(inp), str(outp)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, f"the C consumer failed:\n{r.stdout}\n{r.stderr}"

    raw = open(outp, "rb").read()
    o = 0
    master = np.frombuffer(raw, np.float32, total, o)
    o += 4 * total
    latest = np.frombuffer(raw, np.uint16, total, o)
    o += 2 * total
    stale = np.frombuffer(raw, np.uint16, total, o)
    o += 2 * total
    norm, clip, flags, k = struct.unpack_from("<dfIq", raw, o)

    offs = np.concatenate([[0], np.cumsum(NUMELS)])
    hp = oracle.HParams(lr=LR, ef_lambda=1.0, max_grad_norm=CLIP).as_f32()
    ref = oracle.DelayedOptimizer(np.split(x0.astype(np.float64), offs[1:-1]), hp, ef=True,
                                  x_store=oracle.F32, stash_store=oracle.BF16,
                                  param_store=oracle.BF16, wd_on=[True] * len(NUMELS))
    for g in grads:
        ref.step(synth.bf16_bits_to_f32(g).astype(np.float64), tag=ref.read_weights("stale")[1])
    assert k == STEPS and flags == 0
    assert norm == pytest.approx(np.sqrt(ref.last_sqnorm), rel=1e-6)
    assert clip == pytest.approx(ref.last_clip, rel=1e-6) and clip < 0.5
    assert rel_err(master.astype(np.float64), ref.x) <= TOL_RUN
    ref_latest, _ = ref.read_weights("latest")
    ref_stale, _ = ref.read_weights("stale")
    for got, want in ((latest, ref_latest), (stale, ref_stale)):
        assert bf16_ulps(got, want) <= 1.0
        assert bf16_raw_ulps_above_floor(got, want)[0] <= 1


MUON_SHAPES = [(256, 768), (768, 256), (300, 700)]   # wide, tall (transposed), padded
MUON_STEPS, MUON_NS, MUON_LR = 3, 1, 2e-3


def test_plain_c_muon_consumer_matches_the_oracle(tmp_path):
    """Three calls (EF from the second), one Newton-Schulz step. The bars are
    the Muon parity tests': the momentum at the run bar, the weights
    elementwise except where a bf16 rounding of O flipped, by at most
    lr r 2^-7 per call."""
    exe = _build_consumer(str(tmp_path), "muon_consumer")
    sizes = [r * c for r, c in MUON_SHAPES]
    total = sum(sizes)
    x0 = synth.host_normal(SEED, synth.STREAM_INIT, 0, 0, total, 0.02)
    grads = [synth.host_normal(SEED, synth.STREAM_GRAD, k, 0, total, 1e-3, synth.BF16)
             for k in range(1, MUON_STEPS + 1)]
    inp, outp = tmp_path / "in.bin", tmp_path / "out.bin"
    with open(inp, "wb") as f:
        f.write(struct.pack("<iii", len(MUON_SHAPES), MUON_STEPS, MUON_NS))
        f.write(np.asarray([r for r, _ in MUON_SHAPES], np.int64).tobytes())
        f.write(np.asarray([c for _, c in MUON_SHAPES], np.int64).tobytes())
        f.write(struct.pack("<f", MUON_LR))
        f.write(x0.astype(np.float32).tobytes())
        for g in grads:
            f.write(g.astype(np.uint16).tobytes())
    r = subprocess.run([exe, str(inp), str(outp)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, f"the C consumer failed:\n{r.stdout}\n{r.stderr}"

    raw = open(outp, "rb").read()
    master = np.frombuffer(raw, np.float32, total, 0)
    mom = np.frombuffer(raw, np.float32, total, 4 * total)
    param = np.frombuffer(raw, np.uint16, total, 8 * total)
    stash = np.frombuffer(raw, np.uint16, total, 10 * total)
    status, k = struct.unpack_from("<Iq", raw, 12 * total)

    offs = np.concatenate([[0], np.cumsum(sizes)])
    split = lambda a: [a[offs[i]:offs[i + 1]].reshape(sh) for i, sh in enumerate(MUON_SHAPES)]
    hp = MuonHParams(lr=MUON_LR, ef_lambda=1.0, ns_steps=MUON_NS, ns_store=oracle.BF16).as_f32()
    ref = OracleMuon([x.astype(np.float64) for x in split(x0)], hp, ef=True, x_store=oracle.F32,
                     stash_store=oracle.BF16, param_store=oracle.BF16)
    for g in grads:
        ref.step([m.astype(np.float64) for m in split(synth.bf16_bits_to_f32(g))])
    assert status == 0 and k == MUON_STEPS
    du = MUON_LR * 0.2 * np.sqrt(max(max(sh) for sh in MUON_SHAPES)) * 2.0 ** -7
    as_f64 = lambda bits: synth.bf16_bits_to_f32(np.asarray(bits)).astype(np.float64)
    assert rel_err(mom.astype(np.float64), _flat(ref.mom)) <= TOL_RUN
    close_with_flips(master, _flat(ref.x), TOL_RUN, MUON_STEPS * du, 1e-3)
    close_with_flips(as_f64(param), _flat(ref.param), 2.0 ** -7, MUON_STEPS * du, 1e-3)
    close_with_flips(as_f64(stash), _flat(ref.stash), 2.0 ** -7, (MUON_STEPS - 1) * du, 1e-3)
