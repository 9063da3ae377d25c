"""bench.py's own paths on a GPU, on small sets: each prints one JSON line with
every key its contract asks for (the elementwise step with its end-to-end
figures, delayed Muon with its CUDA-graph replay, and the delayed-Muon entry
the default line carries), with a roofline fraction in a sane range. The
full-size lines are the benchmark's own run; this keeps its code paths
exercised by the test suite."""
from __future__ import annotations

import json
import os
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402

TOP = ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
       "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "cpu_baseline", "e2e",
       "gpu_launches", "clocks")


def _line(capsys, argv):
    assert bench.main(argv) == 0
    out = [x for x in capsys.readouterr().out.splitlines() if x.startswith("{")]
    assert len(out) == 1
    line = json.loads(out[0])
    missing = [k for k in TOP if k not in line]
    assert not missing, missing
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in line["roofline"], k
    for k in ("sm_mhz", "sm_max_mhz", "reasons"):
        assert k in line["clocks"], k
    return line


def test_elementwise_line_with_end_to_end(capsys):
    line = _line(capsys, ["--workload", "gpt2-small-124M", "--steps", "3", "--warmup", "3",
                          "--no-cpu-baseline", "--e2e-steps", "2"])
    r = line["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and 0.3 < r["frac"] < 1.3
    assert line["gpu_launches"] == 3 and line["value"] > 0
    e = line["e2e"]
    assert e["h2d_bytes_per_step"] > 0 and 0 < e["d2h_bytes_per_step"] <= 64
    assert e["value"] > 0
    assert e["link_frac"] is None or 0.1 < e["link_frac"] < 2.0
    w = e["weights_to_host"]
    assert w["d2h_bytes_per_step"] == w["h2d_bytes_per_step"] and w["value"] > 0
    assert e["staged"]["value"] > 0


def test_muon_line_with_graph_replay(capsys):
    line = _line(capsys, ["--optimizer", "muon", "--workload", "gpt2-small-124M", "--steps", "3",
                          "--warmup", "3", "--no-cpu-baseline", "--no-library-ns", "--graph"])
    r = line["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and 0.1 < r["frac"] < 1.3
    # AdamW's step, momentum, norm, apply, one normalisation per shape group
    # (3) and 15 GEMM launches (the three groups share each product's launch)
    assert line["gpu_launches"] == 3 * (1 + 3 + 3 + 15)
    assert line["graph"]["ms_per_step"] > 0


def test_muon_entry_of_the_default_line():
    from paper_2606_30634_gb300.synth import workloads as W
    args = bench.parse_args(["--workload", "gpt2-small-124M", "--muon-steps", "2"])
    entry = bench.run_muon_secondary(args, W.GPT2_SMALL, 1, 0, 0)
    assert entry["value"] > 0 and entry["steps"] == 2
    g = entry["gemm"]
    assert g["bound"] == "tensor" and 0.1 < g["frac"] < 1.3 and g["gemm_ms_per_step"] > 0
