"""Benchmark of the one-step-delayed AdamW step (arXiv 2606.30634, Alg. 1 with
Error Feedback) on a 6.74e9-parameter Llama-7B-shaped tensor set.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dpo|reference]
                    [--workload llama-7B] [--mode ef|std]

A step is one dpo_step over the whole set: every parameter's stale gradient
is consumed and master, m, v, the EF buffer and the bf16 weights are
rewritten; the stale version is the bf16 weights of the previous step, kept
in the second of two weight buffers that swap roles (PipeDream-2BW's double
buffering, --stash pingpong, the default where the layout allows it; --stash
copy writes a separate stash instead) (inputs already resident in HBM when timing
starts; the 148 GB working set is far larger than L2, so no flush is
needed). Prints one JSON line: throughput in parameters updated per second,
the fused kernel's achieved HBM bandwidth against the measured copy peak,
an end-to-end figure through the public API with the gradients coming from
and the new weights going to pinned host memory, and the CPU oracle's
throughput on a bounded sample of the same set.

Under torchrun every rank runs its own full replica on its own GPU (the step
is elementwise, so ranks are independent problems: weak scaling, no
collective on the data path); timing is the maximum over ranks.
"""
from __future__ import annotations

import argparse
import gc
import hashlib
import json
import os
import re
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "params updated/sec and achieved HBM GB/s (% of GB300 peak), 7B-shaped step"
UNIT = "params/s"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
MUON_LR = 2e-3


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=30)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["dpo", "reference"], default="dpo")
    p.add_argument("--workload", default="llama-7B")
    p.add_argument("--mode", choices=["ef", "std", "sapipe-same", "sapipe-updated"],
                   default="ef")
    p.add_argument("--optimizer", choices=["adamw", "nadam", "lion", "adan", "muon"],
                   default="adamw",
                   help="muon: delayed Muon (Alg. 2) on the attention and MLP matrices, "
                        "AdamW on the rest")
    p.add_argument("--ns-steps", type=int, default=5, help="Newton-Schulz steps (muon)")
    p.add_argument("--graph", action="store_true",
                   help="muon: also time the step captured once in a CUDA graph and replayed "
                        "(capturable mode)")
    p.add_argument("--no-library-ns", action="store_true",
                   help="muon: skip timing the cuBLAS Newton-Schulz chain for context")
    p.add_argument("--stash", choices=["auto", "copy", "pingpong"], default="auto",
                   help="pingpong: bf16 param and stash buffers swap roles (no stash store); "
                        "auto: pingpong where the layout allows it (bf16 param and stash, "
                        "standard rule or EF), else copy")
    p.add_argument("--dc-lambda", type=float, default=0.0,
                   help="DC-ASGD compensation strength (Sec. 3.1); 0: off")
    p.add_argument("--wpipe", action="store_true",
                   help="train the second half of the tensor list synchronously (App. B.2)")
    p.add_argument("--e2e-steps", type=int, default=4)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-link-peak", action="store_true",
                   help="skip timing plain pinned-host copies (the e2e path's bound)")
    p.add_argument("--no-secondary", action="store_true",
                   help="skip the clipped Llama-1B step (norm pass and fused step timed apart)")
    p.add_argument("--secondary-steps", type=int, default=10)
    p.add_argument("--no-muon-secondary", action="store_true",
                   help="skip the delayed-Muon step on the same set after the headline")
    p.add_argument("--muon-steps", type=int, default=5,
                   help="timed steps of the delayed-Muon entry of the default line")
    p.add_argument("--parallel", choices=["shard", "replica"], default="shard",
                   help="N > 1: shard (each rank steps its contiguous share of the set, "
                        "ZeRO-1 style; clipping takes one fp64 all-reduce of the squared "
                        "norm; strong scaling) or replica (each rank its own full set; "
                        "weak scaling). One GPU: the whole set either way")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    return p.parse_args(argv)


# ----------------------------------------------------------- distributed --

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Maximum of a per-rank scalar (a timing) over all ranks."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(units_per_rank: float, seconds_per_rank: float, world: int, device=None):
    """Whole-job throughput: units all ranks processed / the slowest rank's time."""
    t = max_over_ranks(seconds_per_rank, world, device)
    return units_per_rank * world / t, t


# ----------------------------------------------------------------- peaks --

def measured_bf16_peak():
    """Sustained dense bf16 TFLOP/s (the Newton-Schulz GEMMs run back to back
    for the whole step), measured on the GB300s."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["bf16_tflops_sustained"]), "measured"
    except Exception:
        return FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


def measured_hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# The device sources each profiled kernel is compiled from.
KERNEL_SOURCES = {
    "fused_step": ("dpo_internal.h", "dpo_device.cuh", "dpo_reduce.cuh", "dpo_step.cuh",
                   "dpo_step_adamw.cu", "dpo_step_nadam.cu", "dpo_step_lion.cu",
                   "dpo_step_adan.cu", "dpo_kernels.cu"),
    "grad_sqnorm": ("dpo_internal.h", "dpo_device.cuh", "dpo_reduce.cuh", "dpo_kernels.cu"),
    "ns_gemm": ("dpo_internal.h", "dpo_device.cuh", "dpo_gemm.cuh", "dpo_muon.cu"),
}


def kernel_source_sha(kernel: str = "fused_step") -> str:
    """First 16 hex digits of the sha256 over the kernel's device sources (in
    name order): a summary taken on other sources describes another kernel."""
    csrc = os.path.join(ROOT, "paper_2606_30634_gb300", "csrc")
    h = hashlib.sha256()
    for name in sorted(KERNEL_SOURCES[kernel]):
        h.update(name.encode() + b"\0")
        h.update(open(os.path.join(csrc, name), "rb").read())
    return h.hexdigest()[:16]


def committed_traffic(kernel_tag: str, key: str = "dram_bytes_per_param"):
    """A DRAM-traffic figure (``key``: bytes per parameter of the fused
    kernel, or bytes per step of the Newton-Schulz GEMMs) from the committed
    ncu summary with this kernel tag, if that summary was taken on the kernel
    source as it is now."""
    kernel = kernel_tag.split(":")[0]
    if kernel not in KERNEL_SOURCES:
        return None
    sha = kernel_source_sha(kernel)
    for name in sorted(os.listdir(os.path.join(ROOT, "profiles"))) if os.path.isdir(
            os.path.join(ROOT, "profiles")) else []:
        if not name.endswith(".md"):
            continue
        text = open(os.path.join(ROOT, "profiles", name)).read()
        m_tag = re.search(r"^kernel_tag:\s*(\S+)", text, re.M)
        m_sha = re.search(r"^kernel_source_sha256_16:\s*(\S+)", text, re.M)
        m_b = re.search(r"^" + re.escape(key) + r":\s*([0-9.eE+-]+)", text, re.M)
        if m_tag and m_sha and m_b and m_tag.group(1) == kernel_tag and m_sha.group(1) == sha:
            return float(m_b.group(1))
    return None


def ns_gemm_tag(workload: str, ns_steps: int) -> str:
    """Kernel tag of the Newton-Schulz GEMM chain's per-step traffic: it
    depends on the matrix set and the number of Newton-Schulz steps, not on
    the delayed rule (which changes only the elementwise apply pass)."""
    return f"ns_gemm:{workload}:ns{ns_steps}"


# ---------------------------------------------------------------- clocks --

class ClockSampler:
    """nvidia-smi samples during the timed region."""
    FIELDS = ("index,pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id=None):
        self.bus_id = (bus_id or "").lower()
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r.split(", ") for r in out.strip().splitlines() if r.count(",") >= 9]
        if self.bus_id:
            mine = [r for r in rows if self.bus_id.endswith(r[1].lower()[-12:]) or
                    r[1].lower().endswith(self.bus_id[-12:])]
            rows = mine or rows
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[6:10]) if v.strip() == "Active"})
        sm = sorted(float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit())
        mx = max((float(r[3]) for r in rows if r[3].strip().replace(".", "").isdigit()), default=None)
        pw = [float(r[4]) for r in rows if re.match(r"^[0-9.]+$", r[4].strip())]
        return {"sm_mhz": sm[len(sm) // 2] if sm else None, "sm_max_mhz": mx,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(pw) if pw else None}


# ----------------------------------------------------------------- modes --

# mode -> (update-history buffer, correction, description)
MODES = {
    "ef": (True, 0, "EF (lambda=1)"),
    "std": (False, 0, "standard delayed rule"),
    "sapipe-same": (True, 1, "SAPipe-WP prediction, same optimizer state"),
    "sapipe-updated": (True, 2, "SAPipe-WP prediction, updated optimizer state"),
}


def rule_settings(args) -> dict:
    """Update rule and its settings (the paper's where it gives them: Lion
    lr 5e-4, wd 0.5, App. E.1; Adan's usual betas)."""
    from paper_2606_30634_gb300 import dpo
    base = {"adamw": dict(optimizer=dpo.DPO_OPT_ADAMW),
            "nadam": dict(optimizer=dpo.DPO_OPT_NADAM, momentum_decay=0.004),
            "lion": dict(optimizer=dpo.DPO_OPT_LION, beta1=0.9, beta2=0.99, lr=5e-4,
                         weight_decay=0.5),
            "adan": dict(optimizer=dpo.DPO_OPT_ADAN, beta1=0.98, beta2=0.92, beta3=0.99),
            }[args.optimizer]
    return dict(base, dc_lambda=args.dc_lambda)


def resolve_stash(args, w) -> str:
    """--stash auto: the ping-pong stash where the layout allows it (bf16
    param and stash buffers, the standard rule or EF, the elementwise path),
    else the copying stash."""
    from paper_2606_30634_gb300.synth import workloads as W
    if args.stash != "auto":
        return args.stash
    ok = (w.param_dtype == W.BF16 and w.stash_dtype == W.BF16
          and args.mode in ("ef", "std") and args.optimizer != "muon")
    return "pingpong" if ok else "copy"


def wpipe_sync(w, args):
    """Per-tensor DPO_SYNC flags: the second half of the tensor list under
    --wpipe (WPipe trains the second half of the model without delay)."""
    n = len(w.tensors)
    return [args.wpipe and i >= n // 2 for i in range(n)]


# ------------------------------------------------------------ CPU oracle --

def extrapolation(n_params: int, timed_params: int, timed_steps: int, timed_s: float,
                  wall_s: float) -> dict:
    """Labels of a CPU figure measured on a sample: its ms_per_step is the
    sample's per-parameter rate scaled to the whole set, not a timed step."""
    return {"extrapolated": timed_params < n_params, "timed_params": timed_params,
            "timed_steps": timed_steps, "timed_s": timed_s, "wall_s": wall_s,
            "ms_per_step_basis": f"{n_params} params / the rate measured on {timed_params} "
                                 f"params over {timed_steps} steps"}


def oracle_sample_run(w, mode: str, seconds: float, max_steps: int = 1000, n: int = 1 << 22,
                      rule: dict = None, threads: int = 0):
    """Time the oracle as it stands on the first n parameters of the set
    (input draws excluded from the timing), on all host cores or on
    ``threads`` of them. Returns (params/s, cores, steps, n)."""
    import numpy as np

    import oracle
    from paper_2606_30634_gb300 import synth
    from paper_2606_30634_gb300.synth import workloads as W

    n = min(n, w.n_params)
    STORE = {0: oracle.F32, 1: oracle.BF16}
    ef, corr, _ = MODES[mode]
    x0 = synth.host_normal(w.seed, synth.STREAM_INIT, 0, 0, n, W.INIT_SIGMA).astype(np.float64)
    rule = dict(rule or {})
    opt = rule.pop("optimizer", 0)
    rule.setdefault("lr", w.lr)
    rule.setdefault("weight_decay", w.weight_decay)
    hp = oracle.HParams(ef_lambda=1.0 if ef and corr == 0 else 0.0,
                        max_grad_norm=w.max_grad_norm, correction=corr,
                        rule={0: oracle.RULE_ADAMW, 1: oracle.RULE_NADAM, 2: oracle.RULE_LION,
                              3: oracle.RULE_ADAN}[opt], **rule).as_f32()
    o = oracle.DelayedOptimizer([x0], hp, ef=ef, x_store=oracle.F32,
                                stash_store=STORE[w.stash_dtype],
                                param_store=oracle.BF16 if w.param_dtype == 1 else None)
    gdt = synth.BF16 if w.grad_dtype == 1 else synth.F32
    all_cores = oracle.num_threads()
    if threads:
        oracle.set_num_threads(threads)
    try:
        cores = oracle.num_threads()
        spent, steps = 0.0, 0
        while steps < max_steps and (spent < seconds or steps < 2):
            g = synth.host_normal(w.seed, synth.STREAM_GRAD, steps + 1, 0, n, W.GRAD_SIGMA, gdt)
            g = (synth.bf16_bits_to_f32(g) if gdt == synth.BF16 else g).astype(np.float64)
            sq = oracle.sqnorm(g) if w.max_grad_norm > 0 else None
            t0 = time.perf_counter()
            o.step(g, sq=sq)
            spent += time.perf_counter() - t0
            steps += 1
    finally:
        oracle.set_num_threads(all_cores)
    return n * steps / spent, cores, steps, n


# ------------------------------------------------------------------- GPU --

def sharded(args, world: int) -> bool:
    """Whether ranks split one set between them (else each steps its own)."""
    return args.parallel == "shard" and world > 1


def build_step(args, w, world, rank, dev, stream, sync=None, **kw):
    """The rank's optimizer over its share of the set (the whole set on one
    GPU or in replica mode) through the product's shard API, start weights
    and the first gradient drawn for its pieces only, and the step function.
    Sharded with clipping, each step sums the ranks' squared norms with one
    fp64 all-reduce (dpo.global_sqnorm) and every rank clips from the total.
    Returns (optimizer, its parameter count, step function)."""
    import numpy as np
    import torch

    from paper_2606_30634_gb300 import dpo, shard, synth
    from paper_2606_30634_gb300.synth import workloads as W

    offs = np.concatenate([[0], np.cumsum(w.numels)]).astype(np.int64)
    world_s, rank_s = (world, rank) if sharded(args, world) else (1, 0)
    fill = lambda start, out: synth.dev_normal(w.seed, synth.STREAM_INIT, 0, int(start), out,
                                               W.INIT_SIGMA)
    with torch.cuda.stream(stream):
        opt, pieces = shard.shard_optimizer(
            w.numels, world_s, rank_s, x0=fill, sync=sync, device=dev,
            stream=stream, param_dtype=w.param_dtype, stash_dtype=w.stash_dtype,
            grad_dtype=w.grad_dtype, max_grad_norm=w.max_grad_norm, delay=1, **kw)
        for j, (i, a, b) in enumerate(pieces):
            synth.dev_normal(w.seed, synth.STREAM_GRAD, 1, int(offs[i]) + a, opt.grads(j),
                             W.GRAD_SIGMA)
    acc = None
    if world_s > 1 and w.max_grad_norm > 0:
        acc = torch.zeros(1, dtype=torch.float64, device=dev)
        opt.set_clip_source(acc)

    def step():
        if acc is not None:
            dpo.global_sqnorm([opt], acc, stream=stream)
        opt.step(stream=stream)

    return opt, sum(b - a for _, a, b in pieces), step


def run_gpu(args, w, world, rank, local):
    import torch

    from paper_2606_30634_gb300 import dpo
    from paper_2606_30634_gb300.synth import workloads as W

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    ef, corr, _ = MODES[args.mode]
    stream = torch.cuda.Stream(dev)
    kw = dict(lr=w.lr, beta1=w.beta1, beta2=w.beta2, eps=w.eps, weight_decay=w.weight_decay,
              stash_mode=(dpo.DPO_STASH_PINGPONG if args.stash == "pingpong"
                          else dpo.DPO_STASH_COPY), ef=ef, ef_lambda=1.0, correction=corr)
    kw.update(rule_settings(args))
    opt, n_local, one_step = build_step(args, w, world, rank, dev, stream,
                                        sync=wpipe_sync(w, args), **kw)
    torch.cuda.synchronize(dev)
    step_bytes, norm_bytes = dpo.dpo_algorithmic_bytes(opt.ctx)
    step_ctas, norm_ctas, threads = dpo.dpo_launch_config(opt.ctx)
    launches_per_step = 2 if w.max_grad_norm > 0 else 1
    if sharded(args, world) and w.max_grad_norm > 0:
        # the norm pass runs through dpo_grad_sqnorm (into the all-reduced
        # scalar), then one thread forms the coefficient: 3 launches
        norm_bytes = (2 if w.grad_dtype == W.BF16 else 4) * n_local
        launches_per_step = 3

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize(dev)

    props = torch.cuda.get_device_properties(dev)
    sampler = ClockSampler(getattr(props, "pci_bus_id", None))
    K = args.steps
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    sampler.start()
    time.sleep(0.25)
    ev[0].record(stream)
    for i in range(K):
        one_step()
        ev[i + 1].record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop()
    per_step_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(K)]
    total_s = ev[0].elapsed_time(ev[K]) / 1e3
    if sharded(args, world):   # all ranks together update the set once per step
        value, t_max = aggregate(w.n_params * K / world, total_s, world, dev)
    else:
        value, t_max = aggregate(w.n_params * K, total_s, world, dev)
    # Without clipping a step is one fused-kernel launch; with clipping it is
    # the norm pass followed by the fused kernel, timed together.
    kernel_ms = sum(per_step_ms) / K
    achieved = (step_bytes + norm_bytes) / (kernel_ms / 1e3) / 1e9

    # End to end through the public API, gradients from and new bf16 weights
    # to pinned host memory, copies inside the timed region.
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, opt, one_step, stream, dev, world, w)

    opt.close()
    return dict(value=value, t_max=t_max, per_step_ms=per_step_ms, kernel_ms=kernel_ms,
                achieved=achieved, step_bytes=step_bytes, norm_bytes=norm_bytes, clocks=clocks,
                launches=K * launches_per_step, step_ctas=step_ctas, threads=threads, e2e=e2e,
                device_name=props.name)


def run_secondary(args, dev, world):
    """The clipped Llama-1B step (global-norm clipping at 1.0 over all 146
    tensors, EF, fp32 stash, one-step delay): the norm pass and the fused
    step each timed by the library's CUDA events on the launch stream
    (dpo_set_timing), and the whole step by events around it."""
    import torch

    from paper_2606_30634_gb300 import dpo
    from paper_2606_30634_gb300.synth import workloads as W

    w = W.LLAMA_1B
    gc.collect()
    torch.cuda.empty_cache()   # the headline set's arenas
    stream = torch.cuda.Stream(dev)
    opt, n_local, one_step = build_step(
        args, w, world, int(os.environ.get("RANK", "0")), dev, stream, ef=True, ef_lambda=1.0,
        lr=w.lr, beta1=w.beta1, beta2=w.beta2, eps=w.eps, weight_decay=w.weight_decay)
    torch.cuda.synchronize(dev)
    step_bytes, norm_bytes = dpo.dpo_algorithmic_bytes(opt.ctx)
    _, norm_ctas, _ = dpo.dpo_launch_config(opt.ctx)
    if sharded(args, world):   # the norm pass runs outside dpo_step (dpo_grad_sqnorm)
        norm_bytes = 2 * n_local
    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize(dev)
    K = max(1, args.secondary_steps)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    opt.set_timing(True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    e0.record(stream)
    for _ in range(K):
        one_step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    norm_ms, fused_ms, calls = opt.kernel_times()
    opt.set_timing(False)
    _, gnorm, coef = dpo.dpo_get_flags(opt.ctx, stream)
    total_ms = e0.elapsed_time(e1)
    opt.close()
    del opt
    torch.cuda.empty_cache()
    total_ms = max_over_ranks(total_ms, world, dev)
    norm_ms = max_over_ranks(norm_ms / calls, world, dev)
    fused_ms = max_over_ranks(fused_ms / calls, world, dev)
    peak, peak_kind = measured_hbm_peak()
    n = n_local

    def kern(bytes_, ms, tag):
        t = committed_traffic(tag)
        return {"avg_launch_ms": ms, "algorithmic_bytes_per_launch": bytes_,
                "bytes_per_param": bytes_ / n, "achieved_gbs": bytes_ / (ms / 1e3) / 1e9,
                "frac": bytes_ / (ms / 1e3) / 1e9 / peak,
                "traffic": None if t is None else t * n, "traffic_tag": tag}

    pair_ms = norm_ms + fused_ms
    units = w.n_params if sharded(args, world) else w.n_params * world
    return {"workload": f"{w.name}: {w.n_params} params in {len(w.tensors)} tensors, EF "
                        f"(lambda=1), global-norm clip at {w.max_grad_norm}, fp32 stash, "
                        "one-step delay",
            "value": units * K / (total_ms / 1e3), "unit": UNIT, "steps": K,
            "params_per_rank": n_local,
            "norm_timing": ("grad_sqnorm_kernel inside dpo_step" if not sharded(args, world)
                            else "dpo_grad_sqnorm + fp64 all-reduce outside dpo_step; "
                                 "grad_sqnorm_kernel's entry times only the coefficient kernel"),
            "ms_per_step": total_ms / K, "grad_norm": gnorm, "clip_coef": coef,
            "peak": peak, "peak_kind": peak_kind, "norm_ctas": norm_ctas,
            "grad_sqnorm_kernel": kern(norm_bytes, norm_ms, f"grad_sqnorm:{w.name}"),
            "fused_step_kernel": kern(step_bytes, fused_ms, f"fused_step:{w.name}:ef"),
            "pair": {"bytes_per_param": (norm_bytes + step_bytes) / n,
                     "achieved_gbs": (norm_bytes + step_bytes) / (pair_ms / 1e3) / 1e9,
                     "frac": (norm_bytes + step_bytes) / (pair_ms / 1e3) / 1e9 / peak,
                     "kernel_ms": pair_ms}}


def run_muon_secondary(args, w, world, rank, local):
    """Delayed Muon (Alg. 2, EF) on the headline set's attention and MLP
    matrices with AdamW EF on the rest, as ``--optimizer muon`` times it: the
    Newton-Schulz GEMM chains by the library's CUDA events against the
    sustained bf16 tensor peak. Runs after the headline's arenas are freed."""
    import torch

    gc.collect()
    torch.cuda.empty_cache()
    a = argparse.Namespace(**vars(args))
    a.mode, a.ns_steps, a.graph, a.no_library_ns = "ef", 5, False, True
    a.steps, a.warmup = max(1, args.muon_steps), max(3, min(args.warmup, 3))
    r = run_muon(a, w, world, rank, local)
    torch.cuda.empty_cache()
    peak, peak_kind = measured_bf16_peak()
    mi, ai = muon_split(w)
    return {"workload": f"{w.name}: {w.n_params} params; delayed Muon (Alg. 2, 5 Newton-Schulz "
                        f"steps, EF) on {len(mi)} attention/MLP matrices ({r['n_muon']} params), "
                        f"AdamW EF on the other {len(ai)} tensors, one-step delay",
            "value": r["value"], "unit": UNIT, "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": r["t_max"] / a.steps * 1e3,
            "gemm": {"kernel": "ns_gemm_kernel", "bound": "tensor",
                     "gemm_ms_per_step": r["gemm_ms"],
                     "algorithmic_flops_per_step": r["flops"],
                     "achieved": r["achieved"], "unit": "TFLOP/s", "peak": peak,
                     "peak_kind": f"{peak_kind} (sustained)", "frac": r["achieved"] / peak,
                     "traffic": committed_traffic(ns_gemm_tag(w.name, 5), "dram_bytes_per_step")},
            "gpu_launches": r["launches"], "clocks": r["clocks"]}


def muon_split(w):
    """(Muon matrix indices, AdamW tensor indices): the attention and MLP
    projection matrices take Muon; embeddings, the LM head, norms and biases
    keep AdamW, the usual division for Muon (Sec. 2.1 trains with it)."""
    hidden = ("_proj", "c_attn.weight", "c_proj.weight", "c_fc.weight")
    mu = [i for i, (name, shape) in enumerate(w.tensors)
          if len(shape) == 2 and name.endswith(hidden)]
    rest = [i for i in range(len(w.tensors)) if i not in set(mu)]
    return mu, rest


def run_muon(args, w, world, rank, local):
    """Delayed Muon (Alg. 2, EF per --mode) on the set's hidden matrices plus
    the fused AdamW step on the rest, one stream; a step is both calls."""
    import numpy as np
    import torch

    from paper_2606_30634_gb300 import dpo, muon, synth
    from paper_2606_30634_gb300.synth import workloads as W

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    ef, corr, _ = MODES[args.mode]   # EF, standard rule, or a SAPipe-WP prediction
    stream = torch.cuda.Stream(dev)
    offs = np.concatenate([[0], np.cumsum(w.numels)]).astype(np.int64)
    mi, ai = muon_split(w)
    shapes = [w.tensors[i][1] for i in mi]
    with torch.cuda.stream(stream):
        mo = muon.DelayedMuon(shapes, stash_dtype=w.stash_dtype, grad_dtype=w.grad_dtype,
                              lr=MUON_LR, ef=ef, ns_steps=args.ns_steps, delay=1, device=dev,
                              init_mode=dpo.DPO_INIT_RESUME, stream=stream, correction=corr)
        for j, i in enumerate(mi):
            synth.dev_normal(w.seed, synth.STREAM_INIT, 0, int(offs[i]),
                             mo.view(mo.master, j).view(-1), W.INIT_SIGMA)
            synth.dev_normal(w.seed, synth.STREAM_GRAD, 1, int(offs[i]),
                             mo.grads(j).view(-1), W.GRAD_SIGMA)
        mo.stash.copy_(mo.master)   # Alg. 1 start: stash = param = x_0, m = U_prev = 0
        mo.param.copy_(mo.master)
        rest = [w.numels[i] for i in ai]
        lay = dpo.Layout.of(rest)
        x0 = torch.empty(lay.total, dtype=torch.float32, device=dev)
        for j, i in enumerate(ai):
            o, n = lay.offsets[j], lay.numels[j]
            synth.dev_normal(w.seed, synth.STREAM_INIT, 0, int(offs[i]), x0[o:o + n],
                             W.INIT_SIGMA)
        ad = dpo.DelayedAdamW(rest, param_dtype=w.param_dtype, stash_dtype=w.stash_dtype,
                              grad_dtype=w.grad_dtype, ef=ef, ef_lambda=1.0, delay=1,
                              device=dev, x0=x0, stream=stream, lr=w.lr, beta1=w.beta1,
                              beta2=w.beta2, eps=w.eps, weight_decay=w.weight_decay,
                              correction=corr)
        del x0
        for j, i in enumerate(ai):
            synth.dev_normal(w.seed, synth.STREAM_GRAD, 1, int(offs[i]), ad.grads(j),
                             W.GRAD_SIGMA)
    torch.cuda.synchronize(dev)
    flops = mo.flops()
    n_groups = len({(min(r, c), max(r, c)) for r, c in shapes})
    # AdamW's fused step; momentum, norm, apply; one normalisation per shape
    # group (the GEMM launches are counted by the library: shape groups may
    # share them)
    other_launches_per_step = 1 + 3 + n_groups
    if corr == 2:   # the updated-state prediction: momentum, norm, predict, normalisations
        other_launches_per_step += 3 + n_groups

    mo.set_timing(True)
    for _ in range(args.warmup):
        ad.step(stream=stream)
        mo.step(stream=stream)
    torch.cuda.synchronize(dev)
    mo.gemm_time()   # start the count at the timed region

    props = torch.cuda.get_device_properties(dev)
    sampler = ClockSampler(getattr(props, "pci_bus_id", None))
    K = args.steps
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    sampler.start()
    time.sleep(0.25)
    ev[0].record(stream)
    for _ in range(K):
        ad.step(stream=stream)
        mo.step(stream=stream)
    ev[1].record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop()
    gemm_ms, gemm_launches = mo.gemm_time()
    status = mo.status()
    total_s = ev[0].elapsed_time(ev[1]) / 1e3
    graph = None
    if args.graph:   # the same step captured once and replayed K times
        mo.set_timing(False)
        for o in (ad, mo):
            o.set_capturable(True, stream=stream)
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            ad.step(stream=stream)
            mo.step(stream=stream)
        with torch.cuda.stream(stream):
            for _ in range(2):
                g.replay()
            torch.cuda.synchronize(dev)
            ev[0].record(stream)
            for _ in range(K):
                g.replay()
            ev[1].record(stream)
        torch.cuda.synchronize(dev)
        graph = {"ms_per_step": ev[0].elapsed_time(ev[1]) / K,
                 "what": "the same step (AdamW call + Muon call) captured once in a CUDA graph "
                         "in capturable mode and replayed"}
        status |= mo.status()
    value, t_max = aggregate(w.n_params * K, total_s, world, dev)
    achieved = flops * K / (gemm_ms / 1e3) / 1e12
    ws = mo.workspace_bytes()
    mo.close()
    ad.close()
    if status != 0:
        raise RuntimeError(f"tensor-core pipeline status {status}")
    library = None if args.no_library_ns else library_ns(shapes, args.ns_steps, dev)
    return dict(value=value, t_max=t_max, achieved=achieved, flops=flops, gemm_ms=gemm_ms / K,
                gemm_launches=gemm_launches, clocks=clocks,
                launches=K * other_launches_per_step + gemm_launches,
                n_muon=sum(w.numels[i] for i in mi), n_matrices=len(mi), workspace=ws,
                device_name=props.name, library=library, graph=graph)


def library_ns(shapes, steps: int, dev, reps: int = 3):
    """Context for the Newton-Schulz roofline: the same iteration on the same
    matrix shapes with cuBLAS (torch.matmul / baddbmm in bf16, full
    products), one batched chain per shape as the library runs it, timed
    with CUDA events. Not part of the measured step."""
    import torch
    a_, b_, c_ = 3.4445, -4.7750, 2.0315
    groups = {}
    for r, c in shapes:
        key = (min(r, c), max(r, c))
        groups[key] = groups.get(key, 0) + 1

    def chain(X):
        for _ in range(steps):
            A = torch.bmm(X, X.transpose(1, 2))
            B = torch.baddbmm(A, A, A, beta=b_, alpha=c_)
            X = torch.baddbmm(X, B, X, beta=a_, alpha=1.0)
        return X

    gen = torch.Generator(device=dev).manual_seed(0)
    Xs = [torch.randn(nb, r, w, device=dev, dtype=torch.bfloat16, generator=gen) * 0.01
          for (r, w), nb in groups.items()]
    full = sum(steps * nb * (4.0 * r * r * w + 2.0 * r * r * r) for (r, w), nb in groups.items())
    for X in Xs:
        chain(X)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        for X in Xs:
            chain(X)
    e1.record()
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / reps
    del Xs
    torch.cuda.empty_cache()
    return {"what": "cuBLAS bf16 Newton-Schulz chain (torch bmm/baddbmm, full products) on the "
                    "same matrix shapes", "ms_per_step": ms, "tflops_full_products": full / ms / 1e9}


def oracle_muon_sample(seconds: float, rows: int = 1024, cols: int = 4096):
    """The Muon oracle as it stands (Newton-Schulz with bf16 iterates, exact
    accumulation) on one rows x cols matrix of the 7B set's width, steps
    until ``seconds`` pass. Returns (params/s, cores, steps, params)."""
    import numpy as np

    import oracle
    from oracle import muon as omuon
    from paper_2606_30634_gb300 import synth

    x0 = synth.host_normal(0xD0D0 + 5, synth.STREAM_INIT, 0, 0, rows * cols, 0.02)
    opt = omuon.DelayedMuon([x0.reshape(rows, cols).astype(np.float64)],
                            omuon.MuonHParams(lr=MUON_LR, ef_lambda=1.0).as_f32(), ef=True,
                            x_store=oracle.F32, stash_store=oracle.BF16, param_store=oracle.BF16)
    steps, spent = 0, 0.0
    while spent < seconds or steps == 0:
        g = synth.bf16_bits_to_f32(synth.host_normal(0xD0D0 + 5, synth.STREAM_GRAD, steps + 1, 0,
                                                     rows * cols, 1e-3, synth.BF16))
        g = g.astype(np.float64).reshape(rows, cols)
        t0 = time.perf_counter()
        opt.step([g])
        spent += time.perf_counter() - t0
        steps += 1
    return rows * cols * steps / spent, oracle.num_threads(), steps, rows * cols


def _host_avail_bytes():
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except Exception:
        pass
    return 0


def e2e_fits(avail: int, io_bytes: int, local_world: int) -> bool:
    """Whether every rank on the node can pin its staged copies and its
    host-I/O arenas (twice the step's input and output bytes each), with
    16 GiB left for the rest of the host."""
    return avail >= local_world * 2 * io_bytes + (16 << 30)


def run_e2e(args, opt, one_step, stream, dev, world, w):
    """End to end through the public API, transfers inside the timed region:
    each step's inputs (the gradients) come from pinned host memory and each
    step's result is read back to the host. The library's host-I/O mode does
    the input transfer inside the fused kernel, over the host link. The main
    figure reads back the step's diagnostics (flags, gradient norm, clip
    coefficient: dpo_get_flags), the new bf16 weights staying on the device
    for the next forward as in training; `weights_to_host` also delivers the
    weights to pinned host memory every step, and `staged` runs cudaMemcpy in,
    the device-resident step and cudaMemcpy out."""
    import torch

    from paper_2606_30634_gb300 import dpo
    gbytes = opt.grad.numel() * opt.grad.element_size()
    pbytes = opt.param.numel() * opt.param.element_size()
    # every rank on this node pins its own copies, and all ranks must agree
    # (the timed region has barriers)
    local_world = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
    ok = e2e_fits(_host_avail_bytes(), gbytes + pbytes, local_world)
    if world > 1:
        t = torch.tensor([1 if ok else 0], dtype=torch.int32, device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MIN)
        ok = bool(t.item())
    if not ok:
        return {"skipped": f"host memory: {(gbytes + pbytes) / 1e9:.1f} GB pinned needed per rank, "
                           f"{local_world} rank(s) on this node"}
    K = max(1, args.e2e_steps)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(one_step):
        one_step()
        torch.cuda.synchronize(dev)
        if world > 1:
            torch.distributed.barrier()
        e0.record(stream)
        for _ in range(K):
            one_step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / 1e3

    # staged copies around the device-resident step
    h_grad = torch.empty(opt.grad.shape, dtype=opt.grad.dtype, pin_memory=True)
    h_param = torch.empty(opt.param.shape, dtype=opt.param.dtype, pin_memory=True)
    with torch.cuda.stream(stream):
        h_grad.copy_(opt.grad, non_blocking=True)
    torch.cuda.synchronize(dev)

    def staged_step():
        with torch.cuda.stream(stream):
            opt.grad.copy_(h_grad, non_blocking=True)
            one_step()
            h_param.copy_(opt.param, non_blocking=True)

    staged_s = timed(staged_step)
    link = None if args.no_link_peak else link_peak(opt, h_grad, h_param, stream, dev)
    del h_grad, h_param

    # host I/O, gradients in: the fused kernel reads them from pinned host
    # memory; the step's diagnostics come back to the host every step
    flags_bytes = 4 + 8 + 4   # uint32 flags, fp64 norm, fp32 clip coefficient
    opt.use_host_io(grad=True, param=False, stream=stream)

    def step_and_result():
        one_step()
        dpo.dpo_get_flags(opt.ctx, stream)

    secs_in = timed(step_and_result)
    # and the new weights out as well
    opt.use_host_io(grad=False, param=True, stream=stream)
    secs_both = timed(one_step)
    units = w.n_params * K / (world if sharded(args, world) else 1)
    value, _ = aggregate(units, secs_in, world, dev)
    both_value, _ = aggregate(units, secs_both, world, dev)
    staged_value, _ = aggregate(units, staged_s, world, dev)
    h2d_ms = None if link is None else gbytes / link["h2d_gbs"] / 1e6
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": gbytes,
            "d2h_bytes_per_step": flags_bytes, "ms_per_step": secs_in / K * 1e3, "steps": K,
            "path": "dpo_step with the gradient arena in pinned host memory: the fused kernel "
                    "reads each step's gradients across the host link; the step's result read "
                    "back every step is its flags, gradient norm and clip coefficient "
                    "(dpo_get_flags); the new bf16 weights stay on the device for the next "
                    "forward",
            "host_link_gbs": gbytes / (secs_in / K) / 1e9,
            "link_peak": link,
            # the bound: the gradients' bytes at the plain pinned copy's rate
            "link_bound_ms": h2d_ms,
            "link_frac": None if h2d_ms is None else h2d_ms / (secs_in / K * 1e3),
            "weights_to_host": {
                "value": both_value, "ms_per_step": secs_both / K * 1e3,
                "h2d_bytes_per_step": gbytes, "d2h_bytes_per_step": pbytes,
                "path": "as above, and the fused kernel also writes the new bf16 weights to "
                        "pinned host memory every step",
                "host_link_gbs": (gbytes + pbytes) / (secs_both / K) / 1e9,
                # each direction at its own measured rate, both at once (the
                # host-I/O kernel overlaps them; two concurrent copy-engine
                # copies do not, see link_peak.both_gbs)
                "link_bound_ms": None if link is None else link["duplex_bound_ms"],
                "link_frac": (None if link is None else
                              link["duplex_bound_ms"] / (secs_both / K * 1e3))},
            "staged": {"value": staged_value, "ms_per_step": staged_s / K * 1e3,
                       "path": "cudaMemcpy grad in, device-resident dpo_step, cudaMemcpy "
                               "weights out, on one stream"}}


def link_peak(opt, h_grad, h_param, stream, dev, reps: int = 2) -> dict:
    """The host link's own rates for the e2e step's transfers, by CUDA
    events: the gradients' bytes host -> device alone, the weights' bytes
    device -> host alone, and both at once on two streams (what the host-I/O
    step needs every step). Plain cudaMemcpyAsync from and to the same pinned
    buffers."""
    import torch
    other = torch.cuda.Stream(dev)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]

    def h2d(s):
        with torch.cuda.stream(s):
            opt.grad.copy_(h_grad, non_blocking=True)

    def d2h(s):
        with torch.cuda.stream(s):
            h_param.copy_(opt.param, non_blocking=True)

    def best(fn):
        ms = []
        for _ in range(reps):
            torch.cuda.synchronize(dev)
            ev[0].record(stream)
            fn()
            ev[1].record(stream)
            torch.cuda.synchronize(dev)
            ms.append(ev[0].elapsed_time(ev[1]))
        return min(ms)

    def both():
        # the second stream starts after the first's start event and the
        # first waits for it at the end, so the interval spans both copies
        other.wait_event(ev[0])
        h2d(stream)
        d2h(other)
        ev[2].record(other)
        stream.wait_event(ev[2])

    gb, pb = opt.grad.numel() * opt.grad.element_size(), opt.param.numel() * opt.param.element_size()
    t_in, t_out, t_both = best(lambda: h2d(stream)), best(lambda: d2h(stream)), best(both)
    torch.cuda.synchronize(dev)
    return {"h2d_gbs": gb / t_in / 1e6, "d2h_gbs": pb / t_out / 1e6,
            "both_gbs": (gb + pb) / t_both / 1e6, "h2d_bytes": gb, "d2h_bytes": pb,
            "duplex_bound_ms": max(t_in, t_out),
            "what": "best of %d: pinned host -> device copy of the gradients alone, device -> "
                    "pinned host copy of the bf16 weights alone, and both at once on two "
                    "streams (combined bytes / elapsed); duplex_bound_ms: the slower "
                    "direction alone, the step's transfer time if both directions ran at "
                    "their own rates at once" % reps}


# ------------------------------------------------------------------ main --

def main_muon(args, w, world, rank, local):
    """--optimizer muon: delayed Muon on the hidden matrices, AdamW on the
    rest; the roofline is the Newton-Schulz GEMMs against the sustained bf16
    tensor peak."""
    mi, ai = muon_split(w)
    n_muon = sum(w.numels[i] for i in mi)
    cfg = {"workload": f"{w.name}: {w.n_params} params; delayed Muon (Alg. 2, "
                       f"{args.ns_steps} Newton-Schulz steps) on {len(mi)} attention/MLP "
                       f"matrices ({n_muon} params), AdamW on the other {len(ai)} tensors, "
                       f"{MODES[args.mode][2]}, one-step delay",
           "mode": args.mode, "optimizer": "muon", "ns_steps": args.ns_steps,
           "param_dtype": "bf16", "stash_dtype": "bf16" if w.stash_dtype else "f32",
           "grad_dtype": "bf16" if w.grad_dtype else "f32",
           "ns_dtype": "bf16 operands, fp32 accumulation (tcgen05)",
           "l2": "inputs larger than L2 (no flush needed)"}
    if args.impl == "reference":
        if rank != 0:
            return 0
        t0 = time.perf_counter()
        v, cores, steps, n = oracle_muon_sample(args.cpu_seconds)
        wall = time.perf_counter() - t0
        line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT,
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": w.n_params / v * 1e3,
                **extrapolation(w.n_params, n, steps, n * steps / v, wall),
                "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": cfg,
                "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                                 "sample": f"one 1024 x 4096 matrix, {steps} Muon oracle steps "
                                           "(plain C, fp64, bf16 Newton-Schulz iterates)"},
                "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0
    import torch
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    r = run_muon(args, w, world, rank, local)
    peak, peak_kind = measured_bf16_peak()
    roof = {"bound": "tensor", "achieved": r["achieved"], "peak": peak, "unit": "TFLOP/s",
            "frac": r["achieved"] / peak, "peak_kind": f"{peak_kind} (sustained)",
            "traffic": committed_traffic(ns_gemm_tag(w.name, args.ns_steps),
                                         "dram_bytes_per_step"),
            "kernel": "ns_gemm_kernel",
            "algorithmic_flops_per_step": r["flops"], "gemm_ms_per_step": r["gemm_ms"],
            "gemm_launches_per_step": r["gemm_launches"] / max(1, args.steps),
            "nominal_peak_tflops": 2250.0, "library_newton_schulz": r["library"]}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:   # the oracle at N=1 only
        v, cores, steps, n = oracle_muon_sample(args.cpu_seconds)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"one 1024 x 4096 matrix, {steps} Muon oracle steps (plain C, fp64, "
                         "bf16 Newton-Schulz iterates)"}
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return 0
    line = {"metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": r["t_max"] / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16+f32", "data": "synthetic",
            "config": cfg, "roofline": roof, "cpu_baseline": cpu, "e2e": None,
            "gpu_launches": r["launches"], "clocks": r["clocks"],
            "workspace_bytes": r["workspace"], "device": r["device_name"]}
    if r["graph"] is not None:
        line["graph"] = r["graph"]
    print(json.dumps(line), flush=True)
    return 0


def main(argv=None):
    args = parse_args(argv)
    from paper_2606_30634_gb300.synth import workloads as W
    w = W.ALL[args.workload]
    args.stash = resolve_stash(args, w)
    world, rank, local = dist_env()
    if args.optimizer == "muon":
        return main_muon(args, w, world, rank, local)
    ef, _, what = MODES[args.mode]
    cfg = {"workload": f"{w.name}: {w.n_params} params in {len(w.tensors)} tensors, "
                       f"{what}, one-step delay",
           "mode": args.mode, "param_dtype": "bf16" if w.param_dtype else "f32",
           "stash_dtype": "bf16" if w.stash_dtype else "f32",
           "grad_dtype": "bf16" if w.grad_dtype else "f32",
           "state": "fp32 master/m/v" + (" + fp32 update-history buffer" if ef else ""),
           "clip": w.max_grad_norm, "l2": "inputs larger than L2 (no flush needed)",
           "wpipe": bool(args.wpipe), "optimizer": args.optimizer,
           "dc_lambda": args.dc_lambda, "stash": args.stash,
           "parallelism": (f"shard{world}: each rank steps 1/{world} of the set (contiguous "
                           "ranges of the flat concatenation), clip norm all-reduced"
                           if sharded(args, world) else
                           f"replica{world}: each rank steps its own full set"
                           if world > 1 else "one GPU, the whole set")}

    if args.impl == "reference":
        if rank != 0:
            return 0
        t0 = time.perf_counter()
        v, cores, steps, n = oracle_sample_run(w, args.mode, args.cpu_seconds,
                                               max_steps=max(1, args.steps + args.warmup),
                                               rule=rule_settings(args))
        wall = time.perf_counter() - t0
        sample = f"first {n} params of the set, {steps} oracle steps (plain C, fp64)"
        line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT,
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": w.n_params / v * 1e3,
                **extrapolation(w.n_params, n, steps, n * steps / v, wall),
                "higher_is_better": True,
                "scaling": "strong" if args.parallel == "shard" else "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": cfg,
                "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                                 "sample": sample},
                "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0

    import torch
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    r = run_gpu(args, w, world, rank, local)
    secondary = muon_entry = None
    # The extra entries never cost the headline its line: a failure is
    # reported in the entry instead.
    if not args.no_secondary and w.name == "llama-7B":
        try:
            secondary = run_secondary(args, torch.device("cuda", local), world)
        except Exception as e:   # noqa: BLE001
            secondary = {"error": f"{type(e).__name__}: {e}"}
    if (not args.no_muon_secondary and w.name == "llama-7B" and args.optimizer == "adamw"
            and not sharded(args, world)):
        try:
            muon_entry = run_muon_secondary(args, w, world, rank, local)
        except Exception as e:   # noqa: BLE001
            muon_entry = {"error": f"{type(e).__name__}: {e}"}
    peak, peak_kind = measured_hbm_peak()
    # the tag names every setting that changes the kernel's traffic; the
    # headline keeps "fused_step:<set>:<mode>[:pingpong]"
    variant = [x for x in (args.optimizer if args.optimizer != "adamw" else None,
                           "dc" if args.dc_lambda else None, "wpipe" if args.wpipe else None) if x]
    kernel_tag = (f"fused_step:{w.name}:{args.mode}" + "".join(":" + v for v in variant) +
                  (":pingpong" if args.stash == "pingpong" else ""))
    traffic = committed_traffic(kernel_tag)
    kernels = "fused_step_kernel" if w.max_grad_norm <= 0 else "grad_sqnorm_kernel+fused_step_kernel"
    roof = {"bound": "hbm", "achieved": r["achieved"], "peak": peak, "unit": "GB/s",
            "frac": r["achieved"] / peak, "peak_kind": peak_kind,
            "traffic": None if traffic is None else traffic * w.n_params,
            "kernel": kernels, "algorithmic_bytes_per_launch": r["step_bytes"] + r["norm_bytes"],
            "bytes_per_param": (r["step_bytes"] + r["norm_bytes"]) / w.n_params,
            "avg_launch_ms": r["kernel_ms"], "nominal_peak_gbs": 8000.0,
            "frac_of_nominal": r["achieved"] / 8000.0}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:   # the oracle at N=1 only
        v, cores, steps, n = oracle_sample_run(w, args.mode, args.cpu_seconds,
                                               rule=rule_settings(args))
        v1, _, steps1, n1 = oracle_sample_run(w, args.mode, args.cpu_seconds / 3,
                                              rule=rule_settings(args), n=1 << 20, threads=1)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"first {n} params of the set, {steps} oracle steps (plain C, fp64)",
               "single_thread": {"value": v1, "unit": UNIT, "cores": 1,
                                 "sample": f"first {n1} params, {steps1} oracle steps"}}
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return 0
    line = {"metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["t_max"] / args.steps * 1e3,
            "higher_is_better": True,
            "scaling": "strong" if args.parallel == "shard" else "weak",
            "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": cfg, "roofline": roof, "cpu_baseline": cpu,
            "e2e": r["e2e"], "gpu_launches": r["launches"], "clocks": r["clocks"],
            "launch": {"ctas": r["step_ctas"], "threads": r["threads"]},
            "hbm_gbs_achieved": r["achieved"], "device": r["device_name"]}
    if secondary is not None:
        line["secondary"] = secondary
    if muon_entry is not None:
        line["muon"] = muon_entry
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
