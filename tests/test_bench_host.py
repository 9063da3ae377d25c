"""Host-side logic of bench.py: the max-over-ranks timing and whole-job
aggregation across processes (gloo, world size 2, CPU only), the JSON of the
reference arm, the committed-traffic lookup, the choice of stash mode and the
division of a set between Muon and AdamW."""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    secs = [2.0, 3.0][rank]
    value, t = bench.aggregate(units_per_rank=600.0, seconds_per_rank=secs, world=world)
    q.put((rank, value, t))
    dist.destroy_process_group()


def test_aggregate_takes_slowest_rank_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, value, t in res:
        assert t == 3.0                      # max over ranks
        assert value == pytest.approx(1200.0 / 3.0)   # all ranks' units / slowest time


def _shard_worker(rank, world, port, q):
    """Partitioned mode: each rank updates its share of one set per step, so
    the whole job's throughput is the set's size over the slowest rank."""
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    args = bench.parse_args(["--gpus", str(world)])
    assert args.parallel == "shard" and bench.sharded(args, world)
    assert not bench.sharded(bench.parse_args(["--parallel", "replica"]), world)
    n_params, steps = 1000, 3
    secs = [0.5, 0.75][rank]
    value, t = bench.aggregate(n_params * steps / world, secs, world)
    q.put((rank, value, t))
    dist.destroy_process_group()


def test_sharded_aggregate_counts_the_set_once_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, value, t in res:
        assert t == 0.75
        assert value == pytest.approx(3000 / 0.75)   # the set's 3 steps / slowest rank


def test_one_gpu_is_never_sharded():
    assert not bench.sharded(bench.parse_args([]), 1)


def test_single_rank_aggregate():
    assert bench.aggregate(10.0, 2.0, 1) == (5.0, 2.0)


def test_reference_arm_json_line():
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0", "--cpu-seconds", "0.5"],
                       capture_output=True, text=True, env=env, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "params/s" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 2
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["higher_is_better"] is True



def test_reference_arm_other_ranks_exit_without_work():
    """Under torchrun only rank 0 runs the oracle arm; another rank prints
    nothing and exits 0 without joining a process group."""
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2", OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "0", "--cpu-seconds", "0.5"],
                       capture_output=True, text=True, env=env, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""

def test_traffic_lookup_ignores_stale_summaries(tmp_path, monkeypatch):
    assert bench.committed_traffic("no-such-kernel") is None


@pytest.mark.parametrize("argv,want", [
    ([], "pingpong"),                                  # llama-7B: bf16 param and stash, EF
    (["--mode", "std"], "pingpong"),
    (["--mode", "sapipe-same"], "copy"),               # the stash holds a prediction
    (["--workload", "gpt2-small-124M"], "copy"),       # fp32 stash
    (["--optimizer", "muon"], "copy"),
    (["--stash", "copy"], "copy"),
])
def test_stash_mode_resolution(argv, want):
    from paper_2606_30634_gb300.synth import workloads as W
    args = bench.parse_args(argv)
    assert bench.resolve_stash(args, W.ALL[args.workload]) == want


def test_muon_takes_the_attention_and_mlp_matrices():
    from paper_2606_30634_gb300.synth import workloads as W
    mi, ai = bench.muon_split(W.LLAMA_7B)
    assert len(mi) == 32 * 7 and len(ai) == len(W.LLAMA_7B.tensors) - 32 * 7
    assert sum(W.LLAMA_7B.numels[i] for i in mi) == 32 * (4 * 4096 * 4096 + 3 * 4096 * 11008)
    names = [W.LLAMA_7B.tensors[i][0] for i in ai]
    assert "embed_tokens" in names and "lm_head" in names and "norm" in names
    mi, _ = bench.muon_split(W.GPT2_SMALL)
    assert len(mi) == 12 * 4 and all(len(W.GPT2_SMALL.tensors[i][1]) == 2 for i in mi)


def test_e2e_host_memory_check_counts_every_rank_on_the_node():
    io = 27 << 30
    assert bench.e2e_fits(2 * io + (16 << 30), io, 1)
    assert not bench.e2e_fits(2 * io + (16 << 30), io, 2)
    assert bench.e2e_fits(8 * 2 * io + (16 << 30), io, 8)


def test_oracle_thread_count_is_settable():
    import oracle
    n = oracle.num_threads()
    oracle.set_num_threads(1)
    try:
        assert oracle.num_threads() == 1
    finally:
        oracle.set_num_threads(n)
    assert oracle.num_threads() == n


def test_committed_traffic_is_per_kernel_variant():
    """The committed headline summary's figure serves the headline only, not
    another rule or mode that runs a different kernel instance: each of those
    takes its own summary's figure, or none."""
    import bench
    head = bench.committed_traffic("fused_step:llama-7B:ef:pingpong")
    assert head is not None
    for tag in ("fused_step:llama-7B:ef:lion:pingpong", "fused_step:llama-7B:std:pingpong",
                "fused_step:llama-7B:ef", "fused_step:llama-7B:ef:dc:pingpong",
                "fused_step:llama-7B:ef:adan:pingpong"):
        got = bench.committed_traffic(tag)
        assert got is None or got != head
    # WPipe's traffic does not scale from one layer to the set: no figure
    assert bench.committed_traffic("fused_step:llama-7B:ef:wpipe:pingpong") is None
    assert bench.committed_traffic("fused_step:llama-7B:ef:pingpong:extra") is None


def test_ns_gemm_traffic_follows_the_newton_schulz_steps():
    """The GEMM chain's committed traffic serves the Newton-Schulz step count
    it was taken with, under any delayed rule, and no other step count."""
    import bench
    got = bench.committed_traffic(bench.ns_gemm_tag("llama-7B", 5), "dram_bytes_per_step")
    assert got is not None and got > 0
    assert bench.committed_traffic(bench.ns_gemm_tag("llama-7B", 3), "dram_bytes_per_step") is None
    assert bench.committed_traffic(bench.ns_gemm_tag("llama-1B", 5), "dram_bytes_per_step") is None
    assert bench.ns_gemm_tag("llama-7B", 5) == "ns_gemm:llama-7B:ns5"
