"""Parameter sets the tests and the benchmark run the step on.

Synthetic stand-ins for the paper's models (arXiv 2606.30634, App. E.2 trains
SmolLM2 135M/360M dense models and 2B/10B MoE models on FineWeb-Edu; no
weights or data are used here): tensor tables with the exact shapes of
GPT-2 small, Llama-3.2-1B and Llama-2-7B, plus a flat vector and a noisy
diagonal quadratic. Values come from the seeded generator (see
``paper_2606_30634_gb300.synth``).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Tuple

F32, BF16 = 0, 1   # same values as DPO_F32 / DPO_BF16


@dataclass(frozen=True)
class Workload:
    name: str
    tensors: Tuple[Tuple[str, Tuple[int, ...]], ...]
    param_dtype: int
    stash_dtype: int
    grad_dtype: int
    steps: int
    max_grad_norm: float = 0.0
    seed: int = 0xD0D0
    lr: float = 3e-4
    beta1: float = 0.9
    beta2: float = 0.95
    eps: float = 1e-8
    weight_decay: float = 0.1
    quadratic: bool = False

    @property
    def numels(self) -> List[int]:
        out = []
        for _, shape in self.tensors:
            n = 1
            for s in shape:
                n *= s
            out.append(n)
        return out

    @property
    def n_params(self) -> int:
        return sum(self.numels)


def _gpt2_small():
    d, ffn, vocab, ctx, layers = 768, 3072, 50257, 1024, 12
    t = [("wte", (vocab, d)), ("wpe", (ctx, d))]
    for i in range(layers):
        p = f"h.{i}."
        t += [(p + "ln_1.weight", (d,)), (p + "ln_1.bias", (d,)),
              (p + "attn.c_attn.weight", (d, 3 * d)), (p + "attn.c_attn.bias", (3 * d,)),
              (p + "attn.c_proj.weight", (d, d)), (p + "attn.c_proj.bias", (d,)),
              (p + "ln_2.weight", (d,)), (p + "ln_2.bias", (d,)),
              (p + "mlp.c_fc.weight", (d, ffn)), (p + "mlp.c_fc.bias", (ffn,)),
              (p + "mlp.c_proj.weight", (ffn, d)), (p + "mlp.c_proj.bias", (d,))]
    t += [("ln_f.weight", (d,)), ("ln_f.bias", (d,))]
    return tuple(t)


def _llama(d, ffn, vocab, layers, n_q, n_kv, tied):
    hd = d // n_q
    t = [("embed_tokens", (vocab, d))]
    for i in range(layers):
        p = f"layers.{i}."
        t += [(p + "q_proj", (n_q * hd, d)), (p + "k_proj", (n_kv * hd, d)),
              (p + "v_proj", (n_kv * hd, d)), (p + "o_proj", (d, n_q * hd)),
              (p + "gate_proj", (ffn, d)), (p + "up_proj", (ffn, d)),
              (p + "down_proj", (d, ffn)),
              (p + "input_layernorm", (d,)), (p + "post_attention_layernorm", (d,))]
    t += [("norm", (d,))]
    if not tied:
        t += [("lm_head", (vocab, d))]
    return tuple(t)


FLAT = Workload("flat-fp32-1M", (("x", (1 << 20,)),), F32, F32, F32, steps=10, seed=0xD0D0 + 1)
QUADRATIC = Workload("quadratic-fp32-16M", (("w", (1 << 24,)),), F32, F32, F32, steps=1000,
                     seed=0xD0D0 + 2, quadratic=True)
GPT2_SMALL = Workload("gpt2-small-124M", _gpt2_small(), BF16, F32, BF16, steps=100,
                      seed=0xD0D0 + 3)
LLAMA_1B = Workload("llama-1B", _llama(2048, 8192, 128256, 16, 32, 8, tied=True), BF16, F32,
                    BF16, steps=50, max_grad_norm=1.0, seed=0xD0D0 + 4)
LLAMA_7B = Workload("llama-7B", _llama(4096, 11008, 32000, 32, 32, 32, tied=False), BF16, BF16,
                    BF16, steps=20, seed=0xD0D0 + 5)

# One decoder layer of the 7B shapes with the 7B dtypes: the same kernel
# instance on a ~4.4 GB working set (profiler captures).
LLAMA_7B_LAYER = Workload("llama-7B-layer", LLAMA_7B.tensors[1:10], BF16, BF16, BF16, steps=20,
                          seed=0xD0D0 + 5)

# Two decoder layers of the 7B shapes: every Newton-Schulz shape group of
# delayed Muon has as many tiles per launch as the full set's keep to their
# own launches (more than 16 rounds over the CTA pairs), so the GEMM chain
# runs as on the full set (profiler captures, about 9 GB on the device).
LLAMA_7B_2LAYERS = Workload("llama-7B-2layers", LLAMA_7B.tensors[1:19], BF16, BF16, BF16,
                            steps=20, seed=0xD0D0 + 5)

# Four decoder layers of the 1B shapes with the 1B dtypes and clipping: the
# same two kernel instances as the clipped 1B step (norm pass, fused step) on
# 243M parameters, whose 486 MB of bf16 gradients exceed the 129 MB L2
# (profiler captures).
LLAMA_1B_4LAYERS = Workload("llama-1B-4layers", LLAMA_1B.tensors[1:37], BF16, F32, BF16,
                            steps=50, max_grad_norm=1.0, seed=0xD0D0 + 4)

ALL = {w.name: w for w in (FLAT, QUADRATIC, GPT2_SMALL, LLAMA_1B, LLAMA_7B, LLAMA_7B_LAYER,
                           LLAMA_7B_2LAYERS, LLAMA_1B_4LAYERS)}

# the quadratic's noise and curvature
QUAD_NOISE_SIGMA = 1e-2
INIT_SIGMA = 0.02
GRAD_SIGMA = 1e-3
