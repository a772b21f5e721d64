"""Seeded synthetic inputs for the ES step: parameter-set shapes, initial
parameters, population seeds and rewards.

This module holds no arithmetic of the method (no noise generator, no
normalisation, no update): it only draws inputs with numpy / torch generators
from fixed seeds, so that the CUDA path and the CPU oracle can be fed the same
values. Rollout rewards are out of scope, so rewards are drawn here from the
distributions of the workloads instead.

Workloads (the paper's LLM checkpoints are stood in for by random weights of
the same shapes):
  toy        1,048,576 fp32 values ~ N(0, 0.02^2), population 8 (seeds 1..8),
             sigma 1e-3, alpha 1e-2, rewards Uniform[0,1]
  quadratic  65,536 fp32, f(theta) = -||theta - theta*||^2, theta* ~ N(0,1),
             32 antithetic pairs, sigma 0.05 -> 0.005 cosine over T = 200,
             alpha 0.01
  qwen4b     Qwen3.5-4B-shaped bf16 set: 36 layers, hidden 2560, 32 query and
             8 KV heads of dim 128, SwiGLU 9728, vocab 151,936, tied
             embeddings (4,022,458,880 parameters, 326 tensors); N = 16,
             sigma 1e-3, Bernoulli(0.3) rewards
  qwen27b    "27B"-shaped bf16 set: 64 layers, hidden 5120, 40 query and 8 KV
             heads of dim 128, SwiGLU 17408, vocab 151,936, untied embeddings
             (22,695,777,280 parameters, 579 tensors); N = 30, sigma_0 5e-4,
             Uniform[0,1] rewards
  qwen4b_fp8 the qwen4b shapes stored as FP8 E4M3 codes with one scale per
             tensor, amax / 448 of its N(0, 0.02^2) weights (norms: 1 / 448,
             so 1.0 is the code 448); N = 16, sigma 1e-3, Bernoulli(0.3)
Weights ~ N(0, 0.02^2), norm weights = 1.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List

import numpy as np


@dataclass(frozen=True)
class TensorSpec:
    name: str
    numel: int
    kind: str  # "weight" or "norm"


def qwen_shapes(layers: int, hidden: int, q_heads: int, kv_heads: int, head_dim: int,
                mlp: int, vocab: int, tied: bool) -> List[TensorSpec]:
    """Parameter tensors of a Qwen-style decoder, in checkpoint order."""
    specs = [TensorSpec("embed_tokens", vocab * hidden, "weight")]
    q, kv = q_heads * head_dim, kv_heads * head_dim
    for l in range(layers):
        p = f"layers.{l}."
        specs += [
            TensorSpec(p + "input_layernorm", hidden, "norm"),
            TensorSpec(p + "q_proj", hidden * q, "weight"),
            TensorSpec(p + "k_proj", hidden * kv, "weight"),
            TensorSpec(p + "v_proj", hidden * kv, "weight"),
            TensorSpec(p + "o_proj", q * hidden, "weight"),
            TensorSpec(p + "post_attention_layernorm", hidden, "norm"),
            TensorSpec(p + "gate_proj", hidden * mlp, "weight"),
            TensorSpec(p + "up_proj", hidden * mlp, "weight"),
            TensorSpec(p + "down_proj", mlp * hidden, "weight"),
        ]
    specs.append(TensorSpec("norm", hidden, "norm"))
    if not tied:
        specs.append(TensorSpec("lm_head", vocab * hidden, "weight"))
    return specs


def qwen4b_shapes() -> List[TensorSpec]:
    return qwen_shapes(36, 2560, 32, 8, 128, 9728, 151_936, tied=True)


def qwen27b_shapes() -> List[TensorSpec]:
    return qwen_shapes(64, 5120, 40, 8, 128, 17_408, 151_936, tied=False)


@dataclass(frozen=True)
class Workload:
    name: str
    dtype: str            # "bf16", "f32" or "e4m3"
    population: int       # N seeds per update
    sigma: float
    alpha: float
    rewards: str          # reward distribution
    description: str


WORKLOADS = {
    "toy": Workload("toy", "f32", 8, 1e-3, 1e-2, "uniform",
                    "1,048,576 fp32 ~ N(0, 0.02^2), N=8, seeds 1..8"),
    "quadratic": Workload("quadratic", "f32", 32, 0.05, 0.01, "quadratic",
                          "65,536 fp32 quadratic, 32 antithetic pairs, T=200"),
    "qwen4b": Workload("qwen4b", "bf16", 16, 1e-3, 5e-4, "bernoulli0.3",
                       "Qwen3.5-4B-shaped bf16 (4,022,458,880 params, 326 tensors), N=16"),
    "qwen27b": Workload("qwen27b", "bf16", 30, 5e-4, 2.5e-4, "uniform",
                        "27B-shaped bf16 (22,695,777,280 params, 579 tensors), N=30"),
    # the 4B shapes in fp32 storage (16.1 GB): the perturb pass moves 8 B per
    # Gaussian there, so HBM rather than the generator bounds it
    "qwen4b_f32": Workload("qwen4b_f32", "f32", 16, 1e-3, 5e-4, "bernoulli0.3",
                           "Qwen3.5-4B-shaped fp32 (4,022,458,880 params, 326 tensors), N=16"),
    # the 4B shapes in FP8 E4M3 storage with a scale per tensor (4.0 GB): the
    # quantized-weight direction of App. A.2 on the config-3 population
    "qwen4b_fp8": Workload("qwen4b_fp8", "e4m3", 16, 1e-3, 5e-4, "bernoulli0.3",
                           "Qwen3.5-4B-shaped FP8 E4M3 with per-tensor scales "
                           "(4,022,458,880 params, 326 tensors), N=16"),
    # profiling case: the 4B shapes cut to 4 layers (about 1.6 GB, larger than L2)
    "qwen4b_4layer": Workload("qwen4b_4layer", "bf16", 16, 1e-3, 5e-4, "bernoulli0.3",
                              "Qwen3.5-4B shapes, 4 layers (792,680,960 params, 38 tensors), N=16"),
}


def shapes_for(name: str) -> List[TensorSpec]:
    if name in ("qwen4b", "qwen4b_f32", "qwen4b_fp8"):
        return qwen4b_shapes()
    if name == "qwen27b":
        return qwen27b_shapes()
    if name == "qwen4b_4layer":
        return qwen_shapes(4, 2560, 32, 8, 128, 9728, 151_936, tied=True)
    if name == "toy":
        return [TensorSpec("theta", 1 << 20, "weight")]
    if name == "quadratic":
        return [TensorSpec("theta", 1 << 16, "weight")]
    raise KeyError(name)


# --- draws ------------------------------------------------------------------------

def normal_f32(n: int, seed: int, std: float = 1.0) -> np.ndarray:
    """n fp32 draws of N(0, std^2) from numpy's PCG64 generator."""
    return (std * np.random.default_rng(seed).standard_normal(n)).astype(np.float32)


def toy_theta() -> np.ndarray:
    """Toy workload: 1,048,576 fp32 values ~ N(0, 0.02^2) from seed 0."""
    return normal_f32(1 << 20, 0, 0.02)


def quadratic_problem(d: int = 1 << 16):
    """(theta_0, theta_star) of the quadratic workload."""
    return normal_f32(d, 0, 0.02), normal_f32(d, 12345, 1.0)


def rewards(kind: str, n: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    if kind == "uniform":
        return rng.uniform(0.0, 1.0, n)
    if kind.startswith("bernoulli"):
        p = float(kind[len("bernoulli"):] or 0.5)
        return (rng.uniform(0.0, 1.0, n) < p).astype(np.float64)
    if kind == "normal":
        return rng.standard_normal(n)
    raise KeyError(kind)


def population_seeds(n: int, generation: int = 0, first: int = 1) -> np.ndarray:
    """Seeds of one generation: first + generation * 1000 + (0..n-1)."""
    start = first + generation * 1000
    return np.arange(start, start + n, dtype=np.uint64)


def init_params_torch(specs: List[TensorSpec], dtype, device, seed: int = 0, std: float = 0.02):
    """One torch tensor per spec: weights ~ N(0, std^2) from a seeded torch
    generator on `device`, norm weights = 1."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    out = []
    for s in specs:
        t = torch.empty(s.numel, dtype=dtype, device=device)
        if s.kind == "norm":
            t.fill_(1.0)
        else:
            t.normal_(0.0, std, generator=gen)
        out.append(t)
    return out


def flat_offsets(specs: List[TensorSpec], align: int = 8) -> List[int]:
    """Element offsets of the tensors packed in one buffer, each rounded up to a
    multiple of `align` elements (16 bytes for bf16 at align 8); the last entry
    is the buffer length."""
    offs, pos = [], 0
    for s in specs:
        offs.append(pos)
        pos = (pos + s.numel + align - 1) // align * align
    offs.append(pos)
    return offs


def init_params_flat(specs: List[TensorSpec], dtype, device, seed: int = 0, std: float = 0.02):
    """The parameter set in one allocation: returns (flat buffer, one view per
    spec). Views start at 16-byte aligned offsets; the padding between them is
    zero and belongs to no tensor. Values as in init_params_torch."""
    import torch
    offs = flat_offsets(specs)
    flat = torch.zeros(offs[-1], dtype=dtype, device=device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    views = []
    for s, o in zip(specs, offs):
        t = flat[o:o + s.numel]
        if s.kind == "norm":
            t.fill_(1.0)
        else:
            t.normal_(0.0, std, generator=gen)
        views.append(t)
    return flat, views


def init_params_flat_e4m3(specs: List[TensorSpec], device, seed: int = 0, std: float = 0.02):
    """The parameter set as FP8 E4M3 codes in one uint8 allocation: returns
    (flat buffer, one view per spec, one scale per spec). Each tensor is drawn
    as in init_params_flat (fp32 here), given the scale amax / 448 (the largest
    E4M3 magnitude is 448) and stored as the nearest E4M3 codes of w / scale
    (torch's float8_e4m3fn conversion). Views start at 16-byte offsets."""
    import torch
    offs = flat_offsets(specs, align=16)
    flat = torch.zeros(offs[-1], dtype=torch.uint8, device=device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    views, scales = [], []
    for s, o in zip(specs, offs):
        w = torch.empty(s.numel, dtype=torch.float32, device=device)
        if s.kind == "norm":
            w.fill_(1.0)
        else:
            w.normal_(0.0, std, generator=gen)
        scale = float(np.float32(max(float(w.abs().max()), 1e-30) / 448.0))
        t = flat[o:o + s.numel]
        t.copy_((w / scale).to(torch.float8_e4m3fn).view(torch.uint8))
        del w
        views.append(t)
        scales.append(scale)
    return flat, views, scales


def sample_offsets(numel: int, n_random: int, seed: int, edge: int = 64) -> np.ndarray:
    """Sorted unique local offsets: the first and last `edge` elements of a
    tensor plus `n_random` uniform ones (parity checks at full size)."""
    rng = np.random.default_rng(seed)
    parts = [np.arange(min(edge, numel)), np.arange(max(0, numel - edge), numel)]
    if n_random:
        parts.append(rng.integers(0, numel, size=n_random))
    return np.unique(np.concatenate(parts)).astype(np.int64)
