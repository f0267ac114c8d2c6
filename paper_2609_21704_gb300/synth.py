"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the oracle.

This module holds none of the method's arithmetic (no quantisation, no
linear algebra of the path, no accept rule): only random draws with the
shapes and distributions of the workloads, so that both sides receive the
same bytes.  Random numbers the method consumes (the uniforms of the accept
step) are drawn here and passed in as inputs.

* weights: fp16 ~ N(0, 0.02) (standard deviation), numpy PCG64 stream.
* activations: fp16 ~ N(0, 1).
* probabilities: softmax of N(0, sigma) logits in fp64, stored fp32; the
  draft distribution is either independent or target + N(0, 0.5) noise.
* uniforms: counter-based splitmix64, u = (z >> 40) * 2^-24, so every
  uniform is a point m * 2^-24 of the 24-bit grid.
* draft tokens: drawn from the draft distribution with numpy's sampler.
"""
from __future__ import annotations

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def splitmix64(seed: int, idx: np.ndarray) -> np.ndarray:
    """The splitmix64 output for counter values idx (Steele, Lea, Flood 2014)."""
    with np.errstate(over="ignore"):
        z = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + (np.asarray(idx, np.uint64) + np.uint64(1)) * _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        z = z ^ (z >> np.uint64(31))
    return z


def uniforms(seed: int, shape) -> np.ndarray:
    """float32 uniforms on the grid m * 2^-24, m in [0, 2^24)."""
    n = int(np.prod(shape))
    z = splitmix64(seed, np.arange(n, dtype=np.uint64))
    m = (z >> np.uint64(40)).astype(np.float64)
    return (m * 2.0 ** -24).astype(np.float32).reshape(shape)


def fp16_normal(seed: int, shape, std: float) -> np.ndarray:
    """fp16 values ~ N(0, std) (numpy PCG64), returned as float16."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal(shape) * std).astype(np.float16)


def weights_fp16(seed: int, n_out: int, k_in: int, std: float = 0.02) -> np.ndarray:
    return fp16_normal(seed, (n_out, k_in), std)


def activations_fp16(seed: int, m: int, k_in: int) -> np.ndarray:
    return fp16_normal(seed, (m, k_in), 1.0)


def _softmax64(z: np.ndarray) -> np.ndarray:
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=-1, keepdims=True)


def spec_block(seed: int, B: int, K: int, V: int, sigma: float = 2.0,
               draft_noise: float | None = 0.5):
    """Synthetic speculative block for the accept step.

    Target logits ~ N(0, sigma) for K+1 positions; draft logits are target +
    N(0, draft_noise) for K positions, or independent N(0, sigma) when
    draft_noise is None.  Returns p [B,K+1,V] f32, q [B,K,V] f32,
    draft [B,K] i32 drawn from q, u [B,K+1] f32 on the 2^-24 grid."""
    rng = np.random.default_rng(seed)
    zt = rng.standard_normal((B, K + 1, V)) * sigma
    if draft_noise is None:
        zd = rng.standard_normal((B, K, V)) * sigma
    else:
        zd = zt[:, :K, :] + rng.standard_normal((B, K, V)) * draft_noise
    p = _softmax64(zt).astype(np.float32)
    q = _softmax64(zd).astype(np.float32)
    draft = np.empty((B, K), np.int32)
    for b in range(B):
        for i in range(K):
            w = q[b, i].astype(np.float64)
            draft[b, i] = rng.choice(V, p=w / w.sum())
    u = uniforms(seed ^ 0x5EED, (B, K + 1))
    return p, q, draft, u


def stack_weight_seed(seed: int, index: int) -> int:
    """Seed of the index-th projection (decoder order, lm_head last) of a
    linear stack built with base seed `seed`."""
    return (seed + index) * 7919 + 17


def rms_gains(seed: int, hidden: int, count: int) -> list:
    """RMSNorm gains 1 + N(0, 0.05), rounded to fp16: two per decoder layer
    (attention, MLP) and then the final norm."""
    return [(1.0 + fp16_normal(seed + i, (hidden,), 0.05).astype(np.float32)).astype(np.float16)
            for i in range(count)]


def prompt_tokens(seed: int, B: int, P: int, vocab: int) -> np.ndarray:
    """Synthetic prompts: int32 [B, P] token ids uniform over the vocabulary."""
    z = splitmix64(seed ^ 0x70C0, np.arange(B * P, dtype=np.uint64))
    return (z % np.uint64(vocab)).astype(np.int32).reshape(B, P)


def weights_fp16_device(seed: int, n_out: int, k_in: int, device, std: float = 0.02):
    """Large fp16 ~ N(0, std) weight matrices drawn on the device with a
    seeded torch generator (used for full-size workloads; tests copy the
    rows they check back to the host for the oracle)."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(seed)
    w = torch.empty((n_out, k_in), dtype=torch.float16, device=device)
    w.normal_(0.0, std, generator=g)
    return w


def activations_fp16_device(seed: int, m: int, k_in: int, device):
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(seed)
    x = torch.empty((m, k_in), dtype=torch.float16, device=device)
    x.normal_(0.0, 1.0, generator=g)
    return x
