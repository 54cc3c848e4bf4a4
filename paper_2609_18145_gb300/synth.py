"""Seeded synthetic inputs shared by the tests, the benchmark and the smoke check.

This module only draws random numbers and lays them out; it holds none of the
mixing layer's arithmetic (no partner rule, no products, no sums), so that the
device path and the CPU oracle can be fed identical inputs without sharing
any code that computes the method.

Recipes (the paper's corpora are not available; these stand in for their
shapes, which is all the mixing cost depends on):

* activations x ~ N(0, 1);
* weights W_self, W_nbr ~ N(0, 1/d) for the tiny check and N(0, 1/(2d)) for
  the timed stacks (keeps the activation scale steady over 16 layers);
* bias ~ N(0, 0.1^2);
* character-LM ids: Zipf(1.1) over a byte vocabulary of 256 (rank r has
  probability proportional to r^-1.1, rank r is byte r-1), embedded through
  an N(0, 1) table [256, d];
* reachability ids: uniform over 16 symbols, embedded through [16, d].

All host draws use numpy's PCG64 with an explicit seed.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def normal(shape, seed: int, std: float = 1.0) -> np.ndarray:
    return (rng(seed).standard_normal(shape) * std).astype(np.float32)


def zipf_ids(B: int, n: int, seed: int, vocab: int = 256, alpha: float = 1.1) -> np.ndarray:
    ranks = np.arange(1, vocab + 1, dtype=np.float64)
    p = ranks ** (-alpha)
    p /= p.sum()
    return rng(seed).choice(vocab, size=(B, n), p=p).astype(np.int64)


def uniform_ids(B: int, n: int, seed: int, vocab: int = 16) -> np.ndarray:
    return rng(seed).integers(0, vocab, size=(B, n)).astype(np.int64)


def embed(ids: np.ndarray, table: np.ndarray) -> np.ndarray:
    """Row lookup table[ids] (input preparation, not part of the mixing path)."""
    return table[ids]


@dataclass
class Problem:
    """Seeded inputs of a stack of L mixing layers (float32, not yet rounded)."""
    x: np.ndarray          # [B, n, d]
    W_self: np.ndarray     # [L, d, d]  (d_out, d_in)
    W_nbr: np.ndarray      # [L, d, d]
    bias: np.ndarray       # [L, d]
    dy: np.ndarray         # [B, n, d]  upstream gradient for backward checks
    z: np.ndarray = field(default=None)  # [L, B, n, d] pre-activations for layer-level bwd checks


def problem(B: int, n: int, d: int, L: int = 1, seed: int = 0, w_std: float | None = None,
            bias_std: float = 0.1, x_ids: str | None = None) -> Problem:
    """Draw one seeded problem.  ``x_ids`` selects token-id inputs
    ("zipf256" or "uniform16") embedded through an N(0,1) table instead of
    x ~ N(0,1)."""
    if w_std is None:
        w_std = (1.0 / d) ** 0.5
    if x_ids == "zipf256":
        ids = zipf_ids(B, n, seed + 11)
        x = embed(ids, normal((256, d), seed + 12))
    elif x_ids == "uniform16":
        ids = uniform_ids(B, n, seed + 11)
        x = embed(ids, normal((16, d), seed + 12))
    else:
        x = normal((B, n, d), seed + 1)
    return Problem(
        x=np.ascontiguousarray(x, dtype=np.float32),
        W_self=normal((L, d, d), seed + 2, w_std),
        W_nbr=normal((L, d, d), seed + 3, w_std),
        bias=normal((L, d), seed + 4, bias_std),
        dy=normal((B, n, d), seed + 5),
        z=normal((L, B, n, d), seed + 6),
    )


def to_bf16_exact(a: np.ndarray):
    """Round a float32 array to bfloat16 (torch's conversion, ties to even)
    and return (bf16 torch tensor on CPU, float64 numpy copy of its exact
    values).  The oracle consumes the float64 copy so both sides see the
    same numbers."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t, t.to(torch.float64).numpy()


def device_normal(shape, seed: int, device):
    """N(0, 1) float32 drawn on `device` by torch's seeded generator, for inputs
    too large to draw on the host (the 2^20-token scaling shapes)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32)


# The workloads, by what they are.  Used by the benchmark and the tests.
WORKLOADS = {
    "tiny_n16_d32": dict(n=16, d=32, L=4, B=4, causal=False, w_std=(1 / 32) ** 0.5),
    "reach_n64_d128": dict(n=64, d=128, L=6, B=256, causal=False, x_ids="uniform16"),
    "charlm_w64_d512": dict(n=64, d=512, L=16, B=64, causal=True, x_ids="zipf256"),
    "charlm_w256_d512": dict(n=256, d=512, L=16, B=64, causal=True, x_ids="zipf256"),
    # scaling sweep: 2^20 tokens per batch, L = log2 n rotated layers, d = 1024
    "scale_n256_d1024": dict(n=256, d=1024, L=8, B=4096, causal=False),
    "scale_n4096_d1024": dict(n=4096, d=1024, L=12, B=256, causal=False),
    "scale_n65536_d1024": dict(n=65536, d=1024, L=16, B=16, causal=False),
}


@dataclass
class BlockProblem:
    """Seeded inputs of the character-LM block around a stack (float32, not yet
    rounded): ids of a window of n + 1 symbols (inputs ids[:, :n], next-symbol
    targets ids[:, 1:]), the token and position tables, per layer the two
    LayerNorms, the mixing maps and the FFN (hidden h), the final LayerNorm
    and the output head."""
    ids: np.ndarray      # [B, n + 1] int64 in [0, V)
    E: np.ndarray        # [V, d]
    P: np.ndarray        # [n, d]
    ln1_g: np.ndarray    # [L, d]
    ln1_b: np.ndarray    # [L, d]
    W_self: np.ndarray   # [L, d, d]
    W_nbr: np.ndarray    # [L, d, d]
    ln2_g: np.ndarray    # [L, d]
    ln2_b: np.ndarray    # [L, d]
    W1: np.ndarray       # [L, h, d]
    b1: np.ndarray       # [L, h]
    W2: np.ndarray       # [L, d, h]
    b2: np.ndarray       # [L, d]
    lnf_g: np.ndarray    # [d]
    lnf_b: np.ndarray    # [d]
    Wh: np.ndarray       # [V, d]
    bh: np.ndarray       # [V]


def block_problem(B: int, n: int, d: int, h: int, V: int, L: int, seed: int = 0) -> BlockProblem:
    """Draw one seeded block problem: Zipf(1.1) ids over V symbols; E ~ N(0, 1);
    P ~ N(0, 0.1^2); LayerNorm scales 1 + N(0, 0.1^2) and shifts N(0, 0.1^2);
    W_self, W_nbr ~ N(0, 1/(2d)); W1 ~ N(0, 1/d), W2 ~ N(0, 1/h), Wh ~ N(0, 1/d);
    biases N(0, 0.1^2)."""
    s = seed * 100

    def nrm(shape, k, std):
        return normal(shape, s + k, std)

    return BlockProblem(
        ids=zipf_ids(B, n + 1, s + 1, vocab=V),
        E=nrm((V, d), 2, 1.0),
        P=nrm((n, d), 3, 0.1),
        ln1_g=(1.0 + nrm((L, d), 4, 0.1)).astype(np.float32),
        ln1_b=nrm((L, d), 5, 0.1),
        W_self=nrm((L, d, d), 6, (1.0 / (2 * d)) ** 0.5),
        W_nbr=nrm((L, d, d), 7, (1.0 / (2 * d)) ** 0.5),
        ln2_g=(1.0 + nrm((L, d), 8, 0.1)).astype(np.float32),
        ln2_b=nrm((L, d), 9, 0.1),
        W1=nrm((L, h, d), 10, (1.0 / d) ** 0.5),
        b1=nrm((L, h), 11, 0.1),
        W2=nrm((L, d, h), 12, (1.0 / h) ** 0.5),
        b2=nrm((L, d), 13, 0.1),
        lnf_g=(1.0 + nrm((d,), 14, 0.1)).astype(np.float32),
        lnf_b=nrm((d,), 15, 0.1),
        Wh=nrm((V, d), 16, (1.0 / d) ** 0.5),
        bh=nrm((V,), 17, 0.1),
    )
