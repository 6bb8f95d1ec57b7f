"""Seeded synthetic inputs, shared by the oracle tests and the CUDA path.

This module only draws random numbers (numpy PCG64, fixed seeds) and rounds
them to bf16. It holds none of the DPB arithmetic: planted codes are returned
as a tree of *choices* (root coordinates, parent slots, generator slots,
coefficients); each consumer turns the choices into feature indices with its
own child map and into activations with its own decoder.

The paper's workloads are residual-stream activations of FineWeb-Edu-trained
models, which are not available here; these distributions stand in for them:

* gaussian_rows: x ~ N(0, 1), optionally with a fraction of rows scaled
  (outlier tokens), the GPT-2-width workload.
* planted_tree: a sparse code with the hierarchy's shape (roots at level 0,
  then children of planted nodes level by level), coefficients +-U[1, 2],
  the wide workload (x = decoded code + N(0, 0.1^2) noise).
"""
from __future__ import annotations

import dataclasses

import numpy as np


def rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(np.random.PCG64(seed))


def to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns
    float32 values that are exactly representable in bf16."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """The upper 16 bits of float32 values already rounded by to_bf16."""
    return (np.ascontiguousarray(a, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def gaussian_rows(T: int, d: int, seed: int, outlier_frac: float = 0.0,
                  outlier_scale: float = 10.0) -> np.ndarray:
    """x[T, d] float32 ~ N(0, 1); a random `outlier_frac` of rows scaled."""
    g = rng(seed)
    x = g.standard_normal((T, d), dtype=np.float32)
    if outlier_frac > 0:
        n = int(round(outlier_frac * T))
        rows = g.choice(T, size=n, replace=False)
        x[rows] *= np.float32(outlier_scale)
    return x


def normal(shape, seed: int, scale: float = 1.0) -> np.ndarray:
    return (rng(seed).standard_normal(shape, dtype=np.float32) * np.float32(scale))


def sample_rows(T: int, n: int, seed: int) -> np.ndarray:
    """min(n, T) distinct row numbers of [0, T), drawn uniformly (int32)."""
    return rng(seed).permutation(T)[: min(n, T)].astype(np.int32)


def coset_generators(bits, levels: int, seed: int, max_children: int = 256) -> np.ndarray:
    """Generator table [8, max_children] uint32 where level l >= 1 holds one
    coset g0 ^ {0, ..., 15}: g0 drawn uniformly from [2^{r_{l-1}}, 2^{r_l})
    with its low 4 bits cleared, g_j = g0 | j (every g_j keeps g0's level bit)."""
    g = rng(seed)
    out = np.zeros((8, max_children), dtype=np.uint32)
    for l in range(1, levels):
        lo, hi = 1 << bits[l - 1], 1 << bits[l]
        g0 = int(g.integers(lo, hi)) & ~15
        if g0 < lo:
            g0 = lo
        out[l, :16] = [g0 | j for j in range(16)]
    return out


def mixed_codes(T: int, d: int, m_bits: int, k: int, hashed_counts, seed: int):
    """Codes idx int32 [T, k] and val float32 [T, k] ~ N(0, 1) in which token t
    has hashed_counts[t % len] distinct entries in [d, 2^m_bits) and the rest
    distinct entries below d (basis), in random order."""
    g = rng(seed)
    counts = list(hashed_counts)
    idx = np.zeros((T, k), dtype=np.int32)
    for t in range(T):
        nh = counts[t % len(counts)]
        if nh > k or k - nh > d:
            raise ValueError("a code of %d entries cannot hold %d hashed ones at d = %d" % (k, nh, d))
        ids = np.concatenate([g.choice(d, k - nh, replace=False),
                              d + g.choice((1 << m_bits) - d, nh, replace=False)])
        g.shuffle(ids)
        idx[t] = ids
    val = g.standard_normal((T, k), dtype=np.float32)
    return idx, val


def moment_tables(m: int, seed: int, mean_scale: float = 0.2, sigma_range=(0.5, 2.0)):
    """Standardisation tables (mu, sigma) fp32 [m]: mu ~ N(0, mean_scale^2),
    sigma uniform in sigma_range."""
    g = rng(seed)
    mu = (g.standard_normal(m) * mean_scale).astype(np.float32)
    sigma = g.uniform(sigma_range[0], sigma_range[1], m).astype(np.float32)
    return mu, sigma


@dataclasses.dataclass
class PlantedTree:
    """Random choices of a planted hierarchical code, per token.

    roots[t, r]            level-0 coordinates (distinct, < d)
    parent[l][t, e]        slot of the parent among level l-1's planted nodes
    gen[l][t, e]           generator slot j < children[l] used for that child
    coef[t, e]             coefficients, level by level (roots first)
    """
    roots: np.ndarray
    parent: list
    gen: list
    coef: np.ndarray


def _distinct_rows(g: np.random.Generator, T: int, n: int, high: int) -> np.ndarray:
    """[T, n] integers below `high`, distinct within each row: a random
    permutation prefix when collisions are likely, else redraws of the rows
    that repeat a value."""
    if n * n > high // 4:
        return np.argsort(g.random((T, high)), axis=1)[:, :n]
    out = g.integers(0, high, size=(T, n))
    while True:
        s = np.sort(out, axis=1)
        bad = np.nonzero(np.any(s[:, 1:] == s[:, :-1], axis=1))[0]
        if len(bad) == 0:
            return out
        out[bad] = g.integers(0, high, size=(len(bad), n))


def planted_tree(T: int, d: int, levels: int, children, per_level, seed: int) -> PlantedTree:
    g = rng(seed)
    roots = _distinct_rows(g, T, per_level[0], d).astype(np.int64)
    parent, gen = [None], [None]
    for l in range(1, levels):
        n_prev, n_here = per_level[l - 1], per_level[l]
        # distinct (parent slot, generator slot) pairs per token
        pairs = _distinct_rows(g, T, n_here, n_prev * children[l])
        parent.append(pairs // children[l])
        gen.append(pairs % children[l])
    k = int(sum(per_level[:levels]))
    mag = g.uniform(1.0, 2.0, size=(T, k))
    sign = np.where(g.random((T, k)) < 0.5, -1.0, 1.0)
    return PlantedTree(roots=roots, parent=parent, gen=gen, coef=(mag * sign))
