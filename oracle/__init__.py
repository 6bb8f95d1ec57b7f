"""CPU oracle of the Deep Parity Bottleneck (DPB) -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The product library never imports,
links or calls it, and the two share no code.

The arithmetic lives in ``dpb_oracle.c`` (plain C, double precision, written
from the paper's definitions; see the header of that file for the sections
and equations each function follows). This module compiles it with gcc on
first use and wraps it with ctypes and numpy.

Config resolution (``resolve``) restates the paper's level layout: level 0 is
the d basis directions (§2.1 Eq. 2) and level l holds the indices
[2^{r_{l-1}}, 2^{r_l}) (§2.2). Where the paper leaves the layout open the same
readings as the C file apply:

* R1  t = max(ceil(log2 d), ceil(r_{L-1} / 2)); rows 0..d-1 of GF(2^t) are used.
* R2  p(z): z^10+z^3+1 (t=10) and z^11+z^2+1 (t=11) as printed in App. A.4
      (Eq. 24); for other t the numerically smallest irreducible polynomial
      with the fewest terms (trinomial, else pentanomial).
* R10 r_l = r_0 + floor(l (N - r_0) / (L - 1)), r_0 = ceil(log2 d).
"""
from __future__ import annotations

import ctypes
import dataclasses
import math
import os
import subprocess
import threading
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dpb_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libdpb_oracle.so")
_lock = threading.Lock()
_lib = None

MAX_LEVELS = 8
GSTRIDE = 1024  # row stride of the generator table (max children per level)

PAPER_POLYS = {10: (1 << 10) | (1 << 3) | 1, 11: (1 << 11) | (1 << 2) | 1}


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/libdpb_oracle.so``."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-Wall", "-shared", "-fPIC",
                    "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        u32, i32, i64, dbl = ctypes.c_uint32, ctypes.c_int, ctypes.c_long, ctypes.c_double
        p = ctypes.c_void_p
        sig = {
            "orc_poly_is_irreducible": (i32, [i32, u32]),
            "orc_gf_mul": (u32, [u32, u32, i32, u32]),
            "orc_gf_inv": (u32, [u32, i32, u32]),
            "orc_gf_trace": (u32, [u32, i32, u32]),
            "orc_kloosterman_bit": (u32, [u32, u32, u32, i32, u32]),
            "orc_seed_matrix": (None, [i32, i32, u32, p]),
            "orc_phi": (None, [i32, p, u32, p]),
            "orc_phi_tilde": (None, [i32, p, u32, p]),
            "orc_generators": (i32, [i32, p, p, ctypes.c_uint64, p, i32]),
            "orc_encode": (i32, [i32, i32, p, p, i32, i32, p, p, i32, p, i64, p, p, p, p, p, p]),
            "orc_encode_per_level": (i32, [i32, i32, p, p, p, p, i32, p, i64, p, p, p, p, p]),
            "orc_decode": (i32, [i32, i32, i32, p, p, p, i64, p, p]),
            "orc_backward": (i32, [i32, i32, i32, p, p, p, p, i64, p, p, p, p]),
            "orc_gf_tables": (None, [i32, u32, p, p, p]),
            "orc_stats_accumulate": (i32, [i32, i32, p, p, p, p, i32, p, i64, p, p, p, i32, p, i64]),
            "orc_stats_update": (None, [i64, p, dbl, p, p]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _i32(seq) -> np.ndarray:
    a = np.zeros(MAX_LEVELS, dtype=np.int32)
    a[: len(seq)] = seq
    return a


# ----------------------------------------------------------------------------
# field and dictionary
# ----------------------------------------------------------------------------

def is_irreducible(t: int, poly: int) -> bool:
    return bool(_load().orc_poly_is_irreducible(t, poly))


def gf_mul(a: int, b: int, t: int, poly: int) -> int:
    return int(_load().orc_gf_mul(a, b, t, poly))


def gf_inv(a: int, t: int, poly: int) -> int:
    return int(_load().orc_gf_inv(a, t, poly))


def gf_trace(y: int, t: int, poly: int) -> int:
    return int(_load().orc_gf_trace(y, t, poly))


def kloosterman_bit(a: int, b: int, xi: int, t: int, poly: int) -> int:
    return int(_load().orc_kloosterman_bit(a, b, xi, t, poly))


def gf_tables(t: int, poly: int, with_mul: bool = True):
    """Whole-field tables (mul[a, b], inv[a], tr[a]) built by the oracle's
    scalar field functions."""
    q = 1 << t
    mul = np.zeros((q, q), dtype=np.uint32) if with_mul else None
    inv = np.zeros(q, dtype=np.uint32)
    tr = np.zeros(q, dtype=np.uint32)
    _load().orc_gf_tables(t, poly, _ptr(mul), _ptr(inv), _ptr(tr))
    return mul, inv, tr


def default_poly(t: int) -> int:
    """Reading R2: the paper's polynomial where it prints one, else the
    numerically smallest irreducible trinomial, else pentanomial."""
    if t in PAPER_POLYS:
        return PAPER_POLYS[t]
    top = 1 << t
    for a in range(1, t):
        p = top | (1 << a) | 1
        if is_irreducible(t, p):
            return p
    best = None
    for a in range(1, t):
        for b in range(1, a):
            for c in range(1, b):
                p = top | (1 << a) | (1 << b) | (1 << c) | 1
                if is_irreducible(t, p) and (best is None or p < best):
                    best = p
    if best is None:
        raise ValueError(f"no irreducible trinomial or pentanomial of degree {t}")
    return best


def seed_matrix(d: int, t: int, poly: int) -> np.ndarray:
    M = np.zeros(d, dtype=np.uint32)
    _load().orc_seed_matrix(d, t, poly, _ptr(M))
    return M


def phi(d: int, M: np.ndarray, i: int) -> np.ndarray:
    out = np.zeros(d, dtype=np.float64)
    _load().orc_phi(d, _ptr(np.ascontiguousarray(M, dtype=np.uint32)), i, _ptr(out))
    return out


def phi_tilde(d: int, M: np.ndarray, i: int) -> np.ndarray:
    out = np.zeros(d, dtype=np.float64)
    _load().orc_phi_tilde(d, _ptr(np.ascontiguousarray(M, dtype=np.uint32)), i, _ptr(out))
    return out


# ----------------------------------------------------------------------------
# configuration
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Config:
    """A resolved DPB configuration as the oracle sees it."""
    d: int
    levels: int
    bits: list          # cumulative r_l, l = 0..levels-1
    children: list      # Delta_l (index 0 unused)
    beam: int
    k: int
    t: int
    poly: int
    seed: int = 0
    norm_match: int = 1
    k_per_level: Optional[list] = None
    M: np.ndarray = dataclasses.field(default=None, repr=False)
    G: np.ndarray = dataclasses.field(default=None, repr=False)

    @property
    def m_bits(self) -> int:
        return self.bits[self.levels - 1]


def resolve(d: int, m_bits: int, levels: int, children: int | Sequence[int], beam: int, k: int,
            seed: int = 0, norm_match: int = 1, t: int = 0, poly: int = 0,
            bits: Optional[Sequence[int]] = None, k_per_level=None,
            generators: Optional[np.ndarray] = None) -> Config:
    r0 = max(1, math.ceil(math.log2(d)))
    if bits is None:
        if levels == 1:
            bits = [r0]
        else:
            bits = [r0 + (l * (m_bits - r0)) // (levels - 1) for l in range(levels)]
    bits = list(bits)
    if isinstance(children, int):
        children = [0] + [children] * (levels - 1)
    children = list(children)
    if t == 0:
        t = max(r0, math.ceil(bits[-1] / 2))
    if poly == 0:
        poly = default_poly(t)
    cfg = Config(d=d, levels=levels, bits=bits, children=children, beam=beam, k=k, t=t,
                 poly=poly, seed=seed, norm_match=norm_match,
                 k_per_level=list(k_per_level) if k_per_level else None)
    cfg.M = seed_matrix(d, t, poly)
    if generators is None:
        cfg.G = generators_table(levels, bits, children, seed)
    else:
        # any [levels, n] table goes into the C side's [MAX_LEVELS, GSTRIDE] rows
        src = np.asarray(generators, dtype=np.uint32)
        cfg.G = np.zeros((MAX_LEVELS, GSTRIDE), dtype=np.uint32)
        cfg.G[: src.shape[0], : src.shape[1]] = src[:, :GSTRIDE]
    return cfg


def generators_table(levels: int, bits: Sequence[int], children: Sequence[int], seed: int) -> np.ndarray:
    G = np.zeros((MAX_LEVELS, GSTRIDE), dtype=np.uint32)
    rc = _load().orc_generators(levels, _ptr(_i32(bits)), _ptr(_i32(children)),
                                ctypes.c_uint64(seed & (2**64 - 1)), _ptr(G), GSTRIDE)
    if rc != 0:
        raise ValueError("generator request exceeds the available generators")
    return G


# ----------------------------------------------------------------------------
# encode / decode / backward
# ----------------------------------------------------------------------------

def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def encode(cfg: Config, x, mu=None, sigma=None):
    """Global-mode encode of rows x[T, d]. Returns idx int32 [T,k], val
    float64 [T,k], xnorm float64 [T], mingap float64 [T]."""
    x = _f64(x)
    T = x.shape[0]
    idx = np.zeros((T, cfg.k), dtype=np.int32)
    val = np.zeros((T, cfg.k), dtype=np.float64)
    xnorm = np.zeros(T, dtype=np.float64)
    gap = np.zeros(T, dtype=np.float64)
    mu = None if mu is None else _f64(mu)
    sigma = None if sigma is None else _f64(sigma)
    rc = _load().orc_encode(cfg.d, cfg.levels, _ptr(_i32(cfg.bits)), _ptr(_i32(cfg.children)),
                            cfg.beam, cfg.k, _ptr(cfg.M), _ptr(cfg.G), GSTRIDE, _ptr(x), T,
                            _ptr(mu), _ptr(sigma), _ptr(idx), _ptr(val), _ptr(xnorm), _ptr(gap))
    if rc != 0:
        raise ValueError(f"oracle encode failed ({rc})")
    return idx, val, xnorm, gap


def encode_per_level(cfg: Config, x, mu=None, sigma=None):
    """Per-level encode (paper form): code = each level's top K_l, level by level."""
    x = _f64(x)
    T = x.shape[0]
    ktot = int(sum(cfg.k_per_level[: cfg.levels]))
    idx = np.zeros((T, ktot), dtype=np.int32)
    val = np.zeros((T, ktot), dtype=np.float64)
    gap = np.zeros(T, dtype=np.float64)
    mu = None if mu is None else _f64(mu)
    sigma = None if sigma is None else _f64(sigma)
    rc = _load().orc_encode_per_level(cfg.d, cfg.levels, _ptr(_i32(cfg.children)),
                                      _ptr(_i32(cfg.k_per_level)), _ptr(cfg.M), _ptr(cfg.G), GSTRIDE,
                                      _ptr(x), T, _ptr(mu), _ptr(sigma), _ptr(idx), _ptr(val), _ptr(gap))
    if rc != 0:
        raise ValueError(f"oracle per-level encode failed ({rc})")
    return idx, val, gap


def decode(cfg: Config, idx, val, xnorm=None, norm_match: Optional[int] = None):
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    val = _f64(val)
    T, k = idx.shape
    nm = cfg.norm_match if norm_match is None else norm_match
    if nm and xnorm is None:
        raise ValueError("norm_match needs xnorm")
    xn = None if xnorm is None else _f64(xnorm)
    y = np.zeros((T, cfg.d), dtype=np.float64)
    _load().orc_decode(cfg.d, k, nm, _ptr(cfg.M), _ptr(idx), _ptr(val), T, _ptr(xn), _ptr(y))
    return y


def backward(cfg: Config, x, idx, val, gy, sigma=None, norm_match: Optional[int] = None):
    x = _f64(x)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    val = _f64(val)
    gy = _f64(gy)
    T, k = idx.shape
    nm = cfg.norm_match if norm_match is None else norm_match
    sg = None if sigma is None else _f64(sigma)
    gx = np.zeros((T, cfg.d), dtype=np.float64)
    gv = np.zeros((T, k), dtype=np.float64)
    _load().orc_backward(cfg.d, k, nm, _ptr(cfg.M), _ptr(x), _ptr(idx), _ptr(val), T, _ptr(sg),
                         _ptr(gy), _ptr(gx), _ptr(gv))
    return gx, gv


# ----------------------------------------------------------------------------
# standardisation moments (§2.2 "Score Standardization")
# ----------------------------------------------------------------------------

def keep_per_level(cfg: Config) -> list:
    """Kept-set size of every level: the beam (global mode) or K_l (per-level)."""
    if cfg.k_per_level:
        return list(cfg.k_per_level[: cfg.levels])
    return [cfg.beam] * cfg.levels


def stats_accumulate(cfg: Config, x, sample, mu=None, sigma=None, acc=None):
    """Moment sums [3, 2^N] (count, sum s, sum s^2): level 0 over every row of
    x, levels >= 1 over the rows listed in ``sample`` (readings R16, R18).
    Adds to ``acc`` when given (float64 [3, 2^N], C order)."""
    x = _f64(x)
    T = x.shape[0]
    m = 1 << cfg.m_bits
    if acc is None:
        acc = np.zeros((3, m), dtype=np.float64)
    assert acc.shape == (3, m) and acc.dtype == np.float64 and acc.flags.c_contiguous
    smp = np.ascontiguousarray(np.asarray(sample, dtype=np.int32).reshape(-1))
    mu = None if mu is None else _f64(mu)
    sigma = None if sigma is None else _f64(sigma)
    rc = _load().orc_stats_accumulate(cfg.d, cfg.levels, _ptr(_i32(cfg.children)),
                                      _ptr(_i32(keep_per_level(cfg))), _ptr(cfg.M), _ptr(cfg.G),
                                      GSTRIDE, _ptr(x), T, _ptr(mu), _ptr(sigma),
                                      _ptr(smp) if smp.size else None, int(smp.size), _ptr(acc), m)
    if rc != 0:
        raise ValueError(f"oracle stats accumulate failed ({rc})")
    return acc


def stats_update(acc, alpha: float, mu, sigma):
    """One EMA step (reading R17). Returns new (mu, sigma) as float64 copies;
    ``acc`` is zeroed in place."""
    assert acc.dtype == np.float64 and acc.flags.c_contiguous and acc.shape[0] == 3
    m = acc.shape[1]
    mu2 = np.array(mu, dtype=np.float64, copy=True).reshape(m)
    sg2 = np.array(sigma, dtype=np.float64, copy=True).reshape(m)
    _load().orc_stats_update(m, _ptr(acc), float(alpha), _ptr(mu2), _ptr(sg2))
    return mu2, sg2
