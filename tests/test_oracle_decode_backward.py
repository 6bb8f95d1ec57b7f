"""Pins of the oracle's decoder (§2.1, normalised output of §2.2) and of the
derived backward: one-hot codes decode to the direction itself (Walsh rows
from scipy where the index has no high half), linearity, norm matching, and
central finite differences of the whole encode-then-decode map with the
selected set held fixed."""
import math

import numpy as np
import pytest
import scipy.linalg

import oracle
from tests import pins


def _cfg(norm_match=1, d=64):
    if d == 64:
        return oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8,
                              norm_match=norm_match)
    return oracle.resolve(d=768, m_bits=20, levels=5, children=16, beam=8, k=64,
                          norm_match=norm_match)


def test_one_hot_decodes_to_direction():
    # North-star pin: decode of a one-hot code equals phi_i. For d = 768 and
    # 768 <= i < 1024 the index has no high half, so phi_i is the Walsh row
    # H_1024[i, :768] / sqrt(768); for i < d it is the basis vector e_i.
    cfg = _cfg(norm_match=0, d=768)
    H = scipy.linalg.hadamard(1024)
    rows = [768, 800, 1000, 1023]
    idx = np.array([[i] for i in rows], dtype=np.int32)
    y = oracle.decode(cfg, idx, np.ones((len(rows), 1)), norm_match=0)
    for r, i in enumerate(rows):
        assert np.allclose(y[r], H[i, :768] / math.sqrt(768), rtol=0, atol=1e-15)
    idx = np.array([[3], [767]], dtype=np.int32)
    y = oracle.decode(cfg, idx, np.full((2, 1), 2.5), norm_match=0)
    assert y[0, 3] == 2.5 and y[1, 767] == 2.5 and np.count_nonzero(y) == 2
    rng = np.random.default_rng(0)
    for i in rng.integers(1024, 1 << 20, 20):
        y = oracle.decode(cfg, np.array([[i]], dtype=np.int32), np.ones((1, 1)), norm_match=0)
        assert np.array_equal(y[0], oracle.phi(768, cfg.M, int(i)))


def test_decode_is_linear_and_norm_matched():
    cfg = _cfg(norm_match=1)
    rng = np.random.default_rng(1)
    x = rng.standard_normal((20, cfg.d))
    idx, val, xnorm, _ = oracle.encode(cfg, x)
    a, b = rng.standard_normal(val.shape), rng.standard_normal(val.shape)
    ya, yb = oracle.decode(cfg, idx, a, norm_match=0), oracle.decode(cfg, idx, b, norm_match=0)
    assert np.allclose(oracle.decode(cfg, idx, a + b, norm_match=0), ya + yb, atol=1e-12)
    y = oracle.decode(cfg, idx, val, xnorm)
    r = oracle.decode(cfg, idx, val, norm_match=0)
    assert np.allclose(np.linalg.norm(y, axis=1), xnorm)                 # |y| = |x|
    cos = np.sum(y * r, axis=1) / (np.linalg.norm(y, axis=1) * np.linalg.norm(r, axis=1))
    assert np.allclose(cos, 1.0)                                          # y parallel to r
    z = oracle.decode(cfg, idx, np.zeros_like(val), xnorm)                # |r| = 0 -> y = 0
    assert np.all(z == 0)


def _val_of(cfg, x, idx, mu, sigma):
    """Coefficients of a fixed index set as functions of x (the encoder's
    val with the selection held fixed)."""
    out = np.zeros(idx.shape)
    for t in range(idx.shape[0]):
        for e, i in enumerate(idx[t]):
            s = float(oracle.phi(cfg.d, cfg.M, int(i)) @ x[t])
            out[t, e] = (s - mu[i]) / sigma[i]
    return out


@pytest.mark.parametrize("norm_match", [0, 1])
@pytest.mark.parametrize("with_stats", [False, True])
def test_backward_matches_finite_differences(norm_match, with_stats):
    cfg = _cfg(norm_match=norm_match)
    rng = np.random.default_rng(2)
    T = 3
    x0 = rng.standard_normal((T, cfg.d))
    m = 1 << cfg.m_bits
    mu = rng.standard_normal(m) * 0.1 if with_stats else np.zeros(m)
    sigma = rng.uniform(0.5, 2.0, m) if with_stats else np.ones(m)
    idx, val, _, _ = oracle.encode(cfg, x0, mu=mu, sigma=sigma)
    w = rng.standard_normal((T, cfg.d))

    def loss_x(x):
        v = _val_of(cfg, x, idx, mu, sigma)
        y = oracle.decode(cfg, idx, v, np.linalg.norm(x, axis=1))
        return float(np.sum(w * y))

    gx, gv = oracle.backward(cfg, x0, idx, val, w, sigma=sigma)
    assert pins.fd_gradient_mismatch(loss_x, x0, gx) < 1e-6

    xn = np.linalg.norm(x0, axis=1)

    def loss_v(v):
        return float(np.sum(w * oracle.decode(cfg, idx, v, xn)))

    assert pins.fd_gradient_mismatch(loss_v, val, gv) < 1e-6


def test_backward_zero_reconstruction_gives_zero_gradient():
    cfg = _cfg(norm_match=1)
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, cfg.d))
    idx, val, _, _ = oracle.encode(cfg, x)
    gx, gv = oracle.backward(cfg, x, idx, np.zeros_like(val), rng.standard_normal(x.shape))
    assert np.all(gx == 0) and np.all(gv == 0)
