"""Each pin must fail on a plausible mistake. These tests plant the mistake in
a copy of the oracle's outputs (on the CPU) and check that the pin notices:
swapped halves of the seed matrix, a flipped sign map, a wrong inverse,
a dropped normalisation, a dropped 1/sigma or norm term in the backward,
sampled rows counted at level 0 and a sample deviation in the EMA step."""
import math

import numpy as np

import oracle
from tests import pins


def test_walsh_pin_catches_swapped_halves_and_flipped_signs():
    d, t, poly = 64, 6, 0x43
    M = oracle.seed_matrix(d, t, poly)
    good = lambda i: oracle.phi_tilde(d, M, i)
    assert pins.walsh_rows_mismatch(good, d, t, range(1 << t)) == 0
    swapped = ((M >> t) | ((M & ((1 << t) - 1)) << t)).astype(np.uint32)   # u1 <-> u2
    assert pins.walsh_rows_mismatch(lambda i: oracle.phi_tilde(d, swapped, i), d, t, range(1 << t)) > 0
    flipped = lambda i: -oracle.phi_tilde(d, M, i)                          # R(0) = -1
    assert pins.walsh_rows_mismatch(flipped, d, t, range(1 << t)) > 0
    unscaled = lambda i: oracle.phi_tilde(d, M, i) * math.sqrt(d)           # 1/sqrt(d) dropped
    assert pins.walsh_rows_mismatch(unscaled, d, t, range(1 << t)) > 0


def test_kloosterman_pin_catches_a_wrong_inverse():
    t, poly, d = 6, 0x43, 64
    mul, inv, tr = oracle.gf_tables(t, poly)
    M = oracle.seed_matrix(d, t, poly)
    pairs = [(a, b) for a in range(d) for b in range(d)]
    assert pins.kloosterman_generation_mismatch(M, t, mul, inv, tr, pairs) == 0
    ident = (np.arange(d) | (np.arange(d) << t)).astype(np.uint32)        # inverse = identity
    assert pins.kloosterman_generation_mismatch(ident, t, mul, inv, tr, pairs) > 0
    one_off = M.copy()
    one_off[5] ^= np.uint32(1 << t)                                         # one row's inverse wrong
    assert pins.kloosterman_generation_mismatch(one_off, t, mul, inv, tr, pairs) > 0
    wrong_poly = oracle.seed_matrix(d, t, 0x49)                             # another field: z^6+z^3+1
    assert pins.kloosterman_generation_mismatch(wrong_poly, t, mul, inv, tr, pairs) > 0


def test_coherence_pin_catches_a_random_seed_matrix():
    # Thm A.1's bound holds for the Kloosterman construction, not for an
    # arbitrary matrix of the same shape (§2.1's random-M alternative).
    d, t = 128, 7
    M = np.random.default_rng(0).integers(0, 1 << (2 * t), d).astype(np.uint32)
    assert pins.coherence_by_linearity(M, d, t) > (1 + 2 * math.sqrt(d)) / d


def test_fd_pin_catches_dropped_terms():
    cfg = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8, norm_match=1)
    rng = np.random.default_rng(1)
    x0 = rng.standard_normal((2, cfg.d))
    m = 1 << cfg.m_bits
    sigma = np.full(m, 2.0)
    idx, val, _, _ = oracle.encode(cfg, x0, sigma=sigma)
    w = rng.standard_normal(x0.shape)

    def loss(x):
        v = np.zeros(idx.shape)
        for t in range(idx.shape[0]):
            for e, i in enumerate(idx[t]):
                v[t, e] = float(oracle.phi(cfg.d, cfg.M, int(i)) @ x[t]) / sigma[i]
        return float(np.sum(w * oracle.decode(cfg, idx, v, np.linalg.norm(x, axis=1))))

    good, _ = oracle.backward(cfg, x0, idx, val, w, sigma=sigma)
    assert pins.fd_gradient_mismatch(loss, x0, good) < 1e-6
    no_sigma, _ = oracle.backward(cfg, x0, idx, val, w, sigma=None)          # 1/sigma dropped
    assert pins.fd_gradient_mismatch(loss, x0, no_sigma) > 1e-2
    no_norm, _ = oracle.backward(cfg, x0, idx, val, w, sigma=sigma, norm_match=0)  # norm term dropped
    assert pins.fd_gradient_mismatch(loss, x0, no_norm) > 1e-2


def test_order_invariant_catches_reversed_tie_break():
    cfg = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8)
    x = np.zeros((1, cfg.d))
    x[0, [3, 9, 20]] = [1.0, -1.0, 1.0]                                     # exact ties
    idx, val, _, _ = oracle.encode(cfg, x)
    keys = [(-abs(v), i) for i, v in zip(idx[0], val[0])]
    assert keys == sorted(keys) and idx[0, :3].tolist() == [3, 9, 20]
    rev = [(-abs(v), -i) for i, v in zip(idx[0], val[0])]                   # index descending
    assert rev != sorted(rev)


def test_moment_pins_catch_level0_and_deviation_mistakes():
    cfg = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8)
    x = np.random.default_rng(7).standard_normal((20, cfg.d))
    acc = oracle.stats_accumulate(cfg, x, sample=[1, 2])
    assert pins.column_moment_mismatch(acc, x, cfg.d) < 1e-10
    twice = acc.copy()
    twice[:, : cfg.d] += oracle.stats_accumulate(cfg, x[[1, 2]], sample=[])[:, : cfg.d]
    assert pins.column_moment_mismatch(twice, x, cfg.d) > 1.0      # sampled rows counted again
    m = 1 << cfg.m_bits
    samples = {i: x[:, i] for i in range(cfg.d)}
    acc0 = oracle.stats_accumulate(cfg, x, sample=[])
    mu, sg = oracle.stats_update(acc0, 0.5, np.zeros(m), np.ones(m))
    assert pins.ema_mismatch(mu, sg, np.zeros(m), np.ones(m), 0.5, samples) < 1e-12
    ddof1 = sg.copy()
    ddof1[: cfg.d] = 0.5 + 0.5 * x.std(axis=0, ddof=1)            # sample (n - 1) deviation
    assert pins.ema_mismatch(mu, ddof1, np.zeros(m), np.ones(m), 0.5, samples) > 1e-3
    raw2 = sg.copy()
    raw2[: cfg.d] = 0.5 + 0.5 * np.sqrt((x * x).mean(axis=0))      # second moment, not deviation
    assert pins.ema_mismatch(mu, raw2, np.zeros(m), np.ones(m), 0.5, samples) > 1e-3
