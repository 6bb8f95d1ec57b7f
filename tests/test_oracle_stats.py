"""Pins of the oracle's standardisation moments (§2.2 "Score
Standardization"; readings R16-R18): level 0 against numpy's column moments,
the EMA step against hand-worked numbers, the sampled candidate sets against
the encoder's own kept sets (per-level mode makes every level's kept set
visible) and against a whole-dictionary search with spanning generators."""
import numpy as np
import pytest

import oracle
from tests import pins


def _sums(acc, c):
    return acc[0, c], acc[1, c], acc[2, c]


def test_level0_moments_are_numpy_column_moments():
    cfg = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8)
    m = 1 << cfg.m_bits
    rng = np.random.default_rng(0)
    x = 0.5 + 2.0 * rng.standard_normal((40, cfg.d))
    acc = oracle.stats_accumulate(cfg, x, sample=[])
    assert pins.column_moment_mismatch(acc, x, cfg.d) < 1e-10 and not acc[:, cfg.d:].any()
    mu0 = rng.standard_normal(m)
    sg0 = rng.uniform(0.5, 2.0, m)
    mu1, sg1 = oracle.stats_update(acc, 0.25, mu0, sg0)
    samples = {i: x[:, i] for i in range(cfg.d)}
    assert pins.ema_mismatch(mu1, sg1, mu0, sg0, 0.25, samples) < 1e-12
    assert not acc.any()                                   # the step consumes the sums


def test_ema_step_by_hand():
    # feature 1: one occurrence s = 4; feature 2: s in {1, 2}; feature 3: s = 2
    # four times (zero deviation); feature 0 untouched.
    acc = np.zeros((3, 4))
    acc[:, 1] = [1, 4, 16]
    acc[:, 2] = [2, 3, 5]
    acc[:, 3] = [4, 8, 16]
    mu0 = np.array([7.0, 0.0, 0.0, 1.0])
    mu, sg = oracle.stats_update(acc, 0.1, mu0, np.ones(4))
    assert np.allclose(mu, [7.0, 0.4, 0.15, 1.1])
    assert np.allclose(sg, [1.0, 1.0, 0.95, 0.9])          # n = 1 leaves sigma alone
    samples = {1: [4.0], 2: [1.0, 2.0], 3: [2.0] * 4}
    assert pins.ema_mismatch(mu, sg, mu0, np.ones(4), 0.1, samples) < 1e-12


def _kids(parents, gens):
    return {int(p) ^ int(g) for p in parents for g in gens}


@pytest.mark.parametrize("tables", [False, True])
def test_sampled_candidates_are_the_children_of_the_kept_sets(tables):
    # Per-level mode exposes each level's kept set in the code, so the
    # considered set of level l must be exactly the children of level l-1's
    # kept set, each with its raw score <phi_c, x_t>.
    cfg = oracle.resolve(d=64, m_bits=15, levels=3, children=16, beam=4, k=8, bits=[6, 10, 15],
                         k_per_level=[4, 6, 5])
    m = 1 << cfg.m_bits
    rng = np.random.default_rng(1)
    x = rng.standard_normal((9, cfg.d))
    mu = sigma = None
    if tables:
        mu = 0.1 * rng.standard_normal(m)
        sigma = rng.uniform(0.5, 1.5, m)
    sample = [2, 7, 4]
    acc = oracle.stats_accumulate(cfg, x, sample, mu=mu, sigma=sigma)
    idx, _, _ = oracle.encode_per_level(cfg, x, mu=mu, sigma=sigma)
    want_n, want_s, want_q = {}, {}, {}
    for t in sample:
        kept = [idx[t, :4], idx[t, 4:10]]
        for l in (1, 2):
            for c in _kids(kept[l - 1], cfg.G[l, :16]):
                s = float(oracle.phi(cfg.d, cfg.M, c) @ x[t])
                want_n[c] = want_n.get(c, 0) + 1
                want_s[c] = want_s.get(c, 0.0) + s
                want_q[c] = want_q.get(c, 0.0) + s * s
    got = {int(c) for c in np.nonzero(acc[0, cfg.d:])[0] + cfg.d}
    assert got == set(want_n)
    for c in want_n:
        n, s, q = _sums(acc, c)
        assert n == want_n[c] and abs(s - want_s[c]) < 1e-12 and abs(q - want_q[c]) < 1e-12


def test_global_mode_candidates_are_those_of_a_per_level_search_with_beam_quotas():
    # Global mode keeps the top `beam` of every level: the same search as
    # per-level mode with K_l = beam, so both must consider the same features.
    common = dict(d=64, m_bits=15, levels=4, children=16, beam=3, k=8, bits=[6, 9, 12, 15])
    g = oracle.resolve(**common)
    p = oracle.resolve(**common, k_per_level=[3, 3, 3, 3])
    x = np.random.default_rng(2).standard_normal((6, g.d))
    a = oracle.stats_accumulate(g, x, [0, 1, 5])
    b = oracle.stats_accumulate(p, x, [0, 1, 5])
    assert np.array_equal(a, b) and a[0, g.d:].sum() > 0


def test_spanning_generators_consider_the_whole_dictionary():
    # With every node kept and generators that reach every index, each sampled
    # token considers every feature exactly once: count = samples, and the
    # sums are those of the dense scores Phi x over the sample.
    G = np.zeros((oracle.MAX_LEVELS, oracle.GSTRIDE), dtype=np.uint32)
    G[1, :16] = [h << 6 for h in range(1, 8)] + [(1 << 6) | s for s in range(1, 10)]
    G[2, :16] = [(h << 9) | s for h in range(1, 8) for s in (0, 64)] + [(1 << 9) | 1, (2 << 9) | 3]
    cfg = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=100000, k=16, generators=G)
    x = np.random.default_rng(3).standard_normal((5, cfg.d))
    sample = [4, 0, 4]                                     # a row may be drawn twice
    acc = oracle.stats_accumulate(cfg, x, sample)
    Phi = np.stack([oracle.phi(cfg.d, cfg.M, c) for c in range(cfg.d, 1 << 12)])
    S = x[sample] @ Phi.T
    assert np.all(acc[0, cfg.d:] == 3)
    assert np.allclose(acc[1, cfg.d:], S.sum(axis=0), atol=1e-12)
    assert np.allclose(acc[2, cfg.d:], (S * S).sum(axis=0), atol=1e-12)


def test_bad_sample_rows_are_rejected():
    cfg = oracle.resolve(d=64, m_bits=12, levels=2, children=16, beam=4, k=8)
    x = np.zeros((3, cfg.d))
    for bad in ([3], [-1]):
        with pytest.raises(ValueError):
            oracle.stats_accumulate(cfg, x, bad)
