"""Pins of the oracle's encoder (§2.2): with a beam wide enough to hold every
node, the beam search must equal a brute-force top-k over the reachable set;
with generators that reach the whole dictionary it must equal a plain flat
top-k; plus ordering invariants, standardisation and planted-code recovery."""
import math

import numpy as np
import pytest

import oracle


def _tiny(beam=4, k=8, generators=None, norm_match=1):
    return oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=beam, k=k,
                          norm_match=norm_match, generators=generators)


def _reachable(cfg):
    """Closure of the child map: R_0 = basis, R_l = {p ^ g : p in R_{l-1}, g in G_l}."""
    levels = [set(range(cfg.d))]
    for l in range(1, cfg.levels):
        gens = cfg.G[l, : cfg.children[l]].tolist()
        levels.append({p ^ g for p in levels[-1] for g in gens})
    return levels


def _brute_topk(cfg, x, universe, k):
    idx = np.array(sorted(universe), dtype=np.int64)
    Phi = np.stack([oracle.phi(cfg.d, cfg.M, int(i)) for i in idx])
    out_i, out_v = [], []
    for row in np.asarray(x, dtype=np.float64):
        s = Phi @ row
        order = sorted(range(len(idx)), key=lambda e: (-abs(s[e]), idx[e]))[:k]
        out_i.append(idx[order])
        out_v.append(s[order])
    return np.array(out_i), np.array(out_v)


def test_generators_follow_the_level_rule():
    # §2.2: g_j < 2^{r_l} with a set bit at or above r_{l-1}; distinct.
    cfg = oracle.resolve(d=768, m_bits=20, levels=5, children=16, beam=8, k=64)
    assert cfg.bits == [10, 12, 15, 17, 20]
    for l in range(1, 5):
        g = cfg.G[l, :16].astype(np.int64)
        assert len(set(g.tolist())) == 16
        assert np.all(g < (1 << cfg.bits[l])) and np.all((g >> cfg.bits[l - 1]) != 0)


def test_wide_beam_equals_brute_force_over_reachable_set():
    cfg = _tiny(beam=100000, k=24)
    R = _reachable(cfg)
    x = np.random.default_rng(0).standard_normal((12, cfg.d))
    idx, val, _, _ = oracle.encode(cfg, x)
    bi, bv = _brute_topk(cfg, x, set().union(*R), cfg.k)
    assert np.array_equal(idx, bi)
    assert np.allclose(val, bv, rtol=0, atol=1e-12)


def test_spanning_generators_give_flat_topk_over_whole_dictionary():
    # Generators whose children reach every index of every level: the wide
    # beam search must then equal a flat TopK over all 2^12 features.
    G = np.zeros((oracle.MAX_LEVELS, oracle.GSTRIDE), dtype=np.uint32)
    g1 = [h << 6 for h in range(1, 8)] + [(1 << 6) | s for s in range(1, 10)]
    g2 = [(h << 9) | s for h in range(1, 8) for s in (0, 64)] + [(1 << 9) | 1, (2 << 9) | 3]
    G[1, :16], G[2, :16] = g1, g2
    cfg = _tiny(beam=100000, k=16, generators=G)
    R = _reachable(cfg)
    assert set().union(*R) == set(range(1 << 12))
    x = np.random.default_rng(1).standard_normal((6, cfg.d))
    idx, val, _, _ = oracle.encode(cfg, x)
    bi, bv = _brute_topk(cfg, x, range(1 << 12), cfg.k)
    assert np.array_equal(idx, bi)
    assert np.allclose(val, bv, rtol=0, atol=1e-12)


@pytest.mark.parametrize("shape", ["tiny", "gpt2"])
def test_code_invariants(shape):
    if shape == "tiny":
        cfg, T = _tiny(), 64
    else:
        cfg, T = oracle.resolve(d=768, m_bits=16, levels=4, children=16, beam=8, k=32), 8
    x = np.random.default_rng(2).standard_normal((T, cfg.d))
    idx, val, xnorm, gap = oracle.encode(cfg, x)
    r0 = cfg.bits[0]
    for t in range(T):
        keys = [(-abs(v), i) for i, v in zip(idx[t], val[t])]
        assert keys == sorted(keys)                               # (|z| desc, idx asc)
        assert len(set(idx[t].tolist())) == cfg.k                 # distinct
        for i in idx[t]:
            assert i < cfg.d or (1 << r0) <= i < (1 << cfg.m_bits)  # no index in [d, 2^r0)
        for i, v in zip(idx[t], val[t]):
            assert abs(float(oracle.phi(cfg.d, cfg.M, int(i)) @ x[t]) - v) < 1e-12
    assert np.allclose(xnorm, np.linalg.norm(x, axis=1))
    assert np.all(gap >= 0)


def test_standardisation_scales_and_shifts():
    # §2.2 "Score Standardization": z = (s - mu)/sigma; |z| selects, signed z
    # is the coefficient.
    cfg = _tiny()
    m = 1 << cfg.m_bits
    x = np.random.default_rng(3).standard_normal((16, cfg.d))
    idx0, val0, _, _ = oracle.encode(cfg, x)
    idx1, val1, _, _ = oracle.encode(cfg, x, mu=np.zeros(m), sigma=np.full(m, 2.0))
    assert np.array_equal(idx0, idx1) and np.allclose(val1, val0 / 2)
    mu = np.zeros(m)
    mu[37] = -100.0                                              # basis index 37 now dominates
    idx2, val2, _, _ = oracle.encode(cfg, x, mu=mu, sigma=np.ones(m))
    assert np.all(idx2[:, 0] == 37) and np.allclose(val2[:, 0], x[:, 37] + 100.0)


def test_planted_tree_is_recovered():
    # x = sum of a planted tree of features (8 basis roots, then children of
    # planted nodes) plus small noise: the encoder finds most of the planted
    # set. (Not all: at d = 768 the cross-talk of 32 features on the basis
    # coordinates reaches ~0.9, comparable to the smallest coefficients.)
    from paper_2607_20652_gb300 import inputs
    from tests.helpers import compose_planted
    cfg = oracle.resolve(d=768, m_bits=16, levels=4, children=16, beam=8, k=32)
    plant = inputs.planted_tree(T=6, d=cfg.d, levels=cfg.levels, children=cfg.children,
                                per_level=[8, 8, 8, 8], seed=4)
    idx_true = compose_planted(plant, cfg.G, cfg.levels)
    clean = oracle.decode(cfg, idx_true, plant.coef, norm_match=0)
    x = clean + 0.01 * np.random.default_rng(5).standard_normal(clean.shape)
    idx, _, _, _ = oracle.encode(cfg, x)
    hits = np.mean([len(set(idx[t]) & set(idx_true[t])) / cfg.k for t in range(len(x))])
    assert hits > 0.8


def test_per_level_mode_levels():
    # Paper's per-level form: level 0 keeps the top K_0 coordinates; level 1
    # keeps the top K_1 of the children of that set.
    cfg = oracle.resolve(d=64, m_bits=12, levels=2, children=16, beam=4, k=8, bits=[6, 12],
                         k_per_level=[4, 6])
    x = np.random.default_rng(6).standard_normal((10, cfg.d))
    idx, val, _ = oracle.encode_per_level(cfg, x)
    gens = cfg.G[1, :16].tolist()
    for t in range(len(x)):
        top0 = sorted(range(cfg.d), key=lambda i: (-abs(x[t, i]), i))[:4]
        assert idx[t, :4].tolist() == top0
        kids = sorted({p ^ g for p in top0 for g in gens})
        s = {c: float(oracle.phi(cfg.d, cfg.M, c) @ x[t]) for c in kids}
        top1 = sorted(kids, key=lambda c: (-abs(s[c]), c))[:6]
        assert idx[t, 4:].tolist() == top1
        assert np.allclose(val[t, 4:], [s[c] for c in top1])


def test_coset_children_scores_are_a_walsh_transform():
    # The coset-generator variant (outside the paper): with g_j = g0 ^ j for
    # j < 16, the 16 child scores of a parent p are the 16-point Walsh-
    # Hadamard transform (scipy's Sylvester matrix) of the bucket sums
    # B_u = sum over iota = u mod 16 of phi~_{p ^ g0}[iota] x[iota].
    import scipy.linalg
    cfg = _tiny()
    rng = np.random.default_rng(8)
    H = scipy.linalg.hadamard(16)
    for _ in range(5):
        g0 = int(rng.integers(1 << 6, 1 << 9)) & ~15
        p = int(rng.integers(0, 1 << 6))
        x = rng.standard_normal(cfg.d)
        y = oracle.phi_tilde(cfg.d, cfg.M, p ^ g0) * x
        B = np.array([y[u::16].sum() for u in range(16)])
        s = np.array([oracle.phi(cfg.d, cfg.M, p ^ g0 ^ j) @ x for j in range(16)])
        assert np.allclose(H @ B, s, atol=1e-12)
