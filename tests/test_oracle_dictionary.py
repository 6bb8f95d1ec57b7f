"""Pins of the oracle's dictionary (§2.1 Eq. 1-5, App. A): Walsh rows from
scipy's Sylvester matrix, the basis override, exact orthogonality cases, the
child factorisation and the coherence theorem with the values the paper
quotes."""
import math
import os

import numpy as np
import pytest

import oracle
from tests import pins

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("d,t,poly", [(64, 6, 0x43), (1024, 10, 0x409), (768, 10, 0x409)])
def test_low_indices_hash_to_walsh_rows(d, t, poly):
    # An index whose high half is zero meets only coord(xi) (Eq. 23), so its
    # sign pattern is row i of Sylvester's Hadamard matrix (first d columns).
    M = oracle.seed_matrix(d, t, poly)
    rows = range(1 << t) if t <= 6 else np.random.default_rng(0).integers(0, 1 << t, 64)
    assert pins.walsh_rows_mismatch(lambda i: oracle.phi_tilde(d, M, i), d, t, rows) == 0


def test_basis_override_and_unit_norm():
    # Eq. 2: phi_i = e_i for the first d indices (0-based, reading R4);
    # every hashed direction has entries +-1/sqrt(d) (Eq. 1) and unit norm.
    d, t, poly = 768, 10, 0x409
    M = oracle.seed_matrix(d, t, poly)
    for i in (0, 1, 500, 767):
        e = np.zeros(d)
        e[i] = 1.0
        assert np.array_equal(oracle.phi(d, M, i), e)
    rng = np.random.default_rng(2)
    for i in rng.integers(d, 1 << 20, 50):
        v = oracle.phi(d, M, int(i))
        assert np.allclose(np.abs(v), 1 / math.sqrt(d), rtol=0, atol=1e-15)
        assert abs(np.linalg.norm(v) - 1.0) < 1e-12
        # a basis vector meets any hashed direction at exactly +-1/sqrt(d)
        assert abs(abs(v[int(i) % d]) - 1 / math.sqrt(d)) < 1e-15


def test_child_factorisation():
    # Eq. 5: phi~_{i xor g} = phi~_i (.) R(M g), for any i and g.
    d, t, poly = 768, 10, 0x409
    M = oracle.seed_matrix(d, t, poly)
    rng = np.random.default_rng(3)
    for i, g in rng.integers(0, 1 << 20, (50, 2)):
        lhs = oracle.phi_tilde(d, M, int(i ^ g))
        rhs = oracle.phi_tilde(d, M, int(i)) * oracle.phi_tilde(d, M, int(g)) * math.sqrt(d)
        assert np.array_equal(lhs, rhs)


def test_hamming_correlation_identity():
    # Eq. 9: <psi_c, psi_c'> = 1 - 2 Hamming(c, c') / d.
    d, t, poly = 64, 6, 0x43
    M = oracle.seed_matrix(d, t, poly)
    rng = np.random.default_rng(4)
    for i, j in rng.integers(0, 1 << 12, (100, 2)):
        a, b = oracle.phi_tilde(d, M, int(i)), oracle.phi_tilde(d, M, int(j))
        ham = int(np.sum(np.sign(a) != np.sign(b)))
        assert abs(float(a @ b) - (1 - 2 * ham / d)) < 1e-12


def test_exact_orthogonality_cases():
    # Proof of Thm A.1, cases 2 and 3: label differences with alpha = 0 or
    # beta = 0 (one half of the message XOR zero) give exactly orthogonal
    # features. Labels differ by u = (u1, u2); case alpha=0 <=> u1 = 0.
    d, t, poly = 64, 6, 0x43
    M = oracle.seed_matrix(d, t, poly)
    base = oracle.phi_tilde(d, M, 0x5A3)
    for u in list(range(1, 64)) + [v << 6 for v in range(1, 64)]:
        other = oracle.phi_tilde(d, M, 0x5A3 ^ u)
        assert abs(float(base @ other)) < 1e-12 * d


def test_coherence_brute_force_full_dictionary_d64():
    # Thm A.1 for d = 64 by brute force over every pair of the full dictionary
    # (64 basis + 4032 hashed), and over all d^2 hashed vectors: mu <= 17/64.
    # With Lachaud-Wolfmann (K = 15 attained) the hashed maximum is 16/64.
    d, t, poly = 64, 6, 0x43
    M = oracle.seed_matrix(d, t, poly)
    Phi = np.stack([oracle.phi(d, M, i) for i in range(1 << 12)])
    G = Phi @ Phi.T
    np.fill_diagonal(G, 0.0)
    bound = (1 + 2 * math.sqrt(d)) / d
    assert np.max(np.abs(G)) <= bound + 1e-12
    Pt = np.stack([oracle.phi_tilde(d, M, i) for i in range(1 << 12)])
    Gt = Pt @ Pt.T
    np.fill_diagonal(Gt, 0.0)
    assert abs(np.max(np.abs(Gt)) - 16 / 64) < 1e-12


@pytest.mark.parametrize("d,t,poly", [(128, 7, 0x83), (1024, 10, 0x409)])
def test_coherence_by_linearity(d, t, poly):
    # Linear code => mu = max over nonzero messages (App. A.1). For d = 1024
    # the bound is 65/1024 and the attained maximum is 64/1024 (K = 63).
    M = oracle.seed_matrix(d, t, poly)
    mu = pins.coherence_by_linearity(M, d, t)
    bound = (1 + 2 * math.sqrt(d)) / d
    assert mu <= bound + 1e-12
    if d == 1024:
        assert abs(mu - 64 / 1024) < 1e-12


def test_paper_quoted_bound_values():
    # The values quoted after Thm A.1 are the bound (1 + 2 sqrt d)/d rounded.
    with open(os.path.join(GOLDEN, "coherence_bounds.txt")) as f:
        rows = [l.split() for l in f if l.strip() and not l.startswith("#")]
    for d_s, quoted, digits in rows:
        d = int(d_s)
        assert round((1 + 2 * math.sqrt(d)) / d, int(digits)) == float(quoted)


def test_truncated_dictionary_coherence_closed_form():
    # Reading R1: d = 768 keeps the first 768 coordinates of the t = 10 code,
    # so Thm A.1 no longer applies. Two indices that differ only in bit 8 of
    # the low half differ by the Walsh character (-1)^{iota_8}, whose sum over
    # iota < 768 is 256 - 256 + 256 = 256: coherence exactly 256/768 = 1/3.
    d, t, poly = 768, 10, 0x409
    M = oracle.seed_matrix(d, t, poly)
    mu = pins.coherence_by_linearity(M, d, t)
    assert abs(mu - 1 / 3) < 1e-12
    a, b = oracle.phi_tilde(d, M, 0x12345), oracle.phi_tilde(d, M, 0x12345 ^ 256)
    assert abs(abs(float(a @ b)) - 1 / 3) < 1e-12
