"""Pins of the oracle's finite-field layer (App. A.2-A.4) against facts that
do not come from the oracle: Gauss's count of irreducible polynomials, a
published worked example of GF(2^8) arithmetic, the field axioms, the trace
lemma, the Kloosterman code's definition, the Weil bound and the values of
binary Kloosterman sums."""
import math
import os

import numpy as np
import pytest

import oracle
from tests import pins

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _mobius(n: int) -> int:
    m, p, res = n, 2, 1
    while p * p <= m:
        if m % p == 0:
            m //= p
            if m % p == 0:
                return 0
            res = -res
        p += 1
    return -res if m > 1 else res


@pytest.mark.parametrize("t", range(2, 11))
def test_irreducible_count_is_gauss_formula(t):
    # Number of monic irreducible binary polynomials of degree t is
    # (1/t) sum_{e | t} mu(e) 2^{t/e} (Gauss). The oracle's trial-division
    # test must find exactly that many among the 2^t monic polynomials.
    want = sum(_mobius(e) * 2 ** (t // e) for e in range(1, t + 1) if t % e == 0) // t
    got = sum(oracle.is_irreducible(t, (1 << t) | low) for low in range(1 << t))
    assert got == want


def test_paper_polynomials_are_irreducible():
    # App. A.4 (Eq. 24) fixes z^10+z^3+1 for d=1024 and z^11+z^2+1 for d=2048.
    rows = _golden_rows("paper_polynomials.txt")
    for t_s, poly_s in rows:
        t, poly = int(t_s), int(poly_s, 16)
        assert oracle.is_irreducible(t, poly)
        assert oracle.default_poly(t) == poly
    # a reducible one is rejected: z^10 + 1 = (z + 1)^2 (z^4+z^3+z^2+z+1)^2
    assert not oracle.is_irreducible(10, (1 << 10) | 1)


def _golden_rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def test_gf256_worked_examples():
    # FIPS-197 (AES) Sec. 4.2 works products in GF(2^8) modulo
    # z^8+z^4+z^3+z+1; the oracle's multiply must reproduce them.
    for a, b, prod in _golden_rows("gf256_fips197.txt"):
        assert oracle.gf_mul(int(a, 16), int(b, 16), 8, 0x11B) == int(prod, 16)


@pytest.mark.parametrize("t,poly", [(6, 0x43), (8, 0x11B)])
def test_field_axioms_exhaustive(t, poly):
    mul, inv, tr = oracle.gf_tables(t, poly)
    q = 1 << t
    a = np.arange(q)
    assert np.array_equal(mul, mul.T)                                   # commutative
    assert np.array_equal(mul[1], a) and np.all(mul[0] == 0)             # identities
    for b in range(q):                                                   # distributive over XOR
        assert np.array_equal(mul[a, b] ^ mul[a, 5 % q], mul[a, b ^ (5 % q)])
    rng = np.random.default_rng(1)
    x, y, z = rng.integers(0, q, (3, 2000))
    assert np.array_equal(mul[mul[x, y], z], mul[x, mul[y, z]])          # associative
    nz = a[1:]
    assert np.all(mul[nz, inv[nz]] == 1) and inv[0] == 0                 # inverses, 0^{-1}=0
    # the nonzero elements form a cyclic group of order q-1: some element
    # has powers that run through all of them.
    found = False
    for g in range(2, q):
        seen, p = set(), 1
        for _ in range(q - 1):
            p = int(mul[p, g])
            seen.add(p)
        if len(seen) == q - 1:
            found = True
            break
    assert found


@pytest.mark.parametrize("t,poly", [(6, 0x43), (7, 0x83), (10, 0x409)])
def test_trace_lemma(t, poly):
    # Lemma A.2: Tr(y) in {0,1}, additive, not identically zero. Additivity
    # with (iii) makes the trace balanced: exactly half the field has Tr = 1.
    _, _, tr = oracle.gf_tables(t, poly, with_mul=False)
    q = 1 << t
    assert set(np.unique(tr)) <= {0, 1}
    rng = np.random.default_rng(t)
    a, b = rng.integers(0, q, (2, 5000))
    assert np.array_equal(tr[a ^ b], tr[a] ^ tr[b])
    assert tr[0] == 0 and int(tr.sum()) == q // 2


@pytest.mark.parametrize("t,poly", [(6, 0x43), (8, 0x11B)])
def test_trace_masks_are_a_bijection(t, poly):
    # App. A.4 (Eq. 20): Tr(a xi) = <coord(xi), tau(a)> for every xi, and
    # a -> tau(a) is a bijection.
    mul, _, tr = oracle.gf_tables(t, poly)
    q = 1 << t
    tau = pins.trace_masks(t, mul, tr)
    assert len(set(tau.tolist())) == q
    xi = np.arange(q)
    for a in range(q):
        par = np.zeros(q, dtype=np.int64)
        v = xi & int(tau[a])
        for p in range(t):
            par ^= (v >> p) & 1
        assert np.array_equal(par, tr[mul[a, xi]])


@pytest.mark.parametrize("t,poly", [(6, 0x43), (7, 0x83)])
def test_seed_matrix_generates_kloosterman_code(t, poly):
    # App. A.4: the seed matrix is a generator matrix of the Kloosterman code;
    # the message (tau(a), tau(b)) gives c_{a,b} of Eq. 12 exactly, and the
    # set of all codewords from M equals the set {c_{a,b}}.
    d = 1 << t
    mul, inv, tr = oracle.gf_tables(t, poly)
    M = oracle.seed_matrix(d, t, poly)
    pairs = [(a, b) for a in range(d) for b in range(d)]
    assert pins.kloosterman_generation_mismatch(M, t, mul, inv, tr, pairs) == 0
    xi = np.arange(d)
    from_def = {tuple(tr[mul[a, xi] ^ mul[b, inv[xi]]]) for a, b in pairs}
    from_m = {tuple(pins.gf2_matvec_bits(M, u)) for u in range(d * d)}
    assert from_def == from_m and len(from_m) == d * d


def test_kloosterman_bit_matches_tables():
    # the scalar codeword bit (Eq. 12) and the table route agree
    t, poly = 6, 0x43
    mul, inv, tr = oracle.gf_tables(t, poly)
    rng = np.random.default_rng(3)
    for a, b, xi in rng.integers(0, 64, (200, 3)):
        assert oracle.kloosterman_bit(int(a), int(b), int(xi), t, poly) == tr[mul[a, xi] ^ mul[b, inv[xi]]]


@pytest.mark.parametrize("t,poly", [(3, 0xB), (4, 0x13), (5, 0x25), (6, 0x43), (7, 0x83),
                                    (8, 0x11B), (9, 0x211), (10, 0x409)])
def test_weil_bound_and_kloosterman_values(t, poly):
    # Thm A.3: |K(a)| <= 2 sqrt(d). Remark A.4 (Lachaud-Wolfmann): K(a) = -1
    # (mod 4) and the values fill every such integer in [-2 sqrt d, 2 sqrt d].
    mul, inv, tr = oracle.gf_tables(t, poly)
    K = pins.kloosterman_sums(t, mul, inv, tr)
    d = 1 << t
    bound = 2 * math.sqrt(d)
    assert np.all(np.abs(K) <= bound + 1e-9)
    assert np.all(K % 4 == 3)
    lo, hi = -bound, bound
    want = {v for v in range(int(math.floor(lo)), int(math.ceil(hi)) + 1) if v % 4 == 3 and lo <= v <= hi}
    assert set(K.tolist()) == want


def test_pair_sums_reduce_to_one_parameter():
    # Eq. 16: K(alpha, beta) = K(alpha beta, 1) for nonzero alpha, beta.
    t, poly = 6, 0x43
    mul, inv, tr = oracle.gf_tables(t, poly)
    xi = np.arange(1, 64)
    rng = np.random.default_rng(5)
    for al, be in rng.integers(1, 64, (100, 2)):
        k2 = np.sum(1 - 2 * tr[mul[al, xi] ^ mul[be, inv[xi]]].astype(np.int64))
        k1 = np.sum(1 - 2 * tr[mul[mul[al, be], xi] ^ inv[xi]].astype(np.int64))
        assert k1 == k2
