"""The comparison rules of tests/parity.py, on CPU: the element-wise check
catches one coordinate that is off by far less than a per-row norm would
allow, accepts bf16 rounding of the reference, and the session report
counts tokens and near-ties."""
import numpy as np
import pytest

from tests import parity


def test_bf16_spacing_matches_the_format():
    # 8 significant bits: spacing 2^-7 on [1, 2), 2^-6 on [2, 4), 2^-8 on [0.5, 1)
    assert parity.bf16_spacing(np.array([1.0, 1.99, 2.0, 0.75, -3.0])).tolist() == \
        [2.0 ** -7, 2.0 ** -7, 2.0 ** -6, 2.0 ** -8, 2.0 ** -6]


def test_one_bad_coordinate_fails_where_the_row_norm_passes():
    rng = np.random.default_rng(0)
    ref = rng.standard_normal((4, 768))
    got = ref.copy()
    got[2, 100] += 0.3 * np.linalg.norm(ref[2]) / np.sqrt(768)   # 0.3 of the row's rms
    assert parity.rel_rows(got, ref).max() < 2e-2                # a per-row L2 bound misses it
    with pytest.raises(AssertionError, match=r"element \[2, 100\]"):
        parity.check_elementwise(got, ref, 2e-2, True, "y")


def test_bf16_rounding_of_the_reference_passes():
    rng = np.random.default_rng(1)
    ref = rng.standard_normal((8, 256))
    # round to bf16 (nearest even on the upper 16 bits of the fp32 pattern)
    b = ref.astype(np.float32).view(np.uint32)
    b = ((b + 0x7FFF + ((b >> 16) & 1)) & 0xFFFF0000).astype(np.uint32)
    got = b.view(np.float32).astype(np.float64)
    worst = parity.check_elementwise(got, ref, 2e-2, True, "y")
    assert 0 < worst < 2 ** -8
    # fp32 storage at 1e-5 does not accept bf16 rounding
    with pytest.raises(AssertionError):
        parity.check_elementwise(got, ref, 1e-5, False, "y")


def test_zero_rows_and_nan():
    z = np.zeros((2, 8))
    assert parity.check_elementwise(z, z, 1e-5) == 0.0
    bad = z.copy()
    bad[1, 3] = np.nan
    with pytest.raises(AssertionError):
        parity.check_elementwise(bad, z, 1e-5)


def test_summary_counts_tokens_and_near_ties():
    rep = [{"test": "a", "tokens": 100, "near_ties": 2, "val": 1e-7, "y": 3e-3},
           {"test": "b", "tokens": 50, "near_ties": 0, "gx": 2e-6}]
    lines = parity.summary_lines(rep)
    assert lines[0].startswith("a: 100 tokens, 2 near-ties")
    assert "150 tokens, 2 near-ties (1.33%)" in lines[-1] and "y 3.0e-03" in lines[-1]


def test_near_tie_values_are_checked_against_each_features_score():
    # a near-tie token's code need not be the oracle's, but each entry's value
    # must be its feature's score <phi_i, x>; a wrong value is caught
    import oracle
    from paper_2607_20652_gb300 import inputs
    ref = oracle.resolve(d=64, m_bits=12, levels=3, children=16, beam=4, k=8)
    x = inputs.gaussian_rows(3, 64, 5).astype(np.float64)
    idx, val, _, _ = oracle.encode(ref, x)
    near = np.array([True, False, True])
    assert parity.check_near_tie_values(ref, x, idx, val, near) == 16
    bad = val.copy()
    bad[2, 5] *= 1.001
    with pytest.raises(AssertionError, match="near-tie token 2"):
        parity.check_near_tie_values(ref, x, idx, bad, near)
