"""The seeded input generators shared by the oracle tests, the GPU parity
tests and the benchmark: shapes, ranges and the structure each promises."""
import numpy as np
import pytest

from paper_2607_20652_gb300 import inputs


def test_mixed_codes_hold_the_requested_split():
    counts = [0, 1, 31, 32, 33, 63, 64, 65, 96]
    idx, val = inputs.mixed_codes(3 * len(counts), 100, 16, 96, counts, 5)
    assert idx.dtype == np.int32 and val.dtype == np.float32 and idx.shape == val.shape == (27, 96)
    for t in range(len(idx)):
        row = idx[t]
        assert len(np.unique(row)) == 96  # distinct entries
        assert row.min() >= 0 and row.max() < (1 << 16)
        assert int((row >= 100).sum()) == counts[t % len(counts)]
    again = inputs.mixed_codes(3 * len(counts), 100, 16, 96, counts, 5)
    assert np.array_equal(again[0], idx) and np.array_equal(again[1], val)  # seeded


def test_mixed_codes_reject_splits_that_cannot_fit():
    with pytest.raises(ValueError):
        inputs.mixed_codes(2, 64, 12, 96, [0], 1)  # 96 basis entries do not fit below d = 64
    with pytest.raises(ValueError):
        inputs.mixed_codes(2, 256, 12, 32, [33], 1)  # more hashed entries than the code holds


def test_outlier_rows_are_scaled():
    x = inputs.gaussian_rows(2000, 64, 3, outlier_frac=0.05, outlier_scale=10.0)
    norms = np.linalg.norm(x, axis=1)
    big = norms > 4 * np.median(norms)
    assert 0.03 < big.mean() < 0.07  # about 5% of the rows, ten times larger


def test_bf16_rounding_is_to_nearest_even():
    a = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -2.5], dtype=np.float32)
    b = inputs.to_bf16(a)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: it goes to the even mantissa (1)
    assert b[0] == 1.0 and b[1] == 1.0 and b[2] == 1.0 + 2.0 ** -6 and b[3] == -2.5
