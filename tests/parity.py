"""Comparison rules between the CUDA path and the oracle.

* Feature indices: bit-exact as a set per token, except tokens whose oracle
  selection has a relative gap below NEAR_TIE at some cut (a beam cut or the
  final top-k cut); those are counted and reported, and on them each code
  entry's value must still equal its feature's score (the code is a valid
  one, not necessarily the oracle's).
* Coefficients (fp32 storage): |val_gpu - val_oracle| <= VAL_TOL * |x_t|.
* Decoded outputs, kept r and gradients, element by element:
  |got_i - ref_i| <= tol * max(|ref_i|, ||ref_row|| / sqrt(n)), plus one bf16
  spacing of ref_i when the output is stored in bf16; tol is 1e-5 for fp32
  storage and 2e-2 for bf16 storage (fp32 accumulation either way). The
  row-RMS floor covers coordinates near zero, whose fp32 sums carry the
  rounding of the row's large terms. Decode and backward are checked by
  running the oracle on the GPU's own code, which isolates each stage from
  selection near-ties.

Every comparison adds a record (tokens, near-ties, worst errors) to REPORT;
the test session prints them in its terminal summary.
"""
from __future__ import annotations

import math
import os

import numpy as np

NEAR_TIE = 1e-5
VAL_TOL = 1e-5
TOL = {"f32": 1e-5, "bf16": 2e-2}

REPORT: list[dict] = []


def _test_name() -> str:
    cur = os.environ.get("PYTEST_CURRENT_TEST", "?")
    return cur.rsplit(" (", 1)[0].split("/")[-1]


def record(**fields) -> dict:
    """Adds one comparison's figures to the session report (keyed by the running test)."""
    rec = {"test": _test_name(), **fields}
    REPORT.append(rec)
    return rec


def check_code_order(idx: np.ndarray, val: np.ndarray):
    """Each row sorted by (|val| desc, idx asc) with distinct indices."""
    for t in range(idx.shape[0]):
        a = np.abs(val[t].astype(np.float64))
        i = idx[t].astype(np.int64)
        assert len(set(i.tolist())) == len(i), f"token {t}: repeated index"
        ok = (a[:-1] > a[1:]) | ((a[:-1] == a[1:]) & (i[:-1] < i[1:]))
        assert np.all(ok), f"token {t}: code not in (|val| desc, idx asc) order"


def compare_codes(idx_g, val_g, idx_o, val_o, gap, xnorm, val_tol=VAL_TOL):
    """Returns (near-tie tokens, worst coefficient error / |x|); asserts on every other token."""
    near = gap < NEAR_TIE
    worst = 0.0
    for t in range(idx_g.shape[0]):
        if near[t]:
            continue
        sg, so = set(idx_g[t].tolist()), set(idx_o[t].tolist())
        assert sg == so, f"token {t}: index sets differ: gpu-only {sorted(sg - so)[:8]}, oracle-only {sorted(so - sg)[:8]}"
        vo = dict(zip(idx_o[t].tolist(), val_o[t].tolist()))
        err = max((abs(float(v) - vo[i]) for i, v in zip(idx_g[t].tolist(), val_g[t].tolist())), default=0.0)
        scale = max(float(xnorm[t]), 1e-30)
        worst = max(worst, err / scale)
        assert err <= val_tol * scale, f"token {t}: coefficient error {err:.3e} > {val_tol} |x| = {val_tol * scale:.3e}"
    return int(near.sum()), worst


def check_near_tie_values(ref, x, idx_g, val_g, near, mu=None, sigma=None, val_tol=VAL_TOL) -> int:
    """For the near-tie tokens (where several codes are correct, so the index
    sets are not compared), what is still unique: each code entry's value is
    the standardised score of its feature, <phi_i, x> by the oracle's own
    dense direction (e_i for a basis index), within val_tol |x|. Returns the
    number of entries checked."""
    import oracle
    n = 0
    for t in np.nonzero(near)[0]:
        ids = np.asarray(idx_g[t], dtype=np.int32)
        phi = oracle.decode(ref, ids.reshape(-1, 1), np.ones((len(ids), 1)), norm_match=0)
        s = phi @ np.asarray(x[t], dtype=np.float64)
        if mu is not None:
            s = (s - mu[ids]) / sigma[ids]
        err = np.abs(np.asarray(val_g[t], dtype=np.float64) - s)
        scale = max(float(np.linalg.norm(np.asarray(x[t], dtype=np.float64))), 1e-30)
        assert err.max() <= val_tol * scale, (
            f"near-tie token {t}: entry {int(np.argmax(err))} (index {ids[np.argmax(err)]}) has value "
            f"{val_g[t][np.argmax(err)]:.7e}, its score is {s[np.argmax(err)]:.7e}")
        n += len(ids)
    return n


def bf16_spacing(v: np.ndarray) -> np.ndarray:
    """Distance between neighbouring bf16 numbers at |v| (8 significant bits):
    2^(e - 7) for |v| in [2^e, 2^(e+1)), the subnormal spacing below 2^-126."""
    a = np.maximum(np.abs(np.asarray(v, np.float64)), 2.0 ** -126)
    return np.ldexp(1.0, np.frexp(a)[1] - 8)


def check_elementwise(got, ref, tol: float, bf16: bool = False, what: str = "output") -> float:
    """Asserts |got_i - ref_i| <= tol * max(|ref_i|, ||ref_row|| / sqrt(n))
    (+ one bf16 spacing of ref_i for bf16 storage) on every element of the
    [rows, n] arrays; returns the worst |got_i - ref_i| / max(|ref_i|, row rms)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, f"{what}: shape {got.shape} != {ref.shape}"
    if got.size == 0:
        return 0.0
    ref2 = ref.reshape(-1, ref.shape[-1])
    got2 = got.reshape(ref2.shape)
    rms = np.linalg.norm(ref2, axis=1, keepdims=True) / math.sqrt(ref2.shape[1])
    scale = np.maximum(np.abs(ref2), rms)
    err = np.abs(got2 - ref2)
    bound = tol * scale + (bf16_spacing(ref2) if bf16 else 0.0)
    bad = ~(err <= bound)                          # NaN counts as out of bound
    if bad.any():
        t, i = np.unravel_index(np.argmax(np.where(bad, np.nan_to_num(err - bound, nan=np.inf), -np.inf)),
                                err.shape)
        raise AssertionError(
            f"{what}: element [{t}, {i}] is {got2[t, i]:.7e}, oracle {ref2[t, i]:.7e} (off by {err[t, i]:.3e}, "
            f"bound {bound[t, i]:.3e}); {int(bad.sum())} of {err.size} elements out of bound")
    rel = np.where(scale > 0, err / np.where(scale > 0, scale, 1.0), 0.0)
    return float(rel.max())


def rel_rows(got: np.ndarray, ref: np.ndarray) -> np.ndarray:
    """Per-row ||got - ref|| / ||ref|| (0 where both are zero)."""
    got = got.astype(np.float64)
    ref = ref.astype(np.float64)
    num = np.linalg.norm(got - ref, axis=1)
    den = np.linalg.norm(ref, axis=1)
    out = np.where(den > 0, num / np.where(den > 0, den, 1.0), num)
    return out


def summary_lines(report=None) -> list[str]:
    """The session report: one line per comparison, then the totals."""
    report = REPORT if report is None else report
    keys = ["val", "y", "r", "gx", "gv"]
    lines = []
    tokens = near = 0
    worst = {k: 0.0 for k in keys}
    for rec in report:
        tokens += rec.get("tokens", 0)
        near += rec.get("near_ties", 0)
        parts = [f"{rec['test']}: {rec.get('tokens', 0)} tokens, {rec.get('near_ties', 0)} near-ties"]
        for k in keys:
            if rec.get(k) is not None:
                worst[k] = max(worst[k], rec[k])
                parts.append(f"{k} {rec[k]:.1e}")
        lines.append("  ".join(parts))
    if report:
        rate = 100.0 * near / max(tokens, 1)
        lines.append(f"TOTAL: {len(report)} comparisons, {tokens} tokens, {near} near-ties ({rate:.2f}%), "
                     "worst relative error " + ", ".join(f"{k} {worst[k]:.1e}" for k in keys))
    return lines
