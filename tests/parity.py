"""Comparison rules between the CUDA path and the oracle.

* Feature indices: bit-exact as a set per token, except tokens whose oracle
  selection has a relative gap below NEAR_TIE at some cut (a beam cut or the
  final top-k cut); those are counted and reported, not failed.
* Coefficients (fp32 storage): |val_gpu - val_oracle| <= VAL_TOL * |x_t|.
* Decoded outputs and gradients: per-token relative L2 error, 1e-5 when they
  are stored in fp32 and 2e-2 when they are stored in bf16 (fp32 accumulation
  either way). Decode and backward are checked by running the oracle on the
  GPU's own code, which isolates each stage from selection near-ties.
"""
from __future__ import annotations

import numpy as np

NEAR_TIE = 1e-5
VAL_TOL = 1e-5
TOL = {"f32": 1e-5, "bf16": 2e-2}


def check_code_order(idx: np.ndarray, val: np.ndarray):
    """Each row sorted by (|val| desc, idx asc) with distinct indices."""
    for t in range(idx.shape[0]):
        a = np.abs(val[t].astype(np.float64))
        i = idx[t].astype(np.int64)
        assert len(set(i.tolist())) == len(i), f"token {t}: repeated index"
        ok = (a[:-1] > a[1:]) | ((a[:-1] == a[1:]) & (i[:-1] < i[1:]))
        assert np.all(ok), f"token {t}: code not in (|val| desc, idx asc) order"


def compare_codes(idx_g, val_g, idx_o, val_o, gap, xnorm, val_tol=VAL_TOL):
    """Returns the number of near-tie tokens; asserts on every other token."""
    near = gap < NEAR_TIE
    worst = 0.0
    for t in range(idx_g.shape[0]):
        if near[t]:
            continue
        sg, so = set(idx_g[t].tolist()), set(idx_o[t].tolist())
        assert sg == so, f"token {t}: index sets differ: gpu-only {sorted(sg - so)[:8]}, oracle-only {sorted(so - sg)[:8]}"
        vo = dict(zip(idx_o[t].tolist(), val_o[t].tolist()))
        err = max(abs(float(v) - vo[i]) for i, v in zip(idx_g[t].tolist(), val_g[t].tolist()))
        scale = max(float(xnorm[t]), 1e-30)
        worst = max(worst, err / scale)
        assert err <= val_tol * scale, f"token {t}: coefficient error {err:.3e} > {val_tol} |x| = {val_tol * scale:.3e}"
    return int(near.sum()), worst


def rel_rows(got: np.ndarray, ref: np.ndarray) -> np.ndarray:
    """Per-row ||got - ref|| / ||ref|| (0 where both are zero)."""
    got = got.astype(np.float64)
    ref = ref.astype(np.float64)
    num = np.linalg.norm(got - ref, axis=1)
    den = np.linalg.norm(ref, axis=1)
    out = np.where(den > 0, num / np.where(den > 0, den, 1.0), num)
    return out
