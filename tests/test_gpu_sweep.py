"""The sweep at d = 768, T = 32768 (features 2^16 / 2^18 / 2^20 / 2^22,
k in {16, 32, 64, 128}, beam in {4, 8, 16}; bf16 x ~ N(0, 1)): every point
runs at its full size through the C ABI, in the launch configuration the
benchmark uses, and a sample of its tokens is compared with the oracle under
the rules of ``tests/parity.py`` (indices as sets except near-ties; values,
decode and both gradients on the GPU's own code). Every point runs the
tensor-core encoder: beam slots past the beam hold no parent, and a beam of
16 gives a warp one token whose two halves of 8 slots fill the tensor-core
rows.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20652_gb300 import build, configs, dpb, inputs
from tests import parity

pytestmark = pytest.mark.gpu

SAMPLED = 24


@pytest.fixture(scope="module", autouse=True)
def _library():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    dpb.load()


def _id(w):
    return f"2^{w['m_bits']}-k{w['k']}-b{w['beam']}"


@pytest.mark.parametrize("w", configs.SWEEP, ids=_id)
def test_sweep_point_full_size_sampled(w):
    plan = dpb.Plan(d=w["d"], levels=w["levels"], m_bits=w["m_bits"], children=w["children"],
                    beam=w["beam"], k=w["k"], dtype=w["dtype"])
    c = plan.config
    ref = oracle.resolve(d=c["d"], m_bits=w["m_bits"], levels=c["levels"], children=c["children"],
                         beam=c["beam"], k=c["k"], seed=c["generator_seed"], norm_match=c["norm_match"],
                         t=c["field_t"], poly=c["field_poly"], bits=c["bits"])
    T, d = w["T"], w["d"]
    seed = w["seed"] + w["m_bits"] * 100 + w["k"] + w["beam"]
    x = inputs.to_bf16(inputs.gaussian_rows(T, d, seed))
    gy = inputs.to_bf16(inputs.normal((T, d), seed + 1))
    dev = torch.device("cuda")
    xt = torch.from_numpy(x).to(dev).to(torch.bfloat16)
    gyt = torch.from_numpy(gy).to(dev).to(torch.bfloat16)
    ws = plan.workspace(T, dev)
    idx, val, xn = dpb.encode(plan, xt, workspace=ws)
    r = torch.empty((T, d), dtype=torch.float32, device=dev)
    y = dpb.decode(plan, idx, val, xn, workspace=ws, r_out=r)
    gx, gv = dpb.backward(plan, xt, idx, val, gyt, workspace=ws, r=r)
    torch.cuda.synchronize()
    assert dpb.workspace_status(ws) == 0
    rows = np.unique(np.concatenate([inputs.sample_rows(T, SAMPLED, seed + 2), [0, T - 1]]))
    gi, gvl = idx.cpu().numpy()[rows], val.cpu().numpy()[rows]
    gxn = xn.cpu().numpy()[rows]
    xr = x[rows].astype(np.float64)
    idx_o, val_o, xn_o, gap = oracle.encode(ref, xr)
    parity.check_code_order(gi, gvl)
    near, worst = parity.compare_codes(gi, gvl, idx_o, val_o, gap, xn_o)
    parity.check_near_tie_values(ref, xr, gi, gvl, gap < parity.NEAR_TIE)
    assert near <= max(2, len(rows) // 10), f"{near} near-ties of {len(rows)} tokens"
    assert np.all(np.abs(gxn - xn_o) <= 1e-5 * xn_o)
    tol = parity.TOL["bf16"]
    y_o = oracle.decode(ref, gi, gvl.astype(np.float64), gxn.astype(np.float64))
    assert parity.rel_rows(y.float().cpu().numpy()[rows], y_o).max() <= tol
    gx_o, gv_o = oracle.backward(ref, xr, gi, gvl.astype(np.float64), gy[rows].astype(np.float64))
    assert parity.rel_rows(gx.float().cpu().numpy()[rows], gx_o).max() <= tol
    assert parity.rel_rows(gv.cpu().numpy()[rows], gv_o).max() <= 1e-5
    parity.record(tokens=len(rows), near_ties=near, val=worst,
                  y=parity.check_elementwise(y.float().cpu().numpy()[rows], y_o, tol, True, "decode y"),
                  r=parity.check_elementwise(r.cpu().numpy()[rows],
                                             oracle.decode(ref, gi, gvl.astype(np.float64), norm_match=0),
                                             1e-5, False, "kept r"),
                  gx=parity.check_elementwise(gx.float().cpu().numpy()[rows], gx_o, tol, True, "grad_x"),
                  gv=parity.check_elementwise(gv.cpu().numpy()[rows], gv_o, 1e-5, False, "grad_val"))
