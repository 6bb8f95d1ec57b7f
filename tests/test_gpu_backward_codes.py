"""The backward (and the decode) on crafted codes, through the C ABI, against
the oracle.

The table-driven backward treats a code's basis entries (index < d) and
hashed entries (index >= d) apart, and gives whole warps to the first
multiple of 32 hashed entries and four lanes each to the rest. These codes
cover every such split (0, 1, 31, 32, 33, 63, 64, 65, 100 and all hashed
entries, of 128, or of 96 where d < 128), rows whose width leaves a partial 32-coordinate block and a
partial chunk of blocks (d = 100, 102, 200; 102 also takes the scalar row path), with and without the decode's r and
with and without standardisation tables. fp32 rows, element by element:
within 1e-5 of max(|ref_i|, row rms), as for every fp32 output.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20652_gb300 import build, dpb, inputs
from tests import parity

pytestmark = pytest.mark.gpu

HASHED = (0, 1, 31, 32, 33, 63, 64, 65, 100, 128)


def _codes_for(d):
    """Code length (k <= d) and the hashed counts that fit it."""
    k = 128 if d >= 128 else 96
    return k, [h for h in HASHED if h < k] + [k]


@pytest.fixture(scope="module", autouse=True)
def _library():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    dpb.load()


@pytest.mark.parametrize("d", [100, 102, 200, 768])
@pytest.mark.parametrize("kept_r", [False, True])
@pytest.mark.parametrize("tables", [False, True])
def test_backward_on_crafted_codes(d, kept_r, tables):
    (k, counts), m_bits = _codes_for(d), 16
    plan = dpb.Plan(d=d, levels=4, m_bits=m_bits, children=16, beam=8, k=k, dtype="f32")
    assert plan.code_len == k
    c = plan.config
    ref = oracle.resolve(d=d, m_bits=m_bits, levels=c["levels"], children=c["children"], beam=c["beam"], k=k,
                         seed=c["generator_seed"], norm_match=c["norm_match"], t=c["field_t"],
                         poly=c["field_poly"], bits=c["bits"])
    T = 6 * len(counts)
    seed = 11 * d + 2 * kept_r + tables
    idx, val = inputs.mixed_codes(T, d, m_bits, k, counts, seed)
    x = inputs.gaussian_rows(T, d, seed + 1)
    gy = inputs.normal((T, d), seed + 2)
    sigma = inputs.moment_tables(1 << m_bits, seed + 3)[1].astype(np.float32) if tables else None
    dev = torch.device("cuda")
    xt, gyt = torch.from_numpy(x).to(dev), torch.from_numpy(gy).to(dev)
    it, vt = torch.from_numpy(idx).to(dev), torch.from_numpy(val).to(dev)
    st = None if sigma is None else torch.from_numpy(sigma).to(dev)
    r = None
    if kept_r:
        xn = torch.linalg.vector_norm(xt, dim=1)
        r = torch.empty((T, d), dtype=torch.float32, device=dev)
        dpb.decode(plan, it, vt, xn, r_out=r)
    ws = plan.workspace(T, dev)
    gx, gv = dpb.backward(plan, xt, it, vt, gyt, sigma=st, workspace=ws, r=r)
    torch.cuda.synchronize()
    assert dpb.workspace_status(ws) == 0
    gx_o, gv_o = oracle.backward(ref, x.astype(np.float64), idx, val.astype(np.float64), gy.astype(np.float64),
                                 sigma=None if sigma is None else sigma.astype(np.float64))
    assert parity.rel_rows(gx.cpu().numpy(), gx_o).max() <= 1e-5
    assert parity.rel_rows(gv.cpu().numpy(), gv_o).max() <= 1e-5
    parity.record(tokens=T, near_ties=0,
                  gx=parity.check_elementwise(gx.cpu().numpy(), gx_o, 1e-5, False, "grad_x"),
                  gv=parity.check_elementwise(gv.cpu().numpy(), gv_o, 1e-5, False, "grad_val"))


@pytest.mark.parametrize("d", [100, 102, 200, 768])
def test_decode_on_crafted_codes(d):
    (k, counts), m_bits = _codes_for(d), 16
    plan = dpb.Plan(d=d, levels=4, m_bits=m_bits, children=16, beam=8, k=k, dtype="f32")
    c = plan.config
    ref = oracle.resolve(d=d, m_bits=m_bits, levels=c["levels"], children=c["children"], beam=c["beam"], k=k,
                         seed=c["generator_seed"], norm_match=c["norm_match"], t=c["field_t"],
                         poly=c["field_poly"], bits=c["bits"])
    T = 6 * len(counts)
    idx, val = inputs.mixed_codes(T, d, m_bits, k, counts, 7 * d)
    xn = np.abs(inputs.normal((T,), 7 * d + 1)) + np.float32(0.5)
    dev = torch.device("cuda")
    r = torch.empty((T, d), dtype=torch.float32, device=dev)
    y = dpb.decode(plan, torch.from_numpy(idx).to(dev), torch.from_numpy(val).to(dev),
                   torch.from_numpy(xn).to(dev), r_out=r)
    torch.cuda.synchronize()
    y_o = oracle.decode(ref, idx, val.astype(np.float64), xn.astype(np.float64))
    r_o = oracle.decode(ref, idx, val.astype(np.float64), norm_match=0)
    assert parity.rel_rows(y.cpu().numpy(), y_o).max() <= 1e-5
    assert parity.rel_rows(r.cpu().numpy(), r_o).max() <= 1e-5
    parity.record(tokens=T, near_ties=0,
                  y=parity.check_elementwise(y.cpu().numpy(), y_o, 1e-5, False, "decode y"),
                  r=parity.check_elementwise(r.cpu().numpy(), r_o, 1e-5, False, "kept r"))
