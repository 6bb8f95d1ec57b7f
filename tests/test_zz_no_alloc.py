"""dpb_encode_noalloc, the encoder entry point that allocates nothing.

It exists for callers that cannot allocate device memory (plug-ins inside a
runtime that owns every allocation and hands them only input and output
buffers). Its scratch lives in a fixed device array inside the library. This
test calls it through the C ABI twice in a row and checks each call against
dpb_encode on the same inputs, within the tolerances of the parity tests, for
the global (mma.sync) and the per-level (tcgen05) encoders; the second call
also shows that the shared scratch starts clean.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_20652_gb300 import build, dpb, inputs
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    return dpb.load()


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _noalloc(lib, plan, x, mu=None, sigma=None):
    T, k = x.shape[0], plan.code_len
    idx = torch.full((T, k), -7, dtype=torch.int32, device=x.device)
    val = torch.full((T, k), float("nan"), dtype=torch.float32, device=x.device)
    xn = torch.empty((T,), dtype=torch.float32, device=x.device)
    st = torch.full((1,), -1, dtype=torch.int32, device=x.device)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.dpb_encode_noalloc(plan.handle, _p(x), T, _p(mu), _p(sigma), _p(idx), _p(val), _p(xn),
                                _p(st), stream)
    assert rc == 0, lib.dpb_last_error()
    torch.cuda.synchronize()
    return idx.cpu().numpy(), val.cpu().numpy(), xn.cpu().numpy(), int(st.item())


@pytest.mark.parametrize("dtype,d,m_bits,levels,beam,k", [("bf16", 768, 20, 5, 8, 64), ("f32", 64, 12, 3, 4, 8)])
def test_noalloc_matches_encode_twice(lib, dtype, d, m_bits, levels, beam, k):
    plan = dpb.Plan(d=d, levels=levels, m_bits=m_bits, children=16, beam=beam, k=k, dtype=dtype)
    T = 777
    x_np = inputs.gaussian_rows(T, d, 42)
    if dtype == "bf16":
        x_np = inputs.to_bf16(x_np)
    x = torch.from_numpy(x_np).cuda().to(plan.torch_dtype)
    ws = plan.workspace(T)
    ri, rv, rxn = (t.cpu().numpy() for t in dpb.encode(plan, x, workspace=ws))
    torch.cuda.synchronize()
    for _ in range(2):
        idx, val, xn, st = _noalloc(lib, plan, x)
        assert st == 0
        parity.check_code_order(idx, val)
        near, _ = parity.compare_codes(idx, val, ri, rv.astype(np.float64), np.full(T, np.inf), rxn)
        assert near == 0
        assert np.array_equal(idx, ri) and np.array_equal(val, rv)
        assert np.allclose(xn, rxn, rtol=1e-6, atol=0)


def test_noalloc_per_level_plan_matches_encode_twice(lib):
    # the paper's per-level selection (tcgen05 scoring): 3L layout of App. G
    plan = dpb.Plan(d=1024, levels=3, bits=[10, 15, 17], children=[0, 256, 256], dtype="bf16",
                    select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[16, 32, 64])
    T = 203                                        # 25 blocks of 8 tokens and a ragged tail
    x = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(T, 1024, 44))).cuda().to(torch.bfloat16)
    ri, rv, rxn = (t.cpu().numpy() for t in dpb.encode(plan, x, workspace=plan.workspace(T)))
    torch.cuda.synchronize()
    for _ in range(2):
        idx, val, xn, st = _noalloc(lib, plan, x)
        assert st == 0
        assert np.array_equal(idx, ri) and np.array_equal(val, rv)
        assert np.allclose(xn, rxn, rtol=1e-6, atol=0)


def test_noalloc_status_is_per_call(lib):
    plan = dpb.Plan(d=64, levels=3, m_bits=12, children=16, beam=4, k=8, dtype="f32")
    x = torch.from_numpy(inputs.gaussian_rows(50, 64, 3)).cuda()
    m = 1 << plan.config["m_bits"]
    mu = torch.zeros(m, device="cuda")
    bad = torch.ones(m, device="cuda")
    bad[5] = 0.0                                   # a sigma <= 0 is flagged
    _, _, _, st1 = _noalloc(lib, plan, x, mu, bad)
    assert st1 & dpb.DEV_BAD_SIGMA
    idx, val, _, st2 = _noalloc(lib, plan, x, mu, torch.ones(m, device="cuda"))
    assert st2 == 0                                # the shared scratch was cleared
    ri, rv, _ = dpb.encode(plan, x)
    assert np.array_equal(idx, ri.cpu().numpy()) and np.array_equal(val, rv.cpu().numpy())


def test_noalloc_rejects_bad_arguments(lib):
    plan = dpb.Plan(d=64, levels=3, m_bits=12, children=16, beam=4, k=8, dtype="f32")
    x = torch.zeros((4, 64), device="cuda")
    idx = torch.empty((4, 8), dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.dpb_encode_noalloc(plan.handle, _p(x), 4, None, None, _p(idx), None, None, None, stream)
    assert rc == dpb.DPBError(1, "").status
