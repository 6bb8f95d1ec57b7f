"""Standardisation moments on the GPU (dpb_stats_accumulate, dpb_stats_update)
against the oracle (§2.2 "Score Standardization", readings R16-R18), on the
same seeded inputs.

* Level 0 (every row): counts exact; sums within the fp32-partial bound
  1e-5 * sum_t |x_t[i]| (squares: 1e-5 * sum_t x_t[i]^2).
* Levels >= 1 (sampled rows): the set of counted features and every count
  exact. The sampled rows are drawn from a larger seeded draw, keeping rows
  whose oracle selection has a relative gap of at least NEAR_TIE at every cut
  (where two scores tie to within rounding, either kept set is correct). Sums
  within count * e with e = 1e-5 * max_t |x_t|_1 / sqrt(d), the fp32 scoring
  bound; squares within count * (2 s_max e + e^2).
* The EMA step on the same seeded sums: mu and sigma within fp32 rounding of
  the oracle's fp64 step, and the sums cleared.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2607_20652_gb300 import build, dpb, inputs
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _library():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    dpb.load()


def _pair(dtype="bf16", **kw):
    plan = dpb.Plan(dtype=dtype, **kw)
    c = plan.config
    per_level = c["select_mode"] == dpb.SELECT_PER_LEVEL
    ref = oracle.resolve(d=c["d"], m_bits=c["bits"][c["levels"] - 1], levels=c["levels"],
                         children=c["children"], beam=c["beam"], k=c["k"], seed=c["generator_seed"],
                         norm_match=c["norm_match"], t=c["field_t"], poly=c["field_poly"], bits=c["bits"],
                         k_per_level=c["k_per_level"] if per_level else None)
    return plan, ref


def _safe_rows(ref, x, n, seed, mu=None, sigma=None):
    """n sampled rows without a near-tie at any cut of the oracle's search."""
    cand = inputs.sample_rows(len(x), 3 * n, seed)
    xr = x[cand].astype(np.float64)
    if ref.k_per_level:
        gap = oracle.encode_per_level(ref, xr, mu=mu, sigma=sigma)[2]
    else:
        gap = oracle.encode(ref, xr, mu=mu, sigma=sigma)[3]
    rows = cand[gap >= parity.NEAR_TIE][:n]
    assert len(rows) == min(n, len(x)) or len(rows) >= n // 2
    return rows.astype(np.int32)


def _gpu_acc(plan, x_np, rows, mu=None, sigma=None):
    dev = torch.device("cuda")
    x = torch.from_numpy(np.ascontiguousarray(x_np)).to(dev).to(plan.torch_dtype)
    ws = plan.workspace(len(x), dev)
    acc = dpb.stats_buffer(plan, dev)
    mu_t = None if mu is None else torch.from_numpy(mu.astype(np.float32)).to(dev)
    sg_t = None if sigma is None else torch.from_numpy(sigma.astype(np.float32)).to(dev)
    smp = torch.from_numpy(np.asarray(rows, dtype=np.int32)).to(dev)
    dpb.stats_accumulate(plan, x, smp, acc, mu=mu_t, sigma=sg_t, workspace=ws)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), dpb.workspace_status(ws)


def _compare(acc_g, acc_o, x, rows, d):
    xr = x.astype(np.float64)
    # level 0: every row
    assert np.array_equal(acc_g[0, :d], acc_o[0, :d])
    b1 = 1e-5 * np.abs(xr).sum(axis=0) + 1e-30
    b2 = 1e-5 * (xr * xr).sum(axis=0) + 1e-30
    assert np.all(np.abs(acc_g[1, :d] - acc_o[1, :d]) <= b1)
    assert np.all(np.abs(acc_g[2, :d] - acc_o[2, :d]) <= b2)
    # levels >= 1: the sampled rows
    hi_g, hi_o = acc_g[:, d:], acc_o[:, d:]
    got, want = np.nonzero(hi_g[0])[0], np.nonzero(hi_o[0])[0]
    assert np.array_equal(got, want), (f"counted sets differ: gpu-only {np.setdiff1d(got, want)[:8]}, "
                                       f"oracle-only {np.setdiff1d(want, got)[:8]}")
    assert np.array_equal(hi_g[0], hi_o[0])
    if len(rows) == 0:
        return dict(level0=d, counted=0)
    n = hi_o[0, want]
    e = 1e-5 * np.abs(xr[rows]).sum(axis=1).max() / math.sqrt(d)
    smax = float(np.sqrt(hi_o[2, want].max()))
    ds = np.abs(hi_g[1, want] - hi_o[1, want])
    dq = np.abs(hi_g[2, want] - hi_o[2, want])
    assert np.all(ds <= n * e), f"sum error {ds.max():.3e} > {e:.3e} per occurrence"
    assert np.all(dq <= n * (2 * smax * e + e * e)), f"square-sum error {dq.max():.3e}"
    return dict(level0=d, counted=len(want), occurrences=int(n.sum()), sum_err=float(ds.max()))


def test_wide_global_moments():
    # the wide global layout: d = 768, 2^20 features, L = 5, beam 8, 16 children
    plan, ref = _pair(d=768, levels=5, m_bits=20, children=16, beam=8, k=64)
    x = inputs.to_bf16(inputs.gaussian_rows(2000, 768, 11))
    rows = _safe_rows(ref, x, 64, 12)
    acc_g, st = _gpu_acc(plan, x, rows)
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), rows)
    assert st == 0
    rep = _compare(acc_g, acc_o, x, rows, 768)
    assert rep["occurrences"] > len(rows) * 4 * 100     # about 128 distinct children per level and row
    print(rep)


def test_global_moments_with_tables_f32():
    plan, ref = _pair(dtype="f32", d=256, levels=4, m_bits=16, children=16, beam=8, k=32)
    m = 1 << 16
    mu, sigma = inputs.moment_tables(m, 13)
    x = inputs.gaussian_rows(300, 256, 14, outlier_frac=0.1)
    rows = _safe_rows(ref, x, 32, 15, mu=mu.astype(np.float64), sigma=sigma.astype(np.float64))
    acc_g, st = _gpu_acc(plan, x, rows, mu, sigma)
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), rows, mu=mu.astype(np.float64),
                                    sigma=sigma.astype(np.float64))
    assert st == 0
    print(_compare(acc_g, acc_o, x, rows, 256))


def test_per_level_paper_3l_moments():
    # PT-Small-3L (App. G): K = 16, 32, 64; Delta = 256; 2^10, 2^15, 2^17
    plan, ref = _pair(d=1024, levels=3, bits=[10, 15, 17], children=[0, 256, 256],
                      select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[16, 32, 64])
    x = inputs.to_bf16(inputs.gaussian_rows(200, 1024, 16))
    rows = _safe_rows(ref, x, 12, 17)
    acc_g, st = _gpu_acc(plan, x, rows)
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), rows)
    assert st == 0
    rep = _compare(acc_g, acc_o, x, rows, 1024)
    assert rep["occurrences"] > len(rows) * 10000       # 16 x 256 + 32 x 256 children per row, less repeats
    print(rep)


@pytest.mark.parametrize("T,d", [(1, 100), (257, 100), (33, 64)])
def test_ragged_level0_and_empty_sample(T, d):
    plan, ref = _pair(dtype="f32", d=d, levels=3, m_bits=12, children=16, beam=4, k=8)
    x = inputs.gaussian_rows(T, d, 18)
    acc_g, st = _gpu_acc(plan, x, [])
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), [])
    assert st == 0
    _compare(acc_g, acc_o, x, [], d)
    assert not acc_g[:, d:].any()


def test_moments_beyond_the_sign_tables():
    # d > 2048: the sampled search scores each child with a warp of popcounts
    plan, ref = _pair(dtype="f32", d=2304, levels=3, m_bits=16, children=16, beam=4, k=8)
    x = inputs.gaussian_rows(40, 2304, 24)
    rows = _safe_rows(ref, x, 6, 25)
    acc_g, st = _gpu_acc(plan, x, rows)
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), rows)
    assert st == 0
    print(_compare(acc_g, acc_o, x, rows, 2304))


def test_bad_rows_are_flagged_and_skipped():
    plan, ref = _pair(dtype="f32", d=64, levels=3, m_bits=12, children=16, beam=4, k=8)
    x = inputs.gaussian_rows(20, 64, 19)
    good = _safe_rows(ref, x, 4, 20)
    acc_g, st = _gpu_acc(plan, x, np.concatenate([good[:2], [-1, 20], good[2:]]))
    acc_o = oracle.stats_accumulate(ref, x.astype(np.float64), good)
    assert st == dpb.DEV_BAD_INDEX
    _compare(acc_g, acc_o, x, good, 64)


def _synthetic_sums(m, seed):
    g = inputs.rng(seed)
    n = g.choice([0, 0, 0, 1, 2, 3, 64], size=m).astype(np.float64)
    s = g.standard_normal(m) * np.sqrt(np.maximum(n, 1)) * (n > 0)
    q = (s * s / np.maximum(n, 1) + n * g.uniform(0.0, 2.0, m)) * (n > 0)
    return np.ascontiguousarray(np.stack([n, s, q]))


def test_ema_update_matches_oracle():
    plan, _ = _pair(dtype="f32", d=64, levels=3, m_bits=16, children=16, beam=4, k=8)
    m = 1 << 16
    acc = _synthetic_sums(m, 21)
    mu, sigma = inputs.moment_tables(m, 22)
    dev = torch.device("cuda")
    acc_t = torch.from_numpy(acc.copy()).to(dev)
    mu_t, sg_t = torch.from_numpy(mu.copy()).to(dev), torch.from_numpy(sigma.copy()).to(dev)
    dpb.stats_update(plan, acc_t, 0.05, mu_t, sg_t)
    torch.cuda.synchronize()
    alpha = float(np.float32(0.05))            # the value the fp32 argument carries
    mu_o, sg_o = oracle.stats_update(acc.copy(), alpha, mu.astype(np.float64), sigma.astype(np.float64))
    assert not acc_t.any().item()
    mu_g, sg_g = mu_t.cpu().numpy().astype(np.float64), sg_t.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(mu_g - mu_o) <= 2 ** -23 * np.abs(mu_o) + 1e-30)
    assert np.all(np.abs(sg_g - sg_o) <= 2 ** -23 * np.abs(sg_o) + 1e-30)
    untouched = acc[0] == 0
    assert np.array_equal(mu_g[untouched], mu[untouched]) and np.array_equal(sg_g[untouched], sigma[untouched])


def test_stats_step_moves_the_tables_like_the_oracle():
    # one EMA step with live tables through the public call (accumulate, then
    # update; one rank, so no all-reduce), twice on two batches
    plan, ref = _pair(d=256, levels=4, m_bits=16, children=16, beam=8, k=32)
    m = 1 << 16
    mu0, sg0 = inputs.moment_tables(m, 23, mean_scale=0.05, sigma_range=(0.8, 1.2))
    dev = torch.device("cuda")
    mu_t, sg_t = torch.from_numpy(mu0.copy()).to(dev), torch.from_numpy(sg0.copy()).to(dev)
    mu_o, sg_o = mu0.astype(np.float64), sg0.astype(np.float64)
    acc = dpb.stats_buffer(plan, dev)
    for step in range(2):
        x = inputs.to_bf16(inputs.gaussian_rows(400, 256, 30 + step))
        # the oracle selects with its own fp32-rounded tables of the previous step
        mu32, sg32 = mu_o.astype(np.float32).astype(np.float64), sg_o.astype(np.float32).astype(np.float64)
        rows = _safe_rows(ref, x, 48, 40 + step, mu=mu32, sigma=sg32)
        xt = torch.from_numpy(x).to(dev).to(torch.bfloat16)
        dpb.stats_step(plan, xt, mu_t, sg_t, 0.1, torch.from_numpy(rows).to(dev), acc=acc)
        a_o = oracle.stats_accumulate(ref, x.astype(np.float64), rows, mu=mu32, sigma=sg32)
        mu_o, sg_o = oracle.stats_update(a_o, float(np.float32(0.1)), mu32, sg32)
    torch.cuda.synchronize()
    assert not acc.any().item()
    mu_g, sg_g = mu_t.cpu().numpy().astype(np.float64), sg_t.cpu().numpy().astype(np.float64)
    moved = (mu_o != mu0.astype(np.float64))
    assert moved.sum() > 256 and np.array_equal(mu_g != mu0, moved)
    assert np.max(np.abs(mu_g - mu_o)) <= 1e-5 and np.max(np.abs(sg_g - sg_o)) <= 1e-5


@pytest.mark.parametrize("layout", ["global", "per_level"])
def test_packed_tables_give_the_same_codes(layout):
    # A workspace of dpb_workspace_size bytes lets the encoder pack (mu, 1/sigma)
    # pairs; the 256-byte minimum makes it read the two tables apart. Both use
    # the same fp32 arithmetic, so the codes must be identical bit for bit.
    if layout == "global":
        plan = dpb.Plan(d=768, levels=5, m_bits=20, children=16, beam=8, k=64, dtype="bf16")
    else:
        plan = dpb.Plan(d=1024, levels=3, bits=[10, 15, 17], children=[0, 256, 256], dtype="bf16",
                        select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[16, 32, 64])
    dev = torch.device("cuda")
    mu, sigma = inputs.moment_tables(plan.n_features, 50)
    mu_t, sg_t = torch.from_numpy(mu).to(dev), torch.from_numpy(sigma).to(dev)
    x = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(3000, plan.d, 51))).to(dev).to(torch.bfloat16)
    full = plan.workspace(len(x), dev)
    assert full.numel() >= 256 + 8 * plan.n_features
    small = torch.zeros(256, dtype=torch.uint8, device=dev)
    a = dpb.encode(plan, x, mu_t, sg_t, workspace=full)
    b = dpb.encode(plan, x, mu_t, sg_t, workspace=small)
    torch.cuda.synchronize()
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    assert dpb.workspace_status(full) == 0 and dpb.workspace_status(small) == 0


def test_bad_sigma_is_flagged_not_faulted():
    # sigma <= 0 (or not finite) for a feature that is used: every path sets
    # DPB_DEV_BAD_SIGMA and carries on
    dev = torch.device("cuda")
    x = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(64, 768, 95))).to(dev).to(torch.bfloat16)
    plan = dpb.Plan(d=768, levels=5, m_bits=20, children=16, beam=8, k=64, dtype="bf16")
    mu = torch.zeros(plan.n_features, device=dev)
    for bad in (0.0, -1.0, float("inf")):
        sg = torch.ones(plan.n_features, device=dev)
        sg[5] = bad                                            # a basis coordinate: every token reads it
        for ws in (plan.workspace(64, dev), torch.zeros(256, dtype=torch.uint8, device=dev)):
            idx, val, xn = dpb.encode(plan, x, mu, sg, workspace=ws)
            assert dpb.workspace_status(ws) & dpb.DEV_BAD_SIGMA
        ws = plan.workspace(64, dev)
        acc = dpb.stats_buffer(plan, dev)
        dpb.stats_accumulate(plan, x, torch.arange(8, dtype=torch.int32, device=dev), acc, mu=mu, sigma=sg,
                             workspace=ws)
        assert dpb.workspace_status(ws) & dpb.DEV_BAD_SIGMA
    # the backward divides grad_val by sigma of each code entry
    idx, val, xn = dpb.encode(plan, x)
    sg = torch.ones(plan.n_features, device=dev)
    sg[idx[0, 0].long()] = 0.0
    ws = plan.workspace(64, dev)
    gy = torch.ones_like(x)
    dpb.backward(plan, x, idx, val, gy, sg, workspace=ws)
    assert dpb.workspace_status(ws) & dpb.DEV_BAD_SIGMA
    # per-level layout
    pl = dpb.Plan(d=64, levels=3, bits=[6, 9, 12], children=[0, 16, 32], dtype="bf16",
                  select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[4, 8, 8])
    x2 = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(16, 64, 96))).to(dev).to(torch.bfloat16)
    sg2 = torch.ones(pl.n_features, device=dev)
    sg2[3] = -2.0
    ws = pl.workspace(16, dev)
    dpb.encode(pl, x2, torch.zeros(pl.n_features, device=dev), sg2, workspace=ws)
    assert dpb.workspace_status(ws) & dpb.DEV_BAD_SIGMA
