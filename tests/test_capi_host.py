"""CPU tests of the C-ABI library: it loads, exports every entry point that
include/dpb.h declares, and its host-side plan builder (field, seed matrix,
generators, config resolution) agrees bit-exactly with the oracle's
independent construction. No compute call is made here."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2607_20652_gb300 import build, dpb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return dpb.load()


def _declared():
    text = open(os.path.join(ROOT, "include", "dpb.h")).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+char\s*\*|dpb_status)\s*(dpb_\w+)\s*\(", text, re.M)))


def test_library_exports_every_declared_symbol(lib):
    names = _declared()
    assert len(names) >= 12
    for name in names:
        assert hasattr(lib, name), name
    out = os.popen(f"nm -D --defined-only {dpb.library_path()}").read()
    exported = set(re.findall(r" T (dpb_\w+)", out))
    assert set(names) <= exported
    assert set(dpb.EXPORTS) == set(names)


def test_status_strings(lib):
    assert lib.dpb_status_string(0) == b"ok"
    assert lib.dpb_status_string(2) == b"unsupported configuration"


CASES = [
    # name, d, m_bits, levels, beam, k
    ("tiny", 64, 12, 3, 4, 8),
    ("gpt2", 768, 16, 4, 8, 32),
    ("wide", 768, 20, 5, 8, 64),
    ("sweep_2^18", 768, 18, 5, 16, 128),
    ("sweep_2^22", 768, 22, 5, 4, 16),
    ("paper_small_3l", 1024, 17, 3, 8, 64),
]


@pytest.mark.parametrize("name,d,m_bits,levels,beam,k", CASES)
def test_plan_tables_match_oracle(lib, name, d, m_bits, levels, beam, k):
    for seed in (0, 12345):
        plan = dpb.Plan(d=d, levels=levels, m_bits=m_bits, children=16, beam=beam, k=k, seed=seed)
        ref = oracle.resolve(d=d, m_bits=m_bits, levels=levels, children=16, beam=beam, k=k, seed=seed)
        cfg = plan.config
        assert cfg["bits"] == ref.bits
        assert cfg["field_t"] == ref.t and cfg["field_poly"] == ref.poly
        M, G = plan.tables()
        assert np.array_equal(M, ref.M)
        for l in range(1, levels):
            assert np.array_equal(G[l, :16], ref.G[l, :16])
            assert np.all(G[l, 16:] == 0)


@pytest.mark.parametrize("t", [6, 7, 8, 9, 12, 13])
def test_default_polynomials_match_oracle(lib, t):
    # the library's and the oracle's default-polynomial rules agree
    d = 1 << min(t, 12)
    plan = dpb.Plan(d=min(d, 4096), levels=2, m_bits=2 * t, children=4, beam=2, k=4, field_t=t)
    assert plan.config["field_poly"] == oracle.default_poly(t)
    M, _ = plan.tables()
    assert np.array_equal(M, oracle.seed_matrix(plan.d, t, oracle.default_poly(t)))


def test_explicit_generators_are_used(lib):
    G = np.zeros((8, 256), dtype=np.uint32)
    G[1, :16] = [(h << 6) | s for h in range(1, 9) for s in (0, 1)]
    plan = dpb.Plan(d=64, levels=2, m_bits=12, children=16, beam=4, k=8, generators=G,
                    bits=[6, 12], dtype="f32")
    _, got = plan.tables()
    assert np.array_equal(got[1, :16], G[1, :16])


@pytest.mark.parametrize("kw,status", [
    (dict(k=65, d=64), 1),                      # k > d
    (dict(beam=33), 2),                         # beam outside [1, 32]
    (dict(k=257, d=512), 2),                    # k outside [1, 256]
    (dict(field_poly=0x41, field_t=6), 1),      # z^6+1 = (z^3+1)^2 is reducible
    (dict(bits=[6, 6, 12]), 1),                 # bits must increase
    (dict(children=[0, 300, 16]), 2),           # children outside [1, 256]
    (dict(d=5000), 2),                          # d outside [2, 4096]
    (dict(m_bits=40), 2),                       # index space beyond 2^31
    (dict(children=[0, 65, 16], bits=[6, 7, 12]), 1),  # only 64 valid generators at level 1
])
def test_invalid_configs_are_rejected(lib, kw, status):
    args = dict(d=64, levels=3, m_bits=12, children=16, beam=4, k=8, dtype="f32")
    args.update(kw)
    with pytest.raises(dpb.DPBError) as e:
        dpb.Plan(**args)
    assert e.value.status == status


@pytest.mark.parametrize("kw,status", [
    (dict(dtype="f32"), 2),                                   # per-level scoring needs bf16 rows
    (dict(d=96, bits=[7, 10, 12]), 2),                        # d a multiple of 64
    (dict(children=[0, 24, 32]), 2),                          # Delta_l a multiple of 16
    (dict(k_per_level=[40, 8, 8]), 2),                        # at most 32 parents per token
    (dict(k_per_level=[4, 65, 8]), 2),                        # K_l at most 64
    (dict(k_per_level=[65, 8, 8], d=64), 2),                  # K_0 beyond [1, 64]
    (dict(k_per_level=[2, 40, 8], children=[0, 16, 32]), 1),  # 40 of 2 x 16 candidates
])
def test_per_level_configs_are_checked(lib, kw, status):
    args = dict(d=64, levels=3, bits=[6, 9, 12], children=[0, 16, 32], dtype="bf16",
                select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[4, 8, 8])
    args.update(kw)
    with pytest.raises(dpb.DPBError) as e:
        dpb.Plan(**args)
    assert e.value.status == status


def test_per_level_code_length(lib):
    # the paper's 3L layout (App. G): K = 16, 32, 64 over 2^10, 2^15, 2^17 indices
    plan = dpb.Plan(d=1024, levels=3, bits=[10, 15, 17], children=[0, 256, 256], dtype="bf16",
                    select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[16, 32, 64])
    assert plan.code_len == 112
    assert plan.config["select_mode"] == dpb.SELECT_PER_LEVEL


def test_stats_arguments_are_checked(lib):
    # Host-side validation of the moment calls runs before any device work, so
    # a plan without a device still reports each bad argument (the pointers
    # below are never dereferenced).
    INVALID, CUDA = 1, 3
    plan = dpb.Plan(d=64, levels=3, m_bits=12, children=16, beam=4, k=8, dtype="f32")
    P = ctypes.c_void_p
    buf, odd = P(0x10000), P(0x10004)
    acc = lib.dpb_stats_accumulate
    # mu without sigma
    assert acc(plan.handle, buf, 4, buf, None, buf, 1, buf, buf, 256, None) == INVALID
    # negative sample count, sampled rows of an empty batch, misaligned acc
    assert acc(plan.handle, buf, 4, None, None, buf, -1, buf, buf, 256, None) == INVALID
    assert acc(plan.handle, buf, 0, None, None, buf, 1, buf, buf, 256, None) == INVALID
    assert acc(plan.handle, buf, 4, None, None, buf, 1, odd, buf, 256, None) == INVALID
    assert acc(plan.handle, buf, 0, None, None, None, 0, buf, buf, 256, None) == 0   # empty batch
    up = lib.dpb_stats_update
    for alpha in (0.0, 1.0, -0.5, float("nan")):
        assert up(plan.handle, buf, alpha, buf, buf, None) == INVALID
    assert up(plan.handle, odd, 0.5, buf, buf, None) == INVALID
    assert up(plan.handle, buf, 0.5, None, buf, None) == INVALID
    # the largest kept sets (32 parents of 256 children each) still fit the sampled
    # search: valid arguments reach the device check
    big = dpb.Plan(d=1024, levels=2, bits=[10, 17], children=[0, 256], dtype="bf16",
                   select_mode=dpb.SELECT_PER_LEVEL, k_per_level=[32, 64])
    assert acc(big.handle, buf, 4, None, None, buf, 1, buf, buf, 256, None) == CUDA


def test_workspace_holds_the_packed_tables(lib):
    # 256 bytes for the status word, then 8 bytes per feature for the
    # standardisation tables packed as (mu, 1 / sigma)
    for m_bits in (12, 20):
        plan = dpb.Plan(d=64, levels=3, m_bits=m_bits, children=16, beam=4, k=8, dtype="f32")
        assert plan.workspace_size(1) == 256 + 8 * (1 << m_bits)


def test_coset_scoring_is_checked(lib):
    # DPB_SCORING_COSET_WHT: every level's 16 generators one coset g0 ^ {0..15},
    # given by the caller, on the tensor-core layout (bf16, beam 8, 16 children)
    from paper_2607_20652_gb300 import inputs
    bits = [10, 12, 15, 17, 20]
    G = inputs.coset_generators(bits, 5, seed=3)
    kw = dict(d=768, levels=5, bits=bits, children=16, beam=8, k=64, dtype="bf16",
              scoring=dpb.SCORING_COSET_WHT)
    plan = dpb.Plan(generators=G, **kw)
    assert plan.config["scoring"] == dpb.SCORING_COSET_WHT
    _, Gp = plan.tables()
    assert np.array_equal(Gp[1:5, :16], G[1:5, :16])
    with pytest.raises(dpb.DPBError) as e:
        dpb.Plan(**kw)                                        # the plan's own random generators
    assert e.value.status == 1
    bad = G.copy()
    bad[2, 5] ^= 1 << 13                                      # not in the coset of g0
    with pytest.raises(dpb.DPBError) as e:
        dpb.Plan(generators=bad, **kw)
    assert e.value.status == 1
    with pytest.raises(dpb.DPBError) as e:
        dpb.Plan(generators=G, **dict(kw, dtype="f32"))       # outside the tensor-core layout
    assert e.value.status == 2
