"""Named DPB workloads (plain data, shared by the tests and the benchmark).

Sizes follow the workloads this build is measured on; the level layout of
each is derived by the plan (r_0 = ceil(log2 d), r_l = r_0 + floor(l (N - r_0)
/ (L - 1))) and children = 16 per parent at every level.
"""

WORKLOADS = {
    # T=256, d=64, 2^12 features as 3 levels of 16 children, beam 4, k=8,
    # fp32 x ~ N(0, 1), seed 0; encode + decode + backward
    "tiny": dict(T=256, d=64, m_bits=12, levels=3, children=16, beam=4, k=8, dtype="f32",
                 inputs="gaussian", seed=0, grad_seed=1, passes="fwd+bwd"),
    # T=8192, d=768, 2^16 features (4 levels x 16), beam 8, k=32, bf16 x ~ N(0,1)
    # with 5% of rows scaled x10; encode + decode
    "gpt2": dict(T=8192, d=768, m_bits=16, levels=4, children=16, beam=8, k=32, dtype="bf16",
                 inputs="gaussian", outlier_frac=0.05, outlier_scale=10.0, seed=0, passes="fwd"),
    # T=65536, d=768, 2^20 features (5 levels x 16), beam 8, k=64, bf16 x = a planted
    # tree of 64 parity directions (8 roots, 8 per level at levels 1-3, 32 at level 4,
    # coefficients +-U[1, 2]) plus N(0, 0.1^2) noise; encode + decode + backward with
    # grad_y ~ N(0, 1) (seed 1)
    "wide": dict(T=65536, d=768, m_bits=20, levels=5, children=16, beam=8, k=64, dtype="bf16",
                 inputs="planted", planted=[8, 8, 8, 8, 32], noise=0.1, seed=0, grad_seed=1,
                 passes="fwd+bwd"),
}

# The paper's own per-level layouts (App. G), per-level selection: PT-Small-3L
# (d = 1024; K = 16, 32, 64 over 2^10, 2^15, 2^17 indices; 256 children per
# parent) and the 2L variants at d = 1024 (K = 16, 32 over 2^10, 2^15); bf16
# x ~ N(0, 1); encode + decode + backward with grad_y ~ N(0, 1)
PER_LEVEL = {
    "paper3l": dict(T=65536, d=1024, levels=3, bits=[10, 15, 17], children=[0, 256, 256],
                    k_per_level=[16, 32, 64], dtype="bf16", inputs="gaussian", seed=0, grad_seed=1,
                    passes="fwd+bwd"),
    "paper2l": dict(T=65536, d=1024, levels=2, bits=[10, 15], children=[0, 256],
                    k_per_level=[16, 32], dtype="bf16", inputs="gaussian", seed=0, grad_seed=1,
                    passes="fwd+bwd"),
}

# d=768, T=32768: features 2^16/2^18/2^20/2^22, k in {16,32,64,128}, beam in {4,8,16}
SWEEP = [dict(T=32768, d=768, m_bits=mb, levels=5, children=16, beam=b, k=k, dtype="bf16",
              inputs="gaussian", seed=0, grad_seed=1, passes="fwd+bwd")
         for mb in (16, 18, 20, 22) for k in (16, 32, 64, 128) for b in (4, 8, 16)]
