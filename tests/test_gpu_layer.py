"""The DPB as a PyTorch layer (autograd around the C ABI) and the
ParityTransformer step built from it.

The layer must give exactly the C-ABI calls' outputs (same kernels): forward
= dpb_encode + dpb_decode (keeping r), the input gradient = dpb_backward with
the code and r of that forward. Its live tables must move like a direct dpb_stats_* sequence.
A small ParityTransformer must train (the loss falls on a fixed batch) with
finite gradients everywhere.
"""
import numpy as np
import pytest
import torch

from paper_2607_20652_gb300 import build, dpb, inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _library():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    dpb.load()


PLAN = dict(d=768, levels=5, m_bits=20, children=16, beam=8, k=64)


def test_layer_is_the_c_abi_calls():
    from paper_2607_20652_gb300.layer import DPBLayer
    dev = torch.device("cuda")
    layer = DPBLayer(device=dev, **PLAN)
    x0 = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(2 * 300, 768, 60))).to(dev).to(torch.bfloat16)
    x = x0.view(2, 300, 768).clone().requires_grad_(True)
    gy = torch.from_numpy(inputs.to_bf16(inputs.normal((2, 300, 768), 61))).to(dev).to(torch.bfloat16)
    y = layer(x)
    y.backward(gy)
    idx, val, xn = dpb.encode(layer.plan, x0)
    r = torch.empty((600, 768), dtype=torch.float32, device=dev)
    y_ref = dpb.decode(layer.plan, idx, val, xn, r_out=r)
    gx_ref, gv_ref = dpb.backward(layer.plan, x0, idx, val, gy.view(-1, 768).contiguous(), r=r)
    torch.cuda.synchronize()
    assert torch.equal(y.view(-1, 768), y_ref)
    assert torch.equal(x.grad.view(-1, 768), gx_ref)
    assert torch.equal(layer.last_grad_val, gv_ref)
    assert dpb.workspace_status(layer._ws) == 0


def test_layer_tables_follow_the_stats_calls():
    from paper_2607_20652_gb300.layer import DPBLayer
    dev = torch.device("cuda")
    layer = DPBLayer(ema=0.1, ema_rows=16, seed=3, device=dev, **PLAN)
    x = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(512, 768, 62))).to(dev).to(torch.bfloat16)
    x.requires_grad_(True)
    layer(x).sum().backward()
    # the same step by hand: accumulate with the starting tables on the same
    # sampled rows, then one update
    mu = torch.zeros(layer.plan.n_features, device=dev)
    sg = torch.ones(layer.plan.n_features, device=dev)
    rows = dpb.sample_rows(512, 16, torch.Generator().manual_seed(3), dev)
    dpb.stats_step(layer.plan, x.detach(), mu, sg, 0.1, rows)
    torch.cuda.synchronize()
    moved = mu != 0
    assert int(moved.sum()) > 768 and torch.equal(moved, layer.mu != 0)
    assert torch.allclose(layer.mu, mu, rtol=0, atol=1e-6) and torch.allclose(layer.sigma, sg, rtol=0, atol=1e-6)
    assert not layer._acc.any().item()


@pytest.mark.parametrize("ema", [None, 0.05])
def test_small_parity_transformer_trains(ema):
    from paper_2607_20652_gb300.transformer import ParityTransformer
    dev = torch.device("cuda")
    torch.manual_seed(0)
    model = ParityTransformer(layers=2, d=64, heads=4, d_mlp=128, vocab=97, context=32,
                              dpb=dict(levels=3, m_bits=12, children=16, beam=8, k=8, ema=ema), device=dev)
    opt = torch.optim.AdamW(model.parameters(), lr=3e-3)
    g = torch.Generator().manual_seed(1)
    ids = torch.randint(0, 97, (4, 32), generator=g).to(dev)
    tgt = torch.randint(0, 97, (4, 32), generator=g).to(dev)
    losses = []
    for _ in range(30):
        opt.zero_grad(set_to_none=True)
        loss = model(ids, tgt)
        loss.backward()
        for p in model.parameters():
            assert p.grad is None or torch.isfinite(p.grad).all()
        opt.step()
        losses.append(float(loss.detach()))
    assert np.isfinite(losses).all() and losses[-1] < losses[0] - 0.5, losses
    for layer in model.dpb_layers():
        assert dpb.workspace_status(layer._ws) == 0
        if ema is not None:
            assert int((layer.mu != 0).sum()) > 64 and torch.all(layer.sigma > 0)
