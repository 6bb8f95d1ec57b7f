"""A ParityTransformer of GPT-2 shape for timing the DPB inside a training step.

§3 of the paper: a GPT-2-style backbone (learned positional embeddings, tied
embedding and unembedding, RMSNorm in place of LayerNorm) with a Deep Parity
Bottleneck inserted before the input of every MLP. Weights are random
(nothing here is trained); attention and the dense layers are PyTorch's own
(cuBLAS / fused attention), the DPB layers are this library's kernels. The
model exists to measure the DPB's share of a forward + backward + optimiser
step at the paper's scale; it is not a training recipe.
"""
from __future__ import annotations

import math
from typing import Optional

import torch
import torch.nn.functional as F
from torch import nn

from .layer import DPBLayer


class _Attention(nn.Module):
    def __init__(self, d: int, heads: int):
        super().__init__()
        self.heads = heads
        self.qkv = nn.Linear(d, 3 * d, bias=False)
        self.out = nn.Linear(d, d, bias=False)

    def forward(self, x):
        B, S, d = x.shape
        q, k, v = self.qkv(x).view(B, S, 3, self.heads, d // self.heads).permute(2, 0, 3, 1, 4)
        o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        return self.out(o.transpose(1, 2).reshape(B, S, d))


class _Block(nn.Module):
    def __init__(self, d: int, heads: int, d_mlp: int, dpb: Optional[DPBLayer]):
        super().__init__()
        self.n1 = nn.RMSNorm(d)
        self.attn = _Attention(d, heads)
        self.n2 = nn.RMSNorm(d)
        self.dpb = dpb
        self.up = nn.Linear(d, d_mlp, bias=False)
        self.down = nn.Linear(d_mlp, d, bias=False)

    def forward(self, x):
        x = x + self.attn(self.n1(x))
        h = self.n2(x)
        if self.dpb is not None:
            h = self.dpb(h)  # the bottleneck sits before the MLP's input (§3)
        return x + self.down(F.gelu(self.up(h)))


class ParityTransformer(nn.Module):
    """GPT-2 shape (12 layers, d = 768, 12 heads, MLP 3072, vocab 50257,
    context 1024 by default) with a DPB before every MLP; ``dpb=None`` gives
    the dense model of the same shape. ``dpb`` holds DPBLayer arguments."""

    def __init__(self, layers: int = 12, d: int = 768, heads: int = 12, d_mlp: int = 3072, vocab: int = 50257,
                 context: int = 1024, dpb: Optional[dict] = None, device=None, dtype=torch.bfloat16):
        super().__init__()
        self.tok = nn.Embedding(vocab, d)
        self.pos = nn.Embedding(context, d)
        blocks = []
        for i in range(layers):
            layer = DPBLayer(seed=i, device=device, d=d, **dpb) if dpb is not None else None
            blocks.append(_Block(d, heads, d_mlp, layer))
        self.blocks = nn.ModuleList(blocks)
        self.norm = nn.RMSNorm(d)
        std = 0.02
        for p in self.parameters():
            if p.dim() >= 2:
                nn.init.normal_(p, std=std)
        for b in self.blocks:  # scaled residual projections, as in GPT-2
            nn.init.normal_(b.attn.out.weight, std=std / math.sqrt(2 * layers))
            nn.init.normal_(b.down.weight, std=std / math.sqrt(2 * layers))
        self.to(device=device)
        for p in self.parameters():  # weights in dtype; the DPB tables stay fp32
            p.data = p.data.to(dtype)

    def dpb_layers(self):
        return [b.dpb for b in self.blocks if b.dpb is not None]

    def forward(self, ids, targets=None):
        B, S = ids.shape
        x = self.tok(ids) + self.pos(torch.arange(S, device=ids.device))
        for b in self.blocks:
            x = b(x)
        logits = F.linear(self.norm(x), self.tok.weight)  # tied unembedding
        if targets is None:
            return logits
        return F.cross_entropy(logits.float().view(-1, logits.shape[-1]), targets.view(-1))
