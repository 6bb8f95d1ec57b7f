"""The DPB as a PyTorch layer: autograd around the C-ABI calls.

Forward runs dpb_forward, i.e. dpb_encode then dpb_decode (the code and the
decode's r are kept for the backward); backward runs dpb_backward, the gradient with the
selected set held fixed. The layer has no trainable parameters: its dictionary is the
parity construction (§2.1). With ``ema`` set, the layer keeps live
standardisation tables (§2.2 "Score Standardization"): forward adds the
batch's moment sums (level 0 over every row, levels >= 1 over a 64-row
sub-sample) with the tables it selected with, and backward, once it has used
sigma, makes the EMA step (summed across data-parallel ranks first).

Every step runs in the library's kernels; this file only moves tensors.
"""
from __future__ import annotations

from typing import Optional

import torch

from . import dpb


class _DPBFunction(torch.autograd.Function):
    @staticmethod
    def forward(ctx, x, layer):
        T = x.shape[0]
        ws = layer._workspace(T, x.device)
        stream = torch.cuda.current_stream(x.device)
        ev = layer._events("forward")
        r = torch.empty((T, layer.d), dtype=torch.float32, device=x.device)  # kept for the backward
        idx, val, xn, y = dpb.forward(layer.plan, x, layer.mu, layer.sigma, workspace=ws, stream=stream, r_out=r)
        if layer.ema is not None and layer.training:
            rows = dpb.sample_rows(T, layer.ema_rows, layer._gen, x.device)
            dpb.stats_accumulate(layer.plan, x, rows, layer._acc, mu=layer.mu, sigma=layer.sigma, workspace=ws,
                                 stream=stream)
        if ev:
            ev[1].record(stream)
        ctx.save_for_backward(x, idx, val, r)
        ctx.layer = layer
        layer.last_code = (idx, val)
        return y

    @staticmethod
    def backward(ctx, gy):
        x, idx, val, r = ctx.saved_tensors
        layer = ctx.layer
        gy = gy.contiguous().to(x.dtype)
        ws = layer._workspace(x.shape[0], x.device)
        stream = torch.cuda.current_stream(x.device)
        ev = layer._events("backward")
        gx, gv = dpb.backward(layer.plan, x, idx, val, gy, layer.sigma, workspace=ws, stream=stream, r=r)
        if layer.ema is not None and layer.training:
            dpb.ema_step(lambda a: None,
                         lambda a: dpb.stats_update(layer.plan, a, layer.ema, layer.mu, layer.sigma, stream=stream),
                         layer._acc, layer.group)
        if ev:
            ev[1].record(stream)
        layer.last_grad_val = gv
        return gx, None


class DPBLayer(torch.nn.Module):
    """y = decode(encode(x)) over the last dimension (d), bf16 rows.

    ``plan_kw`` are dpb.Plan's arguments (d, levels, m_bits, children, beam,
    k, ...). ``ema`` (the EMA weight alpha, or None) turns on live
    standardisation; ``ema_rows`` is the sub-sample size of levels >= 1.
    ``group`` is the data-parallel process group of the moment all-reduce.
    """

    def __init__(self, ema: Optional[float] = None, ema_rows: int = 64, seed: int = 0, group=None,
                 device=None, **plan_kw):
        super().__init__()
        plan_kw.setdefault("dtype", "bf16")
        self.plan = dpb.Plan(**plan_kw)
        self.d = self.plan.d
        self.ema, self.ema_rows, self.group = ema, ema_rows, group
        dev = torch.device(device or "cuda")
        self._acc = None
        if ema is not None:
            m = self.plan.n_features
            self.register_buffer("mu", torch.zeros(m, dtype=torch.float32, device=dev))
            self.register_buffer("sigma", torch.ones(m, dtype=torch.float32, device=dev))
            self._acc = dpb.stats_buffer(self.plan, dev)
            self._gen = torch.Generator().manual_seed(seed)
        else:
            self.register_buffer("mu", None)
            self.register_buffer("sigma", None)
        self._ws = None
        self.timing = None          # set to a list to collect (forward, backward) CUDA event pairs
        self.last_code = None
        self.last_grad_val = None

    def _workspace(self, T, device):
        n = self.plan.workspace_size(T)
        if self._ws is None or self._ws.numel() < n or self._ws.device != device:
            self._ws = torch.zeros(n, dtype=torch.uint8, device=device)
        return self._ws

    def _events(self, which):
        if self.timing is None:
            return None
        ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        ev[0].record(torch.cuda.current_stream())
        self.timing.append((which, ev))
        return ev

    def forward(self, x):
        shape = x.shape
        if shape[-1] != self.d:
            raise ValueError(f"last dimension {shape[-1]} != d = {self.d}")
        rows = x.reshape(-1, self.d).to(self.plan.torch_dtype).contiguous()
        return _DPBFunction.apply(rows, self).view(shape)
