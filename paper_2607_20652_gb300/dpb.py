"""Python binding of the DPB C-ABI library (``include/dpb.h``).

Argument marshalling only: every step of encode, decode and backward runs in
the library's CUDA kernels. PyTorch supplies device memory and the current
stream; tensors are passed to the library as raw pointers. The functions keep
the C names (``dpb_encode`` -> ``encode`` ...). Loading fails loudly if the
library has not been built: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

from . import build as _build

MAX_LEVELS = 8
MAX_CHILDREN = 256
F32, BF16 = 0, 1
SELECT_GLOBAL, SELECT_PER_LEVEL = 0, 1
SCORING_CONTRACTION, SCORING_COSET_WHT = 0, 1
DEV_BAD_INDEX, DEV_BAD_SIGMA, DEV_SHORT_CODE, DEV_TIMEOUT = 0x1, 0x2, 0x4, 0x8

_STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported configuration", 3: "CUDA error",
           4: "device wait timed out", 5: "out of memory", 6: "device-side error flagged"}


class DPBError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [
        ("d", ctypes.c_int32),
        ("levels", ctypes.c_int32),
        ("m_bits", ctypes.c_int32),
        ("bits", ctypes.c_int32 * MAX_LEVELS),
        ("children", ctypes.c_int32 * MAX_LEVELS),
        ("beam", ctypes.c_int32),
        ("k", ctypes.c_int32),
        ("k_per_level", ctypes.c_int32 * MAX_LEVELS),
        ("select_mode", ctypes.c_int32),
        ("norm_match", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("field_t", ctypes.c_int32),
        ("field_poly", ctypes.c_uint32),
        ("generator_seed", ctypes.c_uint64),
        ("scoring", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
    ]

    def as_dict(self) -> dict:
        L = self.levels
        return {"d": self.d, "levels": L, "m_bits": self.m_bits, "bits": list(self.bits[:L]),
                "children": list(self.children[:L]), "beam": self.beam, "k": self.k,
                "k_per_level": list(self.k_per_level[:L]), "select_mode": self.select_mode,
                "norm_match": self.norm_match, "dtype": self.dtype, "field_t": self.field_t,
                "field_poly": self.field_poly, "generator_seed": self.generator_seed, "scoring": self.scoring}


_lib = None
EXPORTS = ("dpb_plan_create", "dpb_plan_destroy", "dpb_plan_config", "dpb_plan_tables",
           "dpb_code_length", "dpb_workspace_size", "dpb_encode", "dpb_decode", "dpb_backward",
           "dpb_workspace_status", "dpb_status_string", "dpb_last_error", "dpb_encode_noalloc",
           "dpb_stats_accumulate", "dpb_stats_update", "dpb_forward", "dpb_debug_set_wait_limit")


def library_path() -> str:
    return _build.LIB


def load(path: Optional[str] = None):
    """Load libdpb.so (built in-tree by ``build.build()``); raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"DPB CUDA library not built ({path} missing); run "
                           "paper_2607_20652_gb300.build.build() first")
    lib = ctypes.CDLL(path)
    vp, i64, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t
    st = ctypes.c_int
    lib.dpb_plan_create.argtypes = [ctypes.POINTER(Config), vp, ctypes.POINTER(vp)]
    lib.dpb_plan_destroy.argtypes = [vp]
    lib.dpb_plan_config.argtypes = [vp, ctypes.POINTER(Config)]
    lib.dpb_plan_tables.argtypes = [vp, vp, vp]
    lib.dpb_code_length.argtypes = [vp, ctypes.POINTER(ctypes.c_int32)]
    lib.dpb_workspace_size.argtypes = [vp, i64, ctypes.POINTER(sz)]
    lib.dpb_encode.argtypes = [vp, vp, i64, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.dpb_decode.argtypes = [vp, vp, vp, i64, vp, vp, vp, vp, sz, vp]
    lib.dpb_backward.argtypes = [vp, vp, vp, vp, i64, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.dpb_workspace_status.argtypes = [vp, ctypes.c_int, ctypes.POINTER(ctypes.c_int32), vp]
    lib.dpb_encode_noalloc.argtypes = [vp, vp, i64, vp, vp, vp, vp, vp, vp, vp]
    lib.dpb_debug_set_wait_limit.argtypes = [ctypes.c_int32]
    lib.dpb_stats_accumulate.argtypes = [vp, vp, i64, vp, vp, vp, ctypes.c_int32, vp, vp, sz, vp]
    lib.dpb_stats_update.argtypes = [vp, vp, ctypes.c_float, vp, vp, vp]
    lib.dpb_forward.argtypes = [vp, vp, i64, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.dpb_status_string.argtypes = [st]
    lib.dpb_status_string.restype = ctypes.c_char_p
    lib.dpb_last_error.argtypes = []
    lib.dpb_last_error.restype = ctypes.c_char_p
    for name in EXPORTS:
        f = getattr(lib, name)
        if f.restype is None or f.restype is ctypes.c_int:
            f.restype = st
    lib.dpb_status_string.restype = ctypes.c_char_p
    lib.dpb_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(status: int):
    if status != 0:
        msg = load().dpb_last_error().decode(errors="replace")
        raise DPBError(status, msg)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


_DTYPES = {"f32": (F32, torch.float32), "fp32": (F32, torch.float32), "float32": (F32, torch.float32),
           "bf16": (BF16, torch.bfloat16), "bfloat16": (BF16, torch.bfloat16)}


class Plan:
    """A DPB plan (``dpb_plan_create``): resolved config, seed matrix M and
    the generators of every level, resident on the current device."""

    def __init__(self, d: int, levels: int, m_bits: int = 0, children: int | Sequence[int] = 16,
                 beam: int = 8, k: int = 64, dtype: str = "bf16", norm_match: int = 1,
                 seed: int = 0, field_t: int = 0, field_poly: int = 0,
                 bits: Optional[Sequence[int]] = None, generators=None,
                 select_mode: int = SELECT_GLOBAL, k_per_level: Optional[Sequence[int]] = None,
                 scoring: int = SCORING_CONTRACTION):
        lib = load()
        c = Config()
        c.d, c.levels, c.m_bits = d, levels, m_bits
        if bits is not None:
            for l, b in enumerate(bits):
                c.bits[l] = b
        if isinstance(children, int):
            children = [0] + [children] * (levels - 1)
        for l, ch in enumerate(children):
            c.children[l] = ch
        c.beam, c.k = beam, k
        if k_per_level is not None:
            for l, kk in enumerate(k_per_level):
                c.k_per_level[l] = kk
        c.select_mode, c.norm_match = select_mode, norm_match
        c.dtype = _DTYPES[dtype][0]
        c.field_t, c.field_poly, c.generator_seed = field_t, field_poly, seed & (2**64 - 1)
        c.scoring = scoring
        gen_buf = None
        if generators is not None:
            import numpy as np
            g = np.zeros((MAX_LEVELS, MAX_CHILDREN), dtype=np.uint32)
            src = np.asarray(generators, dtype=np.uint32)
            g[: src.shape[0], : min(src.shape[1], MAX_CHILDREN)] = src[:, :MAX_CHILDREN]
            gen_buf = g
        handle = ctypes.c_void_p()
        _check(lib.dpb_plan_create(ctypes.byref(c),
                                   None if gen_buf is None else gen_buf.ctypes.data_as(ctypes.c_void_p),
                                   ctypes.byref(handle)))
        self._h = handle
        self._lib = lib
        out = Config()
        _check(lib.dpb_plan_config(self._h, ctypes.byref(out)))
        self.config = out.as_dict()
        kk = ctypes.c_int32()
        _check(lib.dpb_code_length(self._h, ctypes.byref(kk)))
        self.code_len = kk.value
        self.n_features = 1 << self.config["bits"][self.config["levels"] - 1]  # 2^N
        self.d = d
        self.torch_dtype = _DTYPES[dtype][1]

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            try:
                self._lib.dpb_plan_destroy(h)
            except Exception:
                pass
            self._h = None

    @property
    def handle(self):
        return self._h

    def tables(self):
        """(M [d] uint32, G [MAX_LEVELS, MAX_CHILDREN] uint32) as numpy arrays."""
        import numpy as np
        M = np.zeros(self.d, dtype=np.uint32)
        G = np.zeros((MAX_LEVELS, MAX_CHILDREN), dtype=np.uint32)
        _check(self._lib.dpb_plan_tables(self._h, M.ctypes.data_as(ctypes.c_void_p),
                                         G.ctypes.data_as(ctypes.c_void_p)))
        return M, G

    def workspace_size(self, T: int) -> int:
        n = ctypes.c_size_t()
        _check(self._lib.dpb_workspace_size(self._h, T, ctypes.byref(n)))
        return n.value

    def workspace(self, T: int, device=None) -> torch.Tensor:
        """A zero-filled workspace tensor (uint8) for up to T tokens."""
        n = self.workspace_size(T)
        return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")

    def _stream_workspace(self, T: int, device, stream) -> torch.Tensor:
        """The workspace of calls made without one: one per (device, stream),
        kept with the plan (calls on one stream run in order, so they may
        share it; its status bits accumulate until read and cleared)."""
        dev = torch.device(device)
        s = stream if stream is not None else torch.cuda.current_stream(dev)
        key = (dev.index if dev.index is not None else torch.cuda.current_device(), s.cuda_stream)
        cache = self.__dict__.setdefault("_ws_cache", {})
        ws = cache.get(key)
        if ws is None or ws.numel() < self.workspace_size(T):
            # allocated and zeroed on the stream the calls use, so the first
            # kernel cannot start before the fill ends
            with torch.cuda.stream(s):
                ws = cache[key] = self.workspace(T, dev)
        return ws

    def status(self, device=None, stream=None, clear: bool = True) -> int:
        """The DPB_DEV_* bits that calls made without a workspace left on
        ``stream`` (synchronises it); cleared by default."""
        dev = torch.device(device or "cuda")
        s = stream if stream is not None else torch.cuda.current_stream(dev)
        key = (dev.index if dev.index is not None else torch.cuda.current_device(), s.cuda_stream)
        ws = self.__dict__.get("_ws_cache", {}).get(key)
        return 0 if ws is None else workspace_status(ws, clear=clear, stream=s)


def _rows(t: torch.Tensor, plan: Plan, name: str):
    if t.dtype != plan.torch_dtype or not t.is_cuda or not t.is_contiguous() or t.dim() != 2 \
            or t.shape[1] != plan.d:
        raise ValueError(f"{name} must be a contiguous CUDA {plan.torch_dtype} tensor of shape [T, {plan.d}]")


def encode(plan: Plan, x: torch.Tensor, mu=None, sigma=None, idx=None, val=None, xnorm=None,
           workspace=None, stream=None, want_xnorm: bool = True):
    """dpb_encode. Returns (idx int32 [T,k], val fp32 [T,k], xnorm fp32 [T] or None)."""
    _rows(x, plan, "x")
    T, k = x.shape[0], plan.code_len
    dev = x.device
    idx = torch.empty((T, k), dtype=torch.int32, device=dev) if idx is None else idx
    val = torch.empty((T, k), dtype=torch.float32, device=dev) if val is None else val
    if xnorm is None and want_xnorm:
        xnorm = torch.empty((T,), dtype=torch.float32, device=dev)
    ws = plan._stream_workspace(T, dev, stream) if workspace is None else workspace
    _check(plan._lib.dpb_encode(plan.handle, _ptr(x), T, _ptr(mu), _ptr(sigma), _ptr(idx), _ptr(val),
                                _ptr(xnorm), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)))
    return idx, val, xnorm


def decode(plan: Plan, idx: torch.Tensor, val: torch.Tensor, xnorm=None, y=None, workspace=None,
           stream=None, r_out: Optional[torch.Tensor] = None):
    """dpb_decode. Returns y [T, d] in the plan's dtype; with ``r_out`` (fp32
    [T, d]) also keeps r there for dpb_backward."""
    T = idx.shape[0]
    if idx.dtype != torch.int32 or val.dtype != torch.float32 or idx.shape != val.shape \
            or not idx.is_contiguous() or not val.is_contiguous():
        raise ValueError("idx must be int32 and val float32, contiguous, same shape [T, k]")
    if idx.shape[1] != plan.code_len:
        raise ValueError(f"code length {idx.shape[1]} != plan's {plan.code_len}")
    y = torch.empty((T, plan.d), dtype=plan.torch_dtype, device=idx.device) if y is None else y
    ws = plan._stream_workspace(T, idx.device, stream) if workspace is None else workspace
    if r_out is not None and (r_out.dtype != torch.float32 or not r_out.is_contiguous()
                              or tuple(r_out.shape) != (T, plan.d)):
        raise ValueError(f"r_out must be a contiguous float32 tensor of shape [T, {plan.d}]")
    _check(plan._lib.dpb_decode(plan.handle, _ptr(idx), _ptr(val), T, _ptr(xnorm), _ptr(y), _ptr(r_out),
                                _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)))
    return y


def forward(plan: Plan, x: torch.Tensor, mu=None, sigma=None, workspace=None, stream=None,
            r_out: Optional[torch.Tensor] = None):
    """dpb_forward (encode then decode). Returns (idx, val, xnorm, y)."""
    _rows(x, plan, "x")
    T, k, dev = x.shape[0], plan.code_len, x.device
    idx = torch.empty((T, k), dtype=torch.int32, device=dev)
    val = torch.empty((T, k), dtype=torch.float32, device=dev)
    xnorm = torch.empty((T,), dtype=torch.float32, device=dev)
    y = torch.empty_like(x)
    if r_out is not None and (r_out.dtype != torch.float32 or not r_out.is_contiguous()
                              or tuple(r_out.shape) != (T, plan.d)):
        raise ValueError(f"r_out must be a contiguous float32 tensor of shape [T, {plan.d}]")
    ws = plan._stream_workspace(T, dev, stream) if workspace is None else workspace
    _check(plan._lib.dpb_forward(plan.handle, _ptr(x), T, _ptr(mu), _ptr(sigma), _ptr(idx), _ptr(val),
                                 _ptr(xnorm), _ptr(y), _ptr(r_out), _ptr(ws), ws.numel() * ws.element_size(),
                                 _stream(stream)))
    return idx, val, xnorm, y


def backward(plan: Plan, x: torch.Tensor, idx: torch.Tensor, val: torch.Tensor, grad_y: torch.Tensor,
             sigma=None, grad_x=None, grad_val=None, workspace=None, stream=None,
             r: Optional[torch.Tensor] = None):
    """dpb_backward. Returns (grad_x [T, d] plan dtype, grad_val fp32 [T, k]);
    ``r`` is the r_out of the decode of this code (optional)."""
    _rows(x, plan, "x")
    _rows(grad_y, plan, "grad_y")
    T = x.shape[0]
    grad_x = torch.empty_like(x) if grad_x is None else grad_x
    grad_val = torch.empty(idx.shape, dtype=torch.float32, device=x.device) if grad_val is None else grad_val
    ws = plan._stream_workspace(T, x.device, stream) if workspace is None else workspace
    if r is not None and (r.dtype != torch.float32 or not r.is_contiguous() or tuple(r.shape) != (T, plan.d)):
        raise ValueError(f"r must be a contiguous float32 tensor of shape [T, {plan.d}]")
    _check(plan._lib.dpb_backward(plan.handle, _ptr(x), _ptr(idx), _ptr(val), T, _ptr(sigma), _ptr(r),
                                  _ptr(grad_y), _ptr(grad_x), _ptr(grad_val), _ptr(ws),
                                  ws.numel() * ws.element_size(), _stream(stream)))
    return grad_x, grad_val


def stats_buffer(plan: Plan, device=None) -> torch.Tensor:
    """A zeroed moment-sum buffer fp64 [3, 2^N] (count, sum s, sum s^2)."""
    return torch.zeros((3, plan.n_features), dtype=torch.float64, device=device or "cuda")


def stats_accumulate(plan: Plan, x: torch.Tensor, sample: torch.Tensor, acc: torch.Tensor, mu=None,
                     sigma=None, workspace=None, stream=None):
    """dpb_stats_accumulate: adds the batch's moment sums to ``acc`` (level 0
    over every row of x, levels >= 1 over the rows in ``sample``)."""
    _rows(x, plan, "x")
    if sample.dtype != torch.int32 or not sample.is_contiguous() or sample.dim() != 1:
        raise ValueError("sample must be a contiguous 1-D int32 tensor of row numbers")
    if acc.dtype != torch.float64 or not acc.is_contiguous() or acc.numel() != 3 * plan.n_features:
        raise ValueError("acc must be a contiguous float64 tensor of 3 * 2^N entries (stats_buffer)")
    T = x.shape[0]
    ws = plan._stream_workspace(T, x.device, stream) if workspace is None else workspace
    _check(plan._lib.dpb_stats_accumulate(plan.handle, _ptr(x), T, _ptr(mu), _ptr(sigma),
                                          _ptr(sample) if sample.numel() else None, sample.numel(),
                                          _ptr(acc), _ptr(ws), ws.numel() * ws.element_size(),
                                          _stream(stream)))
    return acc


def stats_update(plan: Plan, acc: torch.Tensor, alpha: float, mu: torch.Tensor, sigma: torch.Tensor,
                 stream=None):
    """dpb_stats_update: one EMA step of (mu, sigma) in place; zeroes ``acc``."""
    if acc.dtype != torch.float64 or not acc.is_contiguous():
        raise ValueError("acc must be a contiguous float64 tensor")
    for name, t in (("mu", mu), ("sigma", sigma)):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.numel() * 3 != acc.numel():
            raise ValueError(f"{name} must be a contiguous float32 tensor of 2^N entries")
    _check(plan._lib.dpb_stats_update(plan.handle, _ptr(acc), float(alpha), _ptr(mu), _ptr(sigma),
                                      _stream(stream)))
    return mu, sigma


def ema_step(accumulate, update, acc, group=None):
    """One standardisation step under data parallelism: each rank adds its
    own moment sums (``accumulate(acc)``), the sums are added up across the
    ranks of ``group`` (one all-reduce; skipped when torch.distributed is not
    initialised or the group has one rank), and every rank makes the same EMA
    step (``update(acc)``), so the tables stay identical everywhere."""
    accumulate(acc)
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(acc, op=dist.ReduceOp.SUM, group=group)
    update(acc)


def sample_rows(T: int, n: int, generator: Optional[torch.Generator] = None, device=None) -> torch.Tensor:
    """n distinct row numbers of [0, T) (all of them when T <= n), drawn
    uniformly by ``generator``: the sub-sample of levels >= 1."""
    n = min(n, T)
    rows = torch.randperm(T, generator=generator)[:n].to(torch.int32)
    return rows.to(device) if device is not None else rows


def stats_step(plan: Plan, x: torch.Tensor, mu: torch.Tensor, sigma: torch.Tensor, alpha: float,
               sample: torch.Tensor, acc: Optional[torch.Tensor] = None, workspace=None, stream=None,
               group=None):
    """The whole EMA update of one batch (§2.2 "Score Standardization"):
    moment sums on this rank, summed across ``group``, then the EMA step of
    mu and sigma in place."""
    acc = stats_buffer(plan, x.device) if acc is None else acc
    ema_step(lambda a: stats_accumulate(plan, x, sample, a, mu=mu, sigma=sigma, workspace=workspace,
                                        stream=stream),
             lambda a: stats_update(plan, a, alpha, mu, sigma, stream=stream), acc, group)
    return mu, sigma


def set_wait_limit(tries: int = -1):
    """dpb_debug_set_wait_limit: bound of the per-level encoder's main-loop
    mbarrier waits for the launches that follow (-1 restores the default)."""
    _check(load().dpb_debug_set_wait_limit(int(tries)))


def workspace_status(workspace: torch.Tensor, clear: bool = False, stream=None) -> int:
    """dpb_workspace_status: the sticky device status bits (0 = none)."""
    v = ctypes.c_int32()
    load().dpb_workspace_status(_ptr(workspace), int(clear), ctypes.byref(v), _stream(stream))
    return v.value
