"""Thin Python binding of the VarRate C ABI (include/varrate.h).

Argument marshalling only: every step of the hot path runs in the CUDA library ``libvarrate.so``.
Functions keep the C names and argument order; tensor arguments are torch tensors (device memory
owned by the caller) or ``None`` for NULL, and ``stream`` defaults to torch's current stream.
Importing this module does not load the library; the first call does, and it raises if the
library has not been built (there is no CPU fallback).

Typical use (one encode of a prompt's cache, then one decode call per layer and step)::

    cfg = make_config(n_layers, n_kv_heads, group, n_ctx, batch=B, budget_frac=0.2, r_min=16,
                      window=32, dtype=BF16)
    packed = PackedCache.allocate(cfg, "cuda")            # static upper bound: no host sync later
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    check(varrate_encode(cfg, q_win, k, v, basis_k, basis_v, None, packed, None, status,
                         workspace(cfg, CALL_ENCODE)), "varrate_encode")
    ws = workspace(cfg, CALL_DECODE)                      # zero-filled; reusable by every decode call
    check(varrate_decode_attn(cfg, packed, basis_k, basis_v, q, layer, None, None, 0, out, status,
                              ws), "varrate_decode_attn")
    # after a synchronise: status.item() is OK (0), FLOOR_BINDS (1) or a negative error

Shapes: q_win [B][L][w][H][d], k and v [B][L][G][N][d], bases [L][G][d][d] (row j = basis vector
j), q and out [B][H][d]; every tensor contiguous on the GPU and 16-byte aligned.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libvarrate.so")

OK, FLOOR_BINDS = 0, 1
ERR_ARG, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT, ERR_UNSUPPORTED, ERR_CORRUPT = -1, -2, -3, -4, -5, -6
F32, BF16 = 0, 1
SALIENCE, UNIFORM = 0, 1
CALL_SALIENCE, CALL_PACK, CALL_ENCODE, CALL_DECODE, CALL_DECODE_WINDOW, CALL_DECODE_Q = 0, 1, 2, 3, 4, 5

_c_void_p = ctypes.c_void_p


class varrate_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("group", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("n_ctx", ctypes.c_int64), ("batch", ctypes.c_int32), ("r_min", ctypes.c_int32),
                ("budget_frac", ctypes.c_double), ("window", ctypes.c_int32),
                ("pool_len", ctypes.c_int32), ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32)]


class varrate_packed(ctypes.Structure):
    _fields_ = [("coef", _c_void_p), ("bucket_count", _c_void_p), ("bucket_base", _c_void_p),
                ("perm", _c_void_p), ("pos", _c_void_p), ("ranks", _c_void_p),
                ("cap_elems", ctypes.c_int64)]


class varrate_qpacked(ctypes.Structure):
    _fields_ = [("data", _c_void_p), ("qbase", _c_void_p), ("bucket_count", _c_void_p),
                ("bits", ctypes.c_int32), ("qcap_bytes", ctypes.c_int64)]


_lib = None

_SIGS = {
    "varrate_version": (ctypes.c_int32, []),
    "varrate_status_string": (ctypes.c_char_p, [ctypes.c_int32]),
    "varrate_check_config": (ctypes.c_int32, [ctypes.POINTER(varrate_config)]),
    "varrate_coded_budget": (ctypes.c_int64, [ctypes.POINTER(varrate_config)]),
    "varrate_packed_cap_elems": (ctypes.c_int64, [ctypes.POINTER(varrate_config)]),
    "varrate_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(varrate_config), ctypes.c_int32]),
    "varrate_salience": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                          _c_void_p, _c_void_p, ctypes.c_size_t, _c_void_p]),
    "varrate_allocate": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                          _c_void_p, _c_void_p, _c_void_p]),
    "varrate_pack": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                      _c_void_p, _c_void_p, ctypes.POINTER(varrate_packed),
                                      _c_void_p, _c_void_p, ctypes.c_size_t, _c_void_p]),
    "varrate_encode": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                        _c_void_p, _c_void_p, _c_void_p, _c_void_p,
                                        ctypes.POINTER(varrate_packed), _c_void_p, _c_void_p,
                                        _c_void_p, ctypes.c_size_t, _c_void_p]),
    "varrate_decode_attn": (ctypes.c_int32, [ctypes.POINTER(varrate_config),
                                             ctypes.POINTER(varrate_packed), _c_void_p, _c_void_p,
                                             _c_void_p, ctypes.c_int32, _c_void_p, _c_void_p,
                                             ctypes.c_int32, _c_void_p, _c_void_p, _c_void_p,
                                             ctypes.c_size_t, _c_void_p]),
    "varrate_decode_window": (ctypes.c_int32, [ctypes.POINTER(varrate_config),
                                               ctypes.POINTER(varrate_packed), _c_void_p, _c_void_p,
                                               _c_void_p, ctypes.c_int32, ctypes.c_int32, _c_void_p,
                                               _c_void_p, ctypes.c_int32, _c_void_p, _c_void_p,
                                               _c_void_p, ctypes.c_size_t, _c_void_p]),
    "varrate_qpacked_cap_bytes": (ctypes.c_int64, [ctypes.POINTER(varrate_config), ctypes.c_int32]),
    "varrate_quantize": (ctypes.c_int32, [ctypes.POINTER(varrate_config), ctypes.POINTER(varrate_packed),
                                          ctypes.POINTER(varrate_qpacked), _c_void_p, _c_void_p]),
    "varrate_decode_attn_q": (ctypes.c_int32, [ctypes.POINTER(varrate_config),
                                               ctypes.POINTER(varrate_qpacked), _c_void_p, _c_void_p,
                                               _c_void_p, ctypes.c_int32, _c_void_p, _c_void_p,
                                               ctypes.c_int32, _c_void_p, _c_void_p, _c_void_p,
                                               ctypes.c_size_t, _c_void_p]),
    "varrate_decode_attn_noalloc": (ctypes.c_int32, [ctypes.POINTER(varrate_config),
                                                     ctypes.POINTER(varrate_packed), _c_void_p,
                                                     _c_void_p, _c_void_p, ctypes.c_int32,
                                                     _c_void_p, _c_void_p, ctypes.c_int32,
                                                     _c_void_p, _c_void_p, _c_void_p]),
    "varrate_selftest_wait_timeout": (ctypes.c_int32, [_c_void_p, ctypes.c_uint32, _c_void_p]),
    "varrate_anchor_search_ws_bytes": (ctypes.c_size_t, [ctypes.POINTER(varrate_config), ctypes.c_int32]),
    "varrate_anchor_search": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                               ctypes.c_int32, ctypes.c_int32, _c_void_p, _c_void_p,
                                               _c_void_p, _c_void_p, ctypes.c_size_t, _c_void_p]),
    "varrate_anchor_residual": (ctypes.c_int32, [ctypes.POINTER(varrate_config), _c_void_p, _c_void_p,
                                                 ctypes.c_int32, ctypes.c_int32, _c_void_p, _c_void_p,
                                                 _c_void_p, _c_void_p]),
}

EXPORTED = tuple(_SIGS)


def lib() -> ctypes.CDLL:
    """The loaded CUDA library (loaded on first use; raises if it was never built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2607_15498_gb300.build` (no CPU fallback exists)")
        l = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


class VarrateError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {status_string(status)} ({status})")
        self.status = status


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _nbytes(t) -> int:
    return 0 if t is None else t.numel() * t.element_size()


def check(status: int, what: str = "varrate") -> int:
    """Raise VarrateError on a negative status; return it otherwise (OK or a warning)."""
    if status < 0:
        raise VarrateError(status, what)
    return status


# ------------------------------------------------------------------ plain C functions

def varrate_version() -> int:
    return lib().varrate_version()


def status_string(status: int) -> str:
    return lib().varrate_status_string(status).decode()


varrate_status_string = status_string


def varrate_check_config(cfg: varrate_config) -> int:
    return lib().varrate_check_config(ctypes.byref(cfg))


def varrate_coded_budget(cfg: varrate_config) -> int:
    return lib().varrate_coded_budget(ctypes.byref(cfg))


def varrate_packed_cap_elems(cfg: varrate_config) -> int:
    return lib().varrate_packed_cap_elems(ctypes.byref(cfg))


def varrate_workspace_bytes(cfg: varrate_config, which_call: int) -> int:
    return lib().varrate_workspace_bytes(ctypes.byref(cfg), which_call)


def varrate_salience(cfg, q_win, k, sal_out, ws, stream=None) -> int:
    return lib().varrate_salience(ctypes.byref(cfg), _ptr(q_win), _ptr(k), _ptr(sal_out), _ptr(ws),
                                  _nbytes(ws), _stream(stream))


def varrate_allocate(cfg, sal, ranks, realized_sum, dev_status, stream=None) -> int:
    return lib().varrate_allocate(ctypes.byref(cfg), _ptr(sal), _ptr(ranks), _ptr(realized_sum),
                                  _ptr(dev_status), _stream(stream))


def varrate_pack(cfg, k, v, basis_k, basis_v, packed, dev_status, ws=None, stream=None) -> int:
    return lib().varrate_pack(ctypes.byref(cfg), _ptr(k), _ptr(v), _ptr(basis_k), _ptr(basis_v),
                              ctypes.byref(packed.c), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                              _stream(stream))


def varrate_encode(cfg, q_win, k, v, basis_k, basis_v, sal_out, packed, realized_sum, dev_status,
                   ws, stream=None) -> int:
    return lib().varrate_encode(ctypes.byref(cfg), _ptr(q_win), _ptr(k), _ptr(v), _ptr(basis_k),
                                _ptr(basis_v), _ptr(sal_out), ctypes.byref(packed.c),
                                _ptr(realized_sum), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                                _stream(stream))


def varrate_decode_attn(cfg, packed, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out,
                        dev_status, ws, stream=None) -> int:
    return lib().varrate_decode_attn(ctypes.byref(cfg), ctypes.byref(packed.c), _ptr(basis_k),
                                     _ptr(basis_v), _ptr(q), layer, _ptr(tail_k), _ptr(tail_v),
                                     n_tail, _ptr(out), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                                     _stream(stream))


def varrate_decode_attn_noalloc(cfg, packed, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail,
                                out, dev_status, stream=None) -> int:
    return lib().varrate_decode_attn_noalloc(ctypes.byref(cfg), ctypes.byref(packed.c),
                                             _ptr(basis_k), _ptr(basis_v), _ptr(q), layer,
                                             _ptr(tail_k), _ptr(tail_v), n_tail, _ptr(out),
                                             _ptr(dev_status), _stream(stream))


def varrate_selftest_wait_timeout(dev_status, polls, stream=None) -> int:
    return lib().varrate_selftest_wait_timeout(_ptr(dev_status), polls, _stream(stream))


def varrate_anchor_search_ws_bytes(cfg: varrate_config, stride: int) -> int:
    return lib().varrate_anchor_search_ws_bytes(ctypes.byref(cfg), stride)


def varrate_anchor_search(cfg, k, v, stride, c, idx_out, dist_out, dev_status, ws, stream=None) -> int:
    return lib().varrate_anchor_search(ctypes.byref(cfg), _ptr(k), _ptr(v), stride, c, _ptr(idx_out),
                                       _ptr(dist_out), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                                       _stream(stream))


def varrate_anchor_residual(cfg, k, v, stride, c, idx, e_out, dev_status, stream=None) -> int:
    return lib().varrate_anchor_residual(ctypes.byref(cfg), _ptr(k), _ptr(v), stride, c, _ptr(idx),
                                         _ptr(e_out), _ptr(dev_status), _stream(stream))


def varrate_decode_window(cfg, packed, basis_k, basis_v, q, n_q, layer, tail_k, tail_v, n_tail, out,
                          dev_status, ws, stream=None) -> int:
    return lib().varrate_decode_window(ctypes.byref(cfg), ctypes.byref(packed.c), _ptr(basis_k),
                                       _ptr(basis_v), _ptr(q), n_q, layer, _ptr(tail_k), _ptr(tail_v),
                                       n_tail, _ptr(out), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                                       _stream(stream))


def varrate_qpacked_cap_bytes(cfg: varrate_config, bits: int) -> int:
    return lib().varrate_qpacked_cap_bytes(ctypes.byref(cfg), bits)


def varrate_quantize(cfg, packed, qpacked, dev_status, stream=None) -> int:
    return lib().varrate_quantize(ctypes.byref(cfg), ctypes.byref(packed.c), ctypes.byref(qpacked.c),
                                  _ptr(dev_status), _stream(stream))


def varrate_decode_attn_q(cfg, qpacked, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out,
                          dev_status, ws, stream=None) -> int:
    return lib().varrate_decode_attn_q(ctypes.byref(cfg), ctypes.byref(qpacked.c), _ptr(basis_k),
                                       _ptr(basis_v), _ptr(q), layer, _ptr(tail_k), _ptr(tail_v),
                                       n_tail, _ptr(out), _ptr(dev_status), _ptr(ws), _nbytes(ws),
                                       _stream(stream))


# ------------------------------------------------------------- device-memory plumbing

def make_config(n_layers, n_kv_heads, group, n_ctx, batch=1, budget_frac=0.2, r_min=16, window=32,
                pool_len=5, dtype=BF16, mode=SALIENCE, head_dim=128) -> varrate_config:
    return varrate_config(n_layers=n_layers, n_kv_heads=n_kv_heads, group=group, head_dim=head_dim,
                          n_ctx=n_ctx, batch=batch, r_min=r_min, budget_frac=budget_frac,
                          window=window, pool_len=pool_len, dtype=dtype, mode=mode)


def torch_dtype(cfg: varrate_config) -> torch.dtype:
    return torch.bfloat16 if cfg.dtype == BF16 else torch.float32


@dataclass
class PackedCache:
    """Torch-allocated device buffers of a packed cache plus the C struct pointing at them."""
    coef: torch.Tensor
    bucket_count: torch.Tensor
    bucket_base: torch.Tensor
    perm: torch.Tensor
    pos: torch.Tensor
    ranks: torch.Tensor
    cap_elems: int
    c: varrate_packed

    @staticmethod
    def allocate(cfg: varrate_config, device="cuda") -> "PackedCache":
        cap = varrate_packed_cap_elems(cfg)
        if cap < 0:
            raise VarrateError(ERR_ARG, "varrate_packed_cap_elems")
        B, L, G, N, d = cfg.batch, cfg.n_layers, cfg.n_kv_heads, cfg.n_ctx, cfg.head_dim
        coef = torch.empty((B, L, G, 2, cap), dtype=torch_dtype(cfg), device=device)
        cnt = torch.zeros((B, L, d + 1), dtype=torch.int32, device=device)
        base = torch.zeros((B, L, d + 2), dtype=torch.int64, device=device)
        perm = torch.empty((B, L, N), dtype=torch.int32, device=device)
        pos = torch.empty((B, L, N), dtype=torch.int32, device=device)
        ranks = torch.empty((B, L, N), dtype=torch.uint8, device=device)
        c = varrate_packed(coef.data_ptr(), cnt.data_ptr(), base.data_ptr(), perm.data_ptr(),
                           pos.data_ptr(), ranks.data_ptr(), cap)
        return PackedCache(coef, cnt, base, perm, pos, ranks, cap, c)

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in
                   (self.coef, self.bucket_count, self.bucket_base, self.perm, self.pos, self.ranks))


@dataclass
class QPackedCache:
    """Torch-allocated buffers of a quantized cache (codes and group parameters, bucket byte
    offsets) plus the C struct; the bucket counts are those of the source PackedCache."""
    data: torch.Tensor
    qbase: torch.Tensor
    source: PackedCache
    bits: int
    qcap_bytes: int
    c: varrate_qpacked

    @staticmethod
    def allocate(cfg: varrate_config, source: PackedCache, bits: int, device="cuda") -> "QPackedCache":
        cap = varrate_qpacked_cap_bytes(cfg, bits)
        if cap < 0:
            raise VarrateError(ERR_ARG, "varrate_qpacked_cap_bytes")
        B, L, G, d = cfg.batch, cfg.n_layers, cfg.n_kv_heads, cfg.head_dim
        data = torch.zeros((B, L, G, 2, cap), dtype=torch.uint8, device=device)
        qbase = torch.zeros((B, L, d + 2), dtype=torch.int64, device=device)
        c = varrate_qpacked(data.data_ptr(), qbase.data_ptr(), source.bucket_count.data_ptr(), bits, cap)
        return QPackedCache(data, qbase, source, bits, cap, c)


def workspace(cfg: varrate_config, which_call: int, device="cuda") -> torch.Tensor:
    """Device scratch for one kind of call, zero-filled (the decode workspace's header must be zero
    before the first decode call that uses it; later calls keep it consistent themselves)."""
    n = varrate_workspace_bytes(cfg, which_call)
    return torch.zeros(max(n, 256), dtype=torch.uint8, device=device)
