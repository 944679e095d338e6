"""Python binding of libsonic (include/sonic.h): argument marshalling only.

Every step of the path runs in the CUDA library; this module loads
``_lib/libsonic.so`` with ctypes, mirrors the argument structs, and offers the
three entry points under their C names taking torch tensors on the GPU:

* :func:`sonic_compact_kv`   -- retention (Sec. 3.2 body removal, App. C),
* :func:`sonic_attn_prefill` -- attention under the Sec. 3.2 mask,
* :func:`sonic_attn_decode`  -- one GQA decode step over the retained cache.

The wrappers only fill the C structs, allocate the caller-owned workspace as a
torch tensor, pass the current CUDA stream and raise :class:`SonicError` on a
non-OK status.  Importing this module fails loudly if the library is missing;
there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import _build

ROLE_SYS, ROLE_BODY, ROLE_NEXUS, ROLE_CURR = 0, 1, 2, 3
NEXUS_FULL, NEXUS_CAUSAL_SEGMENTS = 0, 1
KEYS_AS_GIVEN, KEYS_RETAINED_FIRST = 0, 1

STATUS = {0: "SONIC_OK", 1: "SONIC_ERR_INVALID_ARGUMENT", 2: "SONIC_ERR_UNSUPPORTED",
          3: "SONIC_ERR_WORKSPACE", 4: "SONIC_ERR_CAPACITY", 5: "SONIC_ERR_DEVICE_TIMEOUT",
          6: "SONIC_ERR_CUDA", 7: "SONIC_ERR_LAYOUT"}

_P = ctypes.c_void_p
_i32, _i64, _f32, _sz = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t


class SonicError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {STATUS.get(code, code)}")
        self.code = code


class sonic_compact_args(ctypes.Structure):
    _fields_ = [("batch", _i32), ("n_layers", _i32), ("k_start", _P), ("k_len", _P),
                ("reserve", _P), ("row_bytes", _i64), ("in_layer_bytes", _i64),
                ("out_layer_bytes", _i64), ("out_capacity_rows", _i32), ("ret_len", _P),
                ("src_idx", _P), ("out_role", _P), ("out_seg", _P), ("status", _P),
                ("workspace", _P), ("workspace_bytes", _sz), ("total_rows", _i32)]


class sonic_prefill_args(ctypes.Structure):
    _fields_ = [("batch", _i32), ("n_layers", _i32), ("n_heads_q", _i32), ("n_heads_kv", _i32),
                ("head_dim", _i32), ("k_start", _P), ("k_len", _P), ("q_start", _P),
                ("q_len", _P), ("max_q_len", _i32), ("max_k_len", _i32), ("total_q_rows", _i32),
                ("total_k_rows", _i32), ("q_layer_stride", _i64), ("kv_layer_stride", _i64),
                ("o_layer_stride", _i64), ("softmax_scale", _f32), ("nexus_vis", _i32),
                ("lse", _P), ("status", _P), ("workspace", _P), ("workspace_bytes", _sz),
                ("key_order", _i32), ("nexus_mass", _P)]


class sonic_decode_args(ctypes.Structure):
    _fields_ = [("batch", _i32), ("n_layers", _i32), ("n_heads_q", _i32), ("n_heads_kv", _i32),
                ("head_dim", _i32), ("kv_start", _P), ("max_len", _i32), ("total_kv_rows", _i32),
                ("q_layer_stride", _i64), ("kv_layer_stride", _i64), ("o_layer_stride", _i64),
                ("softmax_scale", _f32), ("chunk_len", _i32), ("lse", _P), ("status", _P),
                ("workspace", _P), ("workspace_bytes", _sz), ("role", _P), ("nexus_mass", _P)]


class sonic_out_part(ctypes.Structure):
    _fields_ = [("base", _P), ("row_stride", _i64), ("cols", _i32), ("scatter", _i32),
                ("rows", _i64)]


class sonic_routed_linear_args(ctypes.Structure):
    _fields_ = [("n_rows", _i32), ("d_in", _i32), ("d_out", _i32), ("x_row_stride", _i64),
                ("dst_row", _P), ("n_parts", _i32), ("parts", sonic_out_part * 4),
                ("status", _P), ("workspace", _P), ("workspace_bytes", _sz)]


# Exported C symbols, with their ctypes signatures.
SIGNATURES = {
    "sonic_compact_kv": (_i32, [_P, _P, _P, _P, _P, _P, _P,
                                ctypes.POINTER(sonic_compact_args), _P]),
    "sonic_compact_workspace_size": (_sz, [ctypes.POINTER(sonic_compact_args)]),
    "sonic_attn_prefill": (_i32, [_P, _P, _P, _P, _P, _P,
                                  ctypes.POINTER(sonic_prefill_args), _P]),
    "sonic_prefill_workspace_size": (_sz, [ctypes.POINTER(sonic_prefill_args)]),
    "sonic_attn_prefill_static": (_i32, [_P, _P, _P, _P, _P, _P,
                                         ctypes.POINTER(sonic_prefill_args), _P]),
    "sonic_attn_decode": (_i32, [_P, _P, _P, _P, _P,
                                 ctypes.POINTER(sonic_decode_args), _P]),
    "sonic_decode_workspace_size": (_sz, [ctypes.POINTER(sonic_decode_args)]),
    "sonic_routed_linear": (_i32, [_P, _P, _P, _P, ctypes.POINTER(sonic_routed_linear_args),
                                   _P]),
    "sonic_routed_linear_workspace_size": (_sz, [ctypes.POINTER(sonic_routed_linear_args)]),
    "sonic_read_status": (_i32, [_P, _P]),
    "sonic_status_string": (ctypes.c_char_p, [_i32]),
    "sonic_abi_version": (_i32, []),
}

_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libsonic.so (building it first if asked and it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise ImportError(f"libsonic.so not built ({path}); run __graft_entry__.build()")
        _build.build()
    _lib = open_library(path)
    return _lib


def open_library(path: str) -> ctypes.CDLL:
    """A libsonic build at `path` with the C signatures applied (entry points
    the build lacks are skipped)."""
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        if not hasattr(lib, name):
            continue
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _check(code: int, where: str):
    if code != 0:
        raise SonicError(code, where)


def _workspace(nbytes: int, device, ws: Optional[torch.Tensor]):
    if nbytes == 0:
        return None
    if ws is not None and ws.numel() * ws.element_size() >= nbytes:
        return ws
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def read_status(status: torch.Tensor, stream=None) -> int:
    return int(load().sonic_read_status(_ptr(status), _stream(stream)))


# ---------------------------------------------------------------------------
# Entry points
# ---------------------------------------------------------------------------

def sonic_compact_kv(K: torch.Tensor, V: torch.Tensor, seg_id: Optional[torch.Tensor],
                     role: torch.Tensor, out_K: torch.Tensor, out_V: torch.Tensor,
                     offsets: torch.Tensor, *, k_start: torch.Tensor, k_len: torch.Tensor,
                     reserve: Optional[torch.Tensor] = None, ret_len=None, src_idx=None,
                     out_role=None, out_seg=None, status=None, workspace=None, stream=None):
    """Retention rule over all layers.  K, V: [n_layers, T, ...] (any dtype, rows
    of row_bytes contiguous); out_K, out_V: [n_layers, capacity, ...]."""
    lib = load()
    nl = K.shape[0]
    T = K.shape[1]
    row_bytes = K[0, 0].numel() * K.element_size() if T > 0 else (
        K.numel() // max(nl, 1) * K.element_size())
    a = sonic_compact_args()
    a.batch = k_start.numel()
    a.n_layers = nl
    a.k_start, a.k_len, a.reserve = _ptr(k_start), _ptr(k_len), _ptr(reserve)
    a.row_bytes = row_bytes
    a.in_layer_bytes = K.stride(0) * K.element_size()
    a.out_layer_bytes = out_K.stride(0) * out_K.element_size()
    a.out_capacity_rows = out_K.shape[1]
    a.ret_len, a.src_idx = _ptr(ret_len), _ptr(src_idx)
    a.out_role, a.out_seg, a.status = _ptr(out_role), _ptr(out_seg), _ptr(status)
    a.total_rows = min([T, role.numel()] + ([seg_id.numel()] if seg_id is not None else []))
    need = lib.sonic_compact_workspace_size(ctypes.byref(a))
    ws = _workspace(need, K.device, workspace)
    a.workspace, a.workspace_bytes = _ptr(ws), need
    _check(lib.sonic_compact_kv(_ptr(K), _ptr(V), _ptr(seg_id), _ptr(role), _ptr(out_K),
                                _ptr(out_V), _ptr(offsets), ctypes.byref(a), _stream(stream)),
           "sonic_compact_kv")
    return ws


def sonic_attn_prefill(Q: torch.Tensor, K: torch.Tensor, V: torch.Tensor, seg_id: torch.Tensor,
                       role: torch.Tensor, O: torch.Tensor, *, k_start, k_len, q_start, q_len,
                       max_q_len: int, max_k_len: int, softmax_scale: float = 0.0,
                       nexus_vis: int = NEXUS_FULL, lse=None, status=None, workspace=None,
                       key_order: int = KEYS_AS_GIVEN, nexus_mass=None, stream=None):
    """Masked prefill.  Q, O: [n_layers, Tq, Hq, D] bf16; K, V: [n_layers, Tk, Hkv, D] bf16;
    lse, nexus_mass: [n_layers, Tq, Hq] float32 or None."""
    lib = load()
    nl, tq, hq, d = Q.shape
    _, tk, hkv, _ = K.shape
    a = sonic_prefill_args()
    a.batch = k_start.numel()
    a.n_layers, a.n_heads_q, a.n_heads_kv, a.head_dim = nl, hq, hkv, d
    a.k_start, a.k_len, a.q_start, a.q_len = (_ptr(k_start), _ptr(k_len), _ptr(q_start),
                                              _ptr(q_len))
    a.max_q_len, a.max_k_len, a.total_q_rows, a.total_k_rows = max_q_len, max_k_len, tq, tk
    a.q_layer_stride, a.kv_layer_stride, a.o_layer_stride = Q.stride(0), K.stride(0), O.stride(0)
    a.softmax_scale, a.nexus_vis = softmax_scale, nexus_vis
    a.lse, a.status = _ptr(lse), _ptr(status)
    a.key_order = key_order
    a.nexus_mass = _ptr(nexus_mass)
    need = lib.sonic_prefill_workspace_size(ctypes.byref(a))
    ws = _workspace(need, Q.device, workspace)
    a.workspace, a.workspace_bytes = _ptr(ws), need
    _check(lib.sonic_attn_prefill(_ptr(Q), _ptr(K), _ptr(V), _ptr(seg_id), _ptr(role), _ptr(O),
                                  ctypes.byref(a), _stream(stream)), "sonic_attn_prefill")
    return ws


def sonic_attn_decode(q: torch.Tensor, K_ret: torch.Tensor, V_ret: torch.Tensor,
                      lens: torch.Tensor, O: torch.Tensor, *, kv_start, max_len: int,
                      softmax_scale: float = 0.0, chunk_len: int = 0, lse=None, status=None,
                      workspace=None, role=None, nexus_mass=None, stream=None):
    """One decode step.  q, O: [n_layers, B, Hq, D]; K_ret, V_ret: [n_layers, T, Hkv, D];
    lse, nexus_mass: [n_layers, B, Hq] float32 or None; role: [T] uint8 (with nexus_mass)."""
    lib = load()
    nl, B, hq, d = q.shape
    _, T, hkv, _ = K_ret.shape
    a = sonic_decode_args()
    a.batch, a.n_layers, a.n_heads_q, a.n_heads_kv, a.head_dim = B, nl, hq, hkv, d
    a.kv_start, a.max_len, a.total_kv_rows = _ptr(kv_start), max_len, T
    a.q_layer_stride, a.kv_layer_stride, a.o_layer_stride = q.stride(0), K_ret.stride(0), O.stride(0)
    a.softmax_scale, a.chunk_len = softmax_scale, chunk_len
    a.lse, a.status = _ptr(lse), _ptr(status)
    a.role, a.nexus_mass = _ptr(role), _ptr(nexus_mass)
    need = lib.sonic_decode_workspace_size(ctypes.byref(a))
    ws = _workspace(need, q.device, workspace)
    a.workspace, a.workspace_bytes = _ptr(ws), need
    _check(lib.sonic_attn_decode(_ptr(q), _ptr(K_ret), _ptr(V_ret), _ptr(lens), _ptr(O),
                                 ctypes.byref(a), _stream(stream)), "sonic_attn_decode")
    return ws


def sonic_routed_linear(X: torch.Tensor, W: torch.Tensor, W_nexus: torch.Tensor,
                        role: torch.Tensor, parts, *, dst_row=None, status=None, workspace=None,
                        stream=None):
    """Role-routed linear map.  X: [T, >= d_in] bf16 (row-contiguous); W, W_nexus:
    [d_out, d_in] bf16; role: [T] uint8.  parts: list of (out, scatter) with out a
    2-D bf16 tensor whose columns (out.shape[1]) take the next columns of Y and
    whose rows are indexed by t (scatter False) or dst_row[t] (scatter True)."""
    lib = load()
    T = X.shape[0]
    d_out, d_in = W.shape
    a = sonic_routed_linear_args()
    a.n_rows, a.d_in, a.d_out = T, d_in, d_out
    a.x_row_stride = X.stride(0) if T > 0 else d_in
    a.dst_row = _ptr(dst_row)
    a.n_parts = len(parts)
    for k, (out, scatter) in enumerate(parts):
        a.parts[k].base = _ptr(out)
        a.parts[k].row_stride = out.stride(0)
        a.parts[k].cols = out.shape[1]
        a.parts[k].scatter = 1 if scatter else 0
        a.parts[k].rows = out.shape[0]
    a.status = _ptr(status)
    need = lib.sonic_routed_linear_workspace_size(ctypes.byref(a))
    ws = _workspace(need, X.device, workspace)
    a.workspace, a.workspace_bytes = _ptr(ws), need
    _check(lib.sonic_routed_linear(_ptr(X), _ptr(W), _ptr(W_nexus), _ptr(role), ctypes.byref(a),
                                   _stream(stream)), "sonic_routed_linear")
    return ws


def sonic_attn_prefill_static(Q: torch.Tensor, K: torch.Tensor, V: torch.Tensor,
                              seg_id: torch.Tensor, role: torch.Tensor, O: torch.Tensor, *,
                              k_start, k_len, q_start, q_len, max_q_len: int, max_k_len: int,
                              softmax_scale: float = 0.0, nexus_vis: int = NEXUS_FULL, lse=None,
                              status=None, nexus_mass=None, stream=None):
    """sonic_attn_prefill for callers that cannot allocate device memory: the
    library keeps the tile summaries and masks in a fixed ~9 MiB device array, so
    no workspace is passed (and this wrapper allocates nothing either).
    Calls overlapping on the GPU share that array and must be serialised."""
    lib = load()
    nl, tq, hq, d = Q.shape
    _, tk, hkv, _ = K.shape
    a = sonic_prefill_args()
    a.batch = k_start.numel()
    a.n_layers, a.n_heads_q, a.n_heads_kv, a.head_dim = nl, hq, hkv, d
    a.k_start, a.k_len, a.q_start, a.q_len = (_ptr(k_start), _ptr(k_len), _ptr(q_start),
                                              _ptr(q_len))
    a.max_q_len, a.max_k_len, a.total_q_rows, a.total_k_rows = max_q_len, max_k_len, tq, tk
    a.q_layer_stride, a.kv_layer_stride, a.o_layer_stride = Q.stride(0), K.stride(0), O.stride(0)
    a.softmax_scale, a.nexus_vis = softmax_scale, nexus_vis
    a.lse, a.status = _ptr(lse), _ptr(status)
    a.nexus_mass = _ptr(nexus_mass)
    _check(lib.sonic_attn_prefill_static(_ptr(Q), _ptr(K), _ptr(V), _ptr(seg_id), _ptr(role),
                                         _ptr(O), ctypes.byref(a), _stream(stream)),
           "sonic_attn_prefill_static")
