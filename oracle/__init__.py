"""Double-precision CPU oracle for the SONIC Nexus-KV attention path.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The CUDA library never
imports it, and it shares no code with the library.

The arithmetic lives in ``sonic_oracle.c`` (plain loops, double precision,
each function citing the passage of the paper it restates).  This module only
builds that file with gcc and marshals numpy arrays into it:

* :func:`visible`       -- Sec. 3.2 mask rule for one pair (Eqs. 3-5).
* :func:`visibility`    -- the same rule for every (p, q) pair of a sequence.
* :func:`retain`        -- retention plan (offsets, retained lengths, source rows).
* :func:`compact_copy`  -- byte copy of retained rows for all layers.
* :func:`attn_masked`   -- masked softmax attention for selected query rows.
* :func:`decode`        -- one decode step over a retained cache.
* :func:`nexus_mass`    -- attention mass on Nexus keys per query row and head
                           (the quantity behind A_nexus, Sec. 4.1 Eq. 9).
* :func:`decode_nexus_mass` -- the same for one decode step.
* :func:`routed_linear` -- linear map with the Nexus rows' own weights (Sec. 3.1).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

ROLE_SYS, ROLE_BODY, ROLE_NEXUS, ROLE_CURR = 0, 1, 2, 3
NEXUS_FULL, NEXUS_CAUSAL_SEGMENTS = 0, 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sonic_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_lib")
_SO = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def compile_source(src: str, out: str) -> str:
    """Compile one oracle C source into a shared object with gcc (no fast-math,
    no contraction of multiply-add, so every rounding is the plain one)."""
    tmp = out + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-fPIC", "-shared", "-std=c99",
                    "-fno-fast-math", "-ffp-contract=off", src,
                    "-o", tmp, "-lm"], check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Build oracle/_lib/liboracle.so from sonic_oracle.c if it is stale."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= os.path.getmtime(_SRC)):
        return _SO
    return compile_source(_SRC, _SO)


class Oracle:
    """The oracle functions bound to one compiled shared object."""

    def __init__(self, so_path: str):
        lib = ctypes.CDLL(so_path)
        P = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        lib.orc_visible.argtypes = [i64, i64, P, P, ctypes.c_int]
        lib.orc_visible.restype = ctypes.c_int
        lib.orc_retain.argtypes = [i32, P, P, P, P, P, P, P]
        lib.orc_retain.restype = i64
        lib.orc_compact_copy.argtypes = [i32, i32, P, i64, P, P, P, i64, P, i64]
        lib.orc_compact_copy.restype = None
        lib.orc_attn_masked.argtypes = [i64, i32, i32, i32, P, P, P, P, P, P,
                                        i64, f64, ctypes.c_int, P, P, P]
        lib.orc_attn_masked.restype = None
        lib.orc_decode.argtypes = [i64, i32, i32, i32, P, P, P, f64, P, P, P]
        lib.orc_decode.restype = None
        lib.orc_nexus_mass.argtypes = [i64, i32, i32, i32, P, P, P, P, P, i64, f64,
                                       ctypes.c_int, P, P]
        lib.orc_nexus_mass.restype = None
        lib.orc_decode_nexus_mass.argtypes = [i64, i32, i32, i32, P, P, P, f64, P, P]
        lib.orc_decode_nexus_mass.restype = None
        lib.orc_routed_linear.argtypes = [i64, i32, i32, P, P, P, P, P]
        lib.orc_routed_linear.restype = None
        self.lib = lib
        self.path = so_path

    def visible(self, p: int, q: int, role, seg, nexus_mode: int = NEXUS_FULL) -> bool:
        role = _c(role, np.uint8)
        seg = _c(seg, np.int32)
        return bool(self.lib.orc_visible(p, q, _ptr(role), _ptr(seg), nexus_mode))

    def visibility(self, role, seg, nexus_mode: int = NEXUS_FULL) -> np.ndarray:
        """Boolean [L, L] matrix vis[p, q] of the per-pair rule (small L only)."""
        role = _c(role, np.uint8)
        seg = _c(seg, np.int32)
        L = role.shape[0]
        out = np.zeros((L, L), dtype=bool)
        for p in range(L):
            for q in range(L):
                out[p, q] = self.lib.orc_visible(p, q, _ptr(role), _ptr(seg), nexus_mode)
        return out

    def retain(self, k_start, k_len, role, reserve=None):
        """Retention plan: returns (offsets[B+1], ret_len[B], src_idx[offsets[B]]).

        src_idx holds packed row indices; entries inside a sequence's reserve
        rows are -1 (never written by the rule).
        """
        k_start = _c(k_start, np.int32)
        k_len = _c(k_len, np.int32)
        role = _c(role, np.uint8)
        B = k_start.shape[0]
        res = None if reserve is None else _c(reserve, np.int32)
        total = int(k_len.sum()) + (0 if res is None else int(res.sum()))
        offsets = np.zeros(B + 1, np.int32)
        ret_len = np.zeros(B, np.int32)
        src_idx = np.full(max(total, 1), -1, np.int32)
        n = self.lib.orc_retain(B, _ptr(k_start), _ptr(k_len), _ptr(role), _ptr(res),
                                _ptr(offsets), _ptr(ret_len), _ptr(src_idx))
        return offsets, ret_len, src_idx[:n]

    def compact_copy(self, src: np.ndarray, offsets, ret_len, src_idx, out_rows: int,
                     fill: int = 0) -> np.ndarray:
        """Copy retained rows.  src: uint8 [n_layers, T, row_bytes] (contiguous).

        Returns uint8 [n_layers, out_rows, row_bytes]; rows no sequence fills
        keep ``fill``.
        """
        src = np.ascontiguousarray(src, dtype=np.uint8)
        nl, T, rb = src.shape
        dst = np.full((nl, out_rows, rb), fill, np.uint8)
        offsets = _c(offsets, np.int32)
        ret_len = _c(ret_len, np.int32)
        src_idx = _c(src_idx, np.int32)
        self.lib.orc_compact_copy(ret_len.shape[0], nl, _ptr(src), T * rb, _ptr(offsets),
                                  _ptr(ret_len), _ptr(src_idx), rb, _ptr(dst),
                                  out_rows * rb)
        return dst

    def attn_masked(self, Q, K, V, role, seg, rows, scale=None, nexus_mode=NEXUS_FULL):
        """Masked attention of one sequence.

        Q: [n_rows, Hq, D]; K, V: [L, Hkv, D]; rows: positions of the queries.
        Returns (O [n_rows, Hq, D] float64, lse [n_rows, Hq] float64).
        """
        Q = _c(Q, np.float64)
        K = _c(K, np.float64)
        V = _c(V, np.float64)
        role = _c(role, np.uint8)
        seg = _c(seg, np.int32)
        rows = _c(rows, np.int64)
        n_rows, Hq, D = Q.shape
        L, Hkv, _ = K.shape
        if scale is None:
            scale = 1.0 / np.sqrt(D)
        O = np.zeros((n_rows, Hq, D), np.float64)
        lse = np.zeros((n_rows, Hq), np.float64)
        s_buf = np.zeros(max(L, 1), np.float64)
        self.lib.orc_attn_masked(L, Hq, Hkv, D, _ptr(Q), _ptr(K), _ptr(V), _ptr(role),
                                 _ptr(seg), _ptr(rows), n_rows, float(scale), nexus_mode,
                                 _ptr(s_buf), _ptr(O), _ptr(lse))
        return O, lse

    def decode(self, q, K, V, scale=None):
        """One decode step: q [Hq, D]; K, V [n, Hkv, D]. Returns (O [Hq, D], lse [Hq])."""
        q = _c(q, np.float64)
        K = _c(K, np.float64)
        V = _c(V, np.float64)
        Hq, D = q.shape
        n, Hkv, _ = K.shape
        if scale is None:
            scale = 1.0 / np.sqrt(D)
        O = np.zeros((Hq, D), np.float64)
        lse = np.zeros(Hq, np.float64)
        s_buf = np.zeros(max(n, 1), np.float64)
        self.lib.orc_decode(n, Hq, Hkv, D, _ptr(q), _ptr(K), _ptr(V), float(scale),
                            _ptr(s_buf), _ptr(O), _ptr(lse))
        return O, lse

    def nexus_mass(self, Q, K, role, seg, rows, scale=None, nexus_mode=NEXUS_FULL):
        """Share of each query row's attention (per head) on visible Nexus keys.

        Q: [n_rows, Hq, D]; K: [L, Hkv, D]; rows: positions of the queries.
        Returns mass [n_rows, Hq] float64.
        """
        Q = _c(Q, np.float64)
        K = _c(K, np.float64)
        role = _c(role, np.uint8)
        seg = _c(seg, np.int32)
        rows = _c(rows, np.int64)
        n_rows, Hq, D = Q.shape
        L, Hkv, _ = K.shape
        if scale is None:
            scale = 1.0 / np.sqrt(D)
        mass = np.zeros((n_rows, Hq), np.float64)
        s_buf = np.zeros(max(L, 1), np.float64)
        self.lib.orc_nexus_mass(L, Hq, Hkv, D, _ptr(Q), _ptr(K), _ptr(role), _ptr(seg),
                                _ptr(rows), n_rows, float(scale), nexus_mode, _ptr(s_buf),
                                _ptr(mass))
        return mass

    def decode_nexus_mass(self, q, K, role, scale=None):
        """Decode form: q [Hq, D]; K [n, Hkv, D]; role [n]. Returns mass [Hq]."""
        q = _c(q, np.float64)
        K = _c(K, np.float64)
        role = _c(role, np.uint8)
        Hq, D = q.shape
        n, Hkv, _ = K.shape
        if scale is None:
            scale = 1.0 / np.sqrt(D)
        mass = np.zeros(Hq, np.float64)
        s_buf = np.zeros(max(n, 1), np.float64)
        self.lib.orc_decode_nexus_mass(n, Hq, Hkv, D, _ptr(q), _ptr(K), _ptr(role),
                                       float(scale), _ptr(s_buf), _ptr(mass))
        return mass

    def routed_linear(self, X, W, W_nexus, role):
        """Y [T, d_out] = X @ W.T on rows whose role is not NEXUS, X @ W_nexus.T on
        Nexus rows.  X: [T, d_in]; W, W_nexus: [d_out, d_in]."""
        X = _c(X, np.float64)
        W = _c(W, np.float64)
        W_nexus = _c(W_nexus, np.float64)
        role = _c(role, np.uint8)
        T, d_in = X.shape
        d_out = W.shape[0]
        assert W.shape == (d_out, d_in) and W_nexus.shape == (d_out, d_in)
        Y = np.zeros((T, d_out), np.float64)
        self.lib.orc_routed_linear(T, d_in, d_out, _ptr(X), _ptr(W), _ptr(W_nexus), _ptr(role),
                                   _ptr(Y))
        return Y


def _ptr(a):
    return None if a is None else a.ctypes.data


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def default() -> Oracle:
    """The oracle built from sonic_oracle.c (built on first use)."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = Oracle(build())
        return _lib


def visible(*a, **k):
    return default().visible(*a, **k)


def visibility(*a, **k):
    return default().visibility(*a, **k)


def retain(*a, **k):
    return default().retain(*a, **k)


def compact_copy(*a, **k):
    return default().compact_copy(*a, **k)


def attn_masked(*a, **k):
    return default().attn_masked(*a, **k)


def decode(*a, **k):
    return default().decode(*a, **k)


def nexus_mass(*a, **k):
    return default().nexus_mass(*a, **k)


def decode_nexus_mass(*a, **k):
    return default().decode_nexus_mass(*a, **k)


def routed_linear(*a, **k):
    return default().routed_linear(*a, **k)
