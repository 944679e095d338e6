"""The C ABI (no GPU needed): the library loads, exports every entry point
declared in include/sonic.h, the ctypes structs match the C layout, and host
validation rejects bad arguments before anything is launched."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2601_21927_gb300 import sonic

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sonic.h")


def _declared():
    txt = open(HEADER).read()
    return sorted(set(re.findall(r"SONIC_API\s+[\w\s\*]+?\b(sonic_\w+)\s*\(", txt)))


def test_library_exports_every_declared_symbol():
    lib = sonic.load()
    names = _declared()
    assert len(names) >= 9
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(sonic.SIGNATURES)
    assert lib.sonic_abi_version() == 4
    assert lib.sonic_status_string(4) == b"output capacity exceeded"


def test_struct_layout_matches_c(tmp_path):
    structs = {"sonic_compact_args": sonic.sonic_compact_args,
               "sonic_prefill_args": sonic.sonic_prefill_args,
               "sonic_decode_args": sonic.sonic_decode_args,
               "sonic_out_part": sonic.sonic_out_part,
               "sonic_routed_linear_args": sonic.sonic_routed_linear_args}
    src = ['#include <stdio.h>', '#include <stddef.h>', '#include "sonic.h"', 'int main(void){']
    for name, cls in structs.items():
        src.append(f'printf("{name} %zu\\n", sizeof({name}));')
        for f, _ in cls._fields_:
            src.append(f'printf("{name}.{f} %zu\\n", offsetof({name}, {f}));')
    src.append("return 0;}")
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                 check=True).stdout.splitlines())
    for name, cls in structs.items():
        assert int(out[name]) == ctypes.sizeof(cls), name
        for f, _ in cls._fields_:
            assert int(out[f"{name}.{f}"]) == getattr(cls, f).offset, f"{name}.{f}"


def test_host_validation_rejects_before_launch():
    lib = sonic.load()
    # NULL args / offsets
    assert lib.sonic_compact_kv(None, None, None, None, None, None, None, None, None) == 1
    a = sonic.sonic_compact_args()
    a.batch, a.n_layers = 2, 1
    assert lib.sonic_compact_kv(16, 16, None, 16, 16, 16, None, ctypes.byref(a), None) == 1
    a.row_bytes = 24  # not a multiple of 16
    a.k_start = a.k_len = 16
    assert lib.sonic_compact_kv(16, 16, None, 16, 16, 16, 16, ctypes.byref(a), None) == 1
    a.row_bytes = 32
    assert lib.sonic_compact_kv(17, 16, None, 16, 16, 16, 16, ctypes.byref(a), None) == 1  # misaligned
    assert lib.sonic_compact_kv(16, 16, None, 16, 16, 16, 16, ctypes.byref(a), None) == 1  # no rows
    a.total_rows = 10
    assert lib.sonic_compact_kv(16, 16, None, 16, 16, 16, 16, ctypes.byref(a), None) == 3  # no workspace

    p = sonic.sonic_prefill_args()
    p.batch, p.n_layers, p.n_heads_q, p.n_heads_kv, p.head_dim = 1, 1, 6, 4, 128
    p.max_q_len = p.max_k_len = p.total_q_rows = p.total_k_rows = 8
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 1  # 6 % 4
    p.n_heads_q, p.head_dim = 8, 96
    p.k_start = p.k_len = p.q_start = p.q_len = 16
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 2  # D = 96
    p.head_dim = 128
    p.max_k_len = 300000
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 2  # too long
    p.max_k_len = 8
    p.nexus_vis = 5
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 1
    p.nexus_vis = 0
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 3  # workspace
    # the work-unit counter (256 B), then one key tile: its summary (32 B) and
    # its column masks (256 B), each part rounded up to 256 bytes
    assert lib.sonic_prefill_workspace_size(ctypes.byref(p)) == 256 + 256 + 256
    p.key_order = 7
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 1
    # the fixed-scratch entry point serves only the as-given key order
    p.key_order = sonic.KEYS_RETAINED_FIRST
    assert lib.sonic_attn_prefill_static(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 2
    p.key_order = sonic.KEYS_AS_GIVEN

    d = sonic.sonic_decode_args()
    d.batch, d.n_layers, d.n_heads_q, d.n_heads_kv, d.head_dim = 2, 1, 40, 2, 128
    d.kv_start, d.max_len, d.total_kv_rows = 16, 10, 20
    assert lib.sonic_attn_decode(16, 16, 16, 16, 16, ctypes.byref(d), None) == 2  # G = 20 > 16
    d.n_heads_q = 8
    d.chunk_len = -5
    assert lib.sonic_attn_decode(16, 16, 16, 16, 16, ctypes.byref(d), None) == 1  # negative
    d.chunk_len, d.head_dim = 0, 80
    assert lib.sonic_attn_decode(16, 16, 16, 16, 16, ctypes.byref(d), None) == 2


def test_python_binding_has_no_cpu_path():
    src = open(os.path.join(ROOT, "paper_2601_21927_gb300", "sonic.py")).read()
    assert "import oracle" not in src and "from oracle" not in src
    for f in os.listdir(os.path.join(ROOT, "paper_2601_21927_gb300")):
        if f.endswith(".py"):
            t = open(os.path.join(ROOT, "paper_2601_21927_gb300", f)).read()
            assert "oracle" not in re.findall(r"^\s*(?:import|from)\s+(\w+)", t, re.M), f


def test_retained_first_workspace_size():
    """Workspace of the retained-first order: the work-unit counter (256 B),
    tile summaries (32 B) and column masks (256 B) of one extra tile per
    sequence, 13 bytes of metadata per permuted row, the first input row of
    each tile read in place (4 B per tile), the query chunk table (4 B per
    32 rows of align128(max_q_len) + 1024 rows per sequence), and a K and a V
    copy of every layer; each part rounded up to 256 bytes."""
    lib = sonic.load()
    p = sonic.sonic_prefill_args()
    p.batch, p.n_layers, p.n_heads_q, p.n_heads_kv, p.head_dim = 2, 3, 8, 4, 128
    p.max_q_len, p.max_k_len, p.total_q_rows, p.total_k_rows = 300, 300, 600, 600
    assert lib.sonic_prefill_workspace_size(ctypes.byref(p)) == 256 + 256 + 1536  # 2 * 3 tiles
    p.key_order = sonic.KEYS_RETAINED_FIRST

    def r256(x):
        return (x + 255) // 256 * 256

    def expect(rows):
        return (256 + r256(2 * 4 * 32) + r256(2 * 4 * 256) + r256(3 * 4) + r256(2 * 4) + r256(rows)
                + 3 * r256(4 * rows) + r256(2 * 4 * 4) + r256(2 * (384 + 1024) // 32 * 4)
                + 2 * r256(3 * rows * 4 * 128 * 2))

    # spans of 384 + 128 rows per sequence, below total_k_rows + 256 per sequence
    assert lib.sonic_prefill_workspace_size(ctypes.byref(p)) == expect(1024)
    p.total_k_rows = 300  # two sequences sharing rows: capped at 300 + 512
    assert lib.sonic_prefill_workspace_size(ctypes.byref(p)) == expect(812)
    p.max_k_len = 2047 * 128 + 1  # one extra tile past the 2048-tile list
    p.total_k_rows = p.max_k_len
    p.k_start = p.k_len = p.q_start = p.q_len = 16
    assert lib.sonic_attn_prefill(16, 16, 16, 16, 16, 16, ctypes.byref(p), None) == 2


def test_routed_linear_validation():
    lib = sonic.load()
    a = sonic.sonic_routed_linear_args()
    assert lib.sonic_routed_linear(None, None, None, None, None, None) == 1
    a.n_rows = 0
    assert lib.sonic_routed_linear(None, None, None, None, ctypes.byref(a), None) == 0  # empty
    a.n_rows, a.d_in, a.d_out, a.x_row_stride, a.n_parts = 10, 96, 64, 96, 1  # d_in % 64
    a.parts[0].base, a.parts[0].row_stride, a.parts[0].cols, a.parts[0].rows = 16, 64, 64, 10
    assert lib.sonic_routed_linear(16, 16, 16, 16, ctypes.byref(a), None) == 1
    a.d_in = a.x_row_stride = 128
    a.parts[0].cols = 48                      # parts must cover d_out in 32-column steps
    assert lib.sonic_routed_linear(16, 16, 16, 16, ctypes.byref(a), None) == 1
    a.parts[0].cols = 64
    a.parts[0].scatter = 1                    # scatter without dst_row
    assert lib.sonic_routed_linear(16, 16, 16, 16, ctypes.byref(a), None) == 1
    a.parts[0].scatter = 0
    a.parts[0].rows = 9                       # fewer rows than X for an unscattered part
    assert lib.sonic_routed_linear(16, 16, 16, 16, ctypes.byref(a), None) == 1
    a.parts[0].rows = 10
    assert lib.sonic_routed_linear(16, 16, 16, 16, ctypes.byref(a), None) == 3  # no workspace
    assert lib.sonic_routed_linear_workspace_size(ctypes.byref(a)) == 256 + 256 + 256 + 2560
