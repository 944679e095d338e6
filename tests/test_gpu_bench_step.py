"""Parity of the benchmarked mixed serving step itself: the full-size workload in
the launch configuration bench.py times (28 layers, 28/4 heads, D = 128; 8
sequences compact a 4k-64k raw history and prefill a new turn, 56 decode),
checked on sampled outputs the oracle computes one by one."""
import numpy as np
import pytest
import torch

import bench
import oracle
from tests import harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def step():
    lay = bench.Layout()
    g = bench.GpuStep(lay, H.dev(), seed=3)
    # keep a copy of the rows compaction will overwrite, to check its bytes
    g.step()
    torch.cuda.synchronize()
    from paper_2601_21927_gb300 import sonic
    assert sonic.read_status(g.status) == 0
    yield lay, g
    del g
    torch.cuda.empty_cache()


def test_compaction_in_bench_step(step):
    lay, g = step
    off = g.offsets.cpu().numpy()
    want_off, ret_len, src = oracle.retain(lay.raw.k_start, lay.raw.k_len, lay.raw.role,
                                           lay.q_len)
    assert off.tolist() == want_off.tolist()
    assert (ret_len == lay.ret_pre).all()
    for layer in (0, 13, 27):
        raw = g.rawK[layer].view(torch.int16).cpu().numpy().view(np.uint8)
        raw = raw.reshape(1, lay.raw.total, -1)
        want = oracle.compact_copy(raw, want_off, ret_len, src, int(want_off[-1]))
        got = g.outK[layer].view(torch.int16).cpu().numpy().view(np.uint8)
        got = got.reshape(1, g.outK.shape[1], -1)
        for b in range(lay.n_pre):
            sl = slice(want_off[b], want_off[b] + ret_len[b])
            assert np.array_equal(got[:, sl], want[:, sl]), f"layer {layer} seq {b}"


def test_prefill_in_bench_step(step):
    lay, g = step
    for layer, b in ((0, 0), (27, 5), (13, 7)):
        ks, kl = int(lay.k_start_pre[b]), int(lay.k_len_pre[b])
        ql, qs = int(lay.q_len[b]), int(lay.q_start[b])
        rows = np.unique(np.r_[0, 1, 127, 128, 255, 256, ql // 2, ql - 2, ql - 1])
        rows = rows[rows < ql]
        K = H.f64(g.Kret[layer, ks:ks + kl])
        V = H.f64(g.Vret[layer, ks:ks + kl])
        Q = H.f64(g.Qp[layer, qs + rows])
        O, _ = oracle.attn_masked(Q, K, V, lay.role_ret[ks:ks + kl], lay.seg_ret[ks:ks + kl],
                                  kl - ql + rows)
        H.check_close(H.f64(g.Op[layer, qs + rows]), O, f"layer {layer} seq {b}")


def test_decode_in_bench_step(step):
    lay, g = step
    for layer, b in ((0, 0), (27, 55), (13, 20), (5, int(np.argmax(lay.dec_len)))):
        s, n = int(lay.dec_start[b]), int(lay.dec_len[b])
        O, _ = oracle.decode(H.f64(g.qd[layer, b]), H.f64(g.Kret[layer, s:s + n]),
                             H.f64(g.Vret[layer, s:s + n]))
        H.check_close(H.f64(g.Od[layer, b]), O, f"layer {layer} seq {b}")
