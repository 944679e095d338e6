"""sonic_attn_prefill_static: the masked prefill for callers that cannot
allocate device memory (code inside an allocator or pool callback, runtimes
that plan every device byte in advance, hosts that only hand over fixed input
and output buffers).  Its scratch lives in a fixed array inside the library.

Checked through the C ABI against sonic_attn_prefill (caller workspace) on
two calls in a row with different shapes, so the second call runs on the
array the first one left behind; and an oversized call is refused before
anything runs.  This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _case(batch, hq, hkv, D, seed, q_len=None):
    role, seg, k_start, k_len = H.meta(batch)
    q_len = batch.k_len.copy() if q_len is None else np.asarray(q_len, np.int32)
    q_start = np.concatenate([[0], np.cumsum(q_len)[:-1]]).astype(np.int32)
    K = inputs.randn((1, batch.total, hkv, D), seed=seed + 1, device=H.dev())
    V = inputs.randn((1, batch.total, hkv, D), seed=seed + 2, device=H.dev())
    Q = inputs.randn((1, int(q_len.sum()), hq, D), seed=seed + 3, device=H.dev())
    kw = dict(k_start=k_start, k_len=k_len, q_start=H.i32(q_start), q_len=H.i32(q_len),
              max_q_len=int(q_len.max()), max_k_len=int(batch.k_len.max()))
    return (Q, K, V, seg, role), kw


def _both(args, kw):
    Q = args[0]
    O_ref = torch.full_like(Q, float("nan"))
    O_new = torch.full_like(Q, float("nan"))
    lse_ref = torch.full(Q.shape[:3], float("nan"), device=H.dev())
    lse_new = torch.full(Q.shape[:3], float("nan"), device=H.dev())
    st = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_prefill(*args, O_ref, lse=lse_ref, status=st, **kw)
    sonic.sonic_attn_prefill_static(*args, O_new, lse=lse_new, status=st, **kw)
    torch.cuda.synchronize()
    assert sonic.read_status(st) == 0
    return O_ref, O_new, lse_ref, lse_new


def test_static_scratch_prefill_matches_workspace_prefill_twice():
    rng = np.random.default_rng(4)
    first = inputs.Batch([inputs.random_dialogue(rng, max_segments=6, max_body=300,
                                                 max_nexus=40, max_curr=200) for _ in range(5)])
    second = inputs.Batch([inputs.Dialogue(64, [(500, 60), (300, 0), (20, 20)], 700),
                           inputs.Dialogue(3, [(129, 128)], 257)])
    for batch, hq, hkv, D, seed, ql in ((first, 8, 2, 128, 1, None),
                                        (second, 4, 4, 64, 2, [700, 100])):
        args, kw = _case(batch, hq, hkv, D, seed, ql)
        O_ref, O_new, lse_ref, lse_new = _both(args, kw)
        got, want = H.f64(O_new), H.f64(O_ref)
        assert np.isfinite(got).all()
        H.check_close(got, want, "static-scratch prefill")
        np.testing.assert_allclose(H.f64(lse_new), H.f64(lse_ref), rtol=0, atol=1e-5)


def test_static_scratch_refuses_oversized_calls():
    lib = sonic.load()
    a = sonic.sonic_prefill_args()
    a.batch, a.n_layers, a.n_heads_q, a.n_heads_kv, a.head_dim = 64, 1, 8, 2, 128
    a.max_q_len, a.max_k_len = 128, 128 * 513   # 64 * 513 tiles > 32768
    a.total_q_rows, a.total_k_rows = 128, 128
    a.k_start = a.k_len = a.q_start = a.q_len = 16
    assert lib.sonic_attn_prefill_static(16, 16, 16, 16, 16, 16, ctypes.byref(a), None) == 3
