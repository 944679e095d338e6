"""sonic_attn_prefill_static: the masked prefill for callers that cannot
allocate device memory (code inside an allocator or pool callback, runtimes
that plan every device byte in advance, hosts that only hand over fixed input
and output buffers).  Its scratch lives in a fixed array inside the library.

Checked through the C ABI:
  * against sonic_attn_prefill with a caller workspace, on two calls in a row
    with different shapes (the second call runs on the array the first one
    left behind): the same kernels on the same inputs, so O, lse and the
    Nexus mass must be bit-identical;
  * against the oracle, every row of a small ragged batch;
  * at the array's limit (256 sequences x 16,384 keys = 32,768 key tiles),
    bit-identical to the workspace call and sampled rows of the first and
    last sequences against the oracle, so the top of the array is used;
  * an oversized call is refused before anything runs.
This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
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
    return (Q, K, V, seg, role), kw, q_len, q_start


def _outputs(Q):
    nan = float("nan")
    return (torch.full_like(Q, nan), torch.full(Q.shape[:3], nan, device=H.dev()),
            torch.full(Q.shape[:3], nan, device=H.dev()))


def _both(args, kw, with_mass):
    """The workspace call and the fixed-scratch call on the same inputs."""
    Q = args[0]
    O_ref, lse_ref, m_ref = _outputs(Q)
    O_new, lse_new, m_new = _outputs(Q)
    st = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_prefill(*args, O_ref, lse=lse_ref, status=st,
                             nexus_mass=m_ref if with_mass else None, **kw)
    torch.cuda.synchronize()
    assert sonic.read_status(st) == 0
    sonic.sonic_attn_prefill_static(*args, O_new, lse=lse_new, status=st,
                                    nexus_mass=m_new if with_mass else None, **kw)
    torch.cuda.synchronize()
    assert sonic.read_status(st) == 0
    return (O_ref, lse_ref, m_ref if with_mass else None), (O_new, lse_new,
                                                            m_new if with_mass else None)


def _assert_identical(ref, new):
    O_ref, lse_ref, m_ref = ref
    O_new, lse_new, m_new = new
    assert torch.isfinite(O_new.float()).all()
    assert torch.equal(O_new.view(torch.int16), O_ref.view(torch.int16)), "O differs"
    assert torch.equal(lse_new.view(torch.int32), lse_ref.view(torch.int32)), "lse differs"
    if m_ref is not None:
        assert torch.equal(m_new.view(torch.int32), m_ref.view(torch.int32)), "mass differs"


def _against_oracle(batch, args, q_len, q_start, new, b, rows):
    Q, K, V = args[0], args[1], args[2]
    O_new, lse_new, m_new = new
    ks, kl = int(batch.k_start[b]), int(batch.k_len[b])
    rows = np.asarray(rows, np.int64)
    pos = kl - int(q_len[b]) + rows
    qr = int(q_start[b]) + rows
    Kb, Qb = H.f64(K[0, ks:ks + kl]), H.f64(Q[0, qr])
    Oref, lref = oracle.attn_masked(Qb, Kb, H.f64(V[0, ks:ks + kl]), batch.role[ks:ks + kl],
                                    batch.seg[ks:ks + kl], pos)
    H.check_close(H.f64(O_new[0, qr]), Oref, f"fixed-scratch prefill, sequence {b}")
    np.testing.assert_allclose(H.f64(lse_new[0, qr]), lref, rtol=0, atol=2e-3)
    if m_new is not None:
        mref = oracle.nexus_mass(Qb, Kb, batch.role[ks:ks + kl], batch.seg[ks:ks + kl], pos)
        np.testing.assert_allclose(H.f64(m_new[0, qr]), mref, rtol=0, atol=2e-3)


def test_static_scratch_prefill_matches_workspace_prefill_twice():
    rng = np.random.default_rng(4)
    first = inputs.Batch([inputs.random_dialogue(rng, max_segments=6, max_body=300,
                                                 max_nexus=40, max_curr=200) for _ in range(5)])
    second = inputs.Batch([inputs.Dialogue(64, [(500, 60), (300, 0), (20, 20)], 700),
                           inputs.Dialogue(3, [(129, 128)], 257)])
    for batch, hq, hkv, D, seed, ql, mass in ((first, 8, 2, 128, 1, None, False),
                                              (second, 4, 4, 64, 2, [700, 100], True)):
        args, kw, q_len, q_start = _case(batch, hq, hkv, D, seed, ql)
        ref, new = _both(args, kw, mass)
        _assert_identical(ref, new)
        if batch is first:
            # every row of the small ragged batch against the oracle
            for b in range(batch.B):
                _against_oracle(batch, args, q_len, q_start, new, b, np.arange(q_len[b]))


def test_static_scratch_at_its_tile_limit():
    """256 sequences of 16,384 keys (32,768 key tiles: the whole array), four
    query rows each, with the Nexus-mass output."""
    d = inputs.Dialogue(128, [(1000, 100)] * 14 + [(300, 56)], 500)
    assert d.length == 16384
    batch = inputs.Batch([d] * 256)
    q_len = np.full(batch.B, 4, np.int32)
    args, kw, q_len, q_start = _case(batch, 2, 1, 64, 7, q_len)
    ref, new = _both(args, kw, True)
    _assert_identical(ref, new)
    for b in (0, 1, 254, 255):
        _against_oracle(batch, args, q_len, q_start, new, b, np.arange(4))


def test_static_scratch_refuses_oversized_calls():
    lib = sonic.load()
    a = sonic.sonic_prefill_args()
    a.batch, a.n_layers, a.n_heads_q, a.n_heads_kv, a.head_dim = 64, 1, 8, 2, 128
    a.max_q_len, a.max_k_len = 128, 128 * 513   # 64 * 513 tiles > 32768
    a.total_q_rows, a.total_k_rows = 128, 128
    a.k_start = a.k_len = a.q_start = a.q_len = 16
    assert lib.sonic_attn_prefill_static(16, 16, 16, 16, 16, 16, ctypes.byref(a), None) == 3
