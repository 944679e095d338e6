"""The tiny single-sequence dialogue end to end: compaction, masked prefill of
every row, then eight decode steps over the growing retained cache.

Dialogue: 16 system tokens, 3 history segments of 32 body + 4 Nexus tokens, a
24-token current query (L = 148, 52 retained rows); 1 layer, 2 query / 1 KV
head, head_dim 64; Q/K/V drawn in fp32 ~ N(0, 1).

* Compaction runs on the fp32 bytes with 8 reserve rows after the retained
  ones and must match the oracle bit for bit (Sec. 3.2 body removal, App. C
  effective context I_sys + N + Q_n).
* Attention runs on the fp32 values rounded to bf16 (nearest even); the
  oracle reads the same rounded values in double precision.
* Generation (App. C, Eq. 15): each step draws the new token's q/k/v, writes
  k/v into the next reserve row (the KV append, a plain copy outside the
  library), and decodes over retained rows + the tokens appended so far, so
  the cache grows from 53 to 60 rows.  Every step is checked against the
  oracle's decode on the rows the GPU read.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu

N_STEPS = 8


def _u8(t: torch.Tensor) -> np.ndarray:
    """Raw bytes of a [n_layers, rows, ...] tensor as uint8 [n_layers, rows, row_bytes]."""
    nl, rows = t.shape[0], t.shape[1]
    return t.contiguous().view(torch.int32).cpu().numpy().view(np.uint8).reshape(nl, rows, -1)


def test_tiny_dialogue_compaction_prefill_and_eight_decode_steps():
    batch, hd = inputs.tiny_ref()
    d = batch.dialogues[0]
    L, hq, hkv, D = d.length, hd.hq, hd.hkv, hd.d
    R = d.recipe_retained
    assert (L, R) == (148, 52)
    dev = H.dev()
    K32 = inputs.randn((1, L, hkv, D), seed=11, dtype=torch.float32, device=dev)
    V32 = inputs.randn((1, L, hkv, D), seed=12, dtype=torch.float32, device=dev)
    Q32 = inputs.randn((1, L, hq, D), seed=13, dtype=torch.float32, device=dev)
    role, seg, k_start, k_len = H.meta(batch)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    # ---- compaction of the fp32 rows, 8 reserve rows for the decoded tokens
    cap = R + N_STEPS
    oK32 = torch.zeros((1, cap, hkv, D), dtype=torch.float32, device=dev)
    oV32 = torch.zeros_like(oK32)
    offsets = torch.full((2,), -7, dtype=torch.int32, device=dev)
    ret_len = torch.full((1,), -7, dtype=torch.int32, device=dev)
    reserve = H.i32([N_STEPS])
    sonic.sonic_compact_kv(K32, V32, seg, role, oK32, oV32, offsets, k_start=k_start,
                           k_len=k_len, reserve=reserve, ret_len=ret_len, status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    off, rl, src = oracle.retain(batch.k_start, batch.k_len, batch.role, [N_STEPS])
    assert offsets.cpu().tolist() == off.tolist() == [0, cap]
    assert ret_len.cpu().tolist() == rl.tolist() == [R]
    for got_t, raw in ((oK32, K32), (oV32, V32)):
        want = oracle.compact_copy(_u8(raw), off, rl, src, cap)
        got = _u8(got_t)
        assert np.array_equal(got[:, :R], want[:, :R])
        assert not got[:, R:].any(), "reserve rows must stay untouched"

    # ---- masked prefill of all 148 rows on the bf16-rounded values
    K, V, Q = K32.to(torch.bfloat16), V32.to(torch.bfloat16), Q32.to(torch.bfloat16)
    res = H.run_prefill(batch, hq, hkv, D, K=K, V=V, Q=Q)
    Oref, lref, Ogot, lgot = H.oracle_prefill_rows(batch, res, 0, np.arange(L))
    H.check_close(Ogot, Oref, "prefill, all rows")
    np.testing.assert_allclose(lgot, lref, rtol=0, atol=2e-3)

    # ---- generation: eight decode steps over the growing retained cache
    Kc = oK32.to(torch.bfloat16)
    Vc = oV32.to(torch.bfloat16)
    kv_start = H.i32([0])
    ws = None
    for s in range(N_STEPS):
        q = inputs.randn((1, 1, hq, D), seed=100 + s, dtype=torch.float32, device=dev)
        q = q.to(torch.bfloat16)
        k_new = inputs.randn((hkv, D), seed=200 + s, dtype=torch.float32, device=dev)
        v_new = inputs.randn((hkv, D), seed=300 + s, dtype=torch.float32, device=dev)
        Kc[0, R + s] = k_new.to(torch.bfloat16)   # KV append into the reserve row
        Vc[0, R + s] = v_new.to(torch.bfloat16)
        n = R + s + 1
        O = torch.full_like(q, float("nan"))
        lse = torch.full((1, 1, hq), float("nan"), device=dev)
        ws = sonic.sonic_attn_decode(q, Kc, Vc, H.i32([n]), O, kv_start=kv_start, max_len=n,
                                     lse=lse, status=status, workspace=ws)
        torch.cuda.synchronize()
        assert sonic.read_status(status) == 0
        Dref, dl = oracle.decode(H.f64(q[0, 0]), H.f64(Kc[0, :n]), H.f64(Vc[0, :n]))
        H.check_close(H.f64(O[0, 0]), Dref, f"decode step {s + 1} ({n} rows)")
        np.testing.assert_allclose(H.f64(lse[0, 0]), dl, rtol=0, atol=2e-3)
    assert n == 60
