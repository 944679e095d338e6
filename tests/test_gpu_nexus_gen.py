"""The Nexus-generation loop (Sec. 3.1 / Table 3 "Nexus Gen."): a dialogue is
processed one history segment at a time with the library's own calls.

For segment i the key sequence is [retained cache | body_i | Nexus_i]: the
retained cache holds the system prompt and the Nexus tokens of segments
1..i-1 (earlier bodies are already gone).  The Nexus rows are the queries
(the last K_i rows), sonic_attn_prefill gives their outputs, and
sonic_compact_kv then drops body_i, leaving [retained | Nexus_i] as the next
retained cache.  After the last segment the current turn is prefilled over the
retained cache.

What must hold, by the rules of Sec. 3.2 (a Nexus token sees the retained rows
before it, its own body and, bidirectionally, Nexus tokens):
  * under the causal-segments reading the Nexus outputs of every segment equal
    the oracle on the whole S_aug: nothing after segment i is visible to them;
  * under the full reading they equal the oracle on S_aug cut after segment i
    (the Nexus tokens of later segments do not exist yet when segment i's are
    produced);
  * every retained cache is, byte for byte, the S_aug rows the retention rule
    keeps, and the current turn's outputs equal the oracle on the whole S_aug.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _prefill(Q, K, V, role, seg, q_len, mode):
    nl, T = K.shape[0], K.shape[1]
    O = torch.full_like(Q, float("nan"))
    lse = torch.full(Q.shape[:3], float("nan"), device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_prefill(Q, K, V, seg, role, O, k_start=H.i32([0]), k_len=H.i32([T]),
                             q_start=H.i32([0]), q_len=H.i32([q_len]), max_q_len=q_len,
                             max_k_len=T, nexus_vis=mode, lse=lse, status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    return O, lse


def _compact(K, V, role, seg, cap):
    nl, T = K.shape[0], K.shape[1]
    oK = torch.zeros((nl, cap) + tuple(K.shape[2:]), dtype=K.dtype, device=H.dev())
    oV = torch.zeros_like(oK)
    offsets = torch.zeros(2, dtype=torch.int32, device=H.dev())
    o_role = torch.zeros(cap, dtype=torch.uint8, device=H.dev())
    o_seg = torch.zeros(cap, dtype=torch.int32, device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_compact_kv(K, V, seg, role, oK, oV, offsets, k_start=H.i32([0]),
                           k_len=H.i32([T]), out_role=o_role, out_seg=o_seg, status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    assert int(offsets[1]) == cap
    return oK, oV, o_role, o_seg


def _oracle_rows(Q, K, V, role, seg, pos, mode, layer=0):
    return oracle.attn_masked(H.f64(Q[layer]), H.f64(K[layer]), H.f64(V[layer]), role, seg, pos,
                              nexus_mode=mode)


@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
@pytest.mark.parametrize("D,hq,hkv", [(128, 4, 2), (64, 2, 1)])
def test_nexus_generation_loop(mode, D, hq, hkv):
    d = inputs.Dialogue(70, [(200, 30), (64, 64), (300, 1), (150, 45), (90, 0)], 130)
    role_all, seg_all = d.arrays()
    L = d.length
    nl = 2
    K = inputs.randn((nl, L, hkv, D), seed=41, device=H.dev())
    V = inputs.randn((nl, L, hkv, D), seed=42, device=H.dev())
    Qall = inputs.randn((nl, L, hq, D), seed=43, device=H.dev())
    t_role, t_seg = (torch.from_numpy(role_all).to(H.dev()), torch.from_numpy(seg_all).to(H.dev()))

    # the retained cache (S_aug row numbers, in order) and its K/V/metadata
    kept = list(range(d.sys_len))
    cK, cV = K[:, :d.sys_len].contiguous(), V[:, :d.sys_len].contiguous()
    c_role, c_seg = t_role[:d.sys_len], t_seg[:d.sys_len]
    t = d.sys_len
    for i, (nb, nk) in enumerate(d.segments, start=1):
        body = list(range(t, t + nb))
        nexus = list(range(t + nb, t + nb + nk))
        t += nb + nk
        rows = torch.as_tensor(body + nexus, device=H.dev()).long()
        kK = torch.cat([cK, K[:, rows]], 1).contiguous()
        kV = torch.cat([cV, V[:, rows]], 1).contiguous()
        k_role = torch.cat([c_role, t_role[rows]]).contiguous()
        k_seg = torch.cat([c_seg, t_seg[rows]]).contiguous()
        if nk > 0:
            Q = Qall[:, torch.as_tensor(nexus, device=H.dev()).long()].contiguous()
            O, lse = _prefill(Q, kK, kV, k_role, k_seg, nk, mode)
            # oracle: whole S_aug (causal segments) or S_aug cut after segment i (full)
            end = L if mode == sonic.NEXUS_CAUSAL_SEGMENTS else t
            for layer in range(nl):
                Ow, lw = _oracle_rows(Qall[:, nexus], K[:, :end], V[:, :end], role_all[:end],
                                      seg_all[:end], np.asarray(nexus), mode, layer)
                H.check_close(H.f64(O[layer]), Ow, f"segment {i} layer {layer}")
                np.testing.assert_allclose(H.f64(lse[layer]), lw, rtol=0, atol=2e-3)
        # incremental compaction: body_i goes, Nexus_i joins the retained cache
        cK, cV, c_role, c_seg = _compact(kK, kV, k_role, k_seg, len(kept) + nk)
        kept += nexus
        idx = torch.as_tensor(kept, device=H.dev()).long()
        assert torch.equal(cK.view(torch.int16), K[:, idx].view(torch.int16)), f"K after {i}"
        assert torch.equal(cV.view(torch.int16), V[:, idx].view(torch.int16)), f"V after {i}"
        assert torch.equal(c_role, t_role[idx]) and torch.equal(c_seg, t_seg[idx])
    # the retained cache is exactly the rows the retention rule keeps
    assert kept == [r for r in range(L - d.curr_len) if role_all[r] != inputs.ROLE_BODY]

    # the current turn over the retained cache = the oracle over the whole S_aug
    cur = list(range(L - d.curr_len, L))
    rows = torch.as_tensor(cur, device=H.dev()).long()
    kK = torch.cat([cK, K[:, rows]], 1).contiguous()
    kV = torch.cat([cV, V[:, rows]], 1).contiguous()
    k_role = torch.cat([c_role, t_role[rows]]).contiguous()
    k_seg = torch.cat([c_seg, t_seg[rows]]).contiguous()
    O, lse = _prefill(Qall[:, rows].contiguous(), kK, kV, k_role, k_seg, d.curr_len, mode)
    for layer in range(nl):
        Ow, lw = _oracle_rows(Qall[:, cur], K, V, role_all, seg_all, np.asarray(cur), mode, layer)
        H.check_close(H.f64(O[layer]), Ow, f"current turn layer {layer}")
        np.testing.assert_allclose(H.f64(lse[layer]), lw, rtol=0, atol=2e-3)
