"""The library's calls replayed from CUDA graphs: every call is stream-ordered
with caller-owned workspace and no host synchronisation, so a step can be
captured once and replayed.  Replays must equal the eager calls bit for bit."""
import numpy as np
import pytest
import torch

from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def test_per_layer_decode_graph_equals_batched_launch():
    """Four layers of a decode step as four per-layer launches captured in one
    graph, against one launch over all layers (same split length)."""
    nl, B, hq, hkv, D = 4, 6, 8, 2, 128
    lens = np.array([1, 100, 641, 1000, 2049, 300], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
    T = int(lens.sum())
    K = inputs.randn((nl, T, hkv, D), seed=1, device=H.dev())
    V = inputs.randn((nl, T, hkv, D), seed=2, device=H.dev())
    q = inputs.randn((nl, B, hq, D), seed=3, device=H.dev())
    lt, st = H.i32(lens), H.i32(starts)
    O_all = torch.empty_like(q)
    sonic.sonic_attn_decode(q, K, V, lt, O_all, kv_start=st, max_len=int(lens.max()),
                            chunk_len=512)
    O_g = torch.full_like(q, float("nan"))
    ws = [sonic.sonic_attn_decode(q[l:l + 1], K[l:l + 1], V[l:l + 1], lt, O_g[l:l + 1],
                                  kv_start=st, max_len=int(lens.max()), chunk_len=512)
          for l in range(nl)]
    O_g.fill_(float("nan"))
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(nl):
            sonic.sonic_attn_decode(q[l:l + 1], K[l:l + 1], V[l:l + 1], lt, O_g[l:l + 1],
                                    kv_start=st, max_len=int(lens.max()), chunk_len=512,
                                    workspace=ws[l])
    for _ in range(2):  # replays reuse the captured workspace and counters
        O_g.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(O_g.view(torch.int16), O_all.view(torch.int16))


def test_step_graph_equals_eager():
    """Compaction, prefill and decode of a small batch captured as one graph."""
    batch, hd = inputs.tiny_ref()
    d = batch.dialogues[0]
    L = d.length
    role, seg, ks, kl = H.meta(batch)
    K = inputs.randn((1, L, hd.hkv, hd.d), seed=4, device=H.dev())
    V = inputs.randn((1, L, hd.hkv, hd.d), seed=5, device=H.dev())
    Q = inputs.randn((1, L, hd.hq, hd.d), seed=6, device=H.dev())
    R = d.recipe_retained
    dec_len, dec_start = H.i32([R]), H.i32([0])  # made before the capture (host copies)

    def outputs():
        return (torch.zeros((1, R, hd.hkv, hd.d), dtype=torch.bfloat16, device=H.dev()),
                torch.zeros((1, R, hd.hkv, hd.d), dtype=torch.bfloat16, device=H.dev()),
                torch.zeros(2, dtype=torch.int32, device=H.dev()), torch.empty_like(Q),
                torch.empty((1, 1, hd.hq, hd.d), dtype=torch.bfloat16, device=H.dev()))

    def step(oK, oV, off, O, Od, ws=(None, None, None)):
        w0 = sonic.sonic_compact_kv(K, V, seg, role, oK, oV, off, k_start=ks, k_len=kl,
                                    workspace=ws[0])
        w1 = sonic.sonic_attn_prefill(Q, K, V, seg, role, O, k_start=ks, k_len=kl, q_start=ks,
                                      q_len=kl, max_q_len=L, max_k_len=L, workspace=ws[1])
        w2 = sonic.sonic_attn_decode(Q[:, L - 1:L], oK, oV, dec_len, Od, kv_start=dec_start,
                                     max_len=R, workspace=ws[2])
        return w0, w1, w2

    eager = outputs()
    ws = step(*eager)
    torch.cuda.synchronize()
    replay = outputs()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step(*replay, ws=ws)
    g.replay()
    torch.cuda.synchronize()
    for a, b in zip(eager, replay):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
