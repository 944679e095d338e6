"""GPU parity of sonic_compact_kv (retention rule) against the oracle: bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _bytes(t: torch.Tensor) -> np.ndarray:
    nl = t.shape[0]
    u8 = t.contiguous().view(torch.uint8) if t.element_size() == 1 else \
        t.contiguous().view(torch.int16 if t.element_size() == 2 else torch.int32)
    return u8.cpu().numpy().view(np.uint8).reshape(nl, t.shape[1], -1)


def _run(batch, K, V, reserve=None, cap=None, want_meta=True):
    role, seg, k_start, k_len = H.meta(batch)
    nl = K.shape[0]
    res = None if reserve is None else H.i32(reserve)
    total = sum(d.recipe_retained for d in batch.dialogues) + (0 if reserve is None else int(np.sum(reserve)))
    cap = total if cap is None else cap
    oK = torch.zeros((nl, cap) + tuple(K.shape[2:]), dtype=K.dtype, device=H.dev())
    oV = torch.zeros_like(oK)
    offsets = torch.full((batch.B + 1,), -7, dtype=torch.int32, device=H.dev())
    ret_len = torch.full((batch.B,), -7, dtype=torch.int32, device=H.dev())
    src_idx = torch.full((max(cap, 1),), -7, dtype=torch.int32, device=H.dev())
    o_role = torch.full((max(cap, 1),), 77, dtype=torch.uint8, device=H.dev()) if want_meta else None
    o_seg = torch.full((max(cap, 1),), -7, dtype=torch.int32, device=H.dev()) if want_meta else None
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_compact_kv(K, V, seg, role, oK, oV, offsets, k_start=k_start, k_len=k_len,
                           reserve=res, ret_len=ret_len, src_idx=src_idx, out_role=o_role,
                           out_seg=o_seg, status=status)
    torch.cuda.synchronize()
    return dict(oK=oK, oV=oV, offsets=offsets, ret_len=ret_len, src_idx=src_idx, o_role=o_role,
                o_seg=o_seg, status=sonic.read_status(status), cap=cap)


def _check(batch, K, V, r, reserve=None):
    off, ret_len, src = oracle.retain(batch.k_start, batch.k_len, batch.role, reserve)
    assert r["status"] == 0
    assert r["offsets"].cpu().numpy().tolist() == off.tolist()
    assert r["ret_len"].cpu().numpy().tolist() == ret_len.tolist()
    np.testing.assert_array_equal(r["src_idx"].cpu().numpy()[:len(src)], src)
    if r["o_role"] is not None:
        keep = src >= 0
        np.testing.assert_array_equal(r["o_role"].cpu().numpy()[:len(src)][keep], batch.role[src[keep]])
        np.testing.assert_array_equal(r["o_seg"].cpu().numpy()[:len(src)][keep], batch.seg[src[keep]])
        assert (r["o_seg"].cpu().numpy()[:len(src)][~keep] == -1).all()
    for name, raw in (("oK", K), ("oV", V)):
        want = oracle.compact_copy(_bytes(raw), off, ret_len, src, r["cap"])
        got = _bytes(r[name])
        for b in range(batch.B):
            sl = slice(off[b], off[b] + ret_len[b])
            assert np.array_equal(got[:, sl], want[:, sl]), f"{name} seq {b}"
            # reserve rows untouched
            rs = slice(off[b] + ret_len[b], off[b + 1])
            assert not got[:, rs].any()


def test_tiny_reference_fp32():
    batch, hd = inputs.tiny_ref()
    K = inputs.randn((1, batch.total, hd.hkv, hd.d), seed=1, dtype=torch.float32, device=H.dev())
    V = inputs.randn((1, batch.total, hd.hkv, hd.d), seed=2, dtype=torch.float32, device=H.dev())
    r = _run(batch, K, V, reserve=[8])
    _check(batch, K, V, r, reserve=[8])
    assert int(r["ret_len"][0]) == 52


def test_random_ragged_batch_with_reserve():
    rng = np.random.default_rng(5)
    ds = [inputs.random_dialogue(rng, max_segments=7, max_body=300, max_nexus=20) for _ in range(13)]
    ds.append(inputs.Dialogue(0, [(50, 0)], 0))   # retains nothing
    ds.append(inputs.Dialogue(0, [], 0))          # empty sequence
    batch = inputs.Batch(ds)
    reserve = rng.integers(0, 9, batch.B)
    K = inputs.randn((3, batch.total, 2, 64), seed=3, device=H.dev())
    V = inputs.randn((3, batch.total, 2, 64), seed=4, device=H.dev())
    r = _run(batch, K, V, reserve=reserve)
    _check(batch, K, V, r, reserve=reserve)


def test_capacity_overflow_sets_status_and_stays_in_bounds():
    batch = inputs.Batch([inputs.Dialogue(10, [(20, 5)], 10)] * 3)
    K = inputs.randn((1, batch.total, 1, 64), seed=3, device=H.dev())
    r = _run(batch, K, K, cap=40)
    assert r["status"] == 4  # SONIC_ERR_CAPACITY
    off, ret_len, src = oracle.retain(batch.k_start, batch.k_len, batch.role)
    got = _bytes(r["oK"])
    want = oracle.compact_copy(_bytes(K), off, ret_len, src, int(off[-1]))
    assert np.array_equal(got[:, :40], want[:, :40])


def test_layout_check():
    d = inputs.Dialogue(4, [(6, 2)], 3)
    batch = inputs.Batch([d])
    batch.seg[5] = 0      # a body row in segment 0
    K = inputs.randn((1, batch.total, 1, 64), seed=3, device=H.dev())
    r = _run(batch, K, K)
    assert r["status"] == 7


def test_masked_prefill_workload_all_layers():
    """Batch 8, L = 5632 -> 1536 retained rows, 32 layers, 8 KV heads, D = 128:
    offsets and source rows checked in full, bytes on four layers."""
    batch, hd = inputs.masked_prefill()
    shape = (hd.n_layers, batch.total, hd.hkv, hd.d)
    K = inputs.randn(shape, seed=41, device=H.dev())
    V = inputs.randn(shape, seed=42, device=H.dev())
    r = _run(batch, K, V, want_meta=False)
    assert r["status"] == 0
    off, ret_len, src = oracle.retain(batch.k_start, batch.k_len, batch.role)
    assert r["offsets"].cpu().numpy().tolist() == off.tolist()
    assert (ret_len == 1536).all()
    np.testing.assert_array_equal(r["src_idx"].cpu().numpy(), src)
    for layer in (0, 9, 22, 31):
        for name, raw in (("oK", K), ("oV", V)):
            want = oracle.compact_copy(_bytes(raw[layer:layer + 1]), off, ret_len, src, int(off[-1]))
            assert np.array_equal(_bytes(r[name][layer:layer + 1]), want), f"{name} layer {layer}"


@pytest.mark.parametrize("nexus_div", [2, 5])
def test_long_ragged_histories_two_layers(nexus_div):
    """The 64 long ragged dialogues (turns ~U[4,32] of ~U[64,1024] tokens, 256
    system tokens, Nexus = ceil(len/2) or ceil(len/5) per history turn, 8 KV
    heads, D = 128): their raw S_aug rows compacted for two layers, offsets,
    source rows and every byte of both layers checked."""
    batch, hd = inputs.long_ragged(nexus_div)
    shape = (2, batch.total, hd.hkv, hd.d)
    K = inputs.randn(shape, seed=50 + nexus_div, device=H.dev())
    V = inputs.randn(shape, seed=60 + nexus_div, device=H.dev())
    r = _run(batch, K, V, want_meta=False)
    assert r["status"] == 0
    off, ret_len, src = oracle.retain(batch.k_start, batch.k_len, batch.role)
    assert r["offsets"].cpu().numpy().tolist() == off.tolist()
    assert ret_len.tolist() == [d.recipe_retained for d in batch.dialogues]
    np.testing.assert_array_equal(r["src_idx"].cpu().numpy(), src)
    for layer in (0, 1):
        for name, raw in (("oK", K), ("oV", V)):
            want = oracle.compact_copy(_bytes(raw[layer:layer + 1]), off, ret_len, src,
                                       int(off[-1]))
            assert np.array_equal(_bytes(r[name][layer:layer + 1]), want), f"{name} layer {layer}"


def test_many_sequences_and_long_pieces():
    """1,100 sequences (the base scan runs over more than one 512-wide block
    pass) plus one sequence of about 70,000 rows (each of its 64 scan pieces
    spans several 512-row passes), reserve rows on every sequence."""
    rng = np.random.default_rng(8)
    ds = [inputs.random_dialogue(rng, max_segments=3, max_body=40, max_nexus=6, max_sys=8,
                                 max_curr=9) for _ in range(1100)]
    ds.insert(517, inputs.Dialogue(33, [(700, 13), (1, 0), (0, 9)] * 99 + [(1500, 1)], 77))
    batch = inputs.Batch(ds)
    reserve = rng.integers(0, 5, batch.B)
    K = inputs.randn((1, batch.total, 1, 64), seed=6, device=H.dev())
    V = inputs.randn((1, batch.total, 1, 64), seed=7, device=H.dev())
    r = _run(batch, K, V, reserve=reserve)
    _check(batch, K, V, r, reserve=reserve)


def test_sequence_outside_the_rows_is_refused():
    """k_start past the input rows: the sequence keeps nothing (ret_len 0) and
    the status word says SONIC_ERR_INVALID_ARGUMENT; the others are exact."""
    ds = [inputs.Dialogue(10, [(40, 5)], 8), inputs.Dialogue(6, [(30, 4), (12, 3)], 9)]
    batch = inputs.Batch(ds)
    K = inputs.randn((2, batch.total, 1, 64), seed=9, device=H.dev())
    role, seg, k_start, k_len = H.meta(batch)
    k_start = H.i32([int(batch.k_start[0]), batch.total + 50])
    cap = ds[0].recipe_retained
    oK = torch.zeros((2, cap, 1, 64), dtype=K.dtype, device=H.dev())
    oV = torch.zeros_like(oK)
    offsets = torch.full((3,), -7, dtype=torch.int32, device=H.dev())
    ret_len = torch.full((2,), -7, dtype=torch.int32, device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_compact_kv(K, K, seg, role, oK, oV, offsets, k_start=k_start, k_len=k_len,
                           ret_len=ret_len, status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 1
    assert ret_len.tolist() == [cap, 0] and offsets.tolist() == [0, cap, cap]
    keep = np.nonzero(batch.role[:int(batch.k_len[0])] != inputs.ROLE_BODY)[0]
    assert torch.equal(oK.view(torch.int16), K[:, torch.as_tensor(keep).long().to(H.dev())]
                       .view(torch.int16))
