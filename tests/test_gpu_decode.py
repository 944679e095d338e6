"""GPU parity of sonic_attn_decode (one GQA step over the retained cache)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _decode(lens, hq, hkv, D, n_layers=1, chunk_len=0, seed=0, pad=37):
    """Random retained caches of the given lengths packed with `pad` junk rows
    between sequences; returns tensors and outputs."""
    lens = np.asarray(lens, dtype=np.int32)
    B = len(lens)
    starts = np.zeros(B, np.int32)
    t = pad
    for b in range(B):
        starts[b] = t
        t += int(lens[b]) + pad
    T = t
    K = inputs.randn((n_layers, T, hkv, D), seed=seed + 1, device=H.dev())
    V = inputs.randn((n_layers, T, hkv, D), seed=seed + 2, device=H.dev())
    # junk rows between sequences must never be read: make them non-finite
    mask = torch.ones(T, dtype=torch.bool)
    for b in range(B):
        mask[starts[b]:starts[b] + lens[b]] = False
    K[:, mask.to(H.dev())] = float("nan")
    V[:, mask.to(H.dev())] = float("inf")
    q = inputs.randn((n_layers, B, hq, D), seed=seed + 3, device=H.dev())
    O = torch.full_like(q, float("nan"))
    lse = torch.full((n_layers, B, hq), float("nan"), device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_decode(q, K, V, H.i32(lens), O, kv_start=H.i32(starts),
                            max_len=int(lens.max()) if B else 0, chunk_len=chunk_len, lse=lse,
                            status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    return dict(K=K, V=V, q=q, O=O, lse=lse, starts=starts, lens=lens)


def _check(r, pairs):
    for layer, b in pairs:
        s, n = int(r["starts"][b]), int(r["lens"][b])
        Oref, lref = oracle.decode(H.f64(r["q"][layer, b]), H.f64(r["K"][layer, s:s + n]),
                                   H.f64(r["V"][layer, s:s + n]))
        if n == 0:
            assert (r["O"][layer, b] == 0).all()
            assert torch.isneginf(r["lse"][layer, b]).all()
            continue
        H.check_close(H.f64(r["O"][layer, b]), Oref, f"layer {layer} seq {b}")
        np.testing.assert_allclose(H.f64(r["lse"][layer, b]), lref, rtol=0, atol=2e-3)


def test_decode_llama8b_workload_all_layers():
    """Batch 16, retained 640 + 1 new token, 32 layers, 32/8 heads, D = 128."""
    r = _decode([641] * 16, 32, 8, 128, n_layers=32, seed=3)
    _check(r, [(l, b) for l in (0, 13, 31) for b in range(16)])
    assert torch.isfinite(r["O"]).all()


@pytest.mark.parametrize("chunk_len", [0, 64, 256, 1024])
def test_ragged_lengths_and_splits(chunk_len):
    lens = [1, 63, 64, 65, 700, 2049, 0, 5000, 129]
    r = _decode(lens, 8, 2, 128, n_layers=2, chunk_len=chunk_len, seed=7)
    _check(r, [(l, b) for l in (0, 1) for b in range(len(lens))])


@pytest.mark.parametrize("hq,hkv,D", [(28, 4, 128), (2, 1, 64), (16, 16, 128), (32, 2, 64),
                                      (12, 4, 128)])
def test_head_shapes(hq, hkv, D):
    lens = [300, 1777, 4096]
    r = _decode(lens, hq, hkv, D, n_layers=1, seed=hq + D)
    _check(r, [(0, b) for b in range(3)])


def test_long_ragged_workload_sampled():
    """Batch 64 ragged dialogues (Nexus = ceil(len/2)), 32 layers, 32/8 heads."""
    batch, hd = inputs.long_ragged(2)
    lens = np.array([d.recipe_retained + 1 for d in batch.dialogues])
    r = _decode(lens, hd.hq, hd.hkv, hd.d, n_layers=4, seed=13, pad=0)
    _check(r, [(l, b) for l in (0, 3) for b in (0, 7, 31, 63)])
    assert torch.isfinite(r["O"]).all()
