"""GPU parity of sonic_attn_decode (one GQA step over the retained cache)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _decode(lens, hq, hkv, D, n_layers=1, chunk_len=0, seed=0, pad=37, with_mass=False,
            q=None):
    """Random retained caches of the given lengths packed with `pad` junk rows
    between sequences; returns tensors and outputs.  with_mass: random roles
    (system, Nexus, current) for the rows and the mass on Nexus rows."""
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
    if q is None:
        q = inputs.randn((n_layers, B, hq, D), seed=seed + 3, device=H.dev())
    O = torch.full_like(q, float("nan"))
    lse = torch.full((n_layers, B, hq), float("nan"), device=H.dev())
    role = mass = None
    if with_mass:
        # Nexus runs among system and current rows; junk rows carry any role
        rng = np.random.default_rng(seed + 4)
        role = np.repeat(rng.choice([inputs.ROLE_SYS, inputs.ROLE_NEXUS, inputs.ROLE_CURR],
                                    T // 8 + 1), 8)[:T].astype(np.uint8)
        role[rng.random(T) < 0.1] = inputs.ROLE_NEXUS
        role = torch.from_numpy(role).to(H.dev())
        mass = torch.full((n_layers, B, hq), float("nan"), device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_decode(q, K, V, H.i32(lens), O, kv_start=H.i32(starts),
                            max_len=int(lens.max()) if B else 0, chunk_len=chunk_len, lse=lse,
                            status=status, role=role, nexus_mass=mass)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    return dict(K=K, V=V, q=q, O=O, lse=lse, starts=starts, lens=lens, role=role, mass=mass)


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
                                      (12, 4, 128), (16, 4, 64), (14, 2, 64), (8, 8, 64),
                                      (12, 6, 64), (9, 3, 64)])
def test_head_shapes(hq, hkv, D):
    lens = [300, 1777, 4096]
    r = _decode(lens, hq, hkv, D, n_layers=1, seed=hq + D)
    _check(r, [(0, b) for b in range(3)])


@pytest.mark.parametrize("nexus_div", [2, 5])
def test_long_ragged_workload_sampled(nexus_div):
    """Batch 64 ragged dialogues, 32/8 heads, D = 128, both Nexus budgets:
    ceil(len/2) (50% compression) and ceil(len/5) (80%, Sec. 6 Table 1
    caption); sampled layers and sequences of a 4-layer launch."""
    batch, hd = inputs.long_ragged(nexus_div)
    lens = np.array([d.recipe_retained + 1 for d in batch.dialogues])
    r = _decode(lens, hd.hq, hd.hkv, hd.d, n_layers=4, seed=13 + nexus_div, pad=0)
    _check(r, [(l, b) for l in (0, 3) for b in (0, 7, 31, 63)])
    assert torch.isfinite(r["O"]).all()


def _check_mass(r, pairs, atol=2e-3):
    role = r["role"].cpu().numpy()
    for layer, b in pairs:
        s, n = int(r["starts"][b]), int(r["lens"][b])
        want = oracle.decode_nexus_mass(H.f64(r["q"][layer, b]), H.f64(r["K"][layer, s:s + n]),
                                        role[s:s + n])
        np.testing.assert_allclose(H.f64(r["mass"][layer, b]), want, rtol=0, atol=atol,
                                   err_msg=f"layer {layer} seq {b}")


@pytest.mark.parametrize("hq,hkv,D,chunk_len", [(28, 4, 128, 0), (32, 8, 128, 256),
                                                (8, 2, 64, 0), (8, 2, 64, 96)])
def test_nexus_mass(hq, hkv, D, chunk_len):
    """Attention mass on Nexus rows of a decode step, one chunk per sequence
    and split into chunks (merged by the combine kernel); O and lse as without
    the mass."""
    lens = [1, 63, 129, 700, 2049, 0, 5000]
    r = _decode(lens, hq, hkv, D, n_layers=2, chunk_len=chunk_len, seed=17, with_mass=True)
    pairs = [(l, b) for l in (0, 1) for b in range(len(lens))]
    _check(r, pairs)
    _check_mass(r, pairs)
    assert (r["mass"][:, 5] == 0).all()
    plain = _decode(lens, hq, hkv, D, n_layers=2, chunk_len=chunk_len, seed=17)
    assert torch.equal(plain["O"].view(torch.int16), r["O"].view(torch.int16))
    assert torch.equal(plain["lse"], r["lse"])


@pytest.mark.parametrize("D,chunk_len", [(128, 0), (128, 128), (64, 0)])
def test_nexus_mass_of_uniform_scores_is_the_nexus_share(D, chunk_len):
    """q = 0: every probability is 1, so the mass is the share of Nexus rows
    among the sequence's rows, up to fp32 rounding."""
    lens = [5, 128, 333, 4100]
    q = torch.zeros((1, len(lens), 8, D), dtype=torch.bfloat16, device=H.dev())
    r = _decode(lens, 8, 2, D, chunk_len=chunk_len, seed=19, with_mass=True, q=q)
    _check_mass(r, [(0, b) for b in range(len(lens))], atol=1e-6)


def test_empty_cache_outputs():
    """Every sequence empty (max_len = 0): O = 0, lse = -inf, mass = 0."""
    q = inputs.randn((2, 3, 4, 128), seed=1, device=H.dev())
    K = torch.zeros((2, 1, 2, 128), dtype=torch.bfloat16, device=H.dev())
    O = torch.full_like(q, float("nan"))
    lse = torch.full((2, 3, 4), float("nan"), device=H.dev())
    mass = torch.full((2, 3, 4), float("nan"), device=H.dev())
    role = torch.zeros(1, dtype=torch.uint8, device=H.dev())
    sonic.sonic_attn_decode(q, K, K, H.i32([0, 0, 0]), O, kv_start=H.i32([0, 0, 0]), max_len=0,
                            lse=lse, role=role, nexus_mass=mass)
    torch.cuda.synchronize()
    assert (O == 0).all() and torch.isneginf(lse).all() and (mass == 0).all()


def test_sequence_outside_the_cache_is_refused():
    """kv_start past the cache's rows: the sequence is refused
    (SONIC_ERR_INVALID_ARGUMENT), the others are computed as usual."""
    lens = np.array([300, 200, 129], np.int32)
    starts = np.array([0, 300, 10_000], np.int32)
    T, nl, hq, hkv, D = 500, 1, 8, 2, 128
    K = inputs.randn((nl, T, hkv, D), seed=31, device=H.dev())
    V = inputs.randn((nl, T, hkv, D), seed=32, device=H.dev())
    q = inputs.randn((nl, 3, hq, D), seed=33, device=H.dev())
    O = torch.full_like(q, float("nan"))
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_attn_decode(q, K, V, H.i32(lens), O, kv_start=H.i32(starts), max_len=300,
                            status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 1
    for b in (0, 1):
        s0, n = int(starts[b]), int(lens[b])
        Oref, _ = oracle.decode(H.f64(q[0, b]), H.f64(K[0, s0:s0 + n]), H.f64(V[0, s0:s0 + n]))
        H.check_close(H.f64(O[0, b]), Oref, f"seq {b}")


def test_very_long_cache():
    """One decode step over 500,000 retained rows (split into many chunks and
    merged), next to a one-row sequence."""
    r = _decode([500_000, 1], 8, 2, 128, n_layers=1, seed=41, pad=3)
    _check(r, [(0, 0), (0, 1)])
