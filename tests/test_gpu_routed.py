"""GPU parity of sonic_routed_linear (Sec. 3.1 role-routed projections)
against the oracle, on the very bf16 values the GPU read."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _weights(d_out, d_in, seed):
    """bf16 weights with unit-variance outputs for unit-variance inputs."""
    w = inputs.randn((d_out, d_in), seed=seed, device=H.dev()).float() / math.sqrt(d_in)
    return w.to(torch.bfloat16)


def _run(role, d_in, cols, scatter, seed, cache_rows=None, same_weights=False, x_pad=0):
    """Routed linear of T = len(role) rows into parts of the given widths;
    scattered parts go to rows dst_row[t] of buffers with cache_rows rows
    (a random injective map), the others to rows t."""
    T = len(role)
    d_out = sum(cols)
    Xfull = inputs.randn((T, d_in + x_pad), seed=seed, device=H.dev())
    X = Xfull[:, :d_in]
    W = _weights(d_out, d_in, seed + 1)
    Wn = W if same_weights else _weights(d_out, d_in, seed + 2)
    rng = np.random.default_rng(seed)
    cache_rows = cache_rows or T
    dst = rng.permutation(cache_rows)[:T].astype(np.int32)
    outs = []
    for c, sc in zip(cols, scatter):
        outs.append(torch.full((cache_rows if sc else T, c), float("nan"), dtype=torch.bfloat16,
                               device=H.dev()))
    role_t = torch.from_numpy(np.asarray(role, np.uint8)).to(H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_routed_linear(X, W, Wn, role_t, list(zip(outs, scatter)), dst_row=H.i32(dst),
                              status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 0
    return dict(X=X, W=W, Wn=Wn, role=np.asarray(role, np.uint8), dst=dst, outs=outs,
                cols=cols, scatter=scatter)


def _close(got, want, what):
    """Elementwise bound from the arithmetic: the fp32 sum differs from the
    exact one by far less than 2e-4 at these sizes (unit-variance outputs),
    and rounding it to bf16 (nearest even) moves it by at most half an ulp,
    2^-8 of its magnitude."""
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - want)
    bound = 2.0 ** -8 * np.abs(want) + 2e-4
    worst = int(np.argmax(err - bound))
    assert (err <= bound).all(), (f"{what}: |err| {err.flat[worst]:.3e} > "
                                  f"{bound.flat[worst]:.3e} at {np.unravel_index(worst, err.shape)}")
    rel = np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-30)
    assert rel <= 5e-3, f"{what}: rel-L2 {rel:.3e}"


def _gathered(r):
    """The GPU's Y [T, d_out] read back from the parts."""
    T = len(r["role"])
    ys = []
    for out, sc in zip(r["outs"], r["scatter"]):
        rows = torch.as_tensor(r["dst"] if sc else np.arange(T)).long().to(H.dev())
        ys.append(H.f64(out[rows]))
    return np.concatenate(ys, axis=1)


def _check(r, rows=None):
    rows = np.arange(len(r["role"])) if rows is None else np.asarray(rows)
    want = oracle.routed_linear(H.f64(r["X"][rows]), H.f64(r["W"]), H.f64(r["Wn"]),
                                r["role"][rows])
    got = _gathered(r)[rows]
    _close(got, want, "routed linear")
    # scattered parts: rows no token maps to stay untouched
    for out, sc in zip(r["outs"], r["scatter"]):
        if sc:
            free = np.setdiff1d(np.arange(out.shape[0]), r["dst"])
            assert torch.isnan(out[torch.as_tensor(free).long().to(H.dev())].float()).all()


def _roles(T, seed, p_nexus=0.3):
    rng = np.random.default_rng(seed)
    # runs of ordinary rows and Nexus rows, as in a dialogue's segments
    role = np.repeat(rng.choice([inputs.ROLE_BODY, inputs.ROLE_NEXUS, inputs.ROLE_CURR,
                                 inputs.ROLE_SYS], T // 7 + 1, p=[0.4, p_nexus, 0.3 - p_nexus / 2,
                                                                  0.3 - p_nexus / 2]), 7)[:T]
    return role.astype(np.uint8)


def test_small_partial_tiles():
    """T = 300 (ragged row tiles in both groups), d_out = 96 (one partial
    column tile), a scattered part."""
    _check(_run(_roles(300, 1), 128, [64, 32], [False, True], seed=3, cache_rows=700))


@pytest.mark.parametrize("T", [1, 127, 128, 129, 1000])
def test_qkv_parts_into_cache_rows(T):
    """QKV-shaped: Q (512 columns) to row t, K and V (128 each) to cache rows
    dst_row[t]; d_in = 512, three column tiles."""
    r = _run(_roles(T, T), 512, [512, 128, 128], [False, True, True], seed=5,
             cache_rows=2 * T + 3)
    _check(r)


@pytest.mark.parametrize("x_pad", [0, 64])
@pytest.mark.parametrize("which", ["none", "all"])
def test_one_group_empty(which, x_pad):
    """One role only: every 128-row slab is a run of X's rows, loaded from X
    itself (rows padded or not); nothing is copied."""
    role = np.full(777, inputs.ROLE_NEXUS if which == "all" else inputs.ROLE_CURR, np.uint8)
    _check(_run(role, 256, [256, 64], [False, True], seed=7, cache_rows=900, x_pad=x_pad))


def test_runs_and_copied_slabs_mixed():
    """Long runs of one role (slabs loaded from X) next to short alternating
    runs (slabs copied), group boundaries off the 128-row grid."""
    role = np.r_[np.full(300, inputs.ROLE_BODY), np.full(5, inputs.ROLE_NEXUS),
                 np.tile(np.r_[np.full(3, inputs.ROLE_CURR), np.full(4, inputs.ROLE_NEXUS)], 40),
                 np.full(260, inputs.ROLE_NEXUS), np.full(9, inputs.ROLE_SYS)].astype(np.uint8)
    _check(_run(role, 128, [128, 96], [False, True], seed=13, cache_rows=2000, x_pad=32))


def test_same_weights_is_a_plain_linear_layer_and_strided_x():
    """W_nexus = W (the routing changes nothing) and X rows with padding."""
    r = _run(_roles(500, 9), 192, [320], [False], seed=9, same_weights=True, x_pad=64)
    _check(r)
    plain = H.f64(r["X"]) @ H.f64(r["W"]).T
    _close(_gathered(r), plain, "plain linear")


def test_nexus_generation_projection_sampled_rows():
    """A Nexus-generation segment step at Llama-3-8B-like widths: 8 sequences
    of 256 body + 32 Nexus rows (T = 2304), d_model 4096, Q 4096 + K 1024 +
    V 1024 columns, K and V into cache rows; 96 rows checked against the
    oracle (all Nexus rows of one sequence and rows across both groups)."""
    role = np.tile(np.r_[np.full(256, inputs.ROLE_BODY), np.full(32, inputs.ROLE_NEXUS)],
                   8).astype(np.uint8)
    r = _run(role, 4096, [4096, 1024, 1024], [False, True, True], seed=11, cache_rows=3000)
    rows = np.unique(np.r_[np.arange(256, 288), np.arange(0, 2304, 37)])
    _check(r, rows)


def test_destination_rows_outside_a_part_are_reported():
    """dst_row values past the cache's rows (or negative) are not written: the
    status word says SONIC_ERR_CAPACITY and every row inside is still right."""
    role = _roles(200, 21)
    T, cache_rows = len(role), 300
    X = inputs.randn((T, 128), seed=21, device=H.dev())
    W, Wn = _weights(64, 128, 22), _weights(64, 128, 23)
    dst = np.random.default_rng(21).permutation(cache_rows)[:T].astype(np.int32)
    dst[[3, 77]] = [cache_rows + 5, -1]
    out = torch.full((cache_rows, 64), float("nan"), dtype=torch.bfloat16, device=H.dev())
    status = torch.zeros(1, dtype=torch.int32, device=H.dev())
    sonic.sonic_routed_linear(X, W, Wn, torch.from_numpy(role).to(H.dev()), [(out, True)],
                              dst_row=H.i32(dst), status=status)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == 4
    ok = np.setdiff1d(np.arange(T), [3, 77])
    want = oracle.routed_linear(H.f64(X), H.f64(W), H.f64(Wn), role)[ok]
    got = H.f64(out[torch.as_tensor(dst[ok]).long().to(H.dev())])
    _close(got, want, "rows inside the part")
