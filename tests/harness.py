"""Shared helpers of the GPU parity tests: device buffers for a dialogue batch,
calls into the C ABI through the binding, and oracle evaluation on the very
bytes the GPU consumed."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic

MAX_ABS = 1e-2     # attention tolerance: max |GPU - oracle|
REL_L2 = 5e-3      # attention tolerance: ||GPU - oracle||_2 / ||oracle||_2


def dev():
    return torch.device("cuda:0")


def f64(t: torch.Tensor) -> np.ndarray:
    return t.float().cpu().double().numpy()


def i32(a) -> torch.Tensor:
    return torch.as_tensor(np.asarray(a, dtype=np.int32)).to(dev())


def meta(batch: inputs.Batch):
    return (torch.from_numpy(batch.role).to(dev()), torch.from_numpy(batch.seg).to(dev()),
            i32(batch.k_start), i32(batch.k_len))


def check_close(got: np.ndarray, want: np.ndarray, what: str):
    err = np.abs(got - want)
    mx = float(err.max()) if err.size else 0.0
    den = float(np.linalg.norm(want))
    rel = float(np.linalg.norm(got - want) / den) if den > 0 else float(np.linalg.norm(got))
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    assert mx <= MAX_ABS, f"{what}: max-abs {mx:.3e} > {MAX_ABS}"
    assert rel <= REL_L2, f"{what}: rel-L2 {rel:.3e} > {REL_L2}"
    return mx, rel


def run_prefill(batch: inputs.Batch, hq: int, hkv: int, D: int, q_len=None, seed: int = 0,
                nexus_vis: int = sonic.NEXUS_FULL, n_layers: int = 1, with_lse: bool = True,
                K=None, V=None, Q=None, key_order: int = sonic.KEYS_AS_GIVEN,
                expect_status: int = 0, k_start=None, total_k_rows=None,
                with_mass: bool = False, o_offset: int = 0):
    """Prefill of the last q_len[b] rows of every sequence (all rows if None).
    o_offset > 0: O starts o_offset elements into a NaN-filled buffer whose
    layers are o_offset elements apart (res["O_buf"]).
    Returns a dict with the device tensors and the query layout."""
    role, seg, k_start_b, k_len = meta(batch)
    k_start = k_start_b if k_start is None else i32(k_start)
    T = batch.total if total_k_rows is None else total_k_rows
    if q_len is None:
        q_len = batch.k_len.copy()
    q_len = np.asarray(q_len, dtype=np.int32)
    q_start = np.concatenate([[0], np.cumsum(q_len)[:-1]]).astype(np.int32)
    Tq = int(q_len.sum())
    if K is None:
        K = inputs.randn((n_layers, T, hkv, D), seed=seed + 1, device=dev())
        V = inputs.randn((n_layers, T, hkv, D), seed=seed + 2, device=dev())
    if Q is None:
        Q = inputs.randn((n_layers, Tq, hq, D), seed=seed + 3, device=dev())
    O_buf = None
    if o_offset:
        n = Tq * hq * D
        O_buf = torch.full((n_layers * (n + o_offset) + o_offset,), float("nan"),
                           dtype=torch.bfloat16, device=dev())
        O = O_buf.as_strided((n_layers, Tq, hq, D), (n + o_offset, hq * D, D, 1),
                             storage_offset=o_offset)
    else:
        O = torch.full_like(Q, float("nan"))
    lse = torch.full((n_layers, Tq, hq), float("nan"), device=dev()) if with_lse else None
    mass = torch.full((n_layers, Tq, hq), float("nan"), device=dev()) if with_mass else None
    status = torch.zeros(1, dtype=torch.int32, device=dev())
    sonic.sonic_attn_prefill(Q, K, V, seg, role, O, k_start=k_start, k_len=k_len,
                             q_start=i32(q_start), q_len=i32(q_len),
                             max_q_len=int(q_len.max()), max_k_len=int(batch.k_len.max()),
                             nexus_vis=nexus_vis, lse=lse, status=status, key_order=key_order,
                             nexus_mass=mass)
    torch.cuda.synchronize()
    assert sonic.read_status(status) == expect_status
    return dict(K=K, V=V, Q=Q, O=O, lse=lse, mass=mass, q_len=q_len, q_start=q_start, O_buf=O_buf)


def oracle_prefill_rows(batch: inputs.Batch, res: dict, b: int, rows, layer: int = 0,
                        nexus_vis: int = oracle.NEXUS_FULL):
    """Oracle output for query rows `rows` (indices into sequence b's query
    block) on the bytes the GPU read."""
    ks, kl = int(batch.k_start[b]), int(batch.k_len[b])
    ql, qs = int(res["q_len"][b]), int(res["q_start"][b])
    rows = np.asarray(rows, dtype=np.int64)
    K = f64(res["K"][layer, ks:ks + kl])
    V = f64(res["V"][layer, ks:ks + kl])
    Q = f64(res["Q"][layer, qs + rows])
    pos = kl - ql + rows
    O, lse = oracle.attn_masked(Q, K, V, batch.role[ks:ks + kl], batch.seg[ks:ks + kl], pos,
                                nexus_mode=nexus_vis)
    return O, lse, f64(res["O"][layer, qs + rows]), (
        None if res["lse"] is None else f64(res["lse"][layer, qs + rows]))


def oracle_mass_rows(batch: inputs.Batch, res: dict, b: int, rows, layer: int = 0,
                     nexus_vis: int = oracle.NEXUS_FULL):
    """Oracle attention mass on Nexus keys for query rows `rows` of sequence
    b, and the GPU's."""
    ks, kl = int(batch.k_start[b]), int(batch.k_len[b])
    ql, qs = int(res["q_len"][b]), int(res["q_start"][b])
    rows = np.asarray(rows, dtype=np.int64)
    K = f64(res["K"][layer, ks:ks + kl])
    Q = f64(res["Q"][layer, qs + rows])
    want = oracle.nexus_mass(Q, K, batch.role[ks:ks + kl], batch.seg[ks:ks + kl], kl - ql + rows,
                             nexus_mode=nexus_vis)
    return want, f64(res["mass"][layer, qs + rows])
