"""Pins for the CPU oracle, against things the paper and the mathematics fix.

None of these compare the oracle with itself: the mask is checked against a
matrix built from the paper's index sets rule by rule (tests/paper_rules.py),
attention against torch's scaled-dot-product attention in float64 on the CPU
and against closed forms, retention against the dialogue recipe, and the
three parts against one another through the equivalences the paper implies.
The mutant tests plant plausible mistakes in a copy of the oracle source and
check that these pins catch each one.
"""
import math
import os
import shutil

import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs
from tests.paper_rules import retained_positions, rule_mask

ORC = oracle.default


def _dialogues():
    rng = np.random.default_rng(7)
    ds = [inputs.tiny_ref()[0].dialogues[0],
          inputs.Dialogue(3, [], 5),                 # no history (h = 0)
          inputs.Dialogue(0, [(4, 0), (0, 3)], 2),    # K_i = 0, empty body, no system
          inputs.Dialogue(2, [(1, 1)] * 4, 1)]        # length-1 pieces
    ds += [inputs.random_dialogue(rng) for _ in range(25)]
    return ds


def _qkv(L, hq, hkv, d, seed, nq=None):
    g = torch.Generator().manual_seed(seed)
    Q = torch.randn(L if nq is None else nq, hq, d, generator=g, dtype=torch.float64)
    K = torch.randn(L, hkv, d, generator=g, dtype=torch.float64)
    V = torch.randn(L, hkv, d, generator=g, dtype=torch.float64)
    return Q.numpy(), K.numpy(), V.numpy()


def _sdpa(Q, K, V, add_mask, scale=None):
    """torch SDPA in float64: Q [n, Hq, D], K/V [L, Hkv, D] (GQA expanded)."""
    hq, hkv = Q.shape[1], K.shape[1]
    G = hq // hkv
    q = torch.from_numpy(Q).permute(1, 0, 2)
    k = torch.from_numpy(K).repeat_interleave(G, dim=1).permute(1, 0, 2)
    v = torch.from_numpy(V).repeat_interleave(G, dim=1).permute(1, 0, 2)
    m = torch.from_numpy(add_mask)
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=m, scale=scale)
    return o.permute(1, 0, 2).numpy()


# ---------------------------------------------------------------- mask (Sec. 3.2)

@pytest.mark.parametrize("mode", [oracle.NEXUS_FULL, oracle.NEXUS_CAUSAL_SEGMENTS])
def test_mask_equals_rule_by_rule_matrix(mode):
    for d in _dialogues():
        role, seg = d.arrays()
        vis = ORC().visibility(role, seg, mode)
        M = rule_mask(d, causal_segments=(mode == oracle.NEXUS_CAUSAL_SEGMENTS))
        assert np.array_equal(vis, M == 0.0), d


def test_tiny_ref_visible_pair_count():
    # L = 148: 16 sys, 3 x (32 body + 4 Nexus), 24 current.  Count by hand:
    #  sys rows see the causal prefix: sum_{p<16} (p+1) = 136
    #  body row at offset j of a segment: earlier sys + earlier Nexus + j+1 own body
    #  Nexus rows: sys + own body + all 12 Nexus
    #  current rows: sys + 12 Nexus + causal own
    d = inputs.tiny_ref()[0].dialogues[0]
    total = sum(p + 1 for p in range(16))
    for i in range(3):
        total += sum(16 + 4 * i + j + 1 for j in range(32))
        total += 4 * (16 + 32 + 12)
    total += sum(16 + 12 + j + 1 for j in range(24))
    role, seg = d.arrays()
    assert ORC().visibility(role, seg).sum() == total == 5332


def test_mask_random_roles_total():
    # The per-pair rule is total: arbitrary role/segment arrays are accepted,
    # and every row sees itself (q = p is visible in every branch of the rule).
    rng = np.random.default_rng(3)
    role = rng.integers(0, 4, 40).astype(np.uint8)
    seg = rng.integers(0, 5, 40).astype(np.int32)
    vis = ORC().visibility(role, seg)
    assert vis.diagonal().all()


# ----------------------------------------------------------- attention

@pytest.mark.parametrize("mode", [oracle.NEXUS_FULL, oracle.NEXUS_CAUSAL_SEGMENTS])
def test_attention_equals_sdpa_with_rule_matrix(mode):
    for i, d in enumerate(_dialogues()[:12]):
        role, seg = d.arrays()
        L = d.length
        Q, K, V = _qkv(L, 4, 2, 16, seed=i)
        O, _ = ORC().attn_masked(Q, K, V, role, seg, np.arange(L), nexus_mode=mode)
        M = rule_mask(d, causal_segments=(mode == oracle.NEXUS_CAUSAL_SEGMENTS))
        ref = _sdpa(Q, K, V, M)
        np.testing.assert_allclose(O, ref, rtol=1e-12, atol=1e-12)


def test_zero_history_is_causal_attention():
    d = inputs.Dialogue(37, [], 29)
    role, seg = d.arrays()
    Q, K, V = _qkv(d.length, 8, 2, 32, seed=11)
    O, lse = ORC().attn_masked(Q, K, V, role, seg, np.arange(d.length))
    hq, G = 8, 4
    q = torch.from_numpy(Q).permute(1, 0, 2)
    k = torch.from_numpy(K).repeat_interleave(G, 1).permute(1, 0, 2)
    v = torch.from_numpy(V).repeat_interleave(G, 1).permute(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True)
    np.testing.assert_allclose(O, ref.permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)
    # lse against a log-sum-exp of the causal scores
    s = torch.einsum("hpd,hqd->hpq", q, k) / math.sqrt(32)
    s = s.masked_fill(torch.triu(torch.ones(d.length, d.length, dtype=torch.bool), 1), -math.inf)
    np.testing.assert_allclose(lse, torch.logsumexp(s, -1).T.numpy(), rtol=1e-12, atol=1e-12)


def test_zero_keys_give_mean_of_visible_values():
    d = inputs.tiny_ref()[0].dialogues[0]
    role, seg = d.arrays()
    L = d.length
    Q, _, V = _qkv(L, 2, 1, 8, seed=5)
    K = np.zeros((L, 1, 8))
    O, lse = ORC().attn_masked(Q, K, V, role, seg, np.arange(L))
    vis = rule_mask(d) == 0.0
    for p in range(L):
        want = V[vis[p], 0, :].mean(axis=0)
        np.testing.assert_allclose(O[p, 0], want, rtol=1e-12, atol=1e-12)
        assert abs(lse[p, 0] - math.log(vis[p].sum())) < 1e-12


def test_one_hot_values_read_out_the_mask():
    d = inputs.Dialogue(3, [(5, 2), (4, 3)], 4)
    role, seg = d.arrays()
    L = d.length  # 21 <= D
    D = 32
    Q, _, _ = _qkv(L, 1, 1, D, seed=2)
    K = np.zeros((L, 1, D))
    V = np.zeros((L, 1, D))
    V[np.arange(L), 0, np.arange(L)] = 1.0
    O, _ = ORC().attn_masked(Q, K, V, role, seg, np.arange(L))
    vis = rule_mask(d) == 0.0
    for p in range(L):
        want = np.zeros(D)
        want[:L][vis[p]] = 1.0 / vis[p].sum()
        np.testing.assert_allclose(O[p, 0], want, rtol=1e-13, atol=1e-13)


def test_gqa_equals_replicated_mha():
    d = inputs.Dialogue(6, [(9, 3), (7, 2)], 8)
    role, seg = d.arrays()
    Q, K, V = _qkv(d.length, 6, 2, 16, seed=9)
    O, lse = ORC().attn_masked(Q, K, V, role, seg, np.arange(d.length))
    Kr, Vr = np.repeat(K, 3, axis=1), np.repeat(V, 3, axis=1)
    O2, lse2 = ORC().attn_masked(Q, Kr, Vr, role, seg, np.arange(d.length))
    np.testing.assert_array_equal(O, O2)
    np.testing.assert_array_equal(lse, lse2)
    # and head h reads KV head h // 3: permuting the query heads inside a group
    # leaves each output head's values with its own group
    for h in range(6):
        Oh, _ = ORC().attn_masked(Q[:, h:h + 1], K[:, h // 3:h // 3 + 1], V[:, h // 3:h // 3 + 1],
                                  role, seg, np.arange(d.length))
        np.testing.assert_array_equal(O[:, h:h + 1], Oh)


def test_explicit_scale_and_selected_rows():
    d = inputs.Dialogue(4, [(6, 2)], 5)
    role, seg = d.arrays()
    Q, K, V = _qkv(d.length, 2, 1, 8, seed=4)
    rows = np.array([d.length - 1, 0, 7])
    O, _ = ORC().attn_masked(Q[rows], K, V, role, seg, rows, scale=0.37)
    ref = _sdpa(Q[rows], K, V, rule_mask(d)[rows], scale=0.37)
    np.testing.assert_allclose(O, ref, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------- retention

def test_retained_length_invariant():
    for d in _dialogues():
        b = inputs.Batch([d])
        off, ret_len, src = ORC().retain(b.k_start, b.k_len, b.role)
        assert ret_len[0] == d.recipe_retained == d.sys_len + sum(k for _, k in d.segments) + d.curr_len
        assert list(src) == retained_positions(d)


def test_retention_offsets_with_reserve_and_batch():
    rng = np.random.default_rng(1)
    ds = [inputs.random_dialogue(rng) for _ in range(9)]
    b = inputs.Batch(ds)
    reserve = rng.integers(0, 5, len(ds))
    off, ret_len, src = ORC().retain(b.k_start, b.k_len, b.role, reserve)
    want_off = np.concatenate([[0], np.cumsum([d.recipe_retained + r for d, r in zip(ds, reserve)])])
    np.testing.assert_array_equal(off, want_off)
    for i, d in enumerate(ds):
        got = src[off[i]:off[i] + ret_len[i]]
        np.testing.assert_array_equal(got, b.k_start[i] + np.array(retained_positions(d), dtype=np.int64))
        assert (src[off[i] + ret_len[i]:off[i + 1]] == -1).all()


def test_compact_copy_bytes():
    rng = np.random.default_rng(2)
    ds = [inputs.random_dialogue(rng) for _ in range(5)]
    b = inputs.Batch(ds)
    raw = rng.integers(0, 256, size=(3, b.total, 48), dtype=np.uint8)
    off, ret_len, src = ORC().retain(b.k_start, b.k_len, b.role)
    out = ORC().compact_copy(raw, off, ret_len, src, int(off[-1]))
    keep_rows = np.concatenate([b.k_start[i] + np.array(retained_positions(d), dtype=np.int64)
                                for i, d in enumerate(ds)])
    np.testing.assert_array_equal(out, raw[:, keep_rows, :])


# ------------------------------------------------- cross-part equivalences

def test_current_rows_equal_compacted_causal_and_decode():
    """For current-turn rows, attention over S_aug under the mask equals plain
    causal attention over the compacted sequence (bottom-right aligned) and
    equals decoding the current turn one token at a time."""
    for mode in (oracle.NEXUS_FULL, oracle.NEXUS_CAUSAL_SEGMENTS):
        d = inputs.Dialogue(5, [(11, 3), (6, 2), (9, 4)], 7)
        role, seg = d.arrays()
        L = d.length
        Q, K, V = _qkv(L, 4, 2, 16, seed=21)
        cur = np.arange(L - d.curr_len, L)
        O_full, lse_full = ORC().attn_masked(Q[cur], K, V, role, seg, cur, nexus_mode=mode)
        keep = np.array(retained_positions(d))
        Kc, Vc = K[keep], V[keep]
        R = len(keep)
        # causal over the compacted sequence, via torch (independent routine)
        causal = np.triu(np.full((d.curr_len, R), -np.inf), k=R - d.curr_len + 1)
        ref = _sdpa(Q[cur], Kc, Vc, causal)
        np.testing.assert_allclose(O_full, ref, rtol=1e-12, atol=1e-12)
        # the oracle's own masked attention over the compacted layout
        rr, rs = d.retained_arrays()
        O_c, lse_c = ORC().attn_masked(Q[cur], Kc, Vc, rr, rs, np.arange(R - d.curr_len, R),
                                       nexus_mode=mode)
        np.testing.assert_allclose(O_full, O_c, rtol=1e-12, atol=1e-12)
        # decode one token at a time
        for i in range(d.curr_len):
            n = R - d.curr_len + i + 1
            o, l = ORC().decode(Q[cur[i]], Kc[:n], Vc[:n])
            np.testing.assert_allclose(O_full[i], o, rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(lse_full[i], l, rtol=1e-12, atol=1e-12)


def test_nexus_modes_differ_only_on_nexus_rows():
    d = inputs.Dialogue(4, [(5, 3), (6, 2), (3, 3)], 6)
    role, seg = d.arrays()
    L = d.length
    Q, K, V = _qkv(L, 2, 1, 8, seed=8)
    Of, _ = ORC().attn_masked(Q, K, V, role, seg, np.arange(L), nexus_mode=oracle.NEXUS_FULL)
    Oc, _ = ORC().attn_masked(Q, K, V, role, seg, np.arange(L),
                              nexus_mode=oracle.NEXUS_CAUSAL_SEGMENTS)
    nexus_rows = role == oracle.ROLE_NEXUS
    np.testing.assert_array_equal(Of[~nexus_rows], Oc[~nexus_rows])
    last_seg = seg == seg[nexus_rows].max()
    differs = np.abs(Of - Oc).max(axis=(1, 2)) > 1e-9
    assert differs[nexus_rows & ~last_seg].all()


def test_decode_equals_unmasked_sdpa():
    Q, K, V = _qkv(50, 8, 2, 16, seed=31, nq=1)
    o, lse = ORC().decode(Q[0], K, V)
    ref = _sdpa(Q, K, V, np.zeros((1, 50)))
    np.testing.assert_allclose(o, ref[0], rtol=1e-12, atol=1e-12)
    o0, l0 = ORC().decode(Q[0], K[:0], V[:0])
    assert (o0 == 0).all() and np.isneginf(l0).all()


# ------------------------------------------- Nexus attention mass (Sec. 4.1, Eq. 9)

def _sdpa_nexus_share(Q, K, role, add_mask):
    """Share of the attention on Nexus keys through torch SDPA: with V the
    indicator of a Nexus key (one value channel), the output is the mass."""
    Vn = np.zeros((K.shape[0], K.shape[1], 1))
    Vn[role == inputs.ROLE_NEXUS] = 1.0
    return _sdpa(Q, K, Vn, add_mask, scale=1.0 / math.sqrt(Q.shape[2]))[:, :, 0]


@pytest.mark.parametrize("mode", [oracle.NEXUS_FULL, oracle.NEXUS_CAUSAL_SEGMENTS])
def test_nexus_mass_equals_sdpa_of_nexus_indicator(mode):
    for i, d in enumerate(_dialogues()[:12]):
        role, seg = d.arrays()
        Q, K, _ = _qkv(d.length, 6, 2, 16, seed=60 + i)
        mass = ORC().nexus_mass(Q, K, role, seg, np.arange(d.length), nexus_mode=mode)
        want = _sdpa_nexus_share(Q, K, role, rule_mask(d, mode == oracle.NEXUS_CAUSAL_SEGMENTS))
        np.testing.assert_allclose(mass, want, rtol=0, atol=1e-12)
        assert ((mass >= 0) & (mass <= 1)).all()


def test_nexus_mass_of_uniform_scores_counts_visible_nexus_keys():
    """K = 0: every visible key gets the same weight, so the mass is the
    share of Nexus keys among the keys the row sees."""
    for d in _dialogues()[:12]:
        role, seg = d.arrays()
        Q, _, _ = _qkv(d.length, 2, 1, 8, seed=8)
        K = np.zeros((d.length, 1, 8))
        mass = ORC().nexus_mass(Q, K, role, seg, np.arange(d.length))
        vis = rule_mask(d) == 0.0
        nexus = role == inputs.ROLE_NEXUS
        want = (vis & nexus[None, :]).sum(1) / vis.sum(1)
        np.testing.assert_allclose(mass, np.repeat(want[:, None], 2, 1), rtol=0, atol=1e-14)


def test_nexus_mass_zero_without_nexus_and_one_for_lone_nexus_rows():
    d = inputs.Dialogue(5, [(7, 0), (4, 0)], 6)          # no Nexus at all
    role, seg = d.arrays()
    Q, K, _ = _qkv(d.length, 2, 1, 8, seed=4)
    assert (ORC().nexus_mass(Q, K, role, seg, np.arange(d.length)) == 0).all()
    d = inputs.Dialogue(0, [(0, 3)], 0)                  # only Nexus rows
    role, seg = d.arrays()
    Q, K, _ = _qkv(d.length, 2, 1, 8, seed=4)
    assert (ORC().nexus_mass(Q, K, role, seg, np.arange(d.length)) == 1).all()


def test_decode_nexus_mass_equals_sdpa_and_current_rows_of_prefill():
    """Decode over a retained cache (system, Nexus, current rows): equal to
    SDPA of the Nexus indicator, and to the prefill mass of the last current
    row over the same cache (Sec. 3.2: it sees every retained row)."""
    d = inputs.Dialogue(6, [(0, 4), (0, 5), (0, 3)], 7)  # a retained cache
    role, seg = d.arrays()
    Q, K, _ = _qkv(d.length, 8, 2, 16, seed=33)
    m = ORC().decode_nexus_mass(Q[-1], K, role)
    np.testing.assert_allclose(m, _sdpa_nexus_share(Q[-1:], K, role, np.zeros((1, d.length)))[0],
                               rtol=0, atol=1e-12)
    mp = ORC().nexus_mass(Q[-1:], K, role, seg, np.array([d.length - 1]))
    np.testing.assert_allclose(m, mp[0], rtol=0, atol=1e-13)
    assert (ORC().decode_nexus_mass(Q[-1], K[:0], role[:0]) == 0).all()


# ------------------------------------------- role-routed projections (Sec. 3.1)

def _routed_inputs(T, d_in, d_out, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((T, d_in))
    W = rng.standard_normal((d_out, d_in))
    Wn = rng.standard_normal((d_out, d_in))
    role = rng.choice([inputs.ROLE_SYS, inputs.ROLE_BODY, inputs.ROLE_NEXUS, inputs.ROLE_CURR],
                      T).astype(np.uint8)
    return X, W, Wn, role


def test_routed_linear_equals_matmul_per_role():
    """Nexus rows through W_nexus, all others through W: numpy matmuls of the
    two row subsets (d_in != d_out, so a transposed weight fails)."""
    X, W, Wn, role = _routed_inputs(37, 24, 40, seed=1)
    Y = ORC().routed_linear(X, W, Wn, role)
    nex = role == inputs.ROLE_NEXUS
    np.testing.assert_allclose(Y[nex], X[nex] @ Wn.T, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(Y[~nex], X[~nex] @ W.T, rtol=1e-12, atol=1e-12)
    assert nex.any() and (~nex).any()


def test_routed_linear_special_cases():
    X, W, Wn, role = _routed_inputs(20, 16, 8, seed=2)
    # one weight for both roles: a plain linear layer
    np.testing.assert_allclose(ORC().routed_linear(X, W, W, role), X @ W.T, rtol=1e-12,
                               atol=1e-12)
    # identity weights read the inputs back (d_in = d_out)
    I = np.eye(16)
    np.testing.assert_array_equal(ORC().routed_linear(X, I, 2 * I, role),
                                  np.where((role == inputs.ROLE_NEXUS)[:, None], 2 * X, X))
    assert ORC().routed_linear(X[:0], W, Wn, role[:0]).shape == (0, 8)


# ------------------------------------------------------------ mutants

_MUTANTS = {
    # Eq. 4 dropped: bodies of earlier segments stay visible
    "no_body_removal": ("return seg[q] == seg[p] && q <= p;", "return q <= p;"),
    # off-by-one in Eq. 3: a token no longer sees itself
    "strict_causal": ("    return q <= p;\n}", "    return q < p;\n}"),
    # Eq. 5 dropped: Nexus tokens causal among themselves
    "no_nexus_bidir": ("            return 1;", "            return q <= p;"),
    # wrong grouped-query head mapping
    "gqa_modulo": ("int32_t hk = h / G;\n            const double *qv = Q",
                   "int32_t hk = h % Hkv;\n            const double *qv = Q"),
    # missing softmax scale
    "no_scale": ("                s *= scale;\n                s_buf[q] = s;",
                 "                s_buf[q] = s;"),
    # retention keeps the bodies
    "keep_bodies": ("if (role[row] != ORC_BODY) {", "if (role[row] != 255) {"),
    # Nexus mass counts every retained role, not just Nexus keys
    "mass_any_retained": ("if (role[q] == ORC_NEXUS)\n                    nexus += w;",
                          "if (role[q] != ORC_BODY)\n                    nexus += w;"),
    # Nexus mass of a decode step over the current-turn rows instead
    "decode_mass_curr": ("if (role[t] == ORC_NEXUS)", "if (role[t] == ORC_CURR)"),
    # role routing keyed on body rows instead of Nexus rows
    "route_body": ("const double *w = role[t] == ORC_NEXUS ? W_nexus : W;",
                   "const double *w = role[t] == ORC_BODY ? W_nexus : W;"),
    # weight read transposed
    "route_transposed": ("acc += x[k] * wn[k];", "acc += x[k] * w[(int64_t)k * d_out + n];"),
    # Nexus mass ignores the mask (every key's weight in the denominator)
    "mass_unmasked": ("            double all = 0.0, nexus = 0.0;\n            for (int64_t q = 0; q < L; ++q) {\n                if (s_buf[q] == -INFINITY)\n                    continue;",
                      "            double all = 0.0, nexus = 0.0;\n            for (int64_t q = 0; q < L; ++q) {\n                if (s_buf[q] == -INFINITY)\n                    s_buf[q] = m;"),
}


def _run_pins(orc):
    """A subset of the pins above, run against a given oracle build; returns
    the names of the pins that fail."""
    failed = []
    ds = _dialogues()[:10]
    for d in ds:
        role, seg = d.arrays()
        if not np.array_equal(orc.visibility(role, seg), rule_mask(d) == 0.0):
            failed.append("mask")
            break
    for i, d in enumerate(ds[:6]):
        role, seg = d.arrays()
        Q, K, V = _qkv(d.length, 4, 2, 16, seed=i)
        O, _ = orc.attn_masked(Q, K, V, role, seg, np.arange(d.length))
        if not np.allclose(O, _sdpa(Q, K, V, rule_mask(d)), rtol=1e-10, atol=1e-10):
            failed.append("attention")
            break
    for d in ds:
        b = inputs.Batch([d])
        _, ret_len, _ = orc.retain(b.k_start, b.k_len, b.role)
        if ret_len[0] != d.recipe_retained:
            failed.append("retention")
            break
    for i, d in enumerate(ds[:6]):
        role, seg = d.arrays()
        Q, K, _ = _qkv(d.length, 4, 2, 16, seed=40 + i)
        mass = orc.nexus_mass(Q, K, role, seg, np.arange(d.length))
        if not np.allclose(mass, _sdpa_nexus_share(Q, K, role, rule_mask(d)), rtol=0, atol=1e-12):
            failed.append("nexus mass")
            break
    q, K, _ = _qkv(40, 4, 2, 16, seed=47, nq=1)
    role = np.random.default_rng(3).choice([0, 2, 3], 40).astype(np.uint8)
    if not np.allclose(orc.decode_nexus_mass(q[0], K, role),
                       _sdpa_nexus_share(q, K, role, np.zeros((1, 40)))[0], rtol=0, atol=1e-12):
        failed.append("decode nexus mass")
    X, W, Wn, role = _routed_inputs(23, 12, 20, seed=5)
    Y = orc.routed_linear(X, W, Wn, role)
    nex = role == inputs.ROLE_NEXUS
    if not (np.allclose(Y[nex], X[nex] @ Wn.T) and np.allclose(Y[~nex], X[~nex] @ W.T)):
        failed.append("routed linear")
    return failed


def test_pins_pass_on_oracle():
    assert _run_pins(ORC()) == []


@pytest.mark.parametrize("name", sorted(_MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(os.path.dirname(oracle.__file__), "sonic_oracle.c")).read()
    old, new = _MUTANTS[name]
    # the attention loops of orc_attn_masked and orc_nexus_mass share some
    # sites: a mutation is planted in every copy of its site
    assert src.count(old) >= 1, f"mutation site for {name} not found"
    mutant = tmp_path / f"mutant_{name}.c"
    mutant.write_text(src.replace(old, new))
    so = oracle.compile_source(str(mutant), str(tmp_path / f"mutant_{name}.so"))
    assert _run_pins(oracle.Oracle(so)) != []
