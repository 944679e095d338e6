"""GPU parity of sonic_attn_prefill (Sec. 3.2 masked attention) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


def _all_rows(batch, hq, hkv, D, mode=sonic.NEXUS_FULL, seed=0):
    res = H.run_prefill(batch, hq, hkv, D, seed=seed, nexus_vis=mode)
    for b in range(batch.B):
        n = int(batch.k_len[b])
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(n), nexus_vis=mode)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)


def test_tiny_reference_all_rows():
    batch, hd = inputs.tiny_ref()
    _all_rows(batch, hd.hq, hd.hkv, hd.d)


@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_random_dialogues_multi_tile(mode):
    rng = np.random.default_rng(11)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=120, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(4)]
    ds.append(inputs.Dialogue(5, [(300, 0), (1, 1), (0, 70)], 1))  # K_i = 0, tiny pieces
    _all_rows(inputs.Batch(ds), 4, 2, 128, mode=mode, seed=5)


def test_head_dim_64_and_gqa_ratios():
    rng = np.random.default_rng(3)
    ds = [inputs.random_dialogue(rng, max_segments=4, max_body=200, max_nexus=30) for _ in range(3)]
    _all_rows(inputs.Batch(ds), 6, 2, 64, seed=9)


def test_current_turn_over_compacted_cache():
    """Turn-by-turn form: queries = the current turn, keys = retained cache +
    current turn (bottom-right aligned)."""
    full = [inputs.Dialogue(40, [(200, 30), (150, 20), (90, 45)], 333),
            inputs.Dialogue(7, [(64, 64)] * 3, 129)]
    ret = inputs.Batch([inputs.Dialogue(d.sys_len, [(0, k) for _, k in d.segments], d.curr_len)
                        for d in full])
    q_len = [d.curr_len for d in full]
    res = H.run_prefill(ret, 8, 2, 128, q_len=q_len, seed=21)
    for b in range(ret.B):
        O, lse, got, got_lse = H.oracle_prefill_rows(ret, res, b, np.arange(q_len[b]))
        H.check_close(got, O, f"seq {b}")


def test_masked_prefill_workload_sampled_rows():
    """Batch 8, 32/8 heads, D = 128, L = 5632, every row (full mask); rows
    sampled across tiles, segment edges and the ragged end."""
    batch, hd = inputs.masked_prefill()
    res = H.run_prefill(batch, hd.hq, hd.hkv, hd.d, seed=31)
    L = int(batch.k_len[0])
    rows = np.unique(np.r_[0, 127, 128, 511, 512, 767, 799, 800, 2000, 4000, 5119, 5120, L - 1])
    for b in (0, 5):
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, rows)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)
    # every output is finite and the lse rows are all written
    assert torch.isfinite(res["O"]).all()
    assert torch.isfinite(res["lse"]).all()
