"""The work counts behind the benchmark's rates, checked on CPU against the
paper's mask built rule by rule (tests/paper_rules.py), not against the code
that produced them: the prefill rates divide 4 * D * Hq * (visible pairs) by
time, so a wrong pair count would misstate every TFLOP/s figure."""
import numpy as np
import pytest

import bench
from paper_2601_21927_gb300 import inputs
from tests import paper_rules


def _rule_pairs(d, rows, causal_segments):
    M = paper_rules.rule_mask(d, causal_segments=causal_segments)
    return int(np.isfinite(M[np.asarray(rows)]).sum())


@pytest.mark.parametrize("mode", [0, 1])
def test_visible_pair_count_equals_rule_matrix(mode):
    rng = np.random.default_rng(7)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=50, max_nexus=9, max_sys=20,
                                 max_curr=25) for _ in range(12)]
    ds.append(inputs.Dialogue(16, [(32, 4)] * 3, 24))        # the tiny dialogue
    ds.append(inputs.Dialogue(5, [(40, 0), (0, 6), (3, 3)], 9))  # K_i = 0, empty body
    for d in ds:
        role, seg = d.arrays()
        L = d.length
        for rows in (range(L), range(L - d.curr_len, L)):
            assert bench._visible_pairs(role, seg, rows, mode) == _rule_pairs(d, rows, mode == 1)


def test_masked_prefill_workload_pair_count():
    """The masked-prefill workload: 5,048,832 visible pairs per sequence and
    head over all 5,632 rows (6.617e11 flops per layer for 8 sequences and 32
    heads at D = 128), from the rule matrix."""
    batch, hd = inputs.masked_prefill()
    d = batch.dialogues[0]
    role, seg = d.arrays()
    pairs = _rule_pairs(d, range(d.length), False)
    assert pairs == 5048832
    assert bench._visible_pairs(role, seg, range(d.length), 0) == pairs
    flops = 4.0 * hd.d * hd.hq * pairs * batch.B
    assert flops == pytest.approx(6.617e11, rel=1e-3)


def test_serving_prefill_flops_equal_rule_count():
    """The serving step's prefill rows are a new turn over retained rows plus
    the turn itself; its flop count (Layout.prefill_flops) must equal the
    visible pairs of the rule matrix on a dialogue of the retained rows and
    the new turn, summed over the prefill sequences."""
    lay = bench.Layout(n_layers=1)
    total = 0
    for q, r, d in zip(lay.q_len, lay.ret_pre, lay.ms.raw_hist):
        # the retained cache is I_sys + every N_i (bodies gone) + the new turn
        ret = inputs.Dialogue(d.sys_len, [(0, k) for _, k in d.segments], int(q))
        assert ret.length == int(r) + int(q)
        role, seg = ret.arrays()
        rows = range(ret.length - int(q), ret.length)
        total += bench._visible_pairs(role, seg, rows, 0)
    assert lay.prefill_flops() == pytest.approx(4.0 * lay.D * lay.HQ * total * lay.NL)


def test_decode_and_compaction_bytes():
    """Decode reads every retained K/V row once (plus q and O); compaction reads
    and writes every kept row of K and V once."""
    lay = bench.Layout(n_layers=2)
    row = lay.HKV * lay.D * 2
    kv = 2.0 * row * float(lay.dec_len.sum())
    qo = 2.0 * lay.n_dec * lay.HQ * lay.D * 2
    assert lay.decode_bytes() == pytest.approx((kv + qo + lay.n_dec * 8.0) * lay.NL)
    kept = float(sum(d.recipe_retained for d in lay.ms.raw_hist))
    assert lay.compact_bytes() == pytest.approx(kept * row * 2 * 2 * lay.NL)
