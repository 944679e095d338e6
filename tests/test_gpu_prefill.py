"""GPU parity of sonic_attn_prefill (Sec. 3.2 masked attention) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu


ORDERS = [sonic.KEYS_AS_GIVEN, sonic.KEYS_RETAINED_FIRST]


def _all_rows(batch, hq, hkv, D, mode=sonic.NEXUS_FULL, seed=0, order=sonic.KEYS_AS_GIVEN):
    res = H.run_prefill(batch, hq, hkv, D, seed=seed, nexus_vis=mode, key_order=order)
    for b in range(batch.B):
        n = int(batch.k_len[b])
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(n), nexus_vis=mode)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)


@pytest.mark.parametrize("order", ORDERS)
def test_tiny_reference_all_rows(order):
    batch, hd = inputs.tiny_ref()
    _all_rows(batch, hd.hq, hd.hkv, hd.d, order=order)


@pytest.mark.parametrize("order", ORDERS)
@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_random_dialogues_multi_tile(mode, order):
    rng = np.random.default_rng(11)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=120, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(4)]
    ds.append(inputs.Dialogue(5, [(300, 0), (1, 1), (0, 70)], 1))  # K_i = 0, tiny pieces
    _all_rows(inputs.Batch(ds), 4, 2, 128, mode=mode, seed=5, order=order)


@pytest.mark.parametrize("D", [64, 128])
def test_output_only_16_byte_aligned(D):
    """O 16 bytes past a 32-byte boundary, with a layer stride that is not a
    multiple of 32 bytes: the epilogue takes its 16-byte stores, every row
    matches the oracle on both layers, and no element outside O is written."""
    rng = np.random.default_rng(17)
    batch = inputs.Batch([inputs.random_dialogue(rng, max_segments=4, max_body=150, max_nexus=30,
                                                 max_curr=140) for _ in range(3)])
    off = 8  # bf16 elements: 16 bytes
    res = H.run_prefill(batch, 4, 2, D, seed=21, n_layers=2, o_offset=off)
    assert res["O"].data_ptr() % 32 == 16 and (res["O"].stride(0) * 2) % 32 == 16
    for layer in (0, 1):
        for b in range(batch.B):
            n = int(batch.k_len[b])
            O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(n), layer=layer)
            H.check_close(got, O, f"layer {layer} seq {b}")
            np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)
    n = res["O"][0].numel()
    buf = res["O_buf"]
    gaps = torch.cat([buf[:off], buf[off + n:2 * off + n], buf[2 * off + 2 * n:]])
    assert gaps.numel() == 3 * off and torch.isnan(gaps.float()).all()


@pytest.mark.parametrize("order", ORDERS)
def test_head_dim_64_and_gqa_ratios(order):
    rng = np.random.default_rng(3)
    ds = [inputs.random_dialogue(rng, max_segments=4, max_body=200, max_nexus=30) for _ in range(3)]
    _all_rows(inputs.Batch(ds), 6, 2, 64, seed=9, order=order)


@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_retained_first_many_runs_per_tile(mode):
    """Short segments: a 128-key tile of the retained part holds more than four
    runs of consecutive positions (Nexus groups of 3-6 tokens), and a body tile
    more than four segments, so both take the per-key mask path."""
    ds = [inputs.Dialogue(30, [(20, 5)] * 40, 100),
          inputs.Dialogue(3, [(9, 3), (7, 6), (11, 4)] * 12, 37),
          inputs.Dialogue(128, [(128, 128)] * 3, 128)]  # tile-aligned everything
    _all_rows(inputs.Batch(ds), 4, 1, 128, mode=mode, seed=13, order=sonic.KEYS_RETAINED_FIRST)


@pytest.mark.parametrize("hq,hkv", [(8, 1), (12, 2), (4, 1)])
@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_retained_first_query_runs(mode, hq, hkv):
    """Retained-first query order by runs in 32-row chunks, at head ratios 8,
    6 and 4: Nexus runs shorter and longer than a chunk, empty runs (K_i = 0),
    adjacent Nexus runs of two segments (an empty body between them), bodies
    that are not multiples of 32 rows (padded chunks) and one-token runs."""
    ds = [inputs.Dialogue(40, [(100, 7), (0, 40), (130, 70), (60, 0), (20, 33)], 50),
          inputs.Dialogue(0, [(256, 32)] * 5, 64),
          inputs.Dialogue(9, [(3, 1)] * 6 + [(200, 100)], 1)]
    _all_rows(inputs.Batch(ds), hq, hkv, 128, mode=mode, seed=25, order=sonic.KEYS_RETAINED_FIRST)


def test_retained_first_query_runs_beyond_the_table():
    """Retained-first walks the query rows by runs (one body, or consecutive
    other rows) in 32-row chunks; 520 one-token segments make 1,040 runs,
    more than the run table holds, so that sequence keeps the given query
    order, beside a sequence whose runs fit (chunked order)."""
    ds = [inputs.Dialogue(4, [(1, 1)] * 520, 8), inputs.Dialogue(40, [(200, 40)] * 3, 90)]
    _all_rows(inputs.Batch(ds), 4, 2, 128, seed=15, order=sonic.KEYS_RETAINED_FIRST)


@pytest.mark.parametrize("order", ORDERS)
def test_first_key_tile_not_listed_first(order):
    """No system prompt and a 300-token first body: as given, key tile 0 holds
    body rows only, which the current turn's rows never see, so the first
    listed tile is a later one and key tile 0's copy must not start early;
    all rows (tile 0 then seen by its own segment's rows) and current rows only."""
    ds = [inputs.Dialogue(0, [(300, 4), (50, 3)], 40), inputs.Dialogue(0, [(260, 0), (9, 9)], 200)]
    batch = inputs.Batch(ds)
    _all_rows(batch, 4, 2, 128, seed=23, order=order)
    q_len = np.array([40, 200], dtype=np.int32)
    res = H.run_prefill(batch, 4, 2, 128, q_len=q_len, seed=29, key_order=order)
    for b in range(batch.B):
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(q_len[b]))
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)


@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_as_given_many_segments_per_tile(mode):
    """Key order as given with segments of 10-20 tokens: most 128-key tiles
    hold more than four body segments and more than four position runs of
    Nexus keys, so their column-mask records fall back to the per-key rule and
    the producer stages the keys' roles, segments and positions."""
    ds = [inputs.Dialogue(3, [(9, 3), (7, 6), (11, 4)] * 12, 37),
          inputs.Dialogue(17, [(5, 5)] * 30, 60)]
    _all_rows(inputs.Batch(ds), 4, 2, 128, mode=mode, seed=17, order=sonic.KEYS_AS_GIVEN)


@pytest.mark.parametrize("order", ORDERS)
@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_uniform_scores_count_visible_keys(mode, order):
    """Q = 0 makes every visible score 0 and every probability exactly 1, so
    the GPU's lse is ln |vis(p)| up to fp32 rounding; one key missing or extra
    in any row moves it by about 1 / |vis(p)|.  An exact check of the mask on
    every row, both readings and both key orders."""
    rng = np.random.default_rng(23)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=150, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(4)]
    ds += [inputs.Dialogue(30, [(20, 5)] * 40, 100), inputs.Dialogue(0, [(300, 0), (1, 1)], 2)]
    batch = inputs.Batch(ds)
    Q = torch.zeros((1, batch.total, 4, 128), dtype=torch.bfloat16, device=H.dev())
    res = H.run_prefill(batch, 4, 2, 128, seed=29, nexus_vis=mode, key_order=order, Q=Q)
    for b in range(batch.B):
        n = int(batch.k_len[b])
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(n), nexus_vis=mode)
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-5, err_msg=f"seq {b}")
        H.check_close(got, O, f"seq {b}")


@pytest.mark.parametrize("order", ORDERS)
@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
@pytest.mark.parametrize("hq,hkv,max_q", [(8, 2, 32), (8, 1, 20), (16, 2, 64), (6, 3, 100)])
def test_short_query_blocks_pack_heads(order, mode, hq, hkv, max_q):
    """Short query blocks (the Nexus rows of a segment, a few current-turn
    rows): the kernel packs 2, 4 or 8 query heads of a KV group into one
    128-row tile.  Ragged q_len from 1 to max_q over multi-tile key sequences,
    every query row and head against the oracle, with lse and Nexus mass."""
    rng = np.random.default_rng(hq * 100 + max_q)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=150, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(5)]
    batch = inputs.Batch(ds)
    q_len = np.minimum(rng.integers(1, max_q + 1, batch.B), batch.k_len)
    res = H.run_prefill(batch, hq, hkv, 128, q_len=q_len, seed=51, nexus_vis=mode,
                        key_order=order, with_mass=True)
    for b in range(batch.B):
        rows = np.arange(q_len[b])
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, rows, nexus_vis=mode)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)
        want, gm = H.oracle_mass_rows(batch, res, b, rows, nexus_vis=mode)
        np.testing.assert_allclose(gm, want, rtol=0, atol=2e-3)


MASS_ATOL = 2e-3  # attention mass on Nexus keys: a share in [0, 1]


@pytest.mark.parametrize("order", ORDERS)
@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
@pytest.mark.parametrize("D,hq,hkv,with_lse", [(128, 4, 2, True), (64, 6, 2, False)])
def test_nexus_mass_matches_oracle(order, mode, D, hq, hkv, with_lse):
    """The mass output on every row: random dialogues spanning several tiles,
    a retained cache followed by a current turn (uncut tiles that mix system,
    Nexus and current keys), and short segments (tiles on the per-key path).
    O and lse do not change when the mass is requested."""
    rng = np.random.default_rng(37)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=150, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(3)]
    ds += [inputs.Dialogue(200, [(0, 60), (0, 90), (0, 7)], 400),
           inputs.Dialogue(30, [(20, 5)] * 30, 100)]
    batch = inputs.Batch(ds)
    res = H.run_prefill(batch, hq, hkv, D, seed=41, nexus_vis=mode, key_order=order,
                        with_lse=with_lse, with_mass=True)
    for b in range(batch.B):
        n = int(batch.k_len[b])
        want, got = H.oracle_mass_rows(batch, res, b, np.arange(n), nexus_vis=mode)
        np.testing.assert_allclose(got, want, rtol=0, atol=MASS_ATOL, err_msg=f"seq {b}")
    plain = H.run_prefill(batch, hq, hkv, D, seed=41, nexus_vis=mode, key_order=order,
                          with_lse=with_lse)
    assert torch.equal(plain["O"].view(torch.int16), res["O"].view(torch.int16))
    if with_lse:
        assert torch.equal(plain["lse"], res["lse"])


@pytest.mark.parametrize("order", ORDERS)
def test_nexus_mass_of_uniform_scores_is_the_visible_nexus_share(order):
    """Q = 0: every visible probability is exactly 1, so the mass is the count
    of visible Nexus keys over the count of visible keys, up to one fp32
    division: a key-exact check of the Nexus bits on every tile kind."""
    rng = np.random.default_rng(43)
    ds = [inputs.random_dialogue(rng, max_segments=6, max_body=150, max_nexus=40, max_sys=90,
                                 max_curr=150) for _ in range(3)]
    ds += [inputs.Dialogue(200, [(0, 60), (0, 90), (0, 7)], 400),
           inputs.Dialogue(30, [(20, 5)] * 30, 100), inputs.Dialogue(9, [(300, 0)], 40)]
    batch = inputs.Batch(ds)
    Q = torch.zeros((1, batch.total, 4, 128), dtype=torch.bfloat16, device=H.dev())
    res = H.run_prefill(batch, 4, 2, 128, seed=47, key_order=order, Q=Q, with_mass=True)
    for b in range(batch.B):
        n = int(batch.k_len[b])
        want, got = H.oracle_mass_rows(batch, res, b, np.arange(n))
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-6, err_msg=f"seq {b}")


def test_retained_first_sequences_sharing_key_rows():
    """Two sequences over the same key rows (a shared history, different query
    blocks): each gets its own span of the permuted copy.  The key tensor has
    2 * 560 rows (the second half unused), so the workspace bound of
    total_k_rows + 256 rows per sequence holds both spans of 768 rows."""
    d = inputs.Dialogue(50, [(120, 40), (200, 60)], 90)
    batch = inputs.Batch([d, d])
    kl = int(batch.k_len[0])
    res = H.run_prefill(batch, 4, 2, 128, seed=17, key_order=sonic.KEYS_RETAINED_FIRST,
                        k_start=[0, 0], total_k_rows=2 * kl)
    shared = inputs.Batch([d])
    for b in range(2):
        # both sequences read key rows [0, kl) of the same K, V, role, seg
        O, lse, got, got_lse = H.oracle_prefill_rows(
            shared, dict(res, q_len=res["q_len"][b:b + 1], q_start=res["q_start"][b:b + 1]),
            0, np.arange(kl))
        H.check_close(got, O, f"seq {b}")


def test_retained_first_workspace_overflow_is_reported():
    """Three sequences sharing 1,100 key rows need more permuted rows than the
    workspace bound (total_k_rows + 256 per sequence): the GPU reports
    SONIC_ERR_WORKSPACE in the status word, sequences that fit still run."""
    d = inputs.Dialogue(100, [(400, 100)] * 2, 0)
    batch = inputs.Batch([d, d, d])
    res = H.run_prefill(batch, 2, 1, 128, seed=19, key_order=sonic.KEYS_RETAINED_FIRST,
                        k_start=[0, 0, 0], total_k_rows=int(batch.k_len[0]),
                        expect_status=3, with_lse=False)
    # sequence 0 fits (its span starts at row 0); later ones are left as zeros
    O, _, got, _ = H.oracle_prefill_rows(
        inputs.Batch([d]), dict(res, q_len=res["q_len"][:1], q_start=res["q_start"][:1]), 0,
        np.arange(0, int(batch.k_len[0]), 7))
    H.check_close(got, O, "seq 0")
    n = int(batch.k_len[0])
    assert (res["O"][0, n:].float() == 0).all()


@pytest.mark.parametrize("order", ORDERS)
def test_current_turn_over_compacted_cache(order):
    """Turn-by-turn form: queries = the current turn, keys = retained cache +
    current turn (bottom-right aligned)."""
    full = [inputs.Dialogue(40, [(200, 30), (150, 20), (90, 45)], 333),
            inputs.Dialogue(7, [(64, 64)] * 3, 129)]
    ret = inputs.Batch([inputs.Dialogue(d.sys_len, [(0, k) for _, k in d.segments], d.curr_len)
                        for d in full])
    q_len = [d.curr_len for d in full]
    res = H.run_prefill(ret, 8, 2, 128, q_len=q_len, seed=21, key_order=order)
    for b in range(ret.B):
        O, lse, got, got_lse = H.oracle_prefill_rows(ret, res, b, np.arange(q_len[b]))
        H.check_close(got, O, f"seq {b}")


@pytest.mark.parametrize("order", ORDERS)
def test_masked_prefill_workload_sampled_rows(order):
    """Batch 8, 32/8 heads, D = 128, L = 5632, every row (full mask); rows
    sampled across tiles, segment edges and the ragged end."""
    batch, hd = inputs.masked_prefill()
    res = H.run_prefill(batch, hd.hq, hd.hkv, hd.d, seed=31, key_order=order)
    L = int(batch.k_len[0])
    rows = np.unique(np.r_[0, 127, 128, 511, 512, 767, 799, 800, 2000, 4000, 5119, 5120, L - 1])
    for b in (0, 5):
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, rows)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)
    # every output is finite and the lse rows are all written
    assert torch.isfinite(res["O"]).all()
    assert torch.isfinite(res["lse"]).all()


@pytest.mark.parametrize("order", ORDERS)
def test_sequence_outside_the_arrays_is_refused(order):
    """A sequence whose k_start points past total_k_rows is refused
    (SONIC_ERR_INVALID_ARGUMENT in the status word, none of its rows read);
    the other sequences are computed as usual."""
    ds = [inputs.Dialogue(20, [(60, 10)], 40), inputs.Dialogue(30, [(100, 20), (50, 5)], 70)]
    batch = inputs.Batch(ds)
    bad_start = [int(batch.k_start[0]), batch.total + 1000]
    res = H.run_prefill(batch, 4, 2, 128, seed=61, key_order=order, k_start=bad_start,
                        expect_status=1)
    O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, 0, np.arange(int(batch.k_len[0])))
    H.check_close(got, O, "seq 0")


@pytest.mark.parametrize("mode", [sonic.NEXUS_FULL, sonic.NEXUS_CAUSAL_SEGMENTS])
def test_retained_first_query_suffix_skips_unseen_bodies(mode):
    """Queries are a suffix of S_aug starting inside a history segment: the
    retained-first copy leaves out the body tiles of earlier segments (no
    query row can see them) and every output still equals the oracle."""
    ds = [inputs.Dialogue(64, [(300, 20)] * 6 + [(200, 40)], 90),
          inputs.Dialogue(10, [(128, 16)] * 9, 33), inputs.Dialogue(0, [(700, 7)], 5)]
    batch = inputs.Batch(ds)
    # from the middle of the 5th segment's body / the 7th segment / the current turn
    first = [64 + 4 * 320 + 150, 10 + 6 * 144 + 5, 700 + 7]
    q_len = [int(batch.k_len[b]) - first[b] for b in range(batch.B)]
    res = H.run_prefill(batch, 4, 2, 128, q_len=q_len, seed=71, nexus_vis=mode,
                        key_order=sonic.KEYS_RETAINED_FIRST)
    for b in range(batch.B):
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(q_len[b]),
                                                     nexus_vis=mode)
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)


@pytest.mark.parametrize("order,L", [(sonic.KEYS_AS_GIVEN, 262144),
                                     (sonic.KEYS_RETAINED_FIRST, 262016)])
def test_longest_sequence(order, L):
    """The longest key sequence the call accepts (2047 key tiles; one fewer
    with the retained-first order, whose copy adds a tile), history segments
    of 4000 body + 400 Nexus rows and a 64-row current turn as the queries:
    sampled rows against the oracle."""
    n_seg = (L - 1000 - 64) // 4400
    sys_len = L - 64 - n_seg * 4400
    d = inputs.Dialogue(sys_len, [(4000, 400)] * n_seg, 64)
    assert d.length == L
    batch = inputs.Batch([d])
    res = H.run_prefill(batch, 8, 2, 128, q_len=[64], seed=81, key_order=order)
    O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, 0, np.array([0, 31, 63]))
    H.check_close(got, O, "longest sequence")
    np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)
