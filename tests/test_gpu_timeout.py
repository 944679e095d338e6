"""The bounded-wait failure path on the GPU.

A test copy of the prefill and decode kernels (every prefill instance: paired,
retained-first chunked, unpaired and single-tile units) is built with a wait limit of
200 ns (SONIC_WAIT_LIMIT_NS) checked on every poll, far shorter than a TMA
round trip, so waits run out while the work they wait for is still in flight.  The
call must then report SONIC_ERR_DEVICE_TIMEOUT in the status word, and its
blocks must wind down cleanly: the copies and MMAs already issued are drained
(bounded by time alone) before tensor memory is freed and the blocks exit.
Afterwards the device must still be usable: the normal library, on the same
device and stream, runs the same call and matches the oracle.
"""
import os
import shutil
import tempfile

import numpy as np
import pytest
import torch

import oracle
from paper_2601_21927_gb300 import _build, inputs, sonic
from tests import harness as H

pytestmark = pytest.mark.gpu

TIMEOUT = 5  # SONIC_ERR_DEVICE_TIMEOUT


@pytest.fixture(scope="module")
def short_wait_lib():
    d = tempfile.mkdtemp(prefix="sonic_short_wait_")
    try:
        path = _build.compile_library(os.path.join(d, "libsonic_short_wait.so"),
                                      ["api.cu", "prefill.cu", "decode.cu"],
                                      defines=["SONIC_WAIT_LIMIT_NS=200ull",
                                               "SONIC_WAIT_CHECK_MASK=0u"])
        yield sonic.open_library(path)
    finally:
        shutil.rmtree(d, ignore_errors=True)


def _with(lib, fn):
    saved = sonic.load()
    sonic._lib = lib
    try:
        return fn()
    finally:
        sonic._lib = saved


# Every kind of prefill kernel instance: paired units (head ratio 4, given
# order), the retained-first query chunks, unpaired units with last query blocks
# shared by two heads (head ratio 3), and single-tile units with packed heads
# (32 query rows per sequence), whose K ring has three stages.
PREFILL_CASES = {
    "paired": dict(hq=8, hkv=2, order=sonic.KEYS_AS_GIVEN, short=False),
    "retained_first": dict(hq=8, hkv=2, order=sonic.KEYS_RETAINED_FIRST, short=False),
    "unpaired": dict(hq=6, hkv=2, order=sonic.KEYS_AS_GIVEN, short=False),
    "single_tile": dict(hq=8, hkv=2, order=sonic.KEYS_AS_GIVEN, short=True),
}


@pytest.mark.parametrize("case", sorted(PREFILL_CASES))
def test_prefill_wait_timeout_then_normal_call(short_wait_lib, case):
    c = PREFILL_CASES[case]
    rng = np.random.default_rng(21)
    batch = inputs.Batch([inputs.random_dialogue(rng, max_segments=5, max_body=400,
                                                 max_nexus=40, max_curr=300) for _ in range(6)])
    q_len = np.minimum(batch.k_len, 32).astype(np.int32) if c["short"] else None
    args = dict(hq=c["hq"], hkv=c["hkv"], D=128, seed=3, key_order=c["order"], q_len=q_len)
    _with(short_wait_lib, lambda: H.run_prefill(batch, expect_status=TIMEOUT, **args))
    torch.cuda.synchronize()  # the context is still usable
    res = H.run_prefill(batch, **args)
    for b in range(batch.B):
        O, lse, got, got_lse = H.oracle_prefill_rows(batch, res, b, np.arange(res["q_len"][b]))
        H.check_close(got, O, f"seq {b}")
        np.testing.assert_allclose(got_lse, lse, rtol=0, atol=2e-3)


def test_decode_wait_timeout_then_normal_call(short_wait_lib):
    lens = np.array([700, 2049, 5000, 129], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int32)
    T, hq, hkv, D = int(lens.sum()), 8, 2, 128
    K = inputs.randn((2, T, hkv, D), seed=31, device=H.dev())
    V = inputs.randn((2, T, hkv, D), seed=32, device=H.dev())
    q = inputs.randn((2, len(lens), hq, D), seed=33, device=H.dev())

    def run(expect):
        O = torch.full_like(q, float("nan"))
        status = torch.zeros(1, dtype=torch.int32, device=H.dev())
        sonic.sonic_attn_decode(q, K, V, H.i32(lens), O, kv_start=H.i32(starts),
                                max_len=int(lens.max()), chunk_len=256, status=status)
        torch.cuda.synchronize()
        assert sonic.read_status(status) == expect
        return O

    _with(short_wait_lib, lambda: run(TIMEOUT))
    O = run(0)
    for layer in (0, 1):
        for b in range(len(lens)):
            s0, n = int(starts[b]), int(lens[b])
            Oref, _ = oracle.decode(H.f64(q[layer, b]), H.f64(K[layer, s0:s0 + n]),
                                    H.f64(V[layer, s0:s0 + n]))
            H.check_close(H.f64(O[layer, b]), Oref, f"layer {layer} seq {b}")
