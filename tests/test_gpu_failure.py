"""Failure detection on the GPU without a fault: the kernels' bounded device-side wait.

Every spin of the kernels (grid barriers, the commit barrier) gives up after a time limit,
raises an abort flag that the other CTAs watch, records PD_ETIMEOUT and returns, so that a
broken schedule ends the kernel instead of hanging the GPU.  pd_debug_wait_timeout runs that
wait against a counter that nothing advances, with a short limit: the test checks that it
gives up in time with PD_ETIMEOUT and that the context decodes correctly afterwards.
"""
import os
import time

import numpy as np
import pytest

import synth
import paper_2305_10427_gb300 as pkg
from paper_2305_10427_gb300 import _binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dec():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)
    torch.cuda.set_device(0)
    w = synth.make_weights(synth.TINY, seed=0)
    d = pkg.Decoder(pkg.Config.from_spec(synth.TINY, max_src_len=64, max_tgt_len=64), w.blob)
    yield d
    d.close()


@pytest.mark.parametrize("limit_ms", [20, 200])
def test_wait_gives_up_with_timeout_status(dec, limit_ms):
    t0 = time.perf_counter()
    status = dec.debug_wait_timeout(limit_ms * 1_000_000)
    elapsed = time.perf_counter() - t0
    assert status == B.PD_ETIMEOUT
    assert limit_ms / 1e3 <= elapsed + 1e-3          # it did wait for the limit
    assert elapsed < limit_ms / 1e3 + 2.0            # and returned soon after it


def test_context_usable_after_timeout(dec):
    src = np.array([5, 17, 9, 33, 2, 41, 7], dtype=np.int32)
    dec.encode(src)
    before = dec.decode("greedy", 12)
    assert dec.debug_wait_timeout(10_000_000) == B.PD_ETIMEOUT
    dec.encode(src)
    after = dec.decode("greedy", 12)
    gs = dec.decode("gs_jacobi", 12, b=3)
    assert before.tokens == after.tokens
    assert gs.tokens == after.tokens


def test_invalid_limit_rejected(dec):
    with pytest.raises(pkg.PdError) as e:
        dec.debug_wait_timeout(0)
    assert e.value.status == B.PD_EINVAL
