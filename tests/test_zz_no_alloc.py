"""pd_debug_logits_static: the teacher-forced logits without any device allocation.

Some callers may not allocate device memory at all (their GPU memory is owned by another pool,
or they must not grow their footprint once running); pd_debug_logits allocates a staging
buffer on every call, pd_debug_logits_static uses a fixed array in the library's device image
instead.  These tests call both through the C ABI and require the same logits, within the
tolerance the fp32 parity tests use, on two calls in a row (the second call reuses the array
the first one left behind), and check the documented size limit.
"""
import os

import numpy as np
import pytest

import synth
import paper_2305_10427_gb300 as pkg

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
    d = pkg.Decoder(pkg.Config.from_spec(synth.TINY, max_src_len=64, max_tgt_len=256), w.blob)
    yield d
    d.close()


def _rel_row_err(got, ref):
    return np.abs(got - ref).max(axis=1) / np.abs(ref).max(axis=1)


def test_static_logits_match_the_allocating_entry_point(dec):
    import torch
    rng = np.random.default_rng(7)
    src = rng.integers(3, synth.TINY.vocab, size=23).astype(np.int32)
    dec.encode(src)
    inputs = [np.r_[synth.BOS_ID, rng.integers(0, synth.TINY.vocab, size=T - 1)].astype(np.int32)
              for T in (16, 40)]
    refs = [dec.debug_logits(y) for y in inputs]
    got = []
    free = []
    for y in inputs:                                  # two calls in a row on the one array
        got.append(dec.debug_logits_static(y))
        torch.cuda.synchronize()
        free.append(torch.cuda.mem_get_info()[0])
    for g, r in zip(got, refs):
        assert g.shape == r.shape
        assert np.isfinite(g).all()
        assert _rel_row_err(g, r).max() < 1e-4
    assert abs(free[1] - free[0]) < (2 << 20)         # the second call did not allocate


def test_static_logits_reject_oversized_requests(dec):
    dec.encode(np.array([5, 6, 7], dtype=np.int32))
    y = np.full(200, synth.BOS_ID, dtype=np.int32)   # 200 * 8000 > 1,048,576 floats
    with pytest.raises(pkg.PdError) as e:
        dec.debug_logits_static(y)
    assert e.value.status == -1 and "static logits buffer" in str(e.value)
    ok = dec.debug_logits_static(y[:100])             # 800,000 floats fit
    assert ok.shape == (100, synth.TINY.vocab)
