"""pd_debug_logits_static: the teacher-forced logits without any device allocation.

Some callers may not allocate device memory at all (their GPU memory is owned by another pool,
or they must not grow their footprint once running); pd_debug_logits allocates a staging
buffer on every call, pd_debug_logits_static uses a fixed array in the library's device image
instead.  Both run the same kernel on the same inputs, so their logits must be equal bit for
bit; these tests call both through the C ABI on two calls in a row (the second call reuses the
array the first one left behind), compare them with the float64 oracle at the parity bars
(1e-4 of a row's largest |logit| for fp32, 2e-2 for bf16), check that device free memory does
not move from before the first call to after the last, and check the documented size limit.
"""
import os

import numpy as np
import pytest

import synth
import paper_2305_10427_gb300 as pkg
from oracle import model as om

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)
    torch.cuda.set_device(0)


def _rel_row_err(got, ref):
    return np.abs(got - ref).max(axis=1) / np.abs(ref).max(axis=1)


def _free_bytes():
    import torch
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def _two_calls(spec, max_tgt, lengths, tol, seed):
    import torch
    w = synth.make_weights(spec, seed=0)
    model = om.Model(spec, w.tensors)
    rng = np.random.default_rng(seed)
    src = rng.integers(3, spec.vocab, size=23).astype(np.int32)
    mem = model.encode(src)
    with pkg.Decoder(pkg.Config.from_spec(spec, max_src_len=64, max_tgt_len=max_tgt),
                     w.blob) as dec:
        dec.encode(src)
        inputs = [np.r_[synth.BOS_ID, rng.integers(0, spec.vocab, size=T - 1)].astype(np.int32)
                  for T in lengths]
        refs = [dec.debug_logits(y) for y in inputs]
        torch.cuda.empty_cache()
        free0 = _free_bytes()
        got = []
        for y in inputs:                              # two calls in a row on the one array
            got.append(dec.debug_logits_static(y))
        free1 = _free_bytes()
        for g, r, y in zip(got, refs, inputs):
            assert g.shape == r.shape
            assert np.isfinite(g).all()
            assert np.array_equal(g.view(np.uint32), r.view(np.uint32))
            assert _rel_row_err(g, model.logits(mem, y)).max() < tol
        # no allocation from before the first call to after the second (the driver's
        # granularity is 2 MiB: any allocation of the 4 MiB the logits need would show)
        assert free1 == free0, (free0, free1)


def test_static_logits_fp32_equal_allocating_and_oracle():
    _two_calls(synth.TINY, 256, (16, 40), 1e-4, 7)


def test_static_logits_bf16_equal_allocating_and_oracle():
    # Marian-sized bf16 model: 18 * 58101 = 1,045,818 floats fit the 1,048,576-float array
    _two_calls(synth.MARIAN, 128, (18, 11), 2e-2, 8)


def test_static_logits_reject_oversized_requests():
    w = synth.make_weights(synth.TINY, seed=0)
    with pkg.Decoder(pkg.Config.from_spec(synth.TINY, max_src_len=64, max_tgt_len=256),
                     w.blob) as dec:
        dec.encode(np.array([5, 6, 7], dtype=np.int32))
        y = np.full(200, synth.BOS_ID, dtype=np.int32)   # 200 * 8000 > 1,048,576 floats
        with pytest.raises(pkg.PdError) as e:
            dec.debug_logits_static(y)
        assert e.value.status == -1 and "static logits buffer" in str(e.value)
        ok = dec.debug_logits_static(y[:100])             # 800,000 floats fit
        assert ok.shape == (100, synth.TINY.vocab)
