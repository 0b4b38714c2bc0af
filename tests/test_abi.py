"""The C ABI library loads, exports every symbol include/pd.h declares, and validates its
arguments on the host (no GPU: only calls that return before any CUDA call)."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
import paper_2305_10427_gb300 as pkg
from paper_2305_10427_gb300 import _binding as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "pd.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)
    return pkg.load_library()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pd_[a-z_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert set(names) == set(B.EXPORTED)
    for n in names:
        assert hasattr(lib, n), n


@pytest.mark.parametrize("spec", [synth.TINY, synth.MARIAN, synth.MBART], ids=lambda s: s.name)
def test_blob_size_matches_layout(lib, spec):
    cfg = pkg.Config.from_spec(spec, 64, 128)
    itemsize = 2 if spec.dtype == synth.DTYPE_BF16 else 4
    assert pkg.weights_nbytes(cfg) == synth.n_params(spec) * itemsize


def test_invalid_configs_are_rejected_before_cuda(lib):
    good = pkg.Config.from_spec(synth.TINY, 64, 128)
    assert pkg.weights_nbytes(good) > 0
    import dataclasses
    for bad in (dict(d_model=200), dict(n_heads=3), dict(d_ff=100), dict(n_dec_layers=0),
                dict(n_enc_layers=17), dict(dtype=5), dict(eos_id=9000), dict(max_tgt_len=0),
                dict(n_heads=1)):
        cfg = dataclasses.replace(good, **bad)
        assert pkg.weights_nbytes(cfg) == 0, bad
        c = cfg._c()
        h = ctypes.c_void_p()
        blob = np.zeros(16, dtype=np.float32)
        st = lib.pd_create(ctypes.byref(c), blob.ctypes.data_as(ctypes.c_void_p), blob.nbytes,
                           None, ctypes.byref(h))
        assert st == B.PD_EINVAL and not h.value


def test_wrong_blob_size_is_rejected(lib):
    cfg = pkg.Config.from_spec(synth.TINY, 64, 128)
    c = cfg._c()
    h = ctypes.c_void_p()
    blob = np.zeros(10, dtype=np.float32)
    st = lib.pd_create(ctypes.byref(c), blob.ctypes.data_as(ctypes.c_void_p), blob.nbytes, None,
                       ctypes.byref(h))
    assert st == B.PD_EINVAL


def test_null_context_calls(lib):
    assert lib.pd_encode(None, None, 3) == B.PD_EINVAL
    assert lib.pd_decode_device(None, None, None, None) == B.PD_EINVAL
    assert lib.pd_debug_wait_timeout(None, 1000, None) == B.PD_EINVAL
    assert lib.pd_launch_count(None) == 0
    assert lib.pd_last_error(None) == b"context is NULL"
    lib.pd_destroy(None)
