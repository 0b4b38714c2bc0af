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
                dict(n_heads=1), dict(max_batch=65), dict(max_batch=-1)):
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
    assert lib.pd_encode_batch(None, None, None, 1) == B.PD_EINVAL
    assert lib.pd_encode_batch_device(None, None, None, 1) == B.PD_EINVAL
    assert lib.pd_decode_batch(None, None, 1, None, None, 0, None, None) == B.PD_EINVAL
    assert lib.pd_decode_batch_device(None, None, 1, None, None, 0, None) == B.PD_EINVAL
    assert lib.pd_launch_count(None) == 0
    lib.pd_destroy(None)


def test_create_failure_reason(lib):
    """pd_create keeps the reason of its failure for pd_last_error(NULL)."""
    cfg = pkg.Config.from_spec(synth.TINY, 64, 128)
    c = cfg._c()
    h = ctypes.c_void_p()
    blob = np.zeros(10, dtype=np.float32)
    assert lib.pd_create(ctypes.byref(c), blob.ctypes.data_as(ctypes.c_void_p), blob.nbytes,
                         None, ctypes.byref(h)) == B.PD_EINVAL
    assert b"nbytes is 40" in lib.pd_last_error(None)
    c.d_model = 100
    assert lib.pd_create(ctypes.byref(c), blob.ctypes.data_as(ctypes.c_void_p), blob.nbytes,
                         None, ctypes.byref(h)) == B.PD_EINVAL
    assert lib.pd_last_error(None).startswith(b"invalid config: d_model")


def _header_text():
    return re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)


def _struct_fields(text, name):
    body = re.search(r"typedef struct \{([^{}]*)\}\s*" + name + r"\s*;", text).group(1)
    out = []
    for decl in body.split(";"):
        decl = decl.strip()
        if decl:
            out += [n.strip() for n in decl.split(None, 1)[1].split(",")]
    return out


def _enum_values(text, name):
    body = re.search(r"typedef enum \{([^{}]*)\}\s*" + name + r"\s*;", text).group(1)
    return {k: int(v) for k, v in re.findall(r"(PD_[A-Z0-9_]+)\s*=\s*(-?\d+)", body)}


@pytest.mark.parametrize("cname,cls", [("pd_config", B._Config),
                                       ("pd_decode_params", B._DecodeParams),
                                       ("pd_trace_step", B._TraceStep)])
def test_binding_structs_match_header(cname, cls):
    """The ctypes mirrors declare the header's fields in the header's order (every field is a
    4-byte int or float, so equal order means equal layout)."""
    assert _struct_fields(_header_text(), cname) == [f for f, _ in cls._fields_]
    assert ctypes.sizeof(cls) == 4 * len(cls._fields_)


def test_binding_enums_match_header():
    text = _header_text()
    assert _enum_values(text, "pd_method") == {
        "PD_GREEDY": B.METHODS["greedy"], "PD_JACOBI": B.METHODS["jacobi"],
        "PD_GS_JACOBI": B.METHODS["gs_jacobi"],
        "PD_HYBRID_GS_JACOBI": B.METHODS["hybrid_gs_jacobi"]}
    assert _enum_values(text, "pd_stop_rule") == {"PD_STOP_UNCHANGED": B.STOP_RULES["paper"],
                                                  "PD_STOP_PREFIX": B.STOP_RULES["prefix"],
                                                  "PD_STOP_SUFFIX": B.STOP_RULES["suffix"]}
    assert _enum_values(text, "pd_init_rule") == {"PD_INIT_PAD": B.INITS["pad"],
                                                  "PD_INIT_LAST": B.INITS["last"]}
    assert _enum_values(text, "pd_gemm_engine") == {"PD_ENGINE_AUTO": B.ENGINES["auto"],
                                                    "PD_ENGINE_SIMT": B.ENGINES["simt"],
                                                    "PD_ENGINE_TENSOR": B.ENGINES["tensor"],
                                                    "PD_ENGINE_CLUSTER": B.ENGINES["cluster"]}
    status = _enum_values(text, "pd_status")
    assert {v: k for k, v in status.items()} == B.STATUS_NAMES
