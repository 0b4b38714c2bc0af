"""ctypes binding of the C ABI in include/pd.h: argument marshalling only.

Every step of decoding runs in the CUDA kernels of ``libpd.so``; this module converts numpy
arrays and Python values to the C structs and pointers and raises ``PdError`` on a non-zero
status.  There is no fallback: if the shared library is missing, loading fails loudly.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import List, Optional

import numpy as np

LIB_NAME = "libpd.so"
LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), LIB_NAME)

PD_OK, PD_EINVAL, PD_ENOMEM, PD_ECUDA, PD_ENOTCONV, PD_ENAN, PD_ESTATE, PD_ETIMEOUT = \
    0, -1, -2, -3, -4, -5, -6, -7
STATUS_NAMES = {0: "PD_OK", -1: "PD_EINVAL", -2: "PD_ENOMEM", -3: "PD_ECUDA", -4: "PD_ENOTCONV",
                -5: "PD_ENAN", -6: "PD_ESTATE", -7: "PD_ETIMEOUT"}

METHODS = {"greedy": 0, "jacobi": 1, "gs_jacobi": 2, "hybrid_gs_jacobi": 3}
STOP_RULES = {"paper": 0, "prefix": 1, "suffix": 2}   # pd_stop_rule: Eq. 5 StopC, accepted
#                                                     prefix, accepted prefix with suffix re-runs
INITS = {"pad": 0, "last": 1}                         # pd_init_rule
ENGINES = {"auto": 0, "simt": 1, "tensor": 2, "cluster": 3}   # pd_gemm_engine

# Every symbol include/pd.h declares.
EXPORTED = ("pd_weights_nbytes", "pd_create", "pd_export_weights", "pd_encode",
            "pd_encode_device", "pd_decode", "pd_decode_device", "pd_debug_logits",
            "pd_debug_logits_static", "pd_debug_wait_timeout", "pd_stream", "pd_launch_count",
            "pd_last_error", "pd_destroy", "pd_encode_batch", "pd_encode_batch_device",
            "pd_decode_batch", "pd_decode_batch_device")


class PdError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class _Config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("d_model", "n_heads", "d_ff", "n_enc_layers",
                                            "n_dec_layers", "vocab", "activation", "pre_ln",
                                            "learned_pos", "max_pos", "dtype", "pad_id",
                                            "eos_id", "bos_id")] + \
              [("ln_eps", ctypes.c_float), ("max_src_len", ctypes.c_int),
               ("max_tgt_len", ctypes.c_int), ("max_batch", ctypes.c_int),
               ("gemm_engine", ctypes.c_int), ("seed", ctypes.c_int), ("kv_pages", ctypes.c_int),
               ("cluster_size", ctypes.c_int)]


class _DecodeParams(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("method", "b", "max_len", "h", "stop_at_eos",
                                            "max_passes", "stop_rule", "init")]


class _TraceStep(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("step", "block_start", "block_len", "n_converged",
                                              "stop", "eos_idx", "n_rows")]


_lib = None


def load_library() -> ctypes.CDLL:
    """Load the in-tree libpd.so (built by ``__graft_entry__.build()``); raise if missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    pi32 = ctypes.POINTER(ctypes.c_int32)
    pint = ctypes.POINTER(ctypes.c_int)
    lib.pd_weights_nbytes.argtypes = [ctypes.POINTER(_Config)]
    lib.pd_weights_nbytes.restype = SZ
    lib.pd_create.argtypes = [ctypes.POINTER(_Config), P, SZ, P, ctypes.POINTER(P)]
    lib.pd_create.restype = I
    lib.pd_export_weights.argtypes = [P, P, SZ]
    lib.pd_export_weights.restype = I
    lib.pd_encode.argtypes = [P, pi32, I]
    lib.pd_encode.restype = I
    lib.pd_encode_device.argtypes = [P, P, I]
    lib.pd_encode_device.restype = I
    lib.pd_decode.argtypes = [P, ctypes.POINTER(_DecodeParams), pi32, pint, pint,
                              ctypes.POINTER(_TraceStep), pi32, ctypes.POINTER(ctypes.c_float), I,
                              pint]
    lib.pd_decode.restype = I
    lib.pd_decode_device.argtypes = [P, ctypes.POINTER(_DecodeParams), P, P]
    lib.pd_decode_device.restype = I
    lib.pd_encode_batch.argtypes = [P, pi32, pi32, I]
    lib.pd_encode_batch.restype = I
    lib.pd_encode_batch_device.argtypes = [P, P, pi32, I]
    lib.pd_encode_batch_device.restype = I
    lib.pd_decode_batch.argtypes = [P, ctypes.POINTER(_DecodeParams), I, pi32, pi32, I, pi32, pi32]
    lib.pd_decode_batch.restype = I
    lib.pd_decode_batch_device.argtypes = [P, ctypes.POINTER(_DecodeParams), I, pi32, P, I, P]
    lib.pd_decode_batch_device.restype = I
    lib.pd_debug_logits.argtypes = [P, pi32, I, ctypes.POINTER(ctypes.c_float)]
    lib.pd_debug_logits.restype = I
    lib.pd_debug_logits_static.argtypes = [P, pi32, I, ctypes.POINTER(ctypes.c_float)]
    lib.pd_debug_logits_static.restype = I
    lib.pd_debug_wait_timeout.argtypes = [P, ctypes.c_uint64, pint]
    lib.pd_debug_wait_timeout.restype = I
    lib.pd_stream.argtypes = [P]
    lib.pd_stream.restype = P
    lib.pd_launch_count.argtypes = [P]
    lib.pd_launch_count.restype = ctypes.c_int64
    lib.pd_last_error.argtypes = [P]
    lib.pd_last_error.restype = ctypes.c_char_p
    lib.pd_destroy.argtypes = [P]
    lib.pd_destroy.restype = None
    _lib = lib
    return lib


@dataclasses.dataclass(frozen=True)
class Config:
    """Mirror of ``pd_config``."""

    d_model: int
    n_heads: int
    d_ff: int
    n_enc_layers: int
    n_dec_layers: int
    vocab: int
    activation: int = 0
    pre_ln: bool = False
    learned_pos: bool = False
    max_pos: int = 1024
    dtype: int = 0
    pad_id: int = 1
    eos_id: int = 0
    bos_id: int = 2
    ln_eps: float = 1e-5
    max_src_len: int = 128
    max_tgt_len: int = 256
    max_batch: int = 0
    gemm_engine: int = 0
    seed: int = 0
    kv_pages: int = 0
    cluster_size: int = 0

    @classmethod
    def from_spec(cls, spec, max_src_len: int, max_tgt_len: int, pad_id=1, eos_id=0, bos_id=2,
                  max_batch: int = 0, engine: str = "auto", kv_pages: int = 0, seed: int = 0,
                  cluster_size: int = 0):
        """Build from any object carrying the model fields (d_model, n_heads, ...); seed is
        used only when the Decoder is created without a weight blob, cluster_size only by the
        cluster engine."""
        return cls(spec.d_model, spec.n_heads, spec.d_ff, spec.n_enc_layers, spec.n_dec_layers,
                   spec.vocab, spec.activation, bool(spec.pre_ln), bool(spec.learned_pos),
                   spec.max_pos, spec.dtype, pad_id, eos_id, bos_id, spec.ln_eps, max_src_len,
                   max_tgt_len, max_batch, ENGINES[engine], seed, kv_pages, cluster_size)

    def _c(self) -> _Config:
        c = _Config()
        for f in dataclasses.fields(self):
            v = getattr(self, f.name)
            setattr(c, f.name, float(v) if f.name == "ln_eps" else int(v))
        return c


def weights_nbytes(cfg: Config) -> int:
    c = cfg._c()
    return int(load_library().pd_weights_nbytes(ctypes.byref(c)))


@dataclasses.dataclass
class DecodeResult:
    tokens: List[int]
    n_iters: int
    trace: Optional[List[dict]] = None
    trace_tokens: Optional[np.ndarray] = None     # [n_trace][max_len]
    trace_probs: Optional[np.ndarray] = None


def _i32p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


class Decoder:
    """One decoding context (pd_ctx) on the current CUDA device."""

    def __init__(self, cfg: Config, weights: Optional[np.ndarray], stream: Optional[int] = None):
        """weights: the blob (host array), or None to have the library draw the weights from
        cfg.seed."""
        self._lib = load_library()
        self.cfg = cfg
        self._ccfg = cfg._c()
        h = ctypes.c_void_p()
        if weights is None:
            ptr, nbytes = None, 0
        else:
            blob = np.ascontiguousarray(weights)
            ptr, nbytes = blob.ctypes.data_as(ctypes.c_void_p), blob.nbytes
        st = self._lib.pd_create(ctypes.byref(self._ccfg), ptr, nbytes,
                                 ctypes.c_void_p(stream) if stream else None, ctypes.byref(h))
        if st != PD_OK:
            raise PdError(st, "pd_create: " + self._lib.pd_last_error(None).decode())
        self._h = h
        self.blob_nbytes = weights_nbytes(cfg)

    def _check(self, st: int, what: str):
        if st != PD_OK:
            msg = self._lib.pd_last_error(self._h).decode()
            raise PdError(st, f"{what}: {msg}")

    # -- calls ------------------------------------------------------------------------------
    def encode(self, src) -> None:
        a = np.ascontiguousarray(src, dtype=np.int32)
        self._check(self._lib.pd_encode(self._h, _i32p(a), int(a.size)), "pd_encode")

    def encode_device(self, d_src: int, n_src: int) -> None:
        self._check(self._lib.pd_encode_device(self._h, ctypes.c_void_p(d_src), int(n_src)),
                    "pd_encode_device")

    @staticmethod
    def batch_offsets(sents):
        """Concatenated ids and the offsets array of pd_encode_batch."""
        arrs = [np.ascontiguousarray(s, dtype=np.int32) for s in sents]
        offs = np.zeros(len(arrs) + 1, dtype=np.int32)
        offs[1:] = np.cumsum([a.size for a in arrs])
        return np.concatenate(arrs), offs

    def encode_batch(self, sents) -> None:
        src, offs = self.batch_offsets(sents)
        self._check(self._lib.pd_encode_batch(self._h, _i32p(src), _i32p(offs), len(offs) - 1),
                    "pd_encode_batch")

    def encode_batch_device(self, d_src: int, offsets: np.ndarray) -> None:
        offs = np.ascontiguousarray(offsets, dtype=np.int32)
        self._check(self._lib.pd_encode_batch_device(self._h, ctypes.c_void_p(d_src), _i32p(offs),
                                                     offs.size - 1), "pd_encode_batch_device")

    def decode_batch(self, method: str, max_len, b: int = 1, h: int = 0,
                     stop_at_eos: bool = True, max_passes: int = 0,
                     stop_rule: str = "paper", init: str = "pad") -> List["DecodeResult"]:
        """Decode the sentences of the last encode_batch together; max_len: one value per
        sentence."""
        ml = np.ascontiguousarray(max_len, dtype=np.int32)
        n = ml.size
        p = self.params(method, int(ml.max()), b, h, stop_at_eos, max_passes, stop_rule, init)
        y_ld = int(ml.max())
        y = np.zeros((n, y_ld), dtype=np.int32)
        n_y = np.zeros(n, dtype=np.int32)
        n_it = np.zeros(n, dtype=np.int32)
        self._check(self._lib.pd_decode_batch(self._h, ctypes.byref(p), n, _i32p(ml), _i32p(y), y_ld,
                                              _i32p(n_y), _i32p(n_it)), "pd_decode_batch")
        return [DecodeResult([int(t) for t in y[s, :n_y[s]]], int(n_it[s])) for s in range(n)]

    def decode_batch_device(self, p: _DecodeParams, max_len: np.ndarray, d_y: int, y_ld: int,
                            d_info: int) -> None:
        ml = np.ascontiguousarray(max_len, dtype=np.int32)
        self._check(self._lib.pd_decode_batch_device(self._h, ctypes.byref(p), ml.size, _i32p(ml),
                                                     ctypes.c_void_p(d_y), int(y_ld),
                                                     ctypes.c_void_p(d_info)),
                    "pd_decode_batch_device")

    @staticmethod
    def params(method: str, max_len: int, b: int = 1, h: int = 0, stop_at_eos: bool = True,
               max_passes: int = 0, stop_rule: str = "paper", init: str = "pad") -> _DecodeParams:
        return _DecodeParams(METHODS[method], int(b), int(max_len), int(h), int(stop_at_eos),
                             int(max_passes), STOP_RULES[stop_rule], INITS[init])

    def decode(self, method: str, max_len: int, b: int = 1, h: int = 0,
               stop_at_eos: bool = True, max_passes: int = 0,
               trace: bool = False, stop_rule: str = "paper", init: str = "pad") -> DecodeResult:
        p = self.params(method, max_len, b, h, stop_at_eos, max_passes, stop_rule, init)
        y = np.zeros(max_len, dtype=np.int32)
        n_y, n_it, n_tr = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        if trace:
            cap = max_len
            tr = (_TraceStep * cap)()
            tt = np.full((cap, max_len), -1, dtype=np.int32)
            tp = np.zeros((cap, max_len), dtype=np.float32)
            st = self._lib.pd_decode(self._h, ctypes.byref(p), _i32p(y), ctypes.byref(n_y),
                                     ctypes.byref(n_it), tr, _i32p(tt),
                                     tp.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), cap,
                                     ctypes.byref(n_tr))
        else:
            st = self._lib.pd_decode(self._h, ctypes.byref(p), _i32p(y), ctypes.byref(n_y),
                                     ctypes.byref(n_it), None, None, None, 0, None)
        self._check(st, "pd_decode")
        res = DecodeResult([int(t) for t in y[:n_y.value]], n_it.value)
        if trace:
            k = n_tr.value
            res.trace = [{f: getattr(tr[i], f) for f, _ in _TraceStep._fields_} for i in range(k)]
            res.trace_tokens = tt[:k]
            res.trace_probs = tp[:k]
        return res

    def decode_device(self, p: _DecodeParams, d_y: int, d_info: int) -> None:
        self._check(self._lib.pd_decode_device(self._h, ctypes.byref(p), ctypes.c_void_p(d_y),
                                               ctypes.c_void_p(d_info)), "pd_decode_device")

    def debug_logits(self, y_in) -> np.ndarray:
        a = np.ascontiguousarray(y_in, dtype=np.int32)
        out = np.zeros((a.size, self.cfg.vocab), dtype=np.float32)
        self._check(self._lib.pd_debug_logits(self._h, _i32p(a), int(a.size),
                                               out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
                    "pd_debug_logits")
        return out

    def debug_logits_static(self, y_in) -> np.ndarray:
        """As debug_logits, staging the logits in the library's fixed device array instead of a
        per-call device allocation (for callers that may not allocate device memory)."""
        a = np.ascontiguousarray(y_in, dtype=np.int32)
        out = np.zeros((a.size, self.cfg.vocab), dtype=np.float32)
        self._check(self._lib.pd_debug_logits_static(
            self._h, _i32p(a), int(a.size), out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
            "pd_debug_logits_static")
        return out

    def debug_wait_timeout(self, limit_ns: int) -> int:
        """Run the device wait against a counter nothing advances, limited to limit_ns; returns
        the status the device raised (PD_ETIMEOUT expected)."""
        st = ctypes.c_int(0)
        self._check(self._lib.pd_debug_wait_timeout(self._h, ctypes.c_uint64(int(limit_ns)),
                                                    ctypes.byref(st)), "pd_debug_wait_timeout")
        return int(st.value)

    def export_weights(self, dtype) -> np.ndarray:
        out = np.zeros(self.blob_nbytes // np.dtype(dtype).itemsize, dtype=dtype)
        self._check(self._lib.pd_export_weights(self._h, out.ctypes.data_as(ctypes.c_void_p),
                                                out.nbytes), "pd_export_weights")
        return out

    @property
    def stream(self) -> int:
        return int(self._lib.pd_stream(self._h) or 0)

    @property
    def launch_count(self) -> int:
        return int(self._lib.pd_launch_count(self._h))

    def close(self) -> None:
        if getattr(self, "_h", None):
            self._lib.pd_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
