"""Seeded synthetic inputs shared by the oracle and the CUDA path.

This module holds no arithmetic of the decoding method: it only draws numbers
(weights, source sentences) and packs them in the documented blob order.  Both
sides of every parity test take their inputs from here and nothing else.

Model presets are named by what they are.  The paper evaluates a base
transformer (d=512, 6+6 layers, Opus-MT, 74M parameters) and a big one
(d=1024, 12+12 layers, MBart50, 610M parameters), Section 4.1 "Model
Configuration"; their trained weights and the WMT/IWSLT/FLORES test sets are
not available, so seeded N(0, 0.02) weights and uniform random source ids of
the same shapes stand in for them.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Iterator, List, Tuple

import numpy as np

# Special token ids shared by every preset (the tiny model fixes them).
EOS_ID = 0
PAD_ID = 1
BOS_ID = 2
FIRST_WORD_ID = 3

ACT_RELU = 0
ACT_SILU = 1
ACT_GELU = 2

DTYPE_F32 = 0
DTYPE_BF16 = 1


@dataclasses.dataclass(frozen=True)
class ModelSpec:
    """Shape and structural choices of one encoder-decoder transformer."""

    name: str
    d_model: int
    n_heads: int
    d_ff: int
    n_enc_layers: int
    n_dec_layers: int
    vocab: int
    activation: int          # ACT_*
    pre_ln: bool             # False: x = LN(x + f(x)); True: x = x + f(LN(x)) + final LNs
    learned_pos: bool        # False: sinusoidal; True: learned table of max_pos rows
    max_pos: int             # rows of the learned table (and the position cap)
    dtype: int               # DTYPE_F32 or DTYPE_BF16 (storage of every parameter)
    ln_eps: float = 1e-5

    @property
    def d_head(self) -> int:
        return self.d_model // self.n_heads


TINY = ModelSpec("tiny-f32", 256, 4, 1024, 2, 2, 8000, ACT_RELU, False, False, 1024, DTYPE_F32)
MARIAN = ModelSpec("marian-base-bf16", 512, 8, 2048, 6, 6, 58101, ACT_SILU, False, False, 1024,
                   DTYPE_BF16)
MBART = ModelSpec("mbart-large-bf16", 1024, 16, 4096, 12, 12, 250027, ACT_GELU, True, True, 1024,
                  DTYPE_BF16)

PRESETS = {s.name: s for s in (TINY, MARIAN, MBART)}


def small_spec(name="toy", d_model=32, n_heads=4, d_ff=64, n_enc_layers=1, n_dec_layers=2,
               vocab=24, activation=ACT_RELU, pre_ln=False, learned_pos=False, max_pos=64,
               dtype=DTYPE_F32) -> ModelSpec:
    """A toy model for brute-force and structural tests."""
    return ModelSpec(name, d_model, n_heads, d_ff, n_enc_layers, n_dec_layers, vocab, activation,
                     pre_ln, learned_pos, max_pos, dtype)


# --------------------------------------------------------------------------------------------
# Blob layout.  Every tensor is row-major; linear maps are stored [out_features, in_features]
# and act as y = x W^T + b.  The order below is the on-disk / on-wire order of the blob.
# --------------------------------------------------------------------------------------------

def tensor_layout(s: ModelSpec) -> List[Tuple[str, Tuple[int, ...]]]:
    d, f, V = s.d_model, s.d_ff, s.vocab
    out: List[Tuple[str, Tuple[int, ...]]] = [("embed", (V, d))]
    if s.learned_pos:
        out.append(("pos", (s.max_pos, d)))
    if s.pre_ln:
        out += [("enc.ln_emb.g", (d,)), ("enc.ln_emb.b", (d,)),
                ("dec.ln_emb.g", (d,)), ("dec.ln_emb.b", (d,)),
                ("enc.ln_final.g", (d,)), ("enc.ln_final.b", (d,)),
                ("dec.ln_final.g", (d,)), ("dec.ln_final.b", (d,))]
    for l in range(s.n_enc_layers):
        p = f"enc.{l}."
        out += [(p + "wqkv", (3 * d, d)), (p + "bqkv", (3 * d,)),
                (p + "wo", (d, d)), (p + "bo", (d,)),
                (p + "ln1.g", (d,)), (p + "ln1.b", (d,)),
                (p + "w1", (f, d)), (p + "b1", (f,)),
                (p + "w2", (d, f)), (p + "b2", (d,)),
                (p + "ln2.g", (d,)), (p + "ln2.b", (d,))]
    for l in range(s.n_dec_layers):
        p = f"dec.{l}."
        out += [(p + "wqkv", (3 * d, d)), (p + "bqkv", (3 * d,)),
                (p + "wo", (d, d)), (p + "bo", (d,)),
                (p + "ln1.g", (d,)), (p + "ln1.b", (d,)),
                (p + "wq_c", (d, d)), (p + "bq_c", (d,)),
                (p + "wkv_c", (2 * d, d)), (p + "bkv_c", (2 * d,)),
                (p + "wo_c", (d, d)), (p + "bo_c", (d,)),
                (p + "ln2.g", (d,)), (p + "ln2.b", (d,)),
                (p + "w1", (f, d)), (p + "b1", (f,)),
                (p + "w2", (d, f)), (p + "b2", (d,)),
                (p + "ln3.g", (d,)), (p + "ln3.b", (d,))]
    return out


def n_params(s: ModelSpec) -> int:
    return int(sum(np.prod(shape) for _, shape in tensor_layout(s)))


def _round_to_bf16(f: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (to nearest, ties to even); returns the uint16 bits."""
    u = np.ascontiguousarray(f, dtype=np.float32).view(np.uint32)
    rounding = ((u >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + rounding) >> 16).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class Weights:
    """The generated parameters: named float32 arrays holding exactly the stored values
    (bf16 values are exact in float32) and the packed blob that the C ABI takes."""

    spec: ModelSpec
    tensors: Dict[str, np.ndarray]
    blob: np.ndarray     # uint16 (bf16 bits) or float32, flat, in tensor_layout order


def make_weights(s: ModelSpec, seed: int = 0, std: float = 0.02, ln_noise: float = 0.0,
                 eos_boost: float = 1.0, embed_std: float = None) -> Weights:
    """Draw every tensor of ``tensor_layout(s)`` in order from one numpy PCG64 stream of
    float32 standard normals ``z``.

    Weights and biases are ``std * z``; LayerNorm gains are ``1 + ln_noise * z`` and biases
    ``ln_noise * z`` (``ln_noise = 0`` gives the usual 1 / 0 initialisation).  ``eos_boost``
    scales the EOS row of the (tied) embedding, a knob that makes EOS frequent in tests;
    ``embed_std`` (default ``std``) draws the token embedding (and a learned position table)
    with its own scale, a knob that sets how strongly a prediction follows its input token.
    bf16 presets round each value to nearest-even bf16.
    """
    rng = np.random.default_rng(seed)
    tensors: Dict[str, np.ndarray] = {}
    parts = []
    for name, shape in tensor_layout(s):
        z = rng.standard_normal(shape, dtype=np.float32)
        parts_of_name = name.split(".")
        is_ln = len(parts_of_name) >= 2 and parts_of_name[-2].startswith("ln")
        if is_ln and parts_of_name[-1] == "g":
            v = np.float32(1.0) + np.float32(ln_noise) * z
        elif is_ln and parts_of_name[-1] == "b":
            v = np.float32(ln_noise) * z
        elif name in ("embed", "pos") and embed_std is not None:
            v = np.float32(embed_std) * z
        else:
            v = np.float32(std) * z
        if name == "embed" and eos_boost != 1.0:
            v[EOS_ID] *= np.float32(eos_boost)
        if s.dtype == DTYPE_BF16:
            bits = _round_to_bf16(v).reshape(-1)
            parts.append(bits)
            tensors[name] = bf16_bits_to_f32(bits).reshape(shape)
        else:
            f = np.ascontiguousarray(v, dtype=np.float32).reshape(-1)
            parts.append(f)
            tensors[name] = f.reshape(shape)
    blob = np.concatenate(parts)
    return Weights(s, tensors, blob)


def weights_from_blob(s: ModelSpec, blob: np.ndarray) -> Dict[str, np.ndarray]:
    """Unpack a blob (as exported by the library) into named float32 arrays."""
    out = {}
    off = 0
    for name, shape in tensor_layout(s):
        n = int(np.prod(shape))
        chunk = blob[off:off + n]
        off += n
        if s.dtype == DTYPE_BF16:
            out[name] = bf16_bits_to_f32(chunk.view(np.uint16)).reshape(shape)
        else:
            out[name] = chunk.view(np.float32).reshape(shape)
    if off != blob.size:
        raise ValueError(f"blob has {blob.size} elements, layout needs {off}")
    return out


# --------------------------------------------------------------------------------------------
# Source sentences
# --------------------------------------------------------------------------------------------

def sentences(seed: int, count: int, len_lo: int, len_hi: int, vocab: int) -> List[np.ndarray]:
    """``count`` source sentences with lengths uniform in [len_lo, len_hi] and ids uniform in
    [FIRST_WORD_ID, vocab) (special ids excluded), as int32 arrays."""
    rng = np.random.default_rng(seed)
    lens = rng.integers(len_lo, len_hi + 1, size=count)
    return [rng.integers(FIRST_WORD_ID, vocab, size=int(n)).astype(np.int32) for n in lens]


@dataclasses.dataclass(frozen=True)
class Workload:
    """One benchmark / parity workload: a model, its sentences and the decoding settings."""

    name: str
    spec: ModelSpec
    weight_seed: int
    sentence_seed: int
    n_sentences: int
    len_lo: int
    len_hi: int
    method: str
    b: int
    max_len_factor: int      # max_len = factor * src_len (0: max_len = fixed_max_len)
    fixed_max_len: int = 0
    embed_std: float = None  # token-embedding scale of the weights (None: the weight std)

    def weights(self) -> "Weights":
        return make_weights(self.spec, seed=self.weight_seed, embed_std=self.embed_std)

    def sentences(self) -> List[np.ndarray]:
        return sentences(self.sentence_seed, self.n_sentences, self.len_lo, self.len_hi,
                         self.spec.vocab)

    def max_len(self, src_len: int) -> int:
        return self.max_len_factor * src_len if self.max_len_factor else self.fixed_max_len


# Tiny fp32 model, one 16-id sentence, full-sentence Jacobi with b = max_len = 16.
TINY_JACOBI = Workload("tiny-f32 jacobi b=16, 1 sentence of 16 ids", TINY, 0, 1, 1, 16, 16,
                       "jacobi", 16, 0, 16)
# Marian-like bf16 model, 256 sentences of 8..64 ids, GS-Jacobi b=5, max_len = 2 * src_len.
MARIAN_GS = Workload("marian-base-bf16 gs_jacobi b=5, 256 sentences of 8..64 ids, max_len=2n",
                     MARIAN, 0, 1, 256, 8, 64, "gs_jacobi", 5, 2)
# Same model and sentences: hybrid b=3 and full-sentence Jacobi.
MARIAN_HYBRID = dataclasses.replace(MARIAN_GS, name="marian-base-bf16 hybrid_gs_jacobi b=3",
                                    method="hybrid_gs_jacobi", b=3)
MARIAN_JACOBI = dataclasses.replace(MARIAN_GS, name="marian-base-bf16 jacobi b=max_len",
                                    method="jacobi", b=0)
# The Marian-sized model with a 20x smaller token-embedding scale ("dependency knob"): its
# predictions depend less on the previous token, so Jacobi iterations accept several positions
# per pass -- the mechanism behind the paper's speedups, which random weights otherwise lack.
MARIAN_KNOB = dataclasses.replace(
    MARIAN_GS, name="marian-base-bf16 embed_std=0.001 gs_jacobi b=5, 256 sentences of 8..64 ids, "
                    "max_len=2n", embed_std=0.001)
# mBART-like bf16 model, 128 sentences of 16..128 ids, GS-Jacobi b=5 (and 16).
MBART_GS = Workload("mbart-large-bf16 gs_jacobi b=5, 128 sentences of 16..128 ids, max_len=2n",
                    MBART, 0, 1, 128, 16, 128, "gs_jacobi", 5, 2)


def iter_sentences(w: Workload) -> Iterator[Tuple[int, np.ndarray]]:
    for k, s in enumerate(w.sentences()):
        yield k, s
