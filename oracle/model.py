"""Float64 encoder-decoder transformer: the conditional model p_theta(y_i | y_<i, x) of Eq. 1.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper evaluates pretrained Marian/Opus and MBart50 models (Section 4.1, "Model
Configuration") through a standard library; it does not restate the architecture.  This file
writes out the textbook transformer with the structural choices each preset names:

* token embedding scaled by sqrt(d_model), tied with the output projection (no logits bias);
* positions: sinusoidal with [sin | cos] halves and frequency 10000^(-2k/d) starting at
  position 0, or a learned table indexed by the position itself;
* post-LN blocks x = LN(x + f(x)), or pre-LN blocks x = x + f(LN(x)) with an embedding LN and a
  final LN on each stack;
* multi-head attention with scale 1/sqrt(d_head); causal self-attention in the decoder;
  unmasked cross-attention to the encoder output;
* FFN act(x W1^T + b1) W2^T + b2 with ReLU, SiLU (x * sigmoid(x)) or exact-erf GELU;
* LayerNorm with biased variance and eps = 1e-5.

No KV cache: every call recomputes the whole prefix, so there is no cache to get wrong.
"""
from __future__ import annotations

import math
from typing import Dict

import numpy as np
from scipy.special import erf

import synth


def layer_norm(x: np.ndarray, g: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def sinusoid(positions: np.ndarray, d: int) -> np.ndarray:
    """Row p = [sin(p w_0) .. sin(p w_{d/2-1}) | cos(p w_0) .. cos(p w_{d/2-1})],
    w_k = 10000^(-2k/d)."""
    k = np.arange(d // 2, dtype=np.float64)
    w = 10000.0 ** (-2.0 * k / d)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * w[None, :]
    return np.concatenate([np.sin(ang), np.cos(ang)], axis=1)


def activation(x: np.ndarray, kind: int) -> np.ndarray:
    if kind == synth.ACT_RELU:
        return np.maximum(x, 0.0)
    if kind == synth.ACT_SILU:
        return x / (1.0 + np.exp(-x))
    if kind == synth.ACT_GELU:
        return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))
    raise ValueError(kind)


def attention(xq: np.ndarray, xkv: np.ndarray, wq, bq, wk, bk, wv, bv, wo, bo, n_heads: int,
              causal: bool) -> np.ndarray:
    """Multi-head attention: softmax(Q K^T / sqrt(d_head) [+ causal mask]) V, heads
    concatenated, then the output projection."""
    T, d = xq.shape
    S = xkv.shape[0]
    dh = d // n_heads
    q = xq @ wq.T + bq
    k = xkv @ wk.T + bk
    v = xkv @ wv.T + bv
    out = np.empty((T, d))
    for h in range(n_heads):
        sl = slice(h * dh, (h + 1) * dh)
        s = q[:, sl] @ k[:, sl].T / math.sqrt(dh)
        if causal:
            s = np.where(np.arange(S)[None, :] <= np.arange(T)[:, None], s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, sl] = p @ v[:, sl]
    return out @ wo.T + bo


class Model:
    """The transformer with float64 copies of a ``synth.Weights`` parameter set."""

    def __init__(self, spec: synth.ModelSpec, tensors: Dict[str, np.ndarray]):
        self.s = spec
        self.w = {k: np.asarray(v, dtype=np.float64) for k, v in tensors.items()}

    # -- embeddings -------------------------------------------------------------------------
    def embed(self, ids: np.ndarray, side: str) -> np.ndarray:
        s, w = self.s, self.w
        ids = np.asarray(ids, dtype=np.int64)
        pos = np.arange(len(ids))
        x = w["embed"][ids] * math.sqrt(s.d_model)
        x = x + (w["pos"][pos] if s.learned_pos else sinusoid(pos, s.d_model))
        if s.pre_ln:
            x = layer_norm(x, w[side + ".ln_emb.g"], w[side + ".ln_emb.b"], s.ln_eps)
        return x

    def _ln(self, x, name):
        return layer_norm(x, self.w[name + ".g"], self.w[name + ".b"], self.s.ln_eps)

    def _ffn(self, x, p):
        w = self.w
        return activation(x @ w[p + "w1"].T + w[p + "b1"], self.s.activation) @ w[p + "w2"].T \
            + w[p + "b2"]

    def _self_attn(self, x, p, causal):
        w, d = self.w, self.s.d_model
        wqkv, bqkv = w[p + "wqkv"], w[p + "bqkv"]
        return attention(x, x, wqkv[:d], bqkv[:d], wqkv[d:2 * d], bqkv[d:2 * d],
                         wqkv[2 * d:], bqkv[2 * d:], w[p + "wo"], w[p + "bo"], self.s.n_heads,
                         causal)

    def _cross_attn(self, x, mem, p):
        w, d = self.w, self.s.d_model
        wkv, bkv = w[p + "wkv_c"], w[p + "bkv_c"]
        return attention(x, mem, w[p + "wq_c"], w[p + "bq_c"], wkv[:d], bkv[:d], wkv[d:],
                         bkv[d:], w[p + "wo_c"], w[p + "bo_c"], self.s.n_heads, False)

    # -- stacks -----------------------------------------------------------------------------
    def encode(self, src: np.ndarray) -> np.ndarray:
        """Encoder output for the source ids x_1..x_n (no BOS/EOS added): [n, d]."""
        s = self.s
        x = self.embed(src, "enc")
        for l in range(s.n_enc_layers):
            p = f"enc.{l}."
            if s.pre_ln:
                x = x + self._self_attn(self._ln(x, p + "ln1"), p, False)
                x = x + self._ffn(self._ln(x, p + "ln2"), p)
            else:
                x = self._ln(x + self._self_attn(x, p, False), p + "ln1")
                x = self._ln(x + self._ffn(x, p), p + "ln2")
        if s.pre_ln:
            x = self._ln(x, "enc.ln_final")
        return x

    def decoder_hidden(self, mem: np.ndarray, y_in: np.ndarray) -> np.ndarray:
        """Final decoder hidden states for the input tokens y_in (positions 0..T-1), teacher
        forced with a causal mask: [T, d]."""
        s = self.s
        h = self.embed(y_in, "dec")
        for l in range(s.n_dec_layers):
            p = f"dec.{l}."
            if s.pre_ln:
                h = h + self._self_attn(self._ln(h, p + "ln1"), p, True)
                h = h + self._cross_attn(self._ln(h, p + "ln2"), mem, p)
                h = h + self._ffn(self._ln(h, p + "ln3"), p)
            else:
                h = self._ln(h + self._self_attn(h, p, True), p + "ln1")
                h = self._ln(h + self._cross_attn(h, mem, p), p + "ln2")
                h = self._ln(h + self._ffn(h, p), p + "ln3")
        if s.pre_ln:
            h = self._ln(h, "dec.ln_final")
        return h

    def logits(self, mem: np.ndarray, y_in: np.ndarray) -> np.ndarray:
        """Row t holds the scores of p_theta(y_{t+1} | y_0..y_t, x) (Eq. 1) over the vocabulary,
        with y_0 = BOS: [T, V]."""
        return self.decoder_hidden(mem, y_in) @ self.w["embed"].T


def top2(logits: np.ndarray):
    """Per row: argmax (lowest index among equal maxima, Eq. 2), the top-1 minus top-2 margin,
    and the softmax probability of the argmax token."""
    lg = np.atleast_2d(logits)
    if np.isnan(lg).any():
        raise FloatingPointError("NaN logits")
    idx = np.argmax(lg, axis=1)
    mx = lg[np.arange(lg.shape[0]), idx]
    part = np.partition(lg, -2, axis=1)
    second = part[:, -2]
    prob = 1.0 / np.exp(lg - mx[:, None]).sum(axis=1)
    return idx, mx - second, prob
