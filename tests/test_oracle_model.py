"""Pins of the oracle's transformer (oracle/model.py) against things other than itself.

* torch.nn.TransformerEncoderLayer / TransformerDecoderLayer (an independent implementation
  of the same layers) run in float64 with the same parameters: post-LN and pre-LN, ReLU /
  SiLU / GELU, with LayerNorm gains and biases perturbed so that every parameter matters.
* Closed forms of the sinusoidal position table.
* Causality: the logits at position t do not depend on inputs after t (the structure that
  makes Eq. 4 a triangular system).
* Planted mistakes: each plausible error, planted into the oracle on the CPU, fails a pin.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import model as om

SPECS = [
    synth.small_spec("post-relu", d_model=32, n_heads=4, d_ff=48, n_enc_layers=2, n_dec_layers=2,
                     vocab=40, activation=synth.ACT_RELU),
    synth.small_spec("post-silu", d_model=48, n_heads=6, d_ff=80, n_enc_layers=1, n_dec_layers=2,
                     vocab=33, activation=synth.ACT_SILU),
    synth.small_spec("pre-gelu-learned", d_model=32, n_heads=2, d_ff=64, n_enc_layers=2,
                     n_dec_layers=1, vocab=37, activation=synth.ACT_GELU, pre_ln=True,
                     learned_pos=True, max_pos=32),
]


def _torch_logits(spec, w, src, y_in):
    """The same model assembled from torch.nn layers in float64."""
    dt = torch.float64
    d = spec.d_model
    T = lambda a: torch.tensor(np.asarray(a, dtype=np.float64), dtype=dt)
    act = {synth.ACT_RELU: F.relu, synth.ACT_SILU: F.silu, synth.ACT_GELU: F.gelu}[spec.activation]

    def embed(ids, side):
        x = T(w["embed"])[torch.tensor(ids, dtype=torch.long)] * math.sqrt(d)
        n = len(ids)
        if spec.learned_pos:
            x = x + T(w["pos"])[:n]
        else:
            pos = torch.arange(n, dtype=dt)[:, None]
            freq = torch.exp(-math.log(10000.0) * torch.arange(0, d, 2, dtype=dt) / d)[None, :]
            x = x + torch.cat([torch.sin(pos * freq), torch.cos(pos * freq)], dim=1)
        if spec.pre_ln:
            x = F.layer_norm(x, (d,), T(w[side + ".ln_emb.g"]), T(w[side + ".ln_emb.b"]),
                             spec.ln_eps)
        return x[None]

    def set_ln(ln, name):
        ln.weight.copy_(T(w[name + ".g"]))
        ln.bias.copy_(T(w[name + ".b"]))

    with torch.no_grad():
        x = embed(src, "enc")
        for l in range(spec.n_enc_layers):
            p = f"enc.{l}."
            layer = torch.nn.TransformerEncoderLayer(d, spec.n_heads, spec.d_ff, dropout=0.0,
                                                     activation=act, layer_norm_eps=spec.ln_eps,
                                                     batch_first=True, norm_first=spec.pre_ln,
                                                     dtype=dt).eval()
            layer.self_attn.in_proj_weight.copy_(T(w[p + "wqkv"]))
            layer.self_attn.in_proj_bias.copy_(T(w[p + "bqkv"]))
            layer.self_attn.out_proj.weight.copy_(T(w[p + "wo"]))
            layer.self_attn.out_proj.bias.copy_(T(w[p + "bo"]))
            layer.linear1.weight.copy_(T(w[p + "w1"]))
            layer.linear1.bias.copy_(T(w[p + "b1"]))
            layer.linear2.weight.copy_(T(w[p + "w2"]))
            layer.linear2.bias.copy_(T(w[p + "b2"]))
            set_ln(layer.norm1, p + "ln1")
            set_ln(layer.norm2, p + "ln2")
            x = layer(x)
        if spec.pre_ln:
            x = F.layer_norm(x, (d,), T(w["enc.ln_final.g"]), T(w["enc.ln_final.b"]), spec.ln_eps)
        mem = x
        h = embed(y_in, "dec")
        n = len(y_in)
        mask = torch.nn.Transformer.generate_square_subsequent_mask(n, dtype=dt)
        for l in range(spec.n_dec_layers):
            p = f"dec.{l}."
            layer = torch.nn.TransformerDecoderLayer(d, spec.n_heads, spec.d_ff, dropout=0.0,
                                                     activation=act, layer_norm_eps=spec.ln_eps,
                                                     batch_first=True, norm_first=spec.pre_ln,
                                                     dtype=dt).eval()
            layer.self_attn.in_proj_weight.copy_(T(w[p + "wqkv"]))
            layer.self_attn.in_proj_bias.copy_(T(w[p + "bqkv"]))
            layer.self_attn.out_proj.weight.copy_(T(w[p + "wo"]))
            layer.self_attn.out_proj.bias.copy_(T(w[p + "bo"]))
            layer.multihead_attn.in_proj_weight.copy_(
                T(np.concatenate([w[p + "wq_c"], w[p + "wkv_c"]])))
            layer.multihead_attn.in_proj_bias.copy_(
                T(np.concatenate([w[p + "bq_c"], w[p + "bkv_c"]])))
            layer.multihead_attn.out_proj.weight.copy_(T(w[p + "wo_c"]))
            layer.multihead_attn.out_proj.bias.copy_(T(w[p + "bo_c"]))
            layer.linear1.weight.copy_(T(w[p + "w1"]))
            layer.linear1.bias.copy_(T(w[p + "b1"]))
            layer.linear2.weight.copy_(T(w[p + "w2"]))
            layer.linear2.bias.copy_(T(w[p + "b2"]))
            set_ln(layer.norm1, p + "ln1")
            set_ln(layer.norm2, p + "ln2")
            set_ln(layer.norm3, p + "ln3")
            h = layer(h, mem, tgt_mask=mask, tgt_is_causal=True)
        if spec.pre_ln:
            h = F.layer_norm(h, (d,), T(w["dec.ln_final.g"]), T(w["dec.ln_final.b"]), spec.ln_eps)
        return (h[0] @ T(w["embed"]).T).numpy()


def _case(spec, seed):
    w = synth.make_weights(spec, seed=seed, std=0.3, ln_noise=0.3).tensors
    rng = np.random.default_rng(100 + seed)
    src = rng.integers(3, spec.vocab, size=9)
    y_in = np.concatenate([[synth.BOS_ID], rng.integers(0, spec.vocab, size=6)])
    return w, src, y_in


def _max_rel_err(a, b):
    return float(np.max(np.abs(a - b)) / np.max(np.abs(b)))


@pytest.mark.parametrize("spec", SPECS, ids=lambda s: s.name)
def test_model_matches_torch_nn(spec):
    for seed in (0, 1):
        w, src, y_in = _case(spec, seed)
        m = om.Model(spec, w)
        ours = m.logits(m.encode(src), y_in)
        ref = _torch_logits(spec, w, src, y_in)
        assert _max_rel_err(ours, ref) < 1e-10


def test_sinusoid_closed_forms():
    d = 16
    pe = om.sinusoid(np.arange(50), d)
    # position 0: all sines 0, all cosines 1
    assert np.array_equal(pe[0], np.r_[np.zeros(d // 2), np.ones(d // 2)])
    # each (sin, cos) pair lies on the unit circle
    assert np.allclose(pe[:, :d // 2] ** 2 + pe[:, d // 2:] ** 2, 1.0, atol=1e-15)
    # column k turns by w_k = 10000^(-2k/d) per position: the angle at position 1 is w_k
    ang = np.arctan2(pe[1, :d // 2], pe[1, d // 2:])
    assert np.allclose(ang, 10000.0 ** (-2.0 * np.arange(d // 2) / d), atol=1e-15)
    # column 0 has frequency 1: sin(p) itself
    assert np.allclose(pe[:, 0], np.sin(np.arange(50)), atol=1e-15)


def test_layer_norm_special_cases():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((4, 64)) * 3 + 5
    y = om.layer_norm(x, np.ones(64), np.zeros(64), 0.0)
    assert np.allclose(y.mean(1), 0, atol=1e-13) and np.allclose(y.std(1), 1, atol=1e-13)
    c = om.layer_norm(np.full((1, 8), 7.0), np.ones(8), np.arange(8.0), 1e-5)
    assert np.allclose(c, np.arange(8.0))          # a constant row maps to the bias


def test_activation_closed_forms():
    x = np.array([-2.0, -0.5, 0.0, 0.5, 3.0])
    assert np.array_equal(om.activation(x, synth.ACT_RELU), [0, 0, 0, 0.5, 3.0])
    assert np.allclose(om.activation(x, synth.ACT_SILU), x / (1 + np.exp(-x)))
    # GELU(x) = x * Phi(x): Phi(1) from the normal table, and Phi(-x) = 1 - Phi(x) gives
    # GELU(x) - GELU(-x) = x
    g = om.activation(x, synth.ACT_GELU)
    assert g[2] == 0.0
    assert np.isclose(om.activation(np.array([1.0]), synth.ACT_GELU)[0], 0.8413447460685429)
    assert np.allclose(g - om.activation(-x, synth.ACT_GELU), x, atol=1e-15)


@pytest.mark.parametrize("spec", SPECS[:2], ids=lambda s: s.name)
def test_decoder_is_causal(spec):
    """Logits of row t depend only on inputs 0..t: truncating or changing later inputs leaves
    them unchanged (bit for bit: the computation over earlier rows is the same)."""
    w, src, y_in = _case(spec, 3)
    m = om.Model(spec, w)
    mem = m.encode(src)
    full = m.logits(mem, y_in)
    for t in range(1, len(y_in)):
        part = m.logits(mem, y_in[:t])
        assert np.allclose(part, full[:t], rtol=0, atol=1e-12)
        changed = y_in.copy()
        changed[t:] = (changed[t:] + 1) % spec.vocab
        assert np.allclose(m.logits(mem, changed)[:t], full[:t], rtol=0, atol=1e-12)


def test_top2_tie_break_and_margin():
    lg = np.array([[0.1, 0.5, 0.5, -1.0], [3.0, 1.0, 2.5, 0.0]])
    idx, margin, prob = om.top2(lg)
    assert list(idx) == [1, 0]                      # equal maxima: the lowest index wins
    assert margin[0] == 0.0 and np.isclose(margin[1], 0.5)
    assert np.isclose(prob[1], np.exp(3.0) / np.exp(lg[1]).sum())


# ---- planted mistakes: every one must break a pin above -------------------------------------

def _no_causal_mask(orig):
    def f(*a, **k):
        a = list(a)
        a[-1] = False
        return orig(*a, **k)
    return f


def _bad_scale(orig_attention):
    def f(xq, xkv, wq, bq, *rest):
        return orig_attention(xq * 1.0001, xkv, wq, bq, *rest)
    return f


def _wrap_attention(change):
    """Plant a mistake in the arguments every attention call receives."""
    def patch(mp):
        orig = om.attention

        def f(*args):
            return orig(*change(*args))
        mp.setattr(om, "attention", f)
    return patch


def _wrap_method(name, make):
    def patch(mp):
        mp.setattr(om.Model, name, make(getattr(om.Model, name)))
    return patch


MUTATIONS = {
    "no causal mask": lambda mp: mp.setattr(om, "attention", _no_causal_mask(om.attention)),
    "sin/cos swapped": lambda mp: mp.setattr(
        om, "sinusoid", (lambda orig: lambda p, d: orig(p, d)[:, ::-1])(om.sinusoid)),
    "LN without eps": lambda mp: mp.setattr(
        om, "layer_norm", (lambda orig: lambda x, g, b, eps: orig(x, g, b, 0.0))(om.layer_norm)),
    "LN gain ignored": lambda mp: mp.setattr(
        om, "layer_norm", (lambda orig: lambda x, g, b, eps: orig(x, 1.0, b, eps))(om.layer_norm)),
    "query perturbed": lambda mp: mp.setattr(om, "attention", _bad_scale(om.attention)),
    "relu for silu": lambda mp: mp.setattr(
        om, "activation", (lambda orig: lambda x, k: orig(x, synth.ACT_RELU))(om.activation)),
    "keys and values swapped": _wrap_attention(
        lambda xq, xkv, wq, bq, wk, bk, wv, bv, wo, bo, h, c:
        (xq, xkv, wq, bq, wv, bv, wk, bk, wo, bo, h, c)),
    "output projection transposed": _wrap_attention(
        lambda xq, xkv, wq, bq, wk, bk, wv, bv, wo, bo, h, c:
        (xq, xkv, wq, bq, wk, bk, wv, bv, wo.T, bo, h, c)),
    "heads merged into one": _wrap_attention(
        lambda xq, xkv, wq, bq, wk, bk, wv, bv, wo, bo, h, c:
        (xq, xkv, wq, bq, wk, bk, wv, bv, wo, bo, 1, c)),
    "embedding not scaled by sqrt(d)": _wrap_method(
        "embed", lambda orig: lambda self, ids, side:
        orig(self, ids, side) - self.w["embed"][np.asarray(ids)] * (math.sqrt(self.s.d_model) - 1)),
    "positions shifted by one": _wrap_method(
        "embed", lambda orig: lambda self, ids, side:
        orig(self, ids, side) - om.sinusoid(np.arange(len(ids)), self.s.d_model)
        + om.sinusoid(np.arange(1, len(ids) + 1), self.s.d_model)),
    "cross-attention to the decoder states": _wrap_method(
        "_cross_attn", lambda orig: lambda self, x, mem, p: orig(self, x, x, p)),
}


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistake_is_caught(name, monkeypatch):
    spec = SPECS[1]
    w, src, y_in = _case(spec, 0)
    ref = _torch_logits(spec, w, src, y_in)
    MUTATIONS[name](monkeypatch)
    m = om.Model(spec, w)
    ours = m.logits(m.encode(src), y_in)
    caught_by_torch = _max_rel_err(ours, ref) >= 1e-10
    caught_by_closed_form = False
    try:
        test_sinusoid_closed_forms()
    except AssertionError:
        caught_by_closed_form = True
    assert caught_by_torch or caught_by_closed_form
