"""Pins of the oracle's decoding algorithms (oracle/decode.py).

* Planted dependency structures (mock passes) with closed-form pass counts: a position-only
  model needs 2 passes per block, a chain y_p = g(y_{p-1}) needs exactly blk passes, a skip
  chain y_p = g(y_{p-2}) needs min(blk, ceil(blk/2) + 1) under Eq. 5 and ceil((blk+1)/2) under
  the accepted-prefix rule.
* Brute force over every token sequence of a toy transformer: the triangular system of Eq. 4
  has exactly one solution, and it is the greedy output of Eq. 2.
* Proposition 1: Jacobi, GS-Jacobi and Hybrid GS-Jacobi return the greedy tokens from PAD and
  from random initial drafts, in at most m passes.
* Structural identities: GS-Jacobi with b = 1 is greedy pass for pass; Jacobi is GS-Jacobi
  with b = m; one teacher-forced pass over the greedy output reproduces it (Eq. 4, f = 0).
* Full per-pass traces on the planted structures equal the hand-derived ones of
  tests/golden/planted_traces.txt (StopC flags, unchanged-prefix counts, block starts, EOS
  index, both stop rules, hybrid EOS exit and greedy tail).
* Planted mistakes in the loops are caught.
"""
import itertools
import math
import os

import numpy as np
import pytest

import synth
from oracle import decode as od
from oracle import model as om

PAD, BOS, EOS = synth.PAD_ID, synth.BOS_ID, synth.EOS_ID
V_MOCK = 41          # mock vocabulary; true tokens live in [4, V_MOCK), 3 marks "derived from PAD"


def _g(v):
    """A bijection of [4, V_MOCK) (plus BOS mapped inside it); PAD and 3 map to 3, a value
    no true token takes, so a draft never matches the solution by accident."""
    if v in (PAD, 3):
        return 3
    if v == BOS:
        return 11
    return 4 + ((v - 4) * 7 + 5) % (V_MOCK - 4)


def position_only(eos_at=None):
    def step(inputs):
        p = np.arange(1, len(inputs) + 1)
        pred = 4 + (p * 13 + 2) % (V_MOCK - 4)
        if eos_at is not None:
            pred = np.where(p == eos_at, EOS, pred)
        return od.StepOut(pred)
    return step


def chain(inputs):
    return od.StepOut(np.array([_g(v) for v in inputs]))


def skip_chain(inputs):
    pred = [17] + [_g(inputs[t - 1]) for t in range(1, len(inputs))]
    return od.StepOut(np.array(pred))


def _blocks(m, b):
    return [min(b, m - i + 1) for i in range(1, m + 1, b)]


@pytest.mark.parametrize("m,b", [(1, 1), (5, 1), (7, 3), (10, 5), (12, 4), (9, 9), (16, 16)])
def test_closed_form_pass_counts(m, b):
    blocks = _blocks(m, b)
    for rule in ("paper", "prefix"):
        r = od.gs_jacobi(position_only(), m, b, stop_rule=rule, stop_at_eos=False)
        assert r.n_iters == sum(1 if k == 1 else 2 for k in blocks)
        r = od.gs_jacobi(chain, m, b, stop_rule=rule, stop_at_eos=False)
        assert r.n_iters == sum(blocks)
    r = od.gs_jacobi(skip_chain, m, b, stop_rule="paper", stop_at_eos=False)
    assert r.n_iters == sum(min(k, math.ceil(k / 2) + 1) for k in blocks)
    r = od.gs_jacobi(skip_chain, m, b, stop_rule="prefix", stop_at_eos=False)
    assert r.n_iters == sum(math.ceil((k + 1) / 2) for k in blocks)


def test_mock_solutions_are_the_greedy_ones():
    for step in (position_only(), chain, skip_chain):
        g = od.greedy(step, 13, stop_at_eos=False)
        for b in (1, 2, 3, 5, 13):
            assert od.gs_jacobi(step, 13, b, stop_at_eos=False).tokens == g.tokens
        assert od.hybrid_gs_jacobi(step, 13, 4).tokens == g.tokens


def test_trace_rows_of_a_chain_block():
    r = od.gs_jacobi(chain, 4, 4, stop_at_eos=False)
    assert [t.n_converged for t in r.trace] == [0, 1, 2, 3]
    assert [t.stop for t in r.trace] == [False] * 4
    assert all(t.block_start == 1 and t.block_len == 4 for t in r.trace)
    assert r.trace[-1].tokens == r.tokens


GOLDEN_TRACES = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                             "planted_traces.txt")


def _golden_trace_cases():
    cases = []
    for line in open(GOLDEN_TRACES):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        if line.startswith("case "):
            f = line.split()
            cases.append(dict(kv.split("=") for kv in f[3:]))
            cases[-1].update(structure=f[1], method=f[2], header=line[5:], rows=[])
        else:
            cases[-1]["rows"].append(tuple(int(v) for v in line.split()))
    return cases


@pytest.mark.parametrize("case", _golden_trace_cases(), ids=lambda c: c["header"])
def test_golden_planted_traces(case):
    eos_at = int(case["eos"]) if "eos" in case else None
    step = {"position_only": position_only(eos_at), "chain": chain,
            "skip_chain": skip_chain}[case["structure"]]
    m, b, rule = int(case["m"]), int(case["b"]), case["rule"]
    if case["method"] == "jacobi":
        r = od.jacobi(step, m, stop_at_eos=False, stop_rule=rule)
    elif case["method"] == "gs_jacobi":
        r = od.gs_jacobi(step, m, b, stop_at_eos=False, stop_rule=rule)
    else:
        r = od.hybrid_gs_jacobi(step, m, b, h=int(case["h"]) if "h" in case else None,
                                stop_rule=rule)
    got = [(t.step, t.block_start, t.block_len, t.n_converged, int(t.stop), t.eos_idx)
           for t in r.trace]
    assert got == case["rows"]
    assert r.n_iters == len(case["rows"])
    assert len(r.tokens) == int(case["tokens"])
    assert r.tokens == od.greedy(step, m, stop_at_eos=case["method"] == "hybrid_gs_jacobi").tokens


def test_hybrid_eos_and_tail():
    step = position_only(eos_at=7)
    g = od.greedy(step, 20)
    assert g.tokens[-1] == EOS and len(g.tokens) == 7 and g.n_iters == 7
    r = od.hybrid_gs_jacobi(step, 20, 3)                 # blocks [1,3] [4,6] [7,9]
    assert r.tokens == g.tokens and r.n_iters == 6
    r = od.hybrid_gs_jacobi(step, 20, 3, h=5)            # blocks [1,3] [4,5], then AR 6, 7
    assert r.tokens == g.tokens and r.n_iters == 2 + 2 + 2
    r = od.gs_jacobi(step, 20, 3)                        # m known: solves all 20, cuts at EOS
    assert r.tokens == g.tokens and r.n_iters == 2 * 6 + 2
    r = od.hybrid_gs_jacobi(position_only(), 10, 3, h=4)  # no EOS: blocks to 4, AR to 10
    assert r.tokens == od.greedy(position_only(), 10).tokens and r.n_iters == 2 + 1 + 6


# ---- toy transformers ------------------------------------------------------------------------

TOYS = [
    # post-LN, ReLU: with these scales the model copies its input token, a dependency chain
    # that needs all m passes
    (synth.small_spec("toy-post", d_model=16, n_heads=2, d_ff=32, n_enc_layers=1,
                      n_dec_layers=2, vocab=6),
     dict(std=0.15, embed_std=0.2, ln_noise=0.3)),
    # pre-LN, GELU, learned positions: varied token sequences
    (synth.small_spec("toy-pre", d_model=16, n_heads=2, d_ff=32, n_enc_layers=1,
                      n_dec_layers=2, vocab=6, activation=synth.ACT_GELU, pre_ln=True,
                      learned_pos=True, max_pos=16),
     dict(std=0.8, embed_std=0.1, ln_noise=0.2)),
]


def _toy(toy, seed):
    spec, kw = toy
    w = synth.make_weights(spec, seed=seed, **kw)
    src = np.random.default_rng(seed + 50).integers(3, spec.vocab, size=5)
    m = om.Model(spec, w.tensors)
    return m, src


@pytest.mark.parametrize("toy", TOYS, ids=lambda t: t[0].name)
def test_brute_force_unique_fixed_point_is_greedy(toy):
    """Every y in V^m is checked against the m equations y_i = argmax p(. | y_<i, x) (one
    teacher-forced pass over its own tokens); exactly one satisfies all of them: greedy's."""
    m_len = 4
    spec = toy[0]
    for seed in (0, 1):
        model, src = _toy(toy, seed)
        mem = model.encode(src)
        hits = []
        for cand in itertools.product(range(spec.vocab), repeat=m_len):
            lg = model.logits(mem, np.array((BOS,) + cand[:-1]))
            if tuple(np.argmax(lg, axis=1)) == cand:
                hits.append(list(cand))
        g = od.greedy(od.model_step(model, src), m_len, stop_at_eos=False)
        assert hits == [g.tokens]


@pytest.mark.parametrize("toy", TOYS, ids=lambda t: t[0].name)
def test_proposition_1_any_init(toy):
    m_len = 9
    spec = toy[0]
    rng = np.random.default_rng(7)
    for seed in range(3):
        model, src = _toy(toy, seed)
        step = od.model_step(model, src)
        g = od.greedy(step, m_len, stop_at_eos=False)
        inits = [None] + [list(rng.integers(0, spec.vocab, size=m_len)) for _ in range(3)]
        for init in inits:
            for b in (1, 2, 3, 5, m_len):
                r = od.gs_jacobi(step, m_len, b, init=init, stop_at_eos=False)
                assert r.tokens == g.tokens and r.n_iters <= m_len
            r = od.jacobi(step, m_len, init=init, stop_at_eos=False)
            assert r.tokens == g.tokens and r.n_iters <= m_len
        ge = od.greedy(step, m_len)
        r = od.hybrid_gs_jacobi(step, m_len, 3)
        assert r.tokens == ge.tokens and r.n_iters <= m_len


@pytest.mark.parametrize("toy", TOYS, ids=lambda t: t[0].name)
def test_structural_identities(toy):
    m_len = 8
    model, src = _toy(toy, 4)
    step = od.model_step(model, src)
    g = od.greedy(step, m_len, stop_at_eos=False)
    b1 = od.gs_jacobi(step, m_len, 1, stop_at_eos=False)
    assert b1.tokens == g.tokens and b1.n_iters == g.n_iters == m_len
    assert [t.tokens for t in b1.trace] == [t.tokens for t in g.trace]
    j = od.jacobi(step, m_len, stop_at_eos=False)
    gm = od.gs_jacobi(step, m_len, m_len, stop_at_eos=False)
    assert j.tokens == gm.tokens and j.n_iters == gm.n_iters
    # Eq. 4: one teacher-forced pass over y returns y (f(y_i, y_<i, x) = 0 for all i)
    out = step([BOS] + g.tokens[:-1])
    assert list(out.pred) == g.tokens


def test_tiny_preset_jacobi_matches_greedy():
    """The tiny fp32 preset (2+2 layers, d=256, V=8000), one 16-id sentence: full-sentence
    Jacobi with b = max_len = 16 from PAD returns the greedy tokens in <= 16 passes."""
    w = synth.make_weights(synth.TINY, seed=0)
    src = synth.TINY_JACOBI.sentences()[0]
    model = om.Model(synth.TINY, w.tensors)
    step = od.model_step(model, src)
    g = od.greedy(step, 16)
    j = od.jacobi(step, 16)
    assert j.tokens == g.tokens and j.n_iters <= 16


# ---- planted mistakes in the loops ----------------------------------------------------------

def test_planted_shift_error_breaks_proposition_1():
    model, src = _toy(TOYS[1], 1)
    step = od.model_step(model, src)
    g = od.greedy(step, 6, stop_at_eos=False)

    def shifted(inputs):                       # read the prediction one row too late
        out = step(inputs)
        return od.StepOut(np.r_[out.pred[1:], out.pred[-1:]], out.margin, out.prob)
    assert od.gs_jacobi(shifted, 6, 3, stop_at_eos=False).tokens != g.tokens


def test_planted_missing_cap_breaks_pass_count(monkeypatch):
    def uncapped(step, y, i, blk, n_pass, trace, eos, rule):
        while True:                             # literal StopC with no pass cap
            o = list(y[i:i + blk])
            new = [int(t) for t in step(y[:i + blk - 1]).pred[i - 1:i - 1 + blk]]
            y[i:i + blk] = new
            n_pass += 1
            if o == new:
                return n_pass
    monkeypatch.setattr(od, "_block_passes", uncapped)
    r = od.gs_jacobi(chain, 10, 5, stop_at_eos=False)
    assert r.n_iters != 10                      # the closed form (blk per block) catches it


# ---- options the paper leaves to future work: suffix re-runs, last-token InitT ---------------

def copy_model(inputs):
    """y_p = y_{p-1}: every prediction copies its input token (what the random-weight presets
    do), so the solution is BOS repeated and a draft of y_{i-1} repeated is already exact."""
    return od.StepOut(np.array(list(inputs)))


def _trace_key(r):
    return [(t.step, t.block_start, t.block_len, t.n_converged, t.stop, t.eos_idx, t.tokens)
            for t in r.trace]


@pytest.mark.parametrize("m,b", [(1, 1), (7, 3), (10, 5), (12, 4), (16, 16)])
def test_last_token_init_closed_form(m, b):
    """Copy model: from PAD every block is a dependency chain (blk passes); from y_{i-1}
    repeated the first pass already returns the draft, StopC holds, one pass per block."""
    blocks = _blocks(m, b)
    g = od.greedy(copy_model, m, stop_at_eos=False)
    assert g.tokens == [BOS] * m
    for rule in ("paper", "prefix", "suffix"):
        pad = od.gs_jacobi(copy_model, m, b, stop_rule=rule, stop_at_eos=False)
        last = od.gs_jacobi(copy_model, m, b, stop_rule=rule, stop_at_eos=False,
                            init_rule="last")
        assert pad.tokens == last.tokens == g.tokens
        assert pad.n_iters == sum(blocks)
        assert last.n_iters == len(blocks)
        assert all(t.stop and t.n_converged == t.block_len for t in last.trace)
    # a chain whose map has no fixed point gains nothing from the last token
    assert od.gs_jacobi(chain, m, b, stop_at_eos=False, init_rule="last").n_iters == sum(blocks)


@pytest.mark.parametrize("m,b", [(7, 3), (10, 5), (12, 4), (16, 16)])
def test_suffix_rule_equals_prefix_rule_with_fewer_rows(m, b):
    """The suffix rule re-runs only the positions after a block's exact prefix: the same
    tokens, passes and trace as the accepted-prefix rule; on a chain a block of k positions
    computes k + (k-1) + ... + 1 rows instead of k per pass."""
    for step in (position_only(), chain, skip_chain, copy_model, position_only(eos_at=5)):
        for init_rule in ("pad", "last"):
            pre = od.gs_jacobi(step, m, b, stop_rule="prefix", stop_at_eos=False,
                               init_rule=init_rule)
            suf = od.gs_jacobi(step, m, b, stop_rule="suffix", stop_at_eos=False,
                               init_rule=init_rule)
            assert _trace_key(suf) == _trace_key(pre)
            assert all(s.n_rows <= p.n_rows == p.block_len for s, p in zip(suf.trace, pre.trace))
    r = od.gs_jacobi(chain, m, b, stop_rule="suffix", stop_at_eos=False)
    assert sum(t.n_rows for t in r.trace) == sum(k * (k + 1) // 2 for k in _blocks(m, b))
    h_pre = od.hybrid_gs_jacobi(position_only(eos_at=6), m, b, stop_rule="prefix")
    h_suf = od.hybrid_gs_jacobi(position_only(eos_at=6), m, b, stop_rule="suffix")
    assert _trace_key(h_suf) == _trace_key(h_pre)


@pytest.mark.parametrize("toy", TOYS, ids=lambda t: t[0].name)
def test_proposition_1_new_options(toy):
    """Any InitT and stop rule reach the greedy solution within m passes (Proposition 1) on the
    brute-force toy transformers."""
    m_len = 9
    for seed in range(2):
        model, src = _toy(toy, seed)
        step = od.model_step(model, src)
        g = od.greedy(step, m_len, stop_at_eos=False)
        ge = od.greedy(step, m_len)
        for rule in ("paper", "prefix", "suffix"):
            for b in (1, 2, 3, m_len):
                r = od.gs_jacobi(step, m_len, b, stop_at_eos=False, stop_rule=rule,
                                 init_rule="last")
                assert r.tokens == g.tokens and r.n_iters <= m_len
            r = od.hybrid_gs_jacobi(step, m_len, 3, stop_rule=rule, init_rule="last")
            assert r.tokens == ge.tokens and r.n_iters <= m_len
