"""Greedy, Jacobi, GS-Jacobi and Hybrid GS-Jacobi decoding, step by step as the paper states
them.  TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Every method works against an abstract pass ``step(inputs) -> StepOut``: ``inputs`` are the
decoder input tokens at positions 0..T-1 (position 0 holds BOS); output row t is the model's
argmax prediction for position t+1.  This is the "shift left" of the appendix to Algorithm 2:
the prediction made at input position t is the value of y_{t+1}.

Readings of the paper that this file fixes (each one listed in the design notes):

* Slices y_{i:i+b} are half-open with b elements; the last block is cut to m - i + 1.
* Algorithm 2/3's ``break`` ends the repeated passes over the current block; the outer loop
  over blocks continues.  A block also ends after as many passes as it has positions: after
  k passes its first k positions are exact (the system of Eq. 4 is triangular), so this cap
  keeps the total at most m passes (Proposition 1) and makes b = 1 the greedy decoder.
* Hybrid (Algorithm 3) counts EOS only in a finished block and returns the prefix through
  that EOS; if none appears up to h it continues autoregressively, one token per pass, until
  EOS or max_len.
* Jacobi and GS-Jacobi solve the system for a known m (Section 4.1 "we assume to know
  beforehand the length m"); with ``stop_at_eos`` the returned tokens end at the first EOS.

Options the paper leaves to future work (Section 5, other initialisations and stopping
conditions), with the same solution by Proposition 1:

* ``stop_rule="prefix"``: a block also ends once the first c + 1 new tokens of a pass (c the
  unchanged leading count) cover it; ``stop_rule="suffix"``: the same, and every further pass
  of a block computes only the positions after that exact prefix.
* ``init_rule="last"``: a new block's drafts are the last decided token y_{i-1} repeated
  instead of PAD (greedy steps and Hybrid's greedy tail have no drafts to initialise).
"""
from __future__ import annotations

import dataclasses
from typing import Callable, List, Optional, Sequence

import numpy as np

import synth


@dataclasses.dataclass
class StepOut:
    pred: np.ndarray                       # [T] argmax predictions for positions 1..T
    margin: Optional[np.ndarray] = None    # [T] top-1 minus top-2 logit
    prob: Optional[np.ndarray] = None      # [T] softmax probability of the argmax


Step = Callable[[Sequence[int]], StepOut]


@dataclasses.dataclass
class TraceRow:
    """One decoder pass, in the spirit of DDGviz (Section 3.5): where the block starts, how
    long it is, how many leading positions came out unchanged, whether the stopping condition
    held, the EOS index inside the block and the block's new tokens."""

    step: int
    block_start: int
    block_len: int
    n_converged: int
    stop: bool
    eos_idx: int
    tokens: List[int]
    probs: Optional[List[float]] = None
    min_margin: float = float("inf")
    n_rows: int = 0              # rows the pass computed (fewer than block_len: suffix rule)


@dataclasses.dataclass
class Result:
    tokens: List[int]            # y_1 .. (through the first EOS when stopping at EOS)
    n_iters: int                 # decoder passes, encoder excluded
    trace: List[TraceRow]

    @property
    def min_margin(self) -> float:
        return min((r.min_margin for r in self.trace), default=float("inf"))


def _leading_equal(a: Sequence[int], b: Sequence[int]) -> int:
    c = 0
    while c < len(a) and a[c] == b[c]:
        c += 1
    return c


def _first(seq: Sequence[int], value: int) -> int:
    for t, v in enumerate(seq):
        if v == value:
            return t
    return -1


def _truncate_at_eos(y: List[int], eos: int) -> List[int]:
    e = _first(y, eos)
    return y if e < 0 else y[:e + 1]


def greedy(step: Step, max_len: int, stop_at_eos: bool = True, bos: int = synth.BOS_ID,
           pad: int = synth.PAD_ID, eos: int = synth.EOS_ID) -> Result:
    """Eq. 2: y_i = argmax p(y_i | y_1..y_{i-1}, x), one position per pass, in order."""
    y = [bos]
    trace = []
    for i in range(1, max_len + 1):
        out = step(y)                       # inputs y_0..y_{i-1}
        tok = int(out.pred[i - 1])          # the prediction made at position i-1 is y_i
        y.append(tok)
        mm = float(out.margin[i - 1]) if out.margin is not None else float("inf")
        pr = [float(out.prob[i - 1])] if out.prob is not None else None
        same = int(tok == pad)                    # the one-position "block" vs its PAD draft
        trace.append(TraceRow(i, i, 1, same, bool(same), 0 if tok == eos else -1, [tok], pr, mm,
                              n_rows=1))
        if stop_at_eos and tok == eos:
            break
    return Result(y[1:], len(trace), trace)


def _block_passes(step: Step, y: List[int], i: int, blk: int, n_pass: int, trace: List[TraceRow],
                  eos: int, stop_rule: str):
    """Repeat one decoder pass over the block y_i..y_{i+blk-1} until the stopping condition
    (Eq. 5: the block did not change) or the pass cap; returns the updated pass counter.
    Under the suffix rule a pass takes new tokens only for the block positions after the
    exact prefix a (the first c + 1 tokens of the pass before); positions below a keep theirs."""
    a = 0
    for k in range(1, blk + 1):
        o = list(y[i:i + blk])                          # copy(y_{i:i+b})
        out = step(y[:i + blk - 1])                     # inputs y_0..y_{i+b-2}
        new = o[:a] + [int(t) for t in out.pred[i - 1 + a:i - 1 + blk]]
        y[i:i + blk] = new                              # y_{i:i+b} <- argmax p(. | y_{1:i+b}, x)
        n_pass += 1
        c = _leading_equal(o, new)
        stop = c == blk                                 # StopC(o, y_{i:i+b})
        mm = float(np.min(out.margin[i - 1 + a:i - 1 + blk])) if out.margin is not None \
            else float("inf")
        pr = [float(p) for p in out.prob[i - 1:i - 1 + blk]] if out.prob is not None else None
        trace.append(TraceRow(n_pass, i, blk, c, stop, _first(new, eos), new, pr, mm,
                              n_rows=blk - a))
        if stop:
            break
        if stop_rule in ("prefix", "suffix") and c + 1 >= blk:
            break
        if stop_rule == "suffix":
            a = c + 1
    return n_pass


def gs_jacobi(step: Step, m: int, b: int, init: Optional[Sequence[int]] = None,
              stop_at_eos: bool = True, stop_rule: str = "paper", init_rule: str = "pad",
              bos: int = synth.BOS_ID, pad: int = synth.PAD_ID, eos: int = synth.EOS_ID) -> Result:
    """Algorithm 2 (Parallel GS-Jacobi): Jacobi passes inside blocks of b positions, blocks
    solved one after the other (Gauss-Seidel across blocks).  InitT = all PAD unless ``init``
    gives another draft of length m, or ``init_rule="last"`` re-initialises each block."""
    if b < 1:
        raise ValueError("b must be >= 1")
    y = [bos] + (list(init) if init is not None else [pad] * m)
    if len(y) != m + 1:
        raise ValueError("init must have m tokens")
    trace: List[TraceRow] = []
    n_pass = 0
    i = 1
    while i <= m:
        blk = min(b, m - i + 1)
        if init_rule == "last":
            y[i:i + blk] = [y[i - 1]] * blk
        n_pass = _block_passes(step, y, i, blk, n_pass, trace, eos, stop_rule)
        i += blk
    out = y[1:]
    return Result(_truncate_at_eos(out, eos) if stop_at_eos else out, n_pass, trace)


def jacobi(step: Step, m: int, init: Optional[Sequence[int]] = None, stop_at_eos: bool = True,
           **kw) -> Result:
    """Algorithm 1 (Parallel Jacobi): the whole sentence y_1..y_m is one block."""
    return gs_jacobi(step, m, max(m, 1), init=init, stop_at_eos=stop_at_eos, **kw)


def hybrid_gs_jacobi(step: Step, max_len: int, b: int, h: Optional[int] = None,
                     init: Optional[Sequence[int]] = None, stop_rule: str = "paper",
                     init_rule: str = "pad", bos: int = synth.BOS_ID, pad: int = synth.PAD_ID,
                     eos: int = synth.EOS_ID) -> Result:
    """Algorithm 3 (Hybrid GS-Jacobi): GS-Jacobi blocks up to length h (default max_len); a
    finished block that contains EOS ends decoding with the prefix through that EOS;
    otherwise greedy steps follow from position h+1 until EOS or max_len."""
    h = max_len if h is None else min(h, max_len)
    y = [bos] + (list(init) if init is not None else [pad] * h)
    trace: List[TraceRow] = []
    n_pass = 0
    i = 1
    while i <= h:
        blk = min(b, h - i + 1)
        if init_rule == "last":
            y[i:i + blk] = [y[i - 1]] * blk
        n_pass = _block_passes(step, y, i, blk, n_pass, trace, eos, stop_rule)
        e = _first(y[i:i + blk], eos)
        if e >= 0:
            return Result(y[1:i + e + 1], n_pass, trace)
        i += blk
    y = y[:i]
    while i <= max_len:                                    # autoregressive tail
        out = step(y)
        tok = int(out.pred[i - 1])
        y.append(tok)
        n_pass += 1
        mm = float(out.margin[i - 1]) if out.margin is not None else float("inf")
        pr = [float(out.prob[i - 1])] if out.prob is not None else None
        same = int(tok == pad)
        trace.append(TraceRow(n_pass, i, 1, same, bool(same), 0 if tok == eos else -1, [tok], pr,
                              mm, n_rows=1))
        i += 1
        if tok == eos:
            break
    return Result(y[1:], n_pass, trace)


def decode(step: Step, method: str, max_len: int, b: int = 1, h: Optional[int] = None,
           stop_at_eos: bool = True, init=None, stop_rule: str = "paper",
           init_rule: str = "pad") -> Result:
    if method == "greedy":
        return greedy(step, max_len, stop_at_eos)
    if method == "jacobi":
        return jacobi(step, max_len, init=init, stop_at_eos=stop_at_eos, stop_rule=stop_rule,
                      init_rule=init_rule)
    if method == "gs_jacobi":
        return gs_jacobi(step, max_len, b, init=init, stop_at_eos=stop_at_eos,
                         stop_rule=stop_rule, init_rule=init_rule)
    if method == "hybrid_gs_jacobi":
        return hybrid_gs_jacobi(step, max_len, b, h=h, init=init, stop_rule=stop_rule,
                                init_rule=init_rule)
    raise ValueError(method)


# ---------------------------------------------------------------------------------------------
# The model as a step function
# ---------------------------------------------------------------------------------------------

def model_step(model, src: np.ndarray, with_probs: bool = False) -> Step:
    """A pass of the oracle transformer: encode x once, then for any input prefix return the
    argmax (Eq. 2) of every row of the teacher-forced logits, with margins and probabilities."""
    from oracle.model import top2
    mem = model.encode(src)

    def step(inputs: Sequence[int]) -> StepOut:
        lg = model.logits(mem, np.asarray(inputs, dtype=np.int64))
        idx, margin, prob = top2(lg)
        return StepOut(idx, margin, prob if with_probs else None)

    step.mem = mem
    return step
