"""DDGviz-style JSONL dump (Section 3.5): the records of a decode's trace and the pass at which
each position settled, checked on the oracle's runs of planted dependency structures, where
the settle passes have closed forms.  The GPU decode's dump is checked in test_gpu_parity.py."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, os.path.join(ROOT, "tests"))

from oracle import decode as od  # noqa: E402
from paper_2305_10427_gb300 import ddgviz  # noqa: E402
from paper_2305_10427_gb300._binding import DecodeResult  # noqa: E402
from test_oracle_decode import chain, position_only  # noqa: E402


def as_result(r, max_len):
    """An oracle run in the shape pd_decode returns (trace rows as dicts, token / probability
    rows padded to max_len)."""
    trace = [dict(step=t.step, block_start=t.block_start, block_len=t.block_len,
                  n_converged=t.n_converged, stop=int(t.stop), eos_idx=t.eos_idx,
                  n_rows=t.n_rows) for t in r.trace]
    tt = np.full((len(r.trace), max_len), -1, dtype=np.int32)
    tp = np.zeros((len(r.trace), max_len), dtype=np.float32)
    for k, t in enumerate(r.trace):
        tt[k, :t.block_len] = t.tokens
        tp[k, :t.block_len] = 0.5
    return DecodeResult(list(r.tokens), r.n_iters, trace, tt, tp)


def test_settle_passes_closed_forms(tmp_path):
    m = 8
    # a chain: position i + k of a block of 4 settles at the block's (k + 1)-th pass
    r = od.gs_jacobi(chain, m, 4, stop_at_eos=False)
    path = str(tmp_path / "chain.jsonl")
    recs = ddgviz.dump_jsonl(as_result(r, m), path, method="gs_jacobi", b=4)
    assert ddgviz.load_jsonl(path) == recs
    head, passes = recs[0], recs[1:]
    assert head["settled_at"] == [1, 2, 3, 4, 5, 6, 7, 8]
    assert head["n_passes"] == len(passes) == 8
    assert [p["n_converged"] for p in passes[:4]] == [0, 1, 2, 3]
    assert passes[-1]["tokens"] == r.tokens[4:]
    # position-only predictions: a block settles in its first pass, the second confirms it
    r = od.gs_jacobi(position_only(), m, 4, stop_at_eos=False)
    head = ddgviz.trace_records(as_result(r, m), method="gs_jacobi", b=4)[0]
    assert head["settled_at"] == [1, 1, 1, 1, 3, 3, 3, 3]
    # greedy: position p at pass p
    r = od.greedy(chain, m, stop_at_eos=False)
    head = ddgviz.trace_records(as_result(r, m), method="greedy")[0]
    assert head["settled_at"] == list(range(1, m + 1))


def test_suffix_rule_records_rows(tmp_path):
    r = od.gs_jacobi(chain, 6, 3, stop_at_eos=False, stop_rule="suffix")
    recs = ddgviz.trace_records(as_result(r, 6), method="gs_jacobi", b=3, stop_rule="suffix")
    assert [p["n_rows"] for p in recs[1:]] == [3, 2, 1, 3, 2, 1]
    assert all(len(p["probs"]) == p["block_len"] for p in recs[1:])
