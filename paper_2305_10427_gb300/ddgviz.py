"""DDGviz-style dump of a decode's per-pass trace (the paper's visualisation of the decoding
dependency graph, Section 3.5 and Fig. 4): one JSON object per line.

The first line describes the decode: method, block size, stop rule, the returned tokens, the
pass count, and for every position p (1-based) the pass after which its token never changed
again (``settled_at``: how deep in the chain of passes the position's value was decided; a
greedy decode settles position p at pass p).  Every further line is one decoder pass: its number,
the block it worked on (start, length), how many leading block positions came out unchanged,
the StopC flag of Eq. 5, the EOS index in the block, the rows the pass computed, and the block's
new tokens with the softmax probability of each (the quantity DDGviz colours tokens by).

Usage, from Python::

    res = dec.decode("gs_jacobi", max_len, b=5, trace=True)
    ddgviz.dump_jsonl(res, "trace.jsonl", method="gs_jacobi", b=5)

or from the command line on a GPU (one synthetic sentence of a preset)::

    python -m paper_2305_10427_gb300.ddgviz --preset tiny-f32 --method gs_jacobi --b 5 out.jsonl
"""
from __future__ import annotations

import json
from typing import Dict, List, Optional


def settled_at(trace: List[dict], trace_tokens, n_positions: int) -> List[int]:
    """For positions 1..n_positions: the pass after which the token at the position never
    changed again (0 for a position no pass wrote)."""
    last_val: Dict[int, int] = {}
    settled = [0] * (n_positions + 1)
    for t, row in enumerate(trace):
        i, blk = row["block_start"], row["block_len"]
        for off in range(blk):
            p = i + off
            tok = int(trace_tokens[t][off])
            if last_val.get(p) != tok:
                last_val[p] = tok
                if p <= n_positions:
                    settled[p] = row["step"]
    return settled[1:]


def trace_records(result, method: str, b: int = 1, stop_rule: str = "paper",
                  init: str = "pad", src: Optional[List[int]] = None) -> List[dict]:
    """The records of one decode (a DecodeResult with its trace): a header, then one per pass."""
    if result.trace is None:
        raise ValueError("the decode was run without a trace (decode(..., trace=True))")
    n = len(result.tokens)
    head = {"kind": "decode", "method": method, "b": int(b), "stop_rule": stop_rule,
            "init": init, "n_passes": int(result.n_iters), "n_trace": len(result.trace),
            "tokens": [int(t) for t in result.tokens],
            "settled_at": settled_at(result.trace, result.trace_tokens, n)}
    if src is not None:
        head["src"] = [int(t) for t in src]
    out = [head]
    for t, row in enumerate(result.trace):
        blk = row["block_len"]
        rec = {"kind": "pass", "pass": int(row["step"]), "block_start": int(row["block_start"]),
               "block_len": int(blk), "n_converged": int(row["n_converged"]),
               "stop": bool(row["stop"]), "eos_idx": int(row["eos_idx"]),
               "n_rows": int(row.get("n_rows", blk)),
               "tokens": [int(v) for v in result.trace_tokens[t][:blk]]}
        if result.trace_probs is not None:
            rec["probs"] = [float(v) for v in result.trace_probs[t][:blk]]
        out.append(rec)
    return out


def dump_jsonl(result, path: str, **meta) -> List[dict]:
    """Write trace_records(result, **meta) to path, one JSON object per line."""
    recs = trace_records(result, **meta)
    with open(path, "w") as f:
        for r in recs:
            f.write(json.dumps(r) + "\n")
    return recs


def load_jsonl(path: str) -> List[dict]:
    with open(path) as f:
        return [json.loads(line) for line in f if line.strip()]


def main(argv=None) -> int:
    import argparse

    import numpy as np

    from . import _binding as pkg

    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("out")
    ap.add_argument("--preset", default="tiny-f32")
    ap.add_argument("--method", default="gs_jacobi", choices=list(pkg.METHODS))
    ap.add_argument("--b", type=int, default=5)
    ap.add_argument("--stop-rule", default="paper", choices=list(pkg.STOP_RULES))
    ap.add_argument("--init", default="pad", choices=list(pkg.INITS))
    ap.add_argument("--src-len", type=int, default=16)
    ap.add_argument("--seed", type=int, default=0)
    args = ap.parse_args(argv)
    import os
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import synth
    spec = synth.PRESETS[args.preset]
    w = synth.make_weights(spec, seed=args.seed)
    src = synth.sentences(args.seed + 1, 1, args.src_len, args.src_len, spec.vocab)[0]
    max_len = 2 * len(src)
    cfg = pkg.Config.from_spec(spec, max_src_len=len(src), max_tgt_len=max_len)
    with pkg.Decoder(cfg, w.blob) as dec:
        dec.encode(src)
        res = dec.decode(args.method, max_len, b=args.b, trace=True, stop_rule=args.stop_rule,
                         init=args.init)
    recs = dump_jsonl(res, args.out, method=args.method, b=args.b, stop_rule=args.stop_rule,
                      init=args.init, src=list(np.asarray(src)))
    print(f"{args.out}: {len(recs) - 1} passes, {len(res.tokens)} tokens")
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
