"""Benchmark: translated tokens/s at batch 1, GS-Jacobi (b=5) vs greedy AR, on the Marian-sized
bf16 model (6+6 layers, d=512, 8 heads, FFN 2048 SiLU, V=58101) over 256 synthetic source
sentences of 8..64 ids with max_len = 2 * src_len, plus the decode kernel's HBM roofline.

One step = encode + decode of all 256 sentences, one after the other (batch 1).
  value : tokens/s with source ids resident in device memory, timed with CUDA events on the
          library stream (pd_encode_device / pd_decode_device), L2 flushed between steps.
  e2e   : the same through the host API (pd_encode / pd_decode: ids copied in, tokens copied
          out, every call synchronous), wall clock.
Multi-GPU: replicas (every rank decodes the full sentence set; weak scaling).
``--impl reference`` times the CPU oracle (numpy float64) on a bounded sample instead.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

WORKLOAD = synth.MARIAN_GS
STOP_RULE = "paper"          # "paper": StopC of Eq. 5; "prefix": accepted-prefix rule
ENGINE = "auto"              # pd_gemm_engine (auto = SIMT)
CLUSTER_SIZE = 0             # cluster engine: CTAs per cluster (0 = the library's choice)
ARGS_WORKLOAD = "marian"
METRIC = "translated tokens/s at batch 1, GS-Jacobi vs greedy AR; HBM GB/s % of peak"
FALLBACK_HBM_GBS = 6800.0

# DRAM bytes (read + write) per decoder pass of decode_kernel<bf16> on this workload, from one
# ncu capture of this workload, valid only for the kernel code whose
# SHA-256 (comments and blank lines left out) is recorded here; other code reports traffic null.
DRAM_BYTES_PER_PASS = 13.85e6
DRAM_SOURCES_SHA256 = "47ee6e16305b9dc2b0751d1c762c8e8d44e084b3e6b83005100da254639a7e02"


def code_without_comments(text: str) -> str:
    """CUDA / C++ source with its comments, trailing blanks and empty lines removed (the kernel
    sources hold no string literal with "//" or "/*")."""
    import re
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    lines = (re.sub(r"//.*", "", ln).rstrip() for ln in text.splitlines())
    return "\n".join(ln for ln in lines if ln)


def kernel_sources_sha256(read=None) -> str:
    import hashlib
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2305_10427_gb300", "csrc")
    for f in sorted(os.listdir(d)):
        if f.endswith((".cu", ".cuh")):
            h.update(f.encode())
            text = read(f) if read else open(os.path.join(d, f)).read()
            h.update(code_without_comments(text).encode())
    return h.hexdigest()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def pass_bytes(spec: synth.ModelSpec, L_keys: int, n_src: int, rows: int) -> int:
    """Algorithmic HBM bytes of one decoder pass: every decoder-layer and LM-head parameter
    once, the self-attention keys/values of positions 0..L_keys-1 and the cross keys/values
    of the n_src source positions once, and the K/V written for the pass's rows."""
    d, f, V, Ld = spec.d_model, spec.d_ff, spec.vocab, spec.n_dec_layers
    es = 2 if spec.dtype == synth.DTYPE_BF16 else 4
    layer = 3 * d * d + 3 * d + d * d + d + d * d + d + d * d + d + 2 * d * f + f + d + 6 * d
    weights = Ld * layer + V * d
    kv = Ld * 2 * d * (L_keys + n_src) + Ld * 2 * d * rows
    return es * (weights + kv)


def decode_bytes(spec, n_src, trace):
    """Sum of pass_bytes over the passes of one decode (from its trace)."""
    tot = 0
    for row in trace:
        i, blk = row["block_start"], row["block_len"]
        tot += pass_bytes(spec, i - 1 + blk, n_src, blk)
    return tot


def over_ranks(x: float, op: str, dist=None, device="cpu") -> float:
    """max or sum of a per-rank number over all ranks (identity without a process group)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return x
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def job_rate(units: float, seconds: float, dist=None, device="cpu") -> float:
    """Whole-job throughput of replicas: units done by all ranks / the slowest rank's time."""
    return over_ranks(units, "sum", dist, device) / over_ranks(seconds, "max", dist, device)


class Clocks:
    """nvidia-smi sampling during the timed region.  The raw samples go to a CSV in
    $PD_BENCH_CLOCKS_DIR (default: the temporary directory); the JSON line carries the summary."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        d = os.environ.get("PD_BENCH_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(d, f"pd_clocks_{os.getpid()}_{index}.csv")

    def __enter__(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index),
                                          f"--query-gpu={q}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and --impl reference)
# ---------------------------------------------------------------------------------------------

def oracle_tokens_per_s(weights, sentences, budget_s):
    from oracle import decode as od
    from oracle import model as om
    model = om.Model(WORKLOAD.spec, weights.tensors)
    tokens, t0, used = 0, time.perf_counter(), []
    for k, src in enumerate(sentences):
        step = od.model_step(model, src)
        r = od.gs_jacobi(step, WORKLOAD.max_len(len(src)), WORKLOAD.b, stop_rule=STOP_RULE)
        tokens += len(r.tokens)
        used.append(k)
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    return tokens / dt, tokens, dt, used


def oracle_one_thread(budget_s, shortest_first=True):
    """The oracle timed with one BLAS thread, in a child process (the thread count of a BLAS
    library is fixed when it loads); returns (tokens/s, tokens, seconds, sentences used)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-worker",
           "--cpu-budget", str(budget_s), "--workload", ARGS_WORKLOAD]
    out = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=600)
    if out.returncode != 0:
        raise RuntimeError("one-thread oracle run failed: " + out.stderr[-500:])
    d = json.loads(out.stdout.strip().splitlines()[-1])
    return d["value"], d["tokens"], d["seconds"], d["used"]


def run_oracle_worker(args):
    sents = WORKLOAD.sentences()
    order = sorted(range(len(sents)), key=lambda k: len(sents[k]))
    v, t, d, used = oracle_tokens_per_s(WORKLOAD.weights(), [sents[k] for k in order],
                                        args.cpu_budget)
    print(json.dumps({"value": v, "tokens": t, "seconds": d, "used": len(used)}), flush=True)
    return 0


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    weights = WORKLOAD.weights()
    sents = WORKLOAD.sentences()
    # each step: GS-Jacobi (b=5) of the next sentence of the workload by the float64 oracle
    order = sorted(range(len(sents)), key=lambda k: len(sents[k]))[:args.warmup + args.steps]
    for k in order[:args.warmup]:
        oracle_tokens_per_s(weights, [sents[k]], 0)
    tok, dt = 0, 0.0
    for k in order[args.warmup:]:
        _, t, d, _ = oracle_tokens_per_s(weights, [sents[k]], 0)
        tok += t
        dt += d
    v = tok / dt
    cores = os.cpu_count()
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD.name, "stop_rule": STOP_RULE,
                       "sample": "one sentence per step, the "
                       "shortest sentences of the 256 (CPU oracle is slow)"},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{args.steps} sentences, GS-Jacobi b=5, numpy float64, "
                                       f"BLAS threads = all {cores} cores"},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------------------------

def run_gpu(args):
    import torch
    import paper_2305_10427_gb300 as pkg

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)

    spec = WORKLOAD.spec
    weights = WORKLOAD.weights()
    sents = WORKLOAD.sentences()[:args.sentences] if args.sentences else WORKLOAD.sentences()
    n_s = len(sents)
    max_src = max(len(s) for s in sents)
    max_tgt = max(WORKLOAD.max_len(len(s)) for s in sents)
    stream = torch.cuda.Stream()
    dec = pkg.Decoder(pkg.Config.from_spec(spec, max_src, max_tgt, engine=ENGINE,
                                           cluster_size=CLUSTER_SIZE), weights.blob,
                      stream=stream.cuda_stream)

    offs = np.cumsum([0] + [len(s) for s in sents])
    d_src = torch.tensor(np.concatenate(sents), dtype=torch.int32, device="cuda")
    d_y = torch.zeros((n_s, max_tgt), dtype=torch.int32, device="cuda")
    d_info = torch.zeros((n_s, 4), dtype=torch.int32, device="cuda")
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")
    params = {m: [pkg.Decoder.params(m, WORKLOAD.max_len(len(s)), b=b, stop_rule=STOP_RULE)
                  for s in sents]
              for m, b in (("gs_jacobi", WORKLOAD.b), ("greedy", 1), ("jacobi", 1),
                           ("hybrid_gs_jacobi", 3))}
    # options the paper leaves to future work: suffix-only re-runs, last-token InitT
    params["gs_jacobi+suffix"] = [pkg.Decoder.params("gs_jacobi", WORKLOAD.max_len(len(s)),
                                                     b=WORKLOAD.b, stop_rule="suffix")
                                  for s in sents]
    params["gs_jacobi+init_last"] = [pkg.Decoder.params("gs_jacobi", WORKLOAD.max_len(len(s)),
                                                        b=WORKLOAD.b, stop_rule=STOP_RULE,
                                                        init="last") for s in sents]

    def device_step(method, ev=None):
        for k in range(n_s):
            if ev is not None:
                ev[k][0].record(stream)
            dec.encode_device(d_src.data_ptr() + 4 * int(offs[k]), len(sents[k]))
            if ev is not None:
                ev[k][1].record(stream)
            dec.decode_device(params[method][k], d_y[k].data_ptr(), d_info[k].data_ptr())
            if ev is not None:
                ev[k][2].record(stream)

    def timed(method, steps, warmup):
        for _ in range(warmup):
            device_step(method)
        torch.cuda.synchronize()
        total_ms, dec_ms, launches0 = 0.0, 0.0, dec.launch_count
        tokens = 0
        for _ in range(steps):
            flush.fill_(1)                     # evict L2 (256 MB > 129 MB) between steps
            ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n_s)]
            torch.cuda.synchronize()
            if dist is not None:
                dist.barrier()
            with torch.cuda.stream(stream):
                device_step(method, ev)
            torch.cuda.synchronize()
            total_ms += ev[0][0].elapsed_time(ev[-1][2])
            dec_ms += sum(e[1].elapsed_time(e[2]) for e in ev)
            info = d_info.cpu().numpy()
            assert (info[:, 2] == 0).all(), "decode reported a failure"
            tokens += int(info[:, 0].sum())
        return tokens, total_ms, dec_ms, dec.launch_count - launches0, d_info.cpu().numpy()

    def max_over_ranks(x):
        return over_ranks(x, "max", dist, "cuda")

    def sum_over_ranks(x):
        return over_ranks(x, "sum", dist, "cuda")

    # greedy AR reference point (same kernels, one position per pass)
    g_tok, g_ms, g_dec_ms, _, g_info = timed("greedy", args.steps, args.warmup)
    g_ms = max_over_ranks(g_ms)
    greedy_tps = sum_over_ranks(g_tok) / (g_ms / 1e3)

    with Clocks(local) as clk:
        tok, ms, dec_ms, launches, info = timed("gs_jacobi", args.steps, args.warmup)
    ms_max = max_over_ranks(ms)
    tps = sum_over_ranks(tok) / (ms_max / 1e3)

    # the other methods (one timed step each), for the report
    others = {}
    if args.all_methods:
        for m in ("jacobi", "hybrid_gs_jacobi", "gs_jacobi+suffix", "gs_jacobi+init_last"):
            t_tok, t_ms, _, _, t_info = timed(m, 1, 1)
            others[m] = {"value": sum_over_ranks(t_tok) / (max_over_ranks(t_ms) / 1e3),
                         "unit": "tokens/s",
                         "passes_per_token": float(t_info[:, 1].sum()) / max(1, int(t_info[:, 0].sum()))}

    # roofline of the decode kernel: algorithmic bytes from the traces of one step
    total_bytes, passes = 0, 0
    toks = []
    for k, s in enumerate(sents):
        dec.encode(s)
        r = dec.decode("gs_jacobi", WORKLOAD.max_len(len(s)), b=WORKLOAD.b, trace=True,
                       stop_rule=STOP_RULE)
        assert r.n_iters == int(info[k, 1])
        total_bytes += decode_bytes(spec, len(s), r.trace)
        passes += r.n_iters
        toks.append(len(r.tokens))
    dec_s_per_step = dec_ms / args.steps / 1e3
    achieved = total_bytes / dec_s_per_step / 1e9
    peak, peak_kind = peaks()
    traffic = None                                  # per average decode launch
    if (DRAM_SOURCES_SHA256 and kernel_sources_sha256() == DRAM_SOURCES_SHA256
            and WORKLOAD is synth.MARIAN_GS):
        traffic = DRAM_BYTES_PER_PASS * passes / n_s

    # end to end through the host API
    e2e_tok, h2d, d2h = 0, 0, 0
    for _ in range(args.warmup):
        for k, s in enumerate(sents[:8]):
            dec.encode(s)
            dec.decode("gs_jacobi", WORKLOAD.max_len(len(s)), b=WORKLOAD.b, stop_rule=STOP_RULE)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for k, s in enumerate(sents):
            dec.encode(s)
            r = dec.decode("gs_jacobi", WORKLOAD.max_len(len(s)), b=WORKLOAD.b,
                           stop_rule=STOP_RULE)
            e2e_tok += len(r.tokens)
            h2d += 4 * len(s)
            d2h += 4 + 16 + 4 * len(r.tokens)      # encode status, decode info, tokens
    torch.cuda.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0)
    e2e_tps = sum_over_ranks(e2e_tok) / e2e_s

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        v, t, d, used = oracle_tokens_per_s(weights, [sents[k] for k in
                                                      sorted(range(n_s), key=lambda k:
                                                             len(sents[k]))], args.cpu_budget)
        cpu = {"value": v, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"{len(used)} shortest sentences of the 256 ({t} tokens, {d:.1f} s), "
                         f"GS-Jacobi b=5, numpy float64, BLAS threads = all cores"}
        v1, t1, d1, u1 = oracle_one_thread(args.cpu_budget / 2)
        cpu["one_thread"] = {"value": v1, "unit": "tokens/s", "cores": 1,
                             "sample": f"{u1} shortest sentences ({t1} tokens, {d1:.1f} s), "
                                       f"one BLAS thread"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": tps, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic: seeded N(0,0.02) weights, uniform random source ids",
            "config": {"workload": WORKLOAD.name if n_s == WORKLOAD.n_sentences else
                       f"{WORKLOAD.name} (first {n_s} sentences only)", "sentences_per_step": n_s,
                       "stop_rule": STOP_RULE, "engine": ENGINE, "cluster_size": CLUSTER_SIZE,
                       "timing": "CUDA events on the library stream; L2 flushed (256 MB write) "
                                 "between steps; replicas across GPUs"},
            "greedy": {"value": greedy_tps, "unit": "tokens/s",
                       "gs_jacobi_speedup": tps / greedy_tps,
                       "passes_per_token": float(g_info[:, 1].sum()) / max(1, int(g_info[:, 0].sum()))},
            "passes_per_token": passes / max(1, sum(toks)),
            "us_per_pass": 1e6 * dec_s_per_step / max(1, passes),
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "algorithmic_bytes_per_launch": total_bytes / n_s,
                         "kernel": "decode_kernel<bf16>", "peak_kind": peak_kind},
            "e2e": {"value": e2e_tps, "unit": "tokens/s", "h2d_bytes_per_step": h2d // args.steps,
                    "d2h_bytes_per_step": d2h // args.steps},
            "gpu_launches": launches,
            "clocks": clk.summary(),
        }
        if others:
            line["other_methods"] = others
        if cpu is not None:
            line["cpu_baseline"] = cpu
        print(json.dumps(line), flush=True)
    dec.close()
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_gpu_batch(args):
    """Batched serving: the workload's sentences in groups of args.batch, each group encoded
    (pd_encode_batch_device) and decoded together (pd_decode_batch_device).  value = tokens/s
    over the whole set; the roofline counts the weights once per batched pass (a group runs
    as many passes as its slowest sentence) plus each sentence's own key/value traffic."""
    import torch
    import paper_2305_10427_gb300 as pkg

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)

    S = args.batch
    spec = WORKLOAD.spec
    weights = WORKLOAD.weights()
    sents = WORKLOAD.sentences()[:args.sentences] if args.sentences else WORKLOAD.sentences()
    groups = [sents[k:k + S] for k in range(0, len(sents), S)]
    max_src = max(len(s) for s in sents)
    max_tgt = max(WORKLOAD.max_len(len(s)) for s in sents)
    stream = torch.cuda.Stream()
    dec = pkg.Decoder(pkg.Config.from_spec(spec, max_src, max_tgt, max_batch=S, engine=ENGINE,
                                           cluster_size=CLUSTER_SIZE),
                      weights.blob, stream=stream.cuda_stream)
    offs_all = np.cumsum([0] + [len(s) for s in sents])
    d_src = torch.tensor(np.concatenate(sents), dtype=torch.int32, device="cuda")
    d_y = torch.zeros((len(groups), S, max_tgt), dtype=torch.int32, device="cuda")
    d_info = torch.zeros((len(groups), S, 4), dtype=torch.int32, device="cuda")
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")
    meta = []
    for gi, g in enumerate(groups):
        k0 = gi * S
        offs = np.asarray(offs_all[k0:k0 + len(g) + 1] - offs_all[k0], dtype=np.int32)
        ml = np.asarray([WORKLOAD.max_len(len(s)) for s in g], dtype=np.int32)
        meta.append((int(offs_all[k0]), offs, ml))
    params = {m: pkg.Decoder.params(m, max_tgt, b=b, stop_rule=STOP_RULE)
              for m, b in (("gs_jacobi", WORKLOAD.b), ("greedy", 1))}

    def device_step(method):
        for gi, (o0, offs, ml) in enumerate(meta):
            dec.encode_batch_device(d_src.data_ptr() + 4 * o0, offs)
            dec.decode_batch_device(params[method], ml, d_y[gi].data_ptr(), max_tgt,
                                    d_info[gi].data_ptr())

    def timed(method, steps, warmup):
        for _ in range(warmup):
            device_step(method)
        torch.cuda.synchronize()
        total_ms, tokens, launches0 = 0.0, 0, dec.launch_count
        for _ in range(steps):
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            if dist is not None:
                dist.barrier()
            e0.record(stream)
            with torch.cuda.stream(stream):
                device_step(method)
            e1.record(stream)
            torch.cuda.synchronize()
            total_ms += e0.elapsed_time(e1)
            info = d_info.cpu().numpy()
            for gi, (_, _, ml) in enumerate(meta):
                assert (info[gi, :len(ml), 2] == 0).all(), "decode reported a failure"
                tokens += int(info[gi, :len(ml), 0].sum())
        return tokens, total_ms, dec.launch_count - launches0, d_info.cpu().numpy()

    g_tok, g_ms, _, _ = timed("greedy", args.steps, args.warmup)
    greedy_tps = over_ranks(g_tok, "sum", dist, "cuda") / (over_ranks(g_ms, "max", dist, "cuda") / 1e3)
    with Clocks(local) as clk:
        tok, ms, launches, info = timed("gs_jacobi", args.steps, args.warmup)
    ms_max = over_ranks(ms, "max", dist, "cuda")
    tps = over_ranks(tok, "sum", dist, "cuda") / (ms_max / 1e3)

    # algorithmic bytes of one step: per group, the weights once per batched pass plus every
    # sentence's key/value traffic of its own passes (single-sentence traces, same passes)
    w_bytes = pass_bytes(spec, 0, 0, 0)           # the weights of one pass, no key/value
    total_bytes, batched_passes = 0, 0
    for gi, g in enumerate(groups):
        n_pass = int(info[gi, :len(g), 1].max())
        batched_passes += n_pass
        total_bytes += n_pass * w_bytes
        for s in g:
            dec.encode(s)
            r = dec.decode("gs_jacobi", WORKLOAD.max_len(len(s)), b=WORKLOAD.b, trace=True,
                           stop_rule=STOP_RULE)
            total_bytes += decode_bytes(spec, len(s), r.trace) - r.n_iters * w_bytes
    sec_per_step = ms / args.steps / 1e3
    achieved = total_bytes / sec_per_step / 1e9
    peak, peak_kind = peaks()
    if rank == 0:
        line = {
            "metric": METRIC, "value": tps, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic: seeded N(0,0.02) weights, uniform random source ids",
            "config": {"workload": f"{WORKLOAD.name}, batches of {S} sentences",
                       "sentences_per_step": len(sents), "batch": S, "stop_rule": STOP_RULE,
                       "engine": ENGINE, "cluster_size": CLUSTER_SIZE,
                       "timing": "CUDA events on the library stream around encode + decode of "
                                 "all batches; L2 flushed (256 MB write) between steps"},
            "greedy": {"value": greedy_tps, "unit": "tokens/s",
                       "gs_jacobi_speedup": tps / greedy_tps},
            "batched_passes_per_step": batched_passes,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": None,
                         "algorithmic_bytes_per_step": total_bytes,
                         "kernel": "encode_kernel + decode_kernel<bf16> (whole step)",
                         "peak_kind": peak_kind},
            "gpu_launches": launches,
            "clocks": clk.summary(),
        }
        print(json.dumps(line), flush=True)
    dec.close()
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", default="marian", choices=["marian", "marian-knob", "mbart"],
                    help="marian: the benchmark workload; marian-knob: the same model with a "
                         "small token-embedding scale (Jacobi accepts several tokens per pass); "
                         "mbart: the mBART-large-sized model (pre-LN, GELU, learned positions, "
                         "V = 250027), 128 sentences of 16..128 ids")
    ap.add_argument("--b", type=int, default=0,
                    help="GS-Jacobi block size (default: the workload's, 5)")
    ap.add_argument("--all-methods", action="store_true",
                    help="also time full-sentence Jacobi and Hybrid GS-Jacobi (b=3), one step each")
    ap.add_argument("--stop-rule", default="paper", choices=["paper", "prefix", "suffix"],
                    help="when a block's passes end: paper = StopC of Eq. 5 (the block unchanged, "
                         "or one pass per position); prefix = also once the unchanged leading "
                         "tokens make the whole block exact; suffix = prefix, re-running only "
                         "the rows after the block's exact prefix")
    ap.add_argument("--oracle-worker", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--engine", default="auto", choices=["auto", "simt", "tensor", "cluster"],
                    help="decoder engine of the context (pd_gemm_engine)")
    ap.add_argument("--cluster-size", type=int, default=0, choices=[0, 1, 2, 4, 8],
                    help="cluster engine: CTAs per thread-block cluster (0 = the library's)")
    ap.add_argument("--batch", type=int, default=1,
                    help="sentences decoded together (batched serving); 1 = the batch-1 benchmark")
    ap.add_argument("--sentences", type=int, default=0,
                    help="use only the first N sentences of the workload (profiling runs)")
    args = ap.parse_args()
    global WORKLOAD, STOP_RULE, ENGINE, ARGS_WORKLOAD, CLUSTER_SIZE
    STOP_RULE = args.stop_rule
    ENGINE = args.engine
    CLUSTER_SIZE = args.cluster_size
    ARGS_WORKLOAD = args.workload
    if args.workload == "marian-knob":
        WORKLOAD = synth.MARIAN_KNOB
    elif args.workload == "mbart":
        WORKLOAD = synth.MBART_GS
    if args.b and args.b != WORKLOAD.b:
        WORKLOAD = dataclasses.replace(
            WORKLOAD, b=args.b, name=WORKLOAD.name.replace(f"b={WORKLOAD.b}", f"b={args.b}"))
    if args.oracle_worker:
        return run_oracle_worker(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.batch > 1:
        return run_gpu_batch(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
