"""Per-CTA timeline of one decoder pass (development tool, needs a GPU).

Builds a copy of the library with ``-DPD_TIMELINE`` into a temporary directory, decodes one
synthetic sentence with the Marian-sized bf16 model and prints, for every phase of one pass,
its span (first release to last arrival over the 152 CTAs), the median per-CTA entry / staging
/ product+epilogue times, and the barrier gap to the next phase.  The marks are recorded in
shared memory and written out when the kernel ends, so they barely perturb the kernel.

    python -m paper_2305_10427_gb300.timeline [--method gs_jacobi] [--b 5] [--pass-index 20]
"""
import argparse
import ctypes
import os
import subprocess
import sys
import tempfile

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402
from paper_2305_10427_gb300 import _binding as B  # noqa: E402
from paper_2305_10427_gb300.build import ARCH, nvcc  # noqa: E402

PHASES = ["qkv", "attn", "o", "qc", "xattn", "oc", "ffn1", "ffn2"]
K_TL = 52          # intervals recorded (kTlN in the kernel)
MARKS = 8


def build_timeline_lib(out_dir):
    lib = os.path.join(out_dir, "libpd_timeline.so")
    src = os.path.join(ROOT, "paper_2305_10427_gb300", "csrc", "pd.cu")
    subprocess.run([nvcc(), "-O3", "-std=c++17", *ARCH, "-DPD_TIMELINE", "-shared", "-Xcompiler",
                    "-fPIC", "-I", os.path.join(ROOT, "include"), "-o", lib, src], check=True)
    return lib


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--method", default="gs_jacobi")
    ap.add_argument("--b", type=int, default=5)
    ap.add_argument("--src-len", type=int, default=36)
    ap.add_argument("--pass-index", type=int, default=20)
    args = ap.parse_args(argv)
    import torch
    torch.cuda.set_device(0)
    tmp = tempfile.mkdtemp(prefix="pd_timeline_")
    B.LIB_PATH = build_timeline_lib(tmp)
    B._lib = None
    lib = B.load_library()
    lib.pd_debug_set_tl.argtypes = [ctypes.c_void_p, ctypes.c_int]
    spec = synth.MARIAN
    w = synth.make_weights(spec, seed=0)
    dec = B.Decoder(B.Config.from_spec(spec, 64, 128), w.blob)
    src = synth.MARIAN_GS.sentences()[0][:args.src_len]
    nph = 8 * spec.n_dec_layers + 1
    G = torch.cuda.get_device_properties(0).multi_processor_count    # one CTA per SM
    buf = torch.zeros(K_TL * G * MARKS, dtype=torch.int64, device="cuda")
    # interval 0 runs from the kernel start to the first barrier (phase 0 of pass 0); every
    # pass has nph intervals, the first of which also holds the commit of the pass before
    assert lib.pd_debug_set_tl(buf.data_ptr(), args.pass_index * nph) == 0
    dec.encode(src)
    for _ in range(3):
        buf.zero_()
        torch.cuda.synchronize()
        r = dec.decode(args.method, 2 * len(src), b=args.b)
        torch.cuda.synchronize()
    if r.n_iters <= args.pass_index:
        sys.exit(f"the decode took {r.n_iters} passes; choose --pass-index below that")
    a = buf.cpu().numpy().reshape(K_TL, G, MARKS).astype(np.float64)
    # SM cycles per us, from the clock64 and globaltimer marks of the whole pass
    last = nph - 1
    clk = float(np.median((a[last, :, 3] - a[0, :, 0]) / ((a[last, :, 5] - a[0, :, 4]) / 1e3)))
    names = [f"L{l}.{p}" for l in range(spec.n_dec_layers) for p in PHASES] + ["lm"]
    print(f"{args.method} b={args.b}, {len(src)} source ids, {r.n_iters} passes; "
          f"pass {args.pass_index}, {G} CTAs, SM clock {clk:.0f} MHz")
    print("phase       span | median: entry  stage  dot+epi | max work | barrier  (us)")
    total = 0.0
    for k, nm in enumerate(names):
        rel, arr, nxt = a[k, :, 4], a[k, :, 5], a[k + 1, :, 4]
        span = (arr.max() - rel.min()) / 1e3
        bar = (nxt.min() - arr.max()) / 1e3
        total += span + bar
        c0, c1, c2, c3, c6 = (a[k, :, j] for j in (0, 1, 2, 3, 6))
        work = ((c3 - c0) / clk).max()
        if (c1 > 0).any():
            h = c1 > 0
            med = "%6.2f %6.2f %8.2f" % (np.median((c6 - c0)[h]) / clk,
                                        np.median((c1 - c6)[h]) / clk,
                                        np.median((c2 - c1)[h]) / clk)
        else:
            med = " " * 22
        print(f"{nm:9s} {span:6.2f} | {med} | {work:8.2f} | {bar:6.2f}")
    print(f"pass total {total:.1f} us (globaltimer resolution about 0.25 us)")
    dec.close()


if __name__ == "__main__":
    main()
