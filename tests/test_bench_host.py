"""Host-side rules of bench.py that need no GPU: the DRAM counters it reports as
roofline.traffic are tied to the kernel code by a hash that ignores comments and blank lines,
and the per-pass algorithmic bytes follow the byte model of the decoder pass."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
import synth  # noqa: E402

SRC = """// leading comment
template <typename W>
__device__ int f(int a) {   // trailing comment
  /* block
     comment */ return a + 1;

}
"""


def test_comment_edits_keep_the_hash_and_code_edits_change_it():
    base = bench.code_without_comments(SRC)
    assert base == "template <typename W>\n__device__ int f(int a) {\n   return a + 1;\n}"
    reworded = SRC.replace("trailing comment", "another remark").replace("block", "other")
    assert bench.code_without_comments(reworded) == base
    assert bench.code_without_comments(SRC.replace("a + 1", "a + 2")) != base


def test_sources_hash_reads_every_kernel_file():
    seen = []

    def read(name):
        seen.append(name)
        return SRC
    bench.kernel_sources_sha256(read)
    d = os.path.join(bench.ROOT, "paper_2305_10427_gb300", "csrc")
    assert sorted(seen) == sorted(f for f in os.listdir(d) if f.endswith((".cu", ".cuh")))


def test_pass_bytes_model():
    """Marian-sized bf16 model: 6 decoder layers of 4 d^2 (self QKV + O) + 2 d^2 (cross Q + O)
    + 2 d f weights plus their biases and LayerNorms, the tied V x d table, and the K/V traffic:
    ~103.5 MB of weights per pass."""
    spec = synth.MARIAN
    d, f, V, L = spec.d_model, spec.d_ff, spec.vocab, spec.n_dec_layers
    weights = L * (6 * d * d + 2 * d * f + 3 * d + d + d + d + f + d + 6 * d) + V * d
    got = bench.pass_bytes(spec, L_keys=10, n_src=7, rows=5)
    assert got == 2 * (weights + L * 2 * d * (10 + 7) + L * 2 * d * 5)
    assert 103e6 < 2 * weights < 104e6


def test_reference_arm_prints_one_contract_line():
    """bench.py --impl reference (the CPU oracle arm the driver runs beside the GPU arm)
    prints exactly one JSON line with the contract's keys."""
    import json
    import subprocess
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "1"], capture_output=True, text=True,
                         timeout=600, check=True).stdout.strip().splitlines()
    assert len(out) == 1
    line = json.loads(out[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
