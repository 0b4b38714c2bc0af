"""CPU oracle for parallel (Jacobi / GS-Jacobi) decoding — TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 numpy restatement of what the GPU path computes, written from the
paper ("Accelerating Transformer Inference for Translation via Parallel Decoding",
arXiv 2305.10427):

* ``oracle.model``  — the encoder-decoder transformer p_theta(y_i | y_<i, x) (Eq. 1) with the
  greedy argmax of Eq. 2, recomputed from scratch for every prefix (no KV cache).
* ``oracle.decode`` — greedy autoregressive decoding (Eq. 2), Parallel Jacobi (Algorithm 1),
  Parallel GS-Jacobi (Algorithm 2) and Hybrid GS-Jacobi (Algorithm 3) with PAD initialisation
  (Section 3.3, InitT) and the "unchanged block" stopping condition (Eq. 5).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg (and its
``--impl reference`` arm) may import this package.  The product path never does: the
library in ``paper_2305_10427_gb300`` runs every step in its own CUDA kernels and fails
loudly when its shared library is missing.  The two sides share no code; their only common
dependency is ``synth`` (seeded weights and sentences, no arithmetic of the method).

Pins (tests/test_oracle_*.py): the model forward against torch.nn's independent transformer
layers; the fixed point of the triangular system (Eq. 3-4) by brute force over all token
sequences on toy models; Proposition 1 (every method returns the greedy output in at most m
passes, from any initialisation); closed-form pass counts on planted dependency structures;
sinusoid closed forms.  Paper speedups and BLEU need trained weights and datasets and are
parity unpinned.
"""
