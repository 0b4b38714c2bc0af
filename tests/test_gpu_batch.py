"""Batched decoding (pd_encode_batch / pd_decode_batch) against single-sentence decoding.

Every sentence of a batch must come out exactly as pd_decode returns it alone (same tokens,
same pass count) for every method and stop rule: each row's arithmetic does not depend on the
other rows of a pass (batch invariance) and every sentence keeps its own state, cache slots
and source length.  The single-sentence path itself is checked against the oracle in
test_gpu_parity.py; here the oracle checks one batch directly where its margins allow.
"""
import numpy as np
import pytest

import synth
import paper_2305_10427_gb300 as pkg
from oracle import decode as od
from oracle import model as om

pytestmark = pytest.mark.gpu

RUNS = [("greedy", 1, 0), ("gs_jacobi", 3, 0), ("gs_jacobi", 5, 0), ("hybrid_gs_jacobi", 3, 0),
        ("hybrid_gs_jacobi", 4, 6), ("jacobi", 0, 0)]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import os
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)
    torch.cuda.set_device(0)


def _decoder(spec, max_batch, eos=synth.EOS_ID, engine="auto", **wkw):
    w = synth.make_weights(spec, **wkw)
    cfg = pkg.Config.from_spec(spec, 64, 128, eos_id=eos, max_batch=max_batch, engine=engine)
    return w, pkg.Decoder(cfg, w.blob)


MODELS = {
    "tiny": (synth.TINY, synth.EOS_ID, dict(seed=0)),
    "tiny_vary": (synth.TINY, synth.EOS_ID, dict(seed=5, embed_std=0.005)),
    "tiny_eos": (synth.TINY, 3038, dict(seed=5, embed_std=0.005)),
    "marian": (synth.MARIAN, synth.EOS_ID, dict(seed=0)),
}
# (model, engine) pairs of the batch-versus-single test
BATCH_CASES = [(m, "simt") for m in MODELS] + [("marian", "tensor"), ("tiny_vary", "cluster"),
                                               ("tiny_eos", "cluster"), ("marian", "cluster")]


@pytest.mark.parametrize("name,engine", BATCH_CASES)
def test_batch_equals_single(name, engine):
    spec, eos, kw = MODELS[name]
    _, dec = _decoder(spec, 4, eos=eos, engine=engine, **kw)
    sents = synth.sentences(61, 4, 5, 20, spec.vocab)
    max_len = [2 * len(s) for s in sents]
    single = {}
    for k, s in enumerate(sents):
        dec.encode(s)
        for m, b, h in RUNS:
            for rule in ("paper", "prefix"):
                single[k, m, b, h, rule] = dec.decode(m, max_len[k], b=b, h=h, stop_rule=rule)
    dec.encode_batch(sents)
    for m, b, h in RUNS:
        for rule in ("paper", "prefix"):
            got = dec.decode_batch(m, max_len, b=b, h=h, stop_rule=rule)
            for k in range(len(sents)):
                ref = single[k, m, b, h, rule]
                assert (got[k].tokens, got[k].n_iters) == (ref.tokens, ref.n_iters), \
                    (k, m, b, h, rule)
    # a prefix of the encoded sentences, and one sentence alone
    got = dec.decode_batch("gs_jacobi", max_len[:2], b=5)
    for k in range(2):
        assert got[k].tokens == single[k, "gs_jacobi", 5, 0, "paper"].tokens
    got = dec.decode_batch("greedy", max_len[:1])
    assert got[0].tokens == single[0, "greedy", 1, 0, "paper"].tokens
    dec.close()


def test_batch_against_oracle():
    """One batch of the tiny model: tokens and pass counts of every sentence equal the
    oracle's step-by-step GS-Jacobi run where all its decisions had margin."""
    spec, eos, kw = MODELS["tiny"]
    w, dec = _decoder(spec, 4, eos=eos, **kw)
    model = om.Model(spec, w.tensors)
    sents = synth.sentences(63, 3, 6, 14, spec.vocab)
    max_len = [2 * len(s) for s in sents]
    dec.encode_batch(sents)
    got = dec.decode_batch("gs_jacobi", max_len, b=3)
    compared = 0
    for k, s in enumerate(sents):
        ref = od.gs_jacobi(od.model_step(model, np.asarray(s)), max_len[k], 3, eos=eos)
        if ref.min_margin > 1e-3:
            assert (got[k].tokens, got[k].n_iters) == (ref.tokens, ref.n_iters), k
            compared += 1
    assert compared >= 1
    dec.close()


def test_batch_errors():
    _, dec = _decoder(synth.TINY, 2, seed=0)
    sents = synth.sentences(62, 3, 5, 9, synth.TINY.vocab)
    with pytest.raises(pkg.PdError) as e:
        dec.decode_batch("greedy", [8, 8])                      # nothing encoded yet
    assert e.value.status == -6
    with pytest.raises(pkg.PdError) as e:
        dec.encode_batch(sents)                                 # 3 > max_batch 2
    assert e.value.status == -1
    with pytest.raises(pkg.PdError) as e:
        dec.encode_batch([sents[0], np.zeros(0, dtype=np.int32)])   # an empty sentence
    assert e.value.status == -1
    dec.encode_batch(sents[:1])
    with pytest.raises(pkg.PdError) as e:
        dec.decode_batch("greedy", [8, 8])                      # only one sentence encoded
    assert e.value.status == -6
    dec.encode_batch(sents[:2])
    with pytest.raises(pkg.PdError) as e:
        dec.decode_batch("greedy", [8, 8, 8])                   # 3 > max_batch
    assert e.value.status == -1
    with pytest.raises(pkg.PdError) as e:
        dec.decode_batch("greedy", [8, 0])                      # max_len out of range
    assert e.value.status == -1
    assert len(dec.decode_batch("greedy", [8, 6])) == 2
    dec.close()
    _, dec = _decoder(synth.TINY, 8, seed=0)                    # a pass holds 512 rows at most
    sents = synth.sentences(64, 8, 5, 9, synth.TINY.vocab)
    dec.encode_batch(sents)
    with pytest.raises(pkg.PdError) as e:
        dec.decode_batch("jacobi", [100] * 8)                   # 800 rows
    assert e.value.status == -1
    assert len(dec.decode_batch("jacobi", [60] * 8)) == 8       # 480 rows
    dec.close()


@pytest.mark.parametrize("engine", ["simt", "tensor", "cluster"])
def test_paged_cache_pool(engine):
    """The self-attention keys and values live in a pool of 16-position pages handed out per
    decode (sentence s's pages interleaved with the others', never contiguous in a batch).  A
    pool sized for the batch's actual lengths (here 12 pages instead of the 4 x 8 that max_tgt_len
    would need) decodes every sentence exactly as a context with the default pool decodes it
    alone, and a request that needs more pages than the pool holds is rejected before any
    launch."""
    spec = MODELS["marian"][0] if engine == "tensor" else synth.TINY
    w = synth.make_weights(spec, seed=0)
    big = pkg.Decoder(pkg.Config.from_spec(spec, 64, 128, engine=engine), w.blob)
    small = pkg.Decoder(pkg.Config.from_spec(spec, 64, 128, max_batch=4, engine=engine,
                                             kv_pages=12), w.blob)
    sents = synth.sentences(65, 4, 8, 20, spec.vocab)
    max_len = [min(48, 2 * len(s)) for s in sents]          # <= 3 pages each, 12 in all
    small.encode_batch(sents)
    for m, b in (("gs_jacobi", 5), ("jacobi", 0), ("greedy", 1)):
        got = small.decode_batch(m, max_len, b=b)
        for k, s in enumerate(sents):
            big.encode(s)
            ref = big.decode(m, max_len[k], b=b)
            assert (got[k].tokens, got[k].n_iters) == (ref.tokens, ref.n_iters), (m, k)
    with pytest.raises(pkg.PdError) as e:
        small.decode_batch("greedy", [64, 64, 64, 64])         # 16 pages > 12
    assert e.value.status == -1 and "page pool" in str(e.value)
    small.close()
    big.close()
