"""Weights drawn by the library (pd_create with weights = NULL): Philox-4x32-10 (Salmon et al.,
"Parallel random numbers: as easy as 1, 2, 3", SC 2011) counters per blob element, Box-Muller
normals, std 0.02, LayerNorm gains 1 and biases 0.

The numpy generator below is written from the generator's published definition (test
infrastructure, independent of the CUDA code) and pinned by the published known-answer
vectors; the GPU tests compare the library's exported blob with it element by element, check
the statistics of every tensor, and check that a context built on drawn weights decodes like
one built on the same blob passed in.
"""
import os

import numpy as np
import pytest

import synth

M0, M1 = 0xD2511F53, 0xCD9E8D57
W0, W1 = 0x9E3779B9, 0xBB67AE85
MASK = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Ten Philox rounds on uint64 arrays holding 32-bit words; returns the four output words."""
    c = [np.asarray(x, dtype=np.uint64) & MASK for x in (c0, c1, c2, c3)]
    k0, k1 = np.uint64(k0) & MASK, np.uint64(k1) & MASK
    for _ in range(10):
        p0 = np.uint64(M0) * c[0]
        p1 = np.uint64(M1) * c[2]
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK
        c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
        k0 = (k0 + np.uint64(W0)) & MASK
        k1 = (k1 + np.uint64(W1)) & MASK
    return c


def test_philox_known_answers():
    """The generator's published known-answer vectors (counter, key -> output)."""
    cases = [((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
             ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
             ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
              (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1))]
    for ctr, key, want in cases:
        got = philox4x32_10(*ctr, *key)
        assert tuple(int(x) for x in got) == want


def reference_tensors(spec, seed, std=0.02):
    """The weights pd_create draws for spec from seed, as float32 arrays in blob order."""
    out = []
    for k, (name, shape) in enumerate(synth.tensor_layout(spec)):
        n = int(np.prod(shape))
        parts = name.split(".")
        is_ln = len(parts) >= 2 and parts[-2].startswith("ln")
        if is_ln:
            v = np.full(n, 1.0 if parts[-1] == "g" else 0.0, dtype=np.float32)
        else:
            e = np.arange(n, dtype=np.uint64)
            r = philox4x32_10(e >> np.uint64(1), k, 0, 0, seed, 0x5EED5EED)
            u1 = (r[0].astype(np.float64) + 0.5) / 4294967296.0
            u2 = (r[1].astype(np.float64) + 0.5) / 4294967296.0
            rad = np.sqrt(-2.0 * np.log(u1))
            ang = 2.0 * np.pi * u2
            z = rad * np.where((e & np.uint64(1)) == 0, np.cos(ang), np.sin(ang))
            v = (std * z).astype(np.float32)
        out.append((name, v))
    return out


def test_reference_statistics():
    """Independent of the library: the drawn normals have the moments of N(0, 0.02^2)."""
    spec = synth.small_spec("stat", d_model=256, n_heads=4, d_ff=512, vocab=3000)
    for name, v in reference_tensors(spec, 3):
        if v.size >= 65536:
            assert abs(v.mean()) < 5 * 0.02 / np.sqrt(v.size)
            assert abs(v.std() / 0.02 - 1) < 0.02
            assert abs(np.mean((v / 0.02) ** 4) - 3) < 0.1            # normal kurtosis


# ---- the library's drawn weights (GPU) --------------------------------------------------------

@pytest.fixture(scope="module")
def gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2305_10427_gb300 as pkg
    if not os.path.exists(pkg.LIB_PATH):
        from paper_2305_10427_gb300 import build
        build.build(force=False)
    torch.cuda.set_device(0)
    return pkg


def _drawn(pkg, spec, seed, **kw):
    return pkg.Decoder(pkg.Config.from_spec(spec, 32, 32, seed=seed, **kw), None)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_drawn_weights_equal_the_reference_generator(gpu, dtype):
    pkg = gpu
    spec = synth.small_spec("drawn", d_model=256, n_heads=4, d_ff=512, n_enc_layers=1,
                            n_dec_layers=2, vocab=3000,
                            dtype=synth.DTYPE_F32 if dtype == "f32" else synth.DTYPE_BF16)
    with _drawn(pkg, spec, 7) as a, _drawn(pkg, spec, 7) as b, _drawn(pkg, spec, 8) as c:
        et = np.float32 if dtype == "f32" else np.uint16
        blob_a, blob_b, blob_c = (d.export_weights(et) for d in (a, b, c))
    assert np.array_equal(blob_a, blob_b) and not np.array_equal(blob_a, blob_c)
    got = synth.weights_from_blob(spec, blob_a)
    for name, ref in reference_tensors(spec, 7):
        g = got[name].reshape(-1)
        if dtype == "bf16":
            ref = synth.bf16_bits_to_f32(synth._round_to_bf16(ref))
        same = np.mean(g == ref)
        # the device's and numpy's double-precision log / sin / cos may differ in the last bit,
        # which can move a value by one unit in its last place after the float32 / bf16 rounding
        ulp = np.spacing(np.abs(ref).astype(np.float32)) * (1 if dtype == "f32" else 65536)
        assert same > 0.999 and (np.abs(g - ref) <= ulp).all(), (name, same)


@pytest.mark.gpu
def test_drawn_weights_decode_like_the_same_blob(gpu):
    """A context on drawn weights and one on its exported blob decode identically."""
    pkg = gpu
    spec = synth.TINY
    with _drawn(pkg, spec, 11) as a:
        blob = a.export_weights(np.float32)
        src = synth.sentences(3, 1, 12, 12, spec.vocab)[0]
        a.encode(src)
        ra = a.decode("gs_jacobi", 24, b=5)
        la = a.debug_logits([synth.BOS_ID] + ra.tokens[:-1])
    with pkg.Decoder(pkg.Config.from_spec(spec, 32, 32), blob) as b:
        b.encode(src)
        rb = b.decode("gs_jacobi", 24, b=5)
        lb = b.debug_logits([synth.BOS_ID] + rb.tokens[:-1])
    assert (ra.tokens, ra.n_iters) == (rb.tokens, rb.n_iters)
    assert np.array_equal(la, lb)
