"""Oracle Rslm4Lite codec (Sec. 3.4, Rslm4Lite paragraph; Sec. 3.5) against
what the paper and the plain 4-bit codec fix (CPU)."""

import json
import os

import numpy as np
import pytest

from oracle import codec, constants as K, search
from oracle.rotation import rotation_matrix, rotation_mode


def _data(n, D, seed, P=6):
    rng = np.random.default_rng(seed)
    C = rng.standard_normal((P, D))
    a = rng.integers(0, P, n)
    X = C[a] + 0.4 * rng.standard_normal((n, D))
    return X, C, a


@pytest.mark.parametrize("global_scale", [True, False])
def test_packed_row_is_half_a_byte_per_dimension(global_scale):
    """Sec. 3.4: the scale lives in the codes, so a row packs to exactly
    ceil(D/2) bytes; at D = 256 that is the paper's two cache lines."""
    with open(os.path.join(os.path.dirname(__file__), "golden", "codec_sizes.json")) as f:
        g = json.load(f)
    lite = [c for c in g["cases"] if c["bits"] == 4 and c["scales"] == 0]
    assert lite
    for c in lite:
        X, C, a = _data(5, c["D"], seed=c["D"])
        enc = codec.encode_lite(X, C[a], global_scale)
        assert enc.codes.max() < 16
        assert codec.pack_nibbles(enc.codes).shape[1] == c["bytes"]


def test_small_dimensions_are_rejected():
    X, C, a = _data(3, 48, seed=1)
    with pytest.raises(ValueError):
        codec.encode_lite(X, C[a])


@pytest.mark.parametrize("global_scale,D", [(True, 64), (False, 128), (True, 100), (False, 768)])
def test_head_on_k8_tail_identical_to_rslm4(global_scale, D):
    """Only the first H coordinates change: the tail's codes equal the plain
    4-bit codec's (same rotation, same EVT scale), and the head's levels are
    the nearest of the 8 levels by brute force (a value on a threshold goes
    up)."""
    X, C, a = _data(200, D, seed=D + int(global_scale))
    H = codec.lite_head(global_scale)
    lite = codec.encode_lite(X, C[a], global_scale)
    plain = codec.encode(X, C[a], 4, global_scale=global_scale)
    levels, _, _ = codec.unpack_lite(lite.codes, global_scale)
    assert np.array_equal(levels[:, H:], plain.codes[:, H:])
    assert np.array_equal(lite.u, plain.u[:, :D])
    lv = K.codebook(3).C[:, 0]
    d = np.abs(lite.u[:, :H, None] - lv[None, None, :])
    near = np.argmin(d, axis=-1)
    # argmin takes the lower level on an exact tie; the codec goes up: none here
    gap = np.sort(d, axis=-1)
    assert (gap[..., 1] - gap[..., 0] > 1e-12).all()
    assert np.array_equal(levels[:, :H], near)
    assert np.array_equal(lite.uhat[:, :H], lv[near])


@pytest.mark.parametrize("global_scale", [True, False])
def test_scale_bits_in_the_top_bits(global_scale):
    """Bit i of the UE7M9 code (and, with the global scale, of the UE4M12
    code) is the top bit of code i (code 16 + i); the stored scale codes
    are those of the norm correction."""
    X, C, a = _data(64, 128, seed=7)
    enc = codec.encode_lite(X, C[a], global_scale)
    for row in range(len(X)):
        Lbits = sum(int((enc.codes[row, i] >> 3) & 1) << i for i in range(16))
        assert Lbits == enc.L_u16[row]
        if global_scale:
            Gbits = sum(int((enc.codes[row, 16 + i] >> 3) & 1) << i for i in range(16))
            assert Gbits == enc.G_u16[row]
    # the tail keeps whole 4-bit codes
    H = codec.lite_head(global_scale)
    assert (enc.codes[:, H:] >= 8).any()
    levels, L, G = codec.unpack_lite(enc.codes, global_scale)
    assert np.array_equal(L, enc.L_u16) and np.array_equal(G, enc.G_u16)
    assert levels[:, :H].max() < 8


@pytest.mark.parametrize("global_scale", [True, False])
def test_norm_correction_with_mixed_codebooks(global_scale):
    """Sec. 3.3 / 3.5.2 with the mixed K=8 / K=16 codewords: ||L uhat|| = ||r||
    and ||G (a + rt)|| = ||x|| exactly before rounding, within the UE7M9 /
    UE4M12 steps after."""
    X, C, a = _data(300, 128, seed=11)
    enc = codec.encode_lite(X, C[a], global_scale)
    r = X - C[a]
    nu = np.linalg.norm(enc.uhat, axis=1)
    assert np.allclose(enc.L_exact * nu, np.linalg.norm(r, axis=1), rtol=1e-12)
    assert np.allclose(enc.Lhat * nu, np.linalg.norm(r, axis=1), rtol=2.0 ** -10)
    if global_scale:
        assert np.allclose(np.linalg.norm(enc.recon, axis=1), np.linalg.norm(X, axis=1), rtol=2.0 ** -12)
    else:
        assert (enc.Ghat == 1.0).all()
    # the decode of the stored codes rebuilds the same reconstruction
    assert np.allclose(codec.decode_lite(C[a], enc.codes, 128, global_scale), enc.recon, rtol=0, atol=1e-12)


@pytest.mark.parametrize("global_scale", [True, False])
def test_lite_error_mixes_rslm3_and_rslm4(global_scale):
    """The first H coordinates carry the 3-bit error, the rest the 4-bit
    error: the relative error is the coordinate-weighted mix of the two
    codecs' errors (within 15%), between them."""
    D = 128
    X, C, a = _data(400, D, seed=5)
    H = codec.lite_head(global_scale)
    r2 = np.sum((X - C[a]) ** 2, 1)
    err = {}
    for name, enc in (("3", codec.encode(X, C[a], 3, global_scale=global_scale)),
                      ("4", codec.encode(X, C[a], 4, global_scale=global_scale)),
                      ("lite", codec.encode_lite(X, C[a], global_scale))):
        err[name] = np.mean(np.sum((enc.recon - X) ** 2, 1) / r2)
    mix = (H * err["3"] + (D - H) * err["4"]) / D
    assert err["4"] < err["lite"] < err["3"]
    assert abs(err["lite"] - mix) < 0.15 * mix


def test_lite_score_identity():
    """Sec. 3.5: the oracle scan's scores of a Rslm4Lite index equal
    <q, decoded reconstruction> of the stored codes."""
    X, C, a = _data(300, 128, seed=21)
    idx = search.build_index(X, np.arange(len(X)), a, C, 4, 0, lite=True)
    q = np.random.default_rng(3).standard_normal(128)
    probes, cs, _ = search.probe(q, C, 3)
    rows, s1 = search.stage1_scores(idx, q, probes[0], cs[0])
    recon = codec.decode_lite(C[a], idx.stage1.codes, 128, True)
    assert np.allclose(s1, recon[rows] @ q, rtol=1e-12, atol=1e-12)
    # and the rotation is the 4-bit codec's
    assert np.array_equal(rotation_matrix(128, rotation_mode(4, 128)),
                          rotation_matrix(128, idx.stage1.mode))
