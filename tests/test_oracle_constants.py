"""Pins of the oracle's tables and scalar formats (Sec. 3.1.2, 3.2, 3.3.1, 3.5.2)."""

import json
import math
import os
import struct

import numpy as np
import pytest
from scipy import integrate

from oracle import constants as K


def _golden(name):
    with open(os.path.join(os.path.dirname(__file__), "golden", name)) as f:
        return json.load(f)


def test_splitmix64_published_outputs():
    g = _golden("splitmix64.json")
    out = K.splitmix64(g["seed"], 0, len(g["outputs_hex"]))
    assert [int(v) for v in out] == [int(h, 16) for h in g["outputs_hex"]]
    # counter form: starting at n equals the tail of a longer run
    assert np.array_equal(K.splitmix64(123, 5, 4), K.splitmix64(123, 0, 9)[5:])


def test_sign_tables_and_permutation():
    s1 = K.sign_table_s1()
    assert s1.shape == (256,) and set(np.unique(s1)) == {-1.0, 1.0}
    assert 80 < int((s1 > 0).sum()) < 176  # pseudo-random, not constant
    s2 = K.sign_table_s2()
    assert all(s2[i] == s1[(i + 127) % 256] for i in range(256))
    assert not np.array_equal(s1, s2)
    P = K.perm_p128()
    assert sorted(P) == list(range(128)) and list(P) != list(range(128))
    assert K.bit_reversal(8) == (0, 4, 2, 6, 1, 5, 3, 7)
    assert K.bit_reversal(1) == (0,)
    assert K.block_permutation(128) == P
    assert K.block_permutation(64) == K.bit_reversal(64)
    t = K.tiled_signs(s1, 600)
    assert t[256] == s1[0] and t[599] == s1[599 - 512]


def test_lloyd_max_against_max_1960():
    g = _golden("lloyd_max_gaussian.json")
    for Ks, half in g["levels"].items():
        lv = np.array(K.lloyd_max_gaussian(int(Ks)))
        n = int(Ks)
        assert np.allclose(lv[n // 2:], half, atol=g["tolerance_levels"])
        assert np.allclose(lv, -lv[::-1], atol=1e-13)  # symmetric
    lv16 = np.array(K.lloyd_max_gaussian(16))
    th = 0.5 * (lv16[1:] + lv16[:-1])
    assert np.allclose(th[7:], g["thresholds_16"], atol=g["tolerance_levels"])
    # 2 levels: closed form +-sqrt(2/pi), MSE 1 - 2/pi
    assert abs(K.lloyd_max_gaussian(2)[1] - math.sqrt(2 / math.pi)) < 1e-14


def _mse_1d(levels):
    lv = np.asarray(levels)
    t = np.concatenate([[-np.inf], 0.5 * (lv[1:] + lv[:-1]), [np.inf]])
    pdf = lambda x: math.exp(-x * x / 2) / math.sqrt(2 * math.pi)  # noqa: E731
    tot = 0.0
    for i in range(len(lv)):
        tot += integrate.quad(lambda x: (x - lv[i]) ** 2 * pdf(x), t[i], t[i + 1])[0]
    return tot


def test_lloyd_max_optimality_by_quadrature():
    """Centroid condition checked with plain quadrature (not the erfc closed form)."""
    g = _golden("lloyd_max_gaussian.json")
    pdf = lambda x: math.exp(-x * x / 2) / math.sqrt(2 * math.pi)  # noqa: E731
    for n in (2, 4, 8, 16):
        lv = np.array(K.lloyd_max_gaussian(n))
        t = np.concatenate([[-np.inf], 0.5 * (lv[1:] + lv[:-1]), [np.inf]])
        for i in range(n):
            num = integrate.quad(lambda x: x * pdf(x), t[i], t[i + 1], epsabs=1e-14)[0]
            den = integrate.quad(pdf, t[i], t[i + 1], epsabs=1e-14)[0]
            assert abs(num / den - lv[i]) < 1e-9
        assert abs(_mse_1d(lv) - g["mse"][str(n)]) < g["tolerance_mse"]
    assert abs(_mse_1d(K.lloyd_max_gaussian(2)) - (1 - 2 / math.pi)) < 1e-12


def test_codebook_shapes_and_f16_rounding():
    for bits, (k, gdim) in {1: (16, 4), 2: (16, 2), 3: (8, 1), 4: (16, 1)}.items():
        cb = K.codebook(bits)
        assert (cb.K, cb.g) == (k, gdim)
        assert K.group_size(bits) == gdim
        # every component is an exact binary16 value
        assert np.array_equal(cb.C, cb.C.astype(np.float16).astype(np.float64))
    lv = np.array(K.lloyd_max_gaussian(16))
    cb4 = K.codebook(4)
    assert np.all(np.abs(cb4.C[:, 0] - lv) <= np.abs(lv) * 2.0 ** -11)
    assert np.allclose(cb4.thresholds, 0.5 * (cb4.C[1:, 0] + cb4.C[:-1, 0]), rtol=0, atol=0)


def test_1d_assignment_tie_goes_up():
    cb = K.codebook(4)
    t = cb.thresholds
    U = np.array([t[3], np.nextafter(t[3], -np.inf), -10.0, 10.0])[:, None]
    assert cb.assign(U).tolist() == [4, 3, 0, 15]


@pytest.mark.parametrize("g,product_mse", [(2, 0.11748), (4, 0.36338)])
def test_multid_codebook_optimality(g, product_mse):
    """Centroid condition and distortion of the k-means codebooks (Sec. 3.2).

    On the recipe's own samples the Lloyd iterations converged, so every
    codeword is the mean of its Voronoi cell up to the binary16 rounding.
    On independent samples (numpy default_rng) every codeword is within 5
    combined standard errors (training + test sample) of its cell mean, and
    the MSE per dimension is below that of the product of 1-D Lloyd-Max
    quantizers with the same rate.
    """
    cb = K.codebook({2: 2, 4: 1}[g])
    C = cb.C
    T = K.multid_samples(g)
    dt = ((T[:, None, :] - C[None]) ** 2).sum(-1)
    at = dt.argmin(1)
    n_train = np.bincount(at, minlength=16)
    for k in range(16):
        cell = T[at == k]
        ulp = np.spacing(np.abs(C[k]).astype(np.float16)).astype(np.float64)
        # fp16 rounding moved the boundaries slightly: allow half an ulp + a hair
        assert np.all(np.abs(cell.mean(0) - C[k]) <= 0.5 * ulp + 2e-4)
    rng = np.random.default_rng(1234)
    X = rng.standard_normal((400_000, g))
    d = ((X[:, None, :] - C[None]) ** 2).sum(-1)
    a = d.argmin(1)
    mse = d.min(1).mean() / g
    assert mse < product_mse - 0.005
    for k in range(16):
        m = X[a == k]
        assert len(m) > 1000
        se = m.std(0) * math.sqrt(1.0 / len(m) + 1.0 / n_train[k])
        assert np.all(np.abs(m.mean(0) - C[k]) < 5 * se)
    # lexicographic order of the stored codewords
    keys = [tuple(r) for r in C]
    assert keys == sorted(keys)


def test_multid_samples_recipe():
    X = K.multid_samples(2)
    assert X.shape == (K.MULTID_SAMPLES, 2)
    assert np.array_equal(X, np.round(X / K.MULTID_GRID) * K.MULTID_GRID)
    assert abs(X.mean()) < 0.01 and abs(X.std() - 1) < 0.01


def test_e_max_closed_forms_and_monte_carlo():
    assert abs(K.e_max(1) - math.sqrt(2 / math.pi)) < 1e-12
    assert abs(K.e_max(2) - 2 / math.sqrt(math.pi)) < 1e-12
    rng = np.random.default_rng(7)
    for D in (96, 128):
        m = np.abs(rng.standard_normal((200_000, D))).max(1)
        assert abs(m.mean() - K.e_max(D)) < 4 * m.std() / math.sqrt(len(m))
    assert K.e_max(128) < K.e_max(768) < K.e_max(1536)


def _f32_bits_to_float(b):
    return struct.unpack("<f", struct.pack("<I", b & 0xFFFFFFFF))[0]


def test_ue7m9_and_ue4m12_formats():
    f7, f4 = K.UE7M9, K.UE4M12
    assert (f7.bias, f7.emax, f4.bias, f4.emax) == (63, 127, 7, 15)
    assert f7.encode_one(1.0) == 63 << 9
    assert f7.encode_one(0.75) == (62 << 9) | 256
    assert f4.encode_one(1.0) == 7 << 12
    assert f4.encode_one(1.5) == (7 << 12) | 2048
    assert f7.encode_one(0.0) == 0 and f7.decode(0) == 0.0
    # round half to even on the mantissa
    assert f7.encode_one(1.0 + 0.5 / 512) == 63 << 9
    assert f7.encode_one(1.0 + 1.5 / 512) == (63 << 9) | 2
    assert f7.encode_one(2.0 - 0.25 / 512) == 64 << 9  # rounds up into the next binade
    # saturation and flush
    assert f7.encode_one(1e30) == 0xFFFF
    assert f7.encode_one(2.0 ** -63) == 0 and f7.encode_one(2.0 ** -62) == 1 << 9
    assert f4.encode_one(1e9) == 0xFFFF and f4.encode_one(2.0 ** -7) == 0
    # decode of every code equals the binary32 bit trick (exponent rebias)
    u = np.arange(1, 1 << 16)
    v7 = f7.decode(u)
    v4 = f4.decode(u)
    assert np.all(v7[:511] == 0.0) and np.all(v4[:4095] == 0.0)  # exponent 0 is zero
    for code in list(range(512, 800)) + list(range(30000, 30300)) + [65535]:
        assert v7[code - 1] == _f32_bits_to_float((code << 14) + (64 << 23))
    for code in list(range(4096, 4400)) + list(range(30000, 30300)) + [65535]:
        assert v4[code - 1] == _f32_bits_to_float((code << 11) + (120 << 23))
    # encode(decode(u)) == u for all nonzero codes
    for code in range(512, 1 << 16, 37):
        assert f7.encode_one(float(f7.decode(code))) == code
    for code in range(4096, 1 << 16, 37):
        assert f4.encode_one(float(f4.decode(code))) == code
