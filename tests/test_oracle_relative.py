"""Oracle relative-mode variants (Sec. 3.5; Sec. 5.2): rescoring codes of
x - c ("reading A") next to the default x - (stage-1 reconstruction)
("reading B"), and full-vector codes (approximation 0).  CPU."""

import numpy as np
import pytest

from oracle import codec, constants as K, search
from oracle.rotation import rotation_matrix, rotation_mode


def _data(n, D, seed, P=5, scale=1.0):
    rng = np.random.default_rng(seed)
    C = rng.standard_normal((P, D))
    a = rng.integers(0, P, n)
    X = (C[a] + 0.5 * rng.standard_normal((n, D))) * scale
    return X, C * scale, a


def _index(X, C, a, bits, rescore_bits=0, **kw):
    return search.build_index(X, np.arange(len(X)), a, C, bits, rescore_bits, **kw)


def test_reading_a_codes_are_the_finer_codec_of_x_minus_c():
    """Reading A: the rescoring stage encodes the same residual x - c as the
    scoring stage, independently, with the rescoring bit rate."""
    X, C, a = _data(300, 96, seed=1)
    A = _index(X, C, a, 2, 4, reading="A")
    B = _index(X, C, a, 2, 4, reading="B")
    direct = codec.encode(X, C[a], 4)
    assert np.array_equal(A.stage2.codes, direct.codes)
    assert np.array_equal(A.stage2.L_u16, direct.L_u16) and np.array_equal(A.stage2.G_u16, direct.G_u16)
    assert np.array_equal(A.stage1.codes, B.stage1.codes)
    # reading B's second residual is x - (stage-1 reconstruction), a different code
    assert not np.array_equal(B.stage2.codes, direct.codes)


@pytest.mark.parametrize("reading", ["A", "B"])
def test_rescore_score_identity(reading):
    """Sec. 3.5: the rescoring score equals <q, stage-2 reconstruction> for
    both readings (reading A: Ghat2 (c + Lhat2 R2^T uhat2))."""
    X, C, a = _data(300, 96, seed=2)
    idx = _index(X, C, a, 2, 4, reading=reading)
    q = np.random.default_rng(3).standard_normal(96)
    probes, cs, _ = search.probe(q, C, 5)
    ids, sc = search.scan(idx, q, probes[0], cs[0], 80)
    _, _, s2 = search.rescore(idx, q, ids, sc, 80)
    recon2 = codec.decode(C[a] if reading == "A" else idx.stage1.recon, codec.unpack_nibbles(
        codec.pack_nibbles(idx.stage2.codes), idx.stage2.codes.shape[1]), idx.stage2.L_u16,
        idx.stage2.G_u16, 4, 96)
    assert np.allclose(s2, recon2[ids] @ q, rtol=1e-12, atol=1e-12)


def test_reading_a_rescoring_is_at_least_as_close_as_stage1():
    """The finer independent code of the same residual scores closer to the
    exact <q, x> than the 2-bit stage-1 code, on average."""
    X, C, a = _data(400, 96, seed=4)
    idx = _index(X, C, a, 2, 4, reading="A")
    q = np.random.default_rng(5).standard_normal(96)
    probes, cs, _ = search.probe(q, C, 5)
    ids, sc = search.scan(idx, q, probes[0], cs[0], 200)
    _, _, s2 = search.rescore(idx, q, ids, sc, 200)
    exact = X[ids] @ q
    assert np.mean(np.abs(s2 - exact)) < 0.5 * np.mean(np.abs(sc - exact))


def test_full_vector_codes_encode_x_itself():
    """Approximation 0: the codes are the codec of x, the scores carry no
    <q, c> term, and the global scale is 1 up to the UE7M9 step, because the
    local scale already restores ||x||."""
    X, C, a = _data(300, 128, seed=6)
    idx = _index(X, C, a, 4, 0, full_vector=True)
    direct = codec.encode(X, np.zeros_like(X), 4)
    assert np.array_equal(idx.stage1.codes, direct.codes)
    assert np.all(np.abs(idx.stage1.G_exact - 1.0) <= 2.0 ** -9)
    q = np.random.default_rng(7).standard_normal(128)
    probes, cs, _ = search.probe(q, C, 3)
    rows, s1 = search.stage1_scores(idx, q, probes[0], cs[0])
    assert np.allclose(s1, idx.stage1.recon[rows] @ q, rtol=1e-12, atol=1e-12)
    R = rotation_matrix(128, rotation_mode(4, 128))
    recon = idx.stage1.Ghat[:, None] * idx.stage1.Lhat[:, None] * (idx.stage1.uhat @ R)
    assert np.allclose(idx.stage1.recon, recon, rtol=0, atol=1e-12)


def test_full_vector_identity_quantizer_is_exact_mips():
    """With no quantization error a full-vector index is exact MIPS over the
    probed partitions: the score of a row is <q, x>."""
    X, C, a = _data(400, 64, seed=8, scale=3.0)
    st = codec.encode(X, np.zeros_like(X), 4, quantize=False, round_scales=False)
    assert np.allclose(st.recon, X, atol=1e-12)
    idx = search.OracleIndex(64, 4, 0, True, C, np.arange(400), a, st, None,
                             {int(p): np.nonzero(a == p)[0] for p in range(5)}, "B", True)
    Q = np.random.default_rng(9).standard_normal((5, 64))
    res = search.search(idx, Q, nprobe=5, k=10)
    for i in range(5):
        exact = X @ Q[i]
        o = np.lexsort((np.arange(400), -exact))[:10]
        assert np.array_equal(res["ids"][i], o)
        assert np.allclose(res["scores"][i], exact[o], rtol=1e-12)


def test_bad_reading_is_rejected():
    X, C, a = _data(10, 16, seed=9)
    with pytest.raises(ValueError):
        _index(X, C, a, 4, 0, reading="C")
