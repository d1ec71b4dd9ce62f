"""Pins of the oracle encoder and search (Sec. 3.2-3.5, Sec. 5.5)."""

import json
import math
import os

import numpy as np
import pytest

from oracle import codec, constants as K, search
from oracle.rotation import rotation_matrix, rotation_mode


def _data(n, D, seed=0, scale=1.0):
    rng = np.random.default_rng(seed)
    C = rng.standard_normal((4, D))
    a = rng.integers(0, 4, n)
    X = C[a] + 0.5 * rng.standard_normal((n, D))
    X *= scale
    return X, C * scale, a


@pytest.mark.parametrize("bits,D", [(4, 128), (4, 96), (2, 96), (2, 99), (1, 100), (1, 768), (4, 300), (3, 64)])
def test_evt_normalisation_and_nearest_codeword(bits, D):
    X, C, a = _data(40, D, seed=bits * 1000 + D)
    enc = codec.encode(X, C[a], bits)
    R = rotation_matrix(D, rotation_mode(bits, D))
    z = (X - C[a]) @ R.T
    # Sec. 3.2: after dividing by s_initial = max|z| / E_max(D), max|u| = E_max(D)
    assert np.allclose(np.abs(enc.u[:, :D]).max(1), K.e_max(D), rtol=1e-13)
    assert np.allclose(enc.u[:, :D], z * (K.e_max(D) / np.abs(z).max(1))[:, None], rtol=1e-12, atol=1e-13)
    # zero padding to a multiple of g
    assert np.all(enc.u[:, D:] == 0)
    # nearest codeword by explicit distance to every codeword (independent of thresholds)
    cb = K.codebook(bits)
    g = cb.g
    U = enc.u.reshape(len(X), -1, g)
    d = ((U[:, :, None, :] - cb.C[None, None]) ** 2).sum(-1)
    assert np.array_equal(enc.codes, d.argmin(-1))


@pytest.mark.parametrize("bits,D", [(4, 128), (2, 96), (1, 768), (2, 99)])
def test_norm_correction_invariants(bits, D):
    """Sec. 3.3: ||L uhat|| = ||r||; Sec. 3.5.2: ||G (a + rt)|| = ||x||."""
    X, C, a = _data(30, D, seed=7 + D)
    A = C[a]
    exact = codec.encode(X, A, bits, round_scales=False)
    r = X - A
    assert np.allclose(np.linalg.norm(exact.L_exact[:, None] * exact.uhat, axis=1),
                       np.linalg.norm(r, axis=1), rtol=1e-13)
    assert np.allclose(np.linalg.norm(exact.recon, axis=1), np.linalg.norm(X, axis=1), rtol=1e-13)
    enc = codec.encode(X, A, bits)
    rel = np.abs(np.linalg.norm(enc.Lhat[:, None] * enc.uhat, axis=1) / np.linalg.norm(r, axis=1) - 1)
    assert np.all(rel <= 2.0 ** -10 * (1 + 1e-9))
    rel = np.abs(np.linalg.norm(enc.recon, axis=1) / np.linalg.norm(X, axis=1) - 1)
    assert np.all(rel <= 2.0 ** -13 * (1 + 1e-9))
    # reconstructed residual lives in the original space: Lhat R^T uhat
    R = rotation_matrix(D, rotation_mode(bits, D))
    rt = enc.Lhat[:, None] * (R.T @ enc.uhat.T).T
    assert np.allclose(enc.recon, enc.Ghat[:, None] * (A + rt), atol=1e-12)
    # the stored scale codes reproduce the decoded values
    assert np.array_equal(K.UE7M9.decode(enc.L_u16), enc.Lhat)
    assert np.array_equal(codec.decode(A, enc.codes, enc.L_u16, enc.G_u16, bits, D), enc.recon)


def test_local_mode_has_unit_global_scale():
    X, C, a = _data(10, 64, seed=3)
    enc = codec.encode(X, C[a], 4, global_scale=False)
    assert np.all(enc.G_u16 == 7 << 12) and np.all(enc.Ghat == 1.0)


def test_zero_residual_and_zero_vector():
    D = 64
    C = np.random.default_rng(1).standard_normal((1, D))
    X = np.vstack([C[0], np.zeros(D)])
    A = np.vstack([C[0], np.zeros(D)])
    enc = codec.encode(X, A, 4)
    assert np.all(enc.L_u16 == 0) and np.all(enc.Lhat == 0)
    assert enc.G_u16[0] == 7 << 12  # ||x|| / ||a|| = 1
    assert enc.G_u16[1] == 0        # 0 / 0 -> 0
    assert np.allclose(enc.recon[0], C[0]) and np.all(enc.recon[1] == 0)


def test_scales_from_codes_matches_encode():
    X, C, a = _data(20, 96, seed=11)
    enc = codec.encode(X, C[a], 2)
    L_u16, G_u16, _, _ = codec.scales_from_codes(X, C[a], 2, enc.codes)
    assert np.array_equal(L_u16, enc.L_u16) and np.array_equal(G_u16, enc.G_u16)


def test_pack_nibbles_order():
    codes = np.array([[1, 2, 3], [15, 0, 7]])
    packed = codec.pack_nibbles(codes)
    assert packed.tolist() == [[0x21, 0x03], [0x0F, 0x07]]
    assert np.array_equal(codec.unpack_nibbles(packed, 3), codes)


def test_bytes_per_vector_against_paper():
    with open(os.path.join(os.path.dirname(__file__), "golden", "codec_sizes.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        assert codec.bytes_per_vector(c["D"], c["bits"], c["scales"]) == c["bytes"], c


def test_error_falls_with_bits():
    X, C, a = _data(200, 128, seed=5)
    errs = {}
    for b in (1, 2, 3, 4):
        enc = codec.encode(X, C[a], b)
        errs[b] = np.mean(np.sum((enc.recon - X) ** 2, 1) / np.sum((X - C[a]) ** 2, 1))
    assert errs[4] < errs[3] < errs[2] < errs[1] < 0.5


# ------------------------------------------------------------------- search
def _index(X, C, a, bits, rescore_bits=0, **kw):
    return search.build_index(X, np.arange(len(X)), a, C, bits, rescore_bits, **kw)


def test_score_identity_equals_explicit_reconstruction():
    """Sec. 3.5: Ghat (<q,c> + Lhat <Rq, uhat>) == <q, Ghat (c + Lhat R^T uhat)>."""
    X, C, a = _data(300, 96, seed=21)
    idx = _index(X, C, a, 2, 4)
    q = np.random.default_rng(2).standard_normal(96)
    probes, cs, _ = search.probe(q, C, 4)
    rows, s1 = search.stage1_scores(idx, q, probes[0], cs[0])
    assert np.allclose(s1, idx.stage1.recon[rows] @ q, rtol=1e-12, atol=1e-12)
    ids, sc = search.scan(idx, q, probes[0], cs[0], 50)
    f_ids, f_sc, s2 = search.rescore(idx, q, ids, sc, 50)
    # reading B: <q, a2> is the stage-1 score, so s2 == <q, stage-2 reconstruction>
    assert np.allclose(s2, idx.stage2.recon[ids] @ q, rtol=1e-12, atol=1e-12)
    assert np.allclose(np.sort(f_sc)[::-1], f_sc)


def test_identity_quantizer_search_is_exact_mips():
    """With no quantization error the pipeline is exact brute-force MIPS."""
    X, C, a = _data(400, 64, seed=31, scale=3.0)
    st = codec.encode(X, C[a], 4, quantize=False, round_scales=False)
    assert np.allclose(st.recon, X, atol=1e-12)
    idx = search.OracleIndex(64, 4, 0, True, C, np.arange(400), a, st, None,
                             {int(p): np.nonzero(a == p)[0] for p in range(4)})
    Q = np.random.default_rng(9).standard_normal((5, 64))
    res = search.search(idx, Q, nprobe=4, k=10)
    for i in range(5):
        exact = X @ Q[i]
        o = np.lexsort((np.arange(400), -exact))[:10]
        assert np.array_equal(res["ids"][i], o)
        assert np.allclose(res["scores"][i], exact[o], rtol=1e-12)


def test_16bit_highres_codebook_approaches_exact_mips():
    X, C, a = _data(300, 96, seed=41)
    cb = K.highres_codebook(16)
    st = codec.encode(X, C[a], 4, cb=cb, round_scales=False)
    idx = search.OracleIndex(96, 4, 0, True, C, np.arange(300), a, st, None,
                             {int(p): np.nonzero(a == p)[0] for p in range(4)})
    Q = np.random.default_rng(4).standard_normal((6, 96))
    res = search.search(idx, Q, nprobe=4, k=10)
    for i in range(6):
        exact = X @ Q[i]
        scale = np.linalg.norm(Q[i]) * np.linalg.norm(X, axis=1).max()
        got = res["scores"][i]
        assert np.all(np.abs(got - exact[res["ids"][i]]) < 1e-5 * scale)
        o = np.lexsort((np.arange(300), -exact))[:10]
        # same top-10 except swaps among near-ties
        kth = exact[o[-1]]
        assert np.all(exact[res["ids"][i]] >= kth - 2e-5 * scale)


def test_probe_order_and_padding():
    C = np.array([[1.0, 0.0], [1.0, 0.0], [0.0, 1.0], [2.0, 0.0]])
    q = np.array([1.0, 0.0])
    p, cs, _ = search.probe(q, C, 3)
    assert p[0].tolist() == [3, 0, 1] and cs[0].tolist() == [2.0, 1.0, 1.0]
    ids, sc = search.take_top(np.array([1.0, 3.0]), np.array([5, 9]), 4)
    assert ids.tolist() == [9, 5, -1, -1] and sc[2] == -np.inf
    ids, sc = search.take_top(np.array([2.0, 2.0, 1.0]), np.array([8, 3, 1]), 2)
    assert ids.tolist() == [3, 8]  # equal scores: lower id first


def test_empty_partition_and_fewer_candidates_than_k():
    X, C, a = _data(12, 32, seed=51)
    a = np.where(a == 1, 0, a)  # partition 1 left empty
    idx = _index(X, C, a, 4)
    q = C[1] * 3
    res = search.search(idx, q, nprobe=1, k=10)
    # the best partition for q is the empty one: nothing to return
    assert res["probes"][0, 0] == 1
    assert res["ids"][0].tolist() == [-1] * 10
    res = search.search(idx, q, nprobe=4, k=20)
    assert (res["ids"][0] >= 0).sum() == 12


# --------------------------------------------------------------- Rslm3
def test_rslm3_packing_by_hand_and_round_trip():
    """Rslm3 (Sec. 3.4: 3 bits per dimension, K = 8) packs 8 codes into 3
    bytes, least significant bit first: codes 1, 2, 3, 4, 5, 6, 7, 0 give
    the stream 001 010 011 100 101 110 111 000 read from bit 0 upwards."""
    codes = np.array([[1, 2, 3, 4, 5, 6, 7, 0]])
    packed = codec.pack_bits3(codes)
    bits = "".join(format(int(b), "08b")[::-1] for b in packed[0])  # bit 0 first
    assert bits == "".join(format(c, "03b")[::-1] for c in codes[0])
    assert packed.shape == (1, 3)
    rng = np.random.default_rng(3)
    for ng in (1, 7, 8, 100, 128, 1536):
        c = rng.integers(0, 8, (5, ng))
        p = codec.pack_bits3(c)
        assert p.shape[1] == (3 * ng + 7) // 8 == codec.bytes_per_vector(ng, 3, 0)
        assert np.array_equal(codec.unpack_bits3(p, ng), c)


def test_rslm3_codes_are_the_nearest_of_eight_levels():
    X, C, a = _data(200, 128, seed=17)
    enc = codec.encode(X, C[a], 3)
    lv = K.codebook(3).C[:, 0]
    d = np.abs(enc.u[:, :, None] - lv[None, None, :])
    assert enc.codes.max() < 8
    assert np.array_equal(enc.codes, np.argmin(d, axis=-1))


@pytest.mark.parametrize("bits", [1, 2, 3, 4])
def test_near_threshold_marks_only_boundary_groups(bits):
    """The tolerance set of the code comparisons: groups placed exactly on a
    decision boundary (a 1-D threshold, or the midpoint of two codewords)
    are marked, groups at a codeword are not."""
    cb = K.codebook(bits)
    g = cb.g
    n = cb.K - 1
    at_code = cb.C[:n].reshape(1, n * g)                    # group j = codeword j
    mid = 0.5 * (cb.C[:n] + cb.C[1:n + 1])                  # between codewords j and j + 1
    if g == 1:
        assert np.allclose(mid[:, 0], cb.thresholds)
    # a midpoint is a boundary only if no other codeword is nearer than its two
    d = ((mid[:, None, :] - cb.C[None, :, :]) ** 2).sum(-1)
    own = ((mid - cb.C[:n]) ** 2).sum(-1)
    boundary = np.sort(d, axis=1)[:, 0] >= own - 1e-12
    assert not codec.near_threshold(at_code, bits).any()
    marked = codec.near_threshold(mid.reshape(1, n * g), bits)[0]
    assert np.array_equal(marked, boundary)
    assert boundary.any()
