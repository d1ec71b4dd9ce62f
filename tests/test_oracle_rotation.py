"""Pins of the oracle rotation (Sec. 3.1.1-3.1.3)."""

import numpy as np
import pytest

from oracle import constants as K
from oracle import rotation as R

DIMS = [1, 2, 3, 5, 64, 96, 100, 127, 128, 129, 200, 256, 300, 768, 1536, 2049]


def test_sylvester_by_hand():
    assert np.array_equal(R.hadamard_unnormalized(2), [[1, 1], [1, -1]])
    H4 = [[1, 1, 1, 1], [1, -1, 1, -1], [1, 1, -1, -1], [1, -1, -1, 1]]
    assert np.array_equal(R.hadamard_unnormalized(4), H4)
    for n in (1, 2, 8, 64, 128):
        H = R.hadamard(n)
        assert np.allclose(H @ H, np.eye(n), atol=1e-13)  # symmetric involution
        assert np.allclose(np.abs(H), 1 / np.sqrt(n))
        # entry (i, j) is (-1)^popcount(i & j) / sqrt(n)
        i, j = np.meshgrid(np.arange(n), np.arange(n), indexing="ij")
        par = np.vectorize(lambda a: bin(a).count("1") & 1)(i & j)
        assert np.allclose(H, np.where(par, -1, 1) / np.sqrt(n))


@pytest.mark.parametrize("D,B,starts", [
    (1, 1, [0]), (2, 2, [0]), (3, 2, [0, 1]), (5, 4, [0, 1]), (64, 64, [0]),
    (96, 64, [0, 32]), (100, 64, [0, 36]), (127, 64, [0, 63]), (128, 128, [0]),
    (129, 128, [0, 1]), (200, 128, [0, 72]), (256, 128, [0, 128]),
    (300, 128, [0, 128, 172]), (1536, 128, [128 * m for m in range(12)]),
    (2049, 128, [128 * m for m in range(16)] + [1921]),
])
def test_block_rule(D, B, starts):
    """B shrinks below 128; a last block [D-B, D) overlaps when B does not divide D."""
    assert R.block_size(D) == B
    assert R.block_starts(D) == starts


def test_mode_rule():
    assert R.rotation_mode(4, 256) == "single"
    assert R.rotation_mode(4, 96) == "single"
    assert R.rotation_mode(4, 257) == "two"
    assert R.rotation_mode(3, 100) == "two"
    assert R.rotation_mode(2, 96) == "two"
    assert R.rotation_mode(1, 64) == "two"


@pytest.mark.parametrize("D", DIMS)
@pytest.mark.parametrize("mode", ["single", "two"])
def test_orthogonal_and_inverse(D, mode):
    M = R.rotation_matrix(D, mode)
    assert np.allclose(M @ M.T, np.eye(D), atol=1e-12)
    # the explicit inverse pipeline (blocks in reverse order) is R^T
    inv = R.unrotate_rows(np.eye(D), mode).T
    assert np.allclose(inv, M.T, atol=1e-12)


def _factor_matrices(D, mode):
    """The pipeline as a product of explicit D x D factor matrices."""
    B = R.block_size(D)
    S1 = np.diag(K.tiled_signs(K.sign_table_s1(), D))
    S2 = np.diag(K.tiled_signs(K.sign_table_s2(), D))
    blocks = []
    for s in R.block_starts(D):
        E = np.eye(D)
        E[s:s + B, s:s + B] = R.hadamard(B)
        blocks.append(E)
    Hb = np.eye(D)
    for E in blocks:  # applied in list order: later factors multiply on the left
        Hb = E @ Hb
    M = D // B
    P = K.block_permutation(B)
    Pi = np.eye(D)
    for b in range(M):
        for k in range(B):
            Pi[k * M + b] = 0
            Pi[k * M + b, b * B + P[k]] = 1
    if mode == "single":
        return Hb @ S1
    return Hb @ S2 @ Pi @ Hb @ S1


@pytest.mark.parametrize("D", [3, 96, 100, 128, 200, 300, 1536])
@pytest.mark.parametrize("mode", ["single", "two"])
def test_matches_factor_product(D, mode):
    assert np.allclose(R.rotation_matrix(D, mode), _factor_matrices(D, mode), atol=1e-12)


def test_transpose_index_map_by_hand():
    P = K.perm_p128()
    for D, M in ((256, 2), (300, 2), (1536, 12)):
        src = R._transpose_map(D)
        x = np.arange(D, dtype=float)
        y = x[src]
        assert y[0] == P[0] and y[1] == 128 + P[0]
        assert y[M] == P[1]
        assert y[M * 5 + (M - 1)] == (M - 1) * 128 + P[5]
        for i in range(M * 128, D):  # tail unchanged
            assert y[i] == i
        assert sorted(y.tolist()) == x.tolist()
    # D <= 128: in-block permutation only (bit reversal below 128)
    src = R._transpose_map(96)
    br = K.bit_reversal(64)
    assert [src[k] for k in range(64)] == list(br) and list(src[64:]) == list(range(64, 96))


def test_spike_is_uniformised_by_one_block():
    """Single pass at D=128: R e_i has every coordinate of magnitude 1/sqrt(128)."""
    M = R.rotation_matrix(128, "single")
    assert np.allclose(np.abs(M), 1 / np.sqrt(128))
    # two-pass at D=256 spreads a spike over both blocks
    M2 = R.rotation_matrix(256, "two")
    col = M2[:, 7]
    assert np.count_nonzero(np.abs(col) > 1e-12) == 256


def test_overlap_block_is_applied_last():
    """Non-commutativity (Sec. 3.1.1): overlap-first gives a different map."""
    D, B = 96, 64
    x = np.random.default_rng(0).standard_normal(D)
    y = x * K.tiled_signs(K.sign_table_s1(), D)
    a = y.copy()
    a[0:64] = R.hadamard(B) @ a[0:64]
    a[32:96] = R.hadamard(B) @ a[32:96]
    b = y.copy()
    b[32:96] = R.hadamard(B) @ b[32:96]
    b[0:64] = R.hadamard(B) @ b[0:64]
    got = R.rotate_rows(x[None], "single")[0]
    assert np.allclose(got, a, atol=1e-13)
    assert not np.allclose(got, b, atol=1e-3)
