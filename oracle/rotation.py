"""Block-wise cascaded FWHT rotation as an explicit float64 matrix.

Test infrastructure only: see ``oracle/__init__.py``.

Follows Sec. 3.1 of the paper:

* Sec. 3.1.1: orthonormal Walsh-Hadamard H_n = Hhat_n / sqrt(n) with the
  Sylvester recursion Hhat_2n = [[Hhat_n, Hhat_n], [Hhat_n, -Hhat_n]],
  Hhat_1 = [1]; applied block-wise with B = 128, B shrunk to the largest
  power of two <= D when D < 128; when B does not divide D a last block
  [D-B, D) overlapping its predecessor is applied after the full blocks.
* Sec. 3.1.2: sign flips S1 tiled over the coordinates; the in-block
  permutation P (bit reversal when B < 128); the strided transpose
  x'[k M + b] = x[b B + P(k)] for b < M = floor(D/B), k < B, tail
  coordinates i >= M B unchanged.
* Sec. 3.1.3: the single-pass variant (Rslm4 with D <= 256: S1 then the
  block FWHT) and the two-pass cascade (S1, FWHT, permute + transpose, S2,
  FWHT) used otherwise.

The rotation is materialised by pushing the identity through these steps;
applying it to a vector is then an O(D^2) matrix product.
"""

from __future__ import annotations

import functools

import numpy as np

from oracle.constants import block_permutation, sign_table_s1, sign_table_s2, tiled_signs


def block_size(D: int) -> int:
    """B = 128, or the largest power of two <= D when D < 128."""
    if D >= 128:
        return 128
    return 1 << (D.bit_length() - 1)


def block_starts(D: int) -> list:
    """Start offsets of the FWHT blocks in application order.

    Full blocks [m B, (m+1) B) for m < floor(D/B), then the overlapping
    block [D-B, D) if B does not divide D.
    """
    B = block_size(D)
    M = D // B
    starts = [m * B for m in range(M)]
    if D % B:
        starts.append(D - B)
    return starts


@functools.lru_cache(maxsize=None)
def hadamard_unnormalized(n: int) -> np.ndarray:
    """Hhat_n by the Sylvester recursion (Sec. 3.1.1)."""
    H = np.ones((1, 1))
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    assert H.shape[0] == n, "n must be a power of two"
    return H


def hadamard(n: int) -> np.ndarray:
    """Orthonormal H_n = Hhat_n / sqrt(n)."""
    return hadamard_unnormalized(n) / np.sqrt(n)


def rotation_mode(bits: int, D: int) -> str:
    """'single' for the 4-bit codecs at D <= 256, else 'two' (Sec. 3.1.3)."""
    return "single" if (bits == 4 and D <= 256) else "two"


def _apply_blocks(Y: np.ndarray, D: int, reverse: bool = False) -> np.ndarray:
    """Apply H_B to every block of each row of Y (n x D), in block order."""
    B = block_size(D)
    H = hadamard(B)
    starts = block_starts(D)
    if reverse:
        starts = starts[::-1]
    Y = Y.copy()
    for s in starts:
        Y[:, s:s + B] = Y[:, s:s + B] @ H.T
    return Y


def _transpose_map(D: int) -> np.ndarray:
    """src[i] such that y'[i] = y[src[i]] for the permute + transpose step."""
    B = block_size(D)
    M = D // B
    P = block_permutation(B)
    src = np.arange(D)
    for b in range(M):
        for k in range(B):
            src[k * M + b] = b * B + P[k]
    return src


def rotate_rows(X: np.ndarray, mode: str) -> np.ndarray:
    """Apply the rotation pipeline to every row of X (n x D)."""
    X = np.asarray(X, dtype=np.float64)
    D = X.shape[1]
    Y = X * tiled_signs(sign_table_s1(), D)[None, :]
    Y = _apply_blocks(Y, D)
    if mode == "single":
        return Y
    Y = Y[:, _transpose_map(D)]
    Y = Y * tiled_signs(sign_table_s2(), D)[None, :]
    return _apply_blocks(Y, D)


def unrotate_rows(Z: np.ndarray, mode: str) -> np.ndarray:
    """Inverse pipeline: every step inverted, blocks in reverse order."""
    Z = np.asarray(Z, dtype=np.float64)
    D = Z.shape[1]
    Y = Z
    if mode == "two":
        Y = _apply_blocks(Y, D, reverse=True)
        Y = Y * tiled_signs(sign_table_s2(), D)[None, :]
        out = np.empty_like(Y)
        out[:, _transpose_map(D)] = Y
        Y = out
    Y = _apply_blocks(Y, D, reverse=True)
    return Y * tiled_signs(sign_table_s1(), D)[None, :]


@functools.lru_cache(maxsize=64)
def rotation_matrix(D: int, mode: str) -> np.ndarray:
    """Explicit D x D matrix R with rotate_rows(x) = x R^T (i.e. R x)."""
    R = rotate_rows(np.eye(D), mode).T
    R.setflags(write=False)
    return R
