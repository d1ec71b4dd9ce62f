"""RSLM residual encoding and decoding in float64.

Test infrastructure only: see ``oracle/__init__.py``.

Steps, in the order of Sec. 3.4 ("Codecs Description") applied to the
residual r = x - a of Sec. 3.5:

1. r = x - a, z = R r  (R: the rotation of Sec. 3.1.3 for this bit rate).
2. EVT initial scale (Sec. 3.2): s_initial = max_i |z_i| / E_max(D); the
   normalised vector u = z / s_initial is zero-padded to a multiple of the
   codebook dimension g (Sec. 3.2, last paragraph).
3. Nearest codeword per group of g coordinates (Sec. 3.2).
4. Local norm correction (Sec. 3.3): with uhat the chosen codewords on the D
   valid coordinates, L = ||r|| / ||uhat|| so that ||L uhat|| = ||r||
   (s_initial cancels and is not stored); stored as UE7M9 (Sec. 3.3.1).
5. Reconstructed residual rt = Lhat R^T uhat.
6. Global scale (Sec. 3.5.2): G = ||x|| / ||a + rt|| stored as UE4M12, so
   that ||Ghat (a + rt)|| = ||x||.  In the local mode (Sec. 3.5.1) G is 1.

Codes of K <= 16 codebooks pack two per byte: code of group i goes to the
low nibble of byte i//2 when i is even, the high nibble when i is odd.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

from oracle.constants import UE4M12, UE7M9, Codebook, codebook, e_max
from oracle.rotation import rotation_matrix, rotation_mode


@dataclass
class Encoded:
    """Codes and scales of a batch of rows, plus derived float64 values."""

    bits: int
    mode: str          # rotation mode used ('single' or 'two')
    D: int
    g: int
    codes: np.ndarray  # (n, ngroups) int64 code indices
    L_u16: np.ndarray  # (n,) UE7M9 local scale codes
    G_u16: np.ndarray  # (n,) UE4M12 global scale codes (1.0 in local mode)
    Lhat: np.ndarray   # (n,) decoded local scale
    Ghat: np.ndarray   # (n,) decoded global scale
    uhat: np.ndarray   # (n, D) chosen codewords on the valid coordinates
    u: np.ndarray      # (n, Dp) normalised rotated residual (for tie checks)
    recon: np.ndarray  # (n, D) Ghat * (a + Lhat R^T uhat)
    L_exact: np.ndarray  # (n,) L before UE7M9 rounding
    G_exact: np.ndarray  # (n,) G before UE4M12 rounding


def padded_dim(D: int, g: int) -> int:
    """D rounded up to a multiple of the codebook dimension g."""
    return g * math.ceil(D / g)


def encode(X, A, bits: int, global_scale: bool = True, cb: Codebook | None = None,
           quantize: bool = True, round_scales: bool = True) -> Encoded:
    """Encode residuals X - A (rows) with the ``bits``-per-dimension codec.

    ``cb`` overrides the codebook (tests).  ``quantize=False`` keeps u itself
    as uhat (identity quantizer) and ``round_scales=False`` keeps exact
    scales; both exist only to pin the pipeline against exact arithmetic.
    """
    X = np.asarray(X, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    n, D = X.shape
    cb = cb if cb is not None else codebook(bits)
    g = cb.g
    Dp = padded_dim(D, g)
    mode = rotation_mode(bits, D)
    R = rotation_matrix(D, mode)

    r = X - A                                   # step 1
    z = r @ R.T
    m = np.max(np.abs(z), axis=1) if D else np.zeros(n)
    emax = e_max(D)
    factor = np.where(m > 0, emax / np.where(m > 0, m, 1.0), 0.0)
    u = np.zeros((n, Dp))                       # step 2
    u[:, :D] = z * factor[:, None]

    if quantize:                                # step 3
        codes = cb.assign(u.reshape(n, Dp // g, g))
        uhat = cb.C[codes].reshape(n, Dp)[:, :D]
    else:
        codes = np.zeros((n, Dp // g), dtype=np.int64)
        uhat = u[:, :D].copy()

    nr = np.linalg.norm(r, axis=1)              # step 4
    nu = np.linalg.norm(uhat, axis=1)
    L = np.where(nu > 0, nr / np.where(nu > 0, nu, 1.0), 0.0)
    if round_scales:
        L_u16 = UE7M9.encode(L)
        Lhat = UE7M9.decode(L_u16)
    else:
        L_u16 = np.zeros(n, dtype=np.int64)
        Lhat = L

    rt = Lhat[:, None] * (uhat @ R)             # step 5: rows of R^T uhat

    if global_scale:                            # step 6
        nx = np.linalg.norm(X, axis=1)
        na = np.linalg.norm(A + rt, axis=1)
        G = np.where(na > 0, nx / np.where(na > 0, na, 1.0), 0.0)
    else:
        G = np.ones(n)
    if round_scales:
        G_u16 = UE4M12.encode(G)
        Ghat = UE4M12.decode(G_u16)
    else:
        G_u16 = np.zeros(n, dtype=np.int64)
        Ghat = G
    recon = Ghat[:, None] * (A + rt)
    return Encoded(bits, mode, D, g, codes, L_u16, G_u16, Lhat, Ghat, uhat, u, recon, L, G)


def scales_from_codes(X, A, bits: int, codes, global_scale: bool = True) -> tuple:
    """UE7M9 / UE4M12 scale codes that ``encode`` derives for given codes.

    Steps 4-6 above with the codewords fixed by ``codes`` (n, ngroups).
    """
    X = np.asarray(X, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    n, D = X.shape
    cb = codebook(bits)
    g = cb.g
    Dp = padded_dim(D, g)
    R = rotation_matrix(D, rotation_mode(bits, D))
    uhat = cb.C[np.asarray(codes, dtype=np.int64)].reshape(n, Dp)[:, :D]
    r = X - A
    nr = np.linalg.norm(r, axis=1)
    nu = np.linalg.norm(uhat, axis=1)
    L = np.where(nu > 0, nr / np.where(nu > 0, nu, 1.0), 0.0)
    L_u16 = UE7M9.encode(L)
    rt = UE7M9.decode(L_u16)[:, None] * (uhat @ R)
    if global_scale:
        na = np.linalg.norm(A + rt, axis=1)
        G = np.where(na > 0, np.linalg.norm(X, axis=1) / np.where(na > 0, na, 1.0), 0.0)
    else:
        G = np.ones(n)
    return L_u16, UE4M12.encode(G), L, G


def decode(A, enc_codes, L_u16, G_u16, bits: int, D: int) -> np.ndarray:
    """Reconstruction Ghat (a + Lhat R^T uhat) from stored codes and scales."""
    A = np.asarray(A, dtype=np.float64)
    cb = codebook(bits)
    n = A.shape[0]
    Dp = padded_dim(D, cb.g)
    uhat = cb.C[np.asarray(enc_codes, dtype=np.int64)].reshape(n, Dp)[:, :D]
    R = rotation_matrix(D, rotation_mode(bits, D))
    Lh = UE7M9.decode(L_u16)
    Gh = UE4M12.decode(G_u16)
    return Gh[:, None] * (A + Lh[:, None] * (uhat @ R))


# ------------------------------------------------------------ Rslm4Lite
# Sec. 3.4 (Rslm4Lite paragraph) and Sec. 3.5 (relative quantization): for
# D >= 64 the first 16 rotated coordinates take the K=8 (3-bit) codebook,
# which leaves the top bit of each of their 4-bit codes free; the UE7M9
# local scale is stored in those 16 bits, so the packed row is exactly
# ceil(D/2) bytes.  RelApproxGlobal-Rslm4Lite does the same over the first
# 32 coordinates and stores the UE4M12 global scale in the second 16 bits.

LITE_MIN_D = 64


def lite_head(global_scale: bool) -> int:
    """Leading coordinates on the K=8 codebook: 32 with the global scale, else 16."""
    return 32 if global_scale else 16


def encode_lite(X, A, global_scale: bool = True) -> Encoded:
    """Rslm4Lite encoding of residuals X - A (steps 1-6 of ``encode``).

    The rotation and the EVT scale are those of the 4-bit codec.  Step 3
    quantizes coordinates j < H (H = ``lite_head``) with the K=8 levels and
    the others with the K=16 levels.  After steps 4-6 the scale codes are
    embedded: bit i of the UE7M9 code is the top bit of code i, and with
    the global scale bit i of the UE4M12 code is the top bit of code 16 + i
    (i = 0 .. 15, least significant bit first).  ``codes`` holds the stored
    4-bit values (level index | scale bit << 3).
    """
    X = np.asarray(X, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    n, D = X.shape
    if D < LITE_MIN_D:
        raise ValueError(f"Rslm4Lite needs D >= {LITE_MIN_D}")
    H = lite_head(global_scale)
    cb8, cb16 = codebook(3), codebook(4)
    R = rotation_matrix(D, rotation_mode(4, D))

    r = X - A                                   # step 1
    z = r @ R.T
    m = np.max(np.abs(z), axis=1)
    factor = np.where(m > 0, e_max(D) / np.where(m > 0, m, 1.0), 0.0)
    u = z * factor[:, None]                     # step 2 (g = 1: no padding)

    levels = np.zeros((n, D), dtype=np.int64)   # step 3
    levels[:, :H] = cb8.assign(u[:, :H, None])
    levels[:, H:] = cb16.assign(u[:, H:, None])
    uhat = np.empty((n, D))
    uhat[:, :H] = cb8.C[levels[:, :H], 0]
    uhat[:, H:] = cb16.C[levels[:, H:], 0]

    nr = np.linalg.norm(r, axis=1)              # step 4
    nu = np.linalg.norm(uhat, axis=1)
    L = np.where(nu > 0, nr / np.where(nu > 0, nu, 1.0), 0.0)
    L_u16 = UE7M9.encode(L)
    Lhat = UE7M9.decode(L_u16)
    rt = Lhat[:, None] * (uhat @ R)             # step 5
    if global_scale:                            # step 6
        na = np.linalg.norm(A + rt, axis=1)
        G = np.where(na > 0, np.linalg.norm(X, axis=1) / np.where(na > 0, na, 1.0), 0.0)
    else:
        G = np.ones(n)
    G_u16 = UE4M12.encode(G)
    Ghat = UE4M12.decode(G_u16)
    recon = Ghat[:, None] * (A + rt)

    codes = levels.copy()                       # scale bits into the free top bits
    for i in range(16):
        codes[:, i] |= ((L_u16 >> i) & 1) << 3
        if global_scale:
            codes[:, 16 + i] |= ((G_u16 >> i) & 1) << 3
    return Encoded(4, rotation_mode(4, D), D, 1, codes, L_u16, G_u16, Lhat, Ghat, uhat, u, recon, L, G)


def unpack_lite(codes, global_scale: bool = True):
    """Stored Rslm4Lite codes (n, D) -> (level indices, UE7M9 codes, UE4M12 codes).

    Without the global scale the UE4M12 code is that of 1.0.
    """
    codes = np.asarray(codes, dtype=np.int64)
    H = lite_head(global_scale)
    levels = codes.copy()
    levels[:, :H] &= 7
    L_u16 = np.zeros(codes.shape[0], dtype=np.int64)
    G_u16 = np.zeros(codes.shape[0], dtype=np.int64)
    for i in range(16):
        L_u16 |= ((codes[:, i] >> 3) & 1) << i
        if global_scale:
            G_u16 |= ((codes[:, 16 + i] >> 3) & 1) << i
    if not global_scale:
        G_u16[:] = UE4M12.encode(np.ones(1))[0]
    return levels, L_u16, G_u16


def decode_lite(A, codes, D: int, global_scale: bool = True) -> np.ndarray:
    """Reconstruction Ghat (a + Lhat R^T uhat) from stored Rslm4Lite codes."""
    A = np.asarray(A, dtype=np.float64)
    levels, L_u16, G_u16 = unpack_lite(codes, global_scale)
    H = lite_head(global_scale)
    uhat = np.empty((levels.shape[0], D))
    uhat[:, :H] = codebook(3).C[levels[:, :H], 0]
    uhat[:, H:] = codebook(4).C[levels[:, H:], 0]
    R = rotation_matrix(D, rotation_mode(4, D))
    return UE4M12.decode(G_u16)[:, None] * (A + UE7M9.decode(L_u16)[:, None] * (uhat @ R))


def pack_nibbles(codes: np.ndarray) -> np.ndarray:
    """(n, ngroups) codes < 16 -> (n, ceil(ngroups/2)) uint8, low nibble first."""
    codes = np.asarray(codes, dtype=np.int64)
    n, ng = codes.shape
    nb = (ng + 1) // 2
    out = np.zeros((n, nb), dtype=np.int64)
    for i in range(ng):
        out[:, i // 2] |= codes[:, i] << (4 * (i % 2))
    return out.astype(np.uint8)


def unpack_nibbles(packed: np.ndarray, ngroups: int) -> np.ndarray:
    """Inverse of ``pack_nibbles``."""
    packed = np.asarray(packed, dtype=np.int64)
    out = np.zeros((packed.shape[0], ngroups), dtype=np.int64)
    for i in range(ngroups):
        out[:, i] = (packed[:, i // 2] >> (4 * (i % 2))) & 15
    return out


def pack_bits3(codes: np.ndarray) -> np.ndarray:
    """(n, ngroups) codes < 8 -> (n, ceil(3 ngroups / 8)) uint8: Rslm3's 3-bit
    stream, code i at bits 3i .. 3i + 2 (least significant bit first), byte j
    holding stream bits 8j .. 8j + 7."""
    codes = np.asarray(codes, dtype=np.int64)
    n, ng = codes.shape
    nb = (3 * ng + 7) // 8
    out = np.zeros((n, nb), dtype=np.int64)
    for i in range(ng):
        for t in range(3):
            bit = 3 * i + t
            out[:, bit // 8] |= ((codes[:, i] >> t) & 1) << (bit % 8)
    return out.astype(np.uint8)


def unpack_bits3(packed: np.ndarray, ngroups: int) -> np.ndarray:
    """Inverse of ``pack_bits3``."""
    packed = np.asarray(packed, dtype=np.int64)
    out = np.zeros((packed.shape[0], ngroups), dtype=np.int64)
    for i in range(ngroups):
        for t in range(3):
            bit = 3 * i + t
            out[:, i] |= ((packed[:, bit // 8] >> (bit % 8)) & 1) << t
    return out


def bytes_per_vector(D: int, bits: int, n_scales: int = 1) -> int:
    """Packed size: ceil(D b / 8) code bytes plus 2 bytes per stored scale."""
    return math.ceil(D * bits / 8) + 2 * n_scales


def near_threshold(u: np.ndarray, bits: int, eps: float = 1e-5) -> np.ndarray:
    """Groups whose code is decided within ``eps`` of a decision boundary.

    1-D codebooks: |u - t| < eps for some threshold t.  Multi-D codebooks:
    the gap between the two smallest squared distances is below eps.
    ``u`` is (n, Dp); returns (n, ngroups) bool.
    """
    cb = codebook(bits)
    g = cb.g
    n, Dp = u.shape
    U = u.reshape(n, Dp // g, g)
    if g == 1:
        d = np.abs(U[..., 0][..., None] - cb.thresholds[None, None, :])
        return d.min(axis=-1) < eps
    dist = ((U[..., None, :] - cb.C[None, None, :, :]) ** 2).sum(-1)
    part = np.sort(dist, axis=-1)
    return (part[..., 1] - part[..., 0]) < eps
