"""Static tables and scalar formats of the RSLM codec (float64 oracle).

Test infrastructure only: see ``oracle/__init__.py``.

Readings of the paper taken here, where it leaves a value or a rule open:

* Sec. 3.1.2 fixes a 256-entry pseudo-random sign table S1 and a 128-entry
  permutation P but does not print them.  They are drawn here from the
  SplitMix64 generator (Steele, Lea, Flood 2014; counter form: output n is
  mix(seed + (n+1)*0x9E3779B97F4A7C15)) with seed 0x52534C4D ("RSLM"):
  outputs 0..255 give S1 (top bit set -> -1), outputs 256..382 drive a
  Fisher-Yates shuffle of 0..127 (step t swaps P[127-t] with
  P[out mod (128-t)]).
* "S2 is S1 offset by 127 elements" (Sec. 3.1.3, step 4) is read as
  S2[i] = S1[(i + 127) mod 256].  Coordinate i uses S[i mod 256].
* The 1-D codebooks (b=4: K=16, b=3: K=8) are the exact Gaussian Lloyd-Max
  quantizers, the limit of the k-means-on-samples recipe of Sec. 3.2, found
  by the Lloyd fixed point on the exact N(0,1) density.
* The 2-D (b=2) and 4-D (b=1) K=16 codebooks follow the recipe of Sec. 3.2
  (k-means on synthetic N(0, I) samples) with a fixed, fully specified
  procedure, see ``multid_codebook``.
* All codebook components are rounded to the nearest IEEE binary16 value so
  that a decoded code is an exact f16 tensor-core operand; 1-D decision
  thresholds are midpoints of the rounded levels.
* E_max(D) (Sec. 3.2) is the exact expectation of max_i |Z_i| over D iid
  N(0,1): integral_0^inf (1 - erf(t/sqrt 2)^D) dt.
* UE7M9 / UE4M12 (Sec. 3.3.1, Sec. 3.5.2): unsigned, e exponent bits and m
  mantissa bits, bias 2^(e-1)-1 (63 and 7), code 0 means 0, no subnormals,
  round-to-nearest-even on the mantissa, values below the smallest normal
  flush to 0, values above the largest saturate.
"""

from __future__ import annotations

import functools
import json
import math
import os

import numpy as np
from scipy import integrate, special

SEED = 0x52534C4D  # "RSLM"
_GAMMA = 0x9E3779B97F4A7C15
_MASK64 = (1 << 64) - 1


# ---------------------------------------------------------------- SplitMix64
def splitmix64(seed: int, start: int, count: int) -> np.ndarray:
    """Outputs start .. start+count-1 of SplitMix64 seeded with ``seed``.

    Counter form of the published generator: state_n = seed + (n+1)*gamma
    (mod 2^64), output = mix(state_n) with the two xor-shift-multiply rounds
    (30, 0xBF58476D1CE4E5B9), (27, 0x94D049BB133111EB) and a final xor-shift
    by 31.
    """
    n = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed & _MASK64) + n * np.uint64(_GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        z = z ^ (z >> np.uint64(31))
    return z


# ----------------------------------------------------- sign flips, permutation
@functools.lru_cache(maxsize=None)
def sign_table_s1() -> np.ndarray:
    """S1: 256 static pseudo-random signs (Sec. 3.1.2, first bullet)."""
    out = splitmix64(SEED, 0, 256)
    return np.where((out >> np.uint64(63)) == 1, -1.0, 1.0)


@functools.lru_cache(maxsize=None)
def sign_table_s2() -> np.ndarray:
    """S2: S1 offset by 127 elements (Sec. 3.1.3, step 4)."""
    s1 = sign_table_s1()
    return np.array([s1[(i + 127) % 256] for i in range(256)])


def tiled_signs(table: np.ndarray, D: int) -> np.ndarray:
    """The 256-entry table tiled across D coordinates (Sec. 3.1.2)."""
    return np.array([table[i % 256] for i in range(D)])


@functools.lru_cache(maxsize=None)
def perm_p128() -> tuple:
    """P: static 128-element permutation (Sec. 3.1.2, second bullet)."""
    out = splitmix64(SEED, 256, 127)
    p = list(range(128))
    for t in range(127):
        i = 127 - t
        j = int(out[t] % np.uint64(i + 1))
        p[i], p[j] = p[j], p[i]
    return tuple(p)


def bit_reversal(B: int) -> tuple:
    """Bit-reversal permutation of 0..B-1 on log2(B) bits (Sec. 3.1.2)."""
    bits = B.bit_length() - 1
    out = []
    for k in range(B):
        r = 0
        for b in range(bits):
            if k >> b & 1:
                r |= 1 << (bits - 1 - b)
        out.append(r)
    return tuple(out)


def block_permutation(B: int) -> tuple:
    """In-block permutation: P for B = 128, bit reversal for B < 128."""
    return perm_p128() if B == 128 else bit_reversal(B)


# ----------------------------------------------------------- Lloyd-Max (1-D)
def _gauss_pdf(t):
    return np.exp(-0.5 * t * t) / math.sqrt(2.0 * math.pi)


def _gauss_cdf(t):
    return 0.5 * special.erfc(-t / math.sqrt(2.0))


@functools.lru_cache(maxsize=None)
def lloyd_max_gaussian(K: int) -> tuple:
    """Exact K-level Lloyd-Max quantizer of N(0, 1) (Sec. 3.2), float64.

    Alternates the two optimality conditions: thresholds are midpoints of
    adjacent levels, each level is the conditional mean of its cell,
    E[Z | a < Z < b] = (pdf(a) - pdf(b)) / (cdf(b) - cdf(a)), until no level
    moves by more than 1e-15.
    """
    lv = np.linspace(-2.5, 2.5, K)
    for _ in range(200000):
        t = np.concatenate([[-np.inf], 0.5 * (lv[1:] + lv[:-1]), [np.inf]])
        pdf = _gauss_pdf(t)
        cdf = _gauss_cdf(t)
        new = (pdf[:-1] - pdf[1:]) / (cdf[1:] - cdf[:-1])
        done = np.max(np.abs(new - lv)) < 1e-15
        lv = new
        if done:
            break
    return tuple(float(v) for v in lv)


def round_to_f16(v) -> np.ndarray:
    """Nearest IEEE binary16 value (round half to even), as float64."""
    return np.asarray(v, dtype=np.float64).astype(np.float16).astype(np.float64)


# ------------------------------------------------- multi-dimensional codebooks
_MULTID_FILE = os.path.join(os.path.dirname(__file__), "data", "codebooks_multid.json")

# Recipe of the 2-D / 4-D k-means codebooks (Sec. 3.2: k-means with K
# clusters on a large set of synthetic N(0, I) samples).
MULTID_SAMPLES = 1 << 17
MULTID_RESTARTS = 8
MULTID_MAX_ITERS = 400
MULTID_GRID = 2.0 ** -20


def multid_samples(g: int) -> np.ndarray:
    """MULTID_SAMPLES x g standard-normal samples for the g-D codebook.

    Box-Muller on SplitMix64 (seed SEED + 1000 + g): pair i uses outputs 2i
    and 2i+1 as u = ((out >> 11) + 0.5) * 2^-53, giving
    sqrt(-2 ln u1) * (cos(2 pi u2), sin(2 pi u2)).  Gaussians fill the rows
    in order and are rounded to the 2^-20 grid so that cluster sums are
    exact in float64 whatever the summation order.
    """
    n = MULTID_SAMPLES * g
    out = splitmix64(SEED + 1000 + g, 0, n)
    u = ((out >> np.uint64(11)).astype(np.float64) + 0.5) * 2.0 ** -53
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    th = 2.0 * math.pi * u2
    z = np.empty(n)
    z[0::2] = r * np.cos(th)
    z[1::2] = r * np.sin(th)
    z = np.round(z / MULTID_GRID) * MULTID_GRID
    return z.reshape(MULTID_SAMPLES, g)


def _sq_dist(X: np.ndarray, c: np.ndarray) -> np.ndarray:
    """sum_j (x_j - c_j)^2 accumulated in coordinate order j = 0, 1, ..."""
    d = (X[:, 0] - c[0]) ** 2
    for j in range(1, X.shape[1]):
        d = d + (X[:, j] - c[j]) ** 2
    return d


def _kmeans_pp_init(X: np.ndarray, K: int, seed: int) -> np.ndarray:
    """k-means++ seeding (Arthur & Vassilvitskii 2007).

    Uniforms u_k = (out_k >> 11) * 2^-53 from SplitMix64(seed).  First center
    = sample floor(u_0 * n); center k = first sample whose running sum of
    squared distances to the chosen centers exceeds u_k * total.
    """
    n = X.shape[0]
    out = splitmix64(seed, 0, K)
    u = (out >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
    idx = [int(u[0] * n)]
    d = _sq_dist(X, X[idx[0]])
    for k in range(1, K):
        cum = np.cumsum(d)
        j = int(np.searchsorted(cum, u[k] * cum[-1], side="right"))
        j = min(j, n - 1)
        idx.append(j)
        d = np.minimum(d, _sq_dist(X, X[j]))
    return X[idx].copy()


def _assign(X: np.ndarray, C: np.ndarray):
    """Nearest center of every sample (ties: lowest index) and its distance."""
    best = _sq_dist(X, C[0])
    arg = np.zeros(X.shape[0], dtype=np.int64)
    for k in range(1, C.shape[0]):
        d = _sq_dist(X, C[k])
        better = d < best
        best = np.where(better, d, best)
        arg = np.where(better, k, arg)
    return arg, best


def kmeans_lloyd(X: np.ndarray, C0: np.ndarray, max_iters: int):
    """Lloyd's k-means: assign, re-center, stop when assignments repeat.

    An empty cluster keeps its previous center.  Returns (centers, mse per
    coordinate, iterations).
    """
    C = C0.copy()
    K = C.shape[0]
    prev = None
    for it in range(max_iters):
        arg, _ = _assign(X, C)
        if prev is not None and np.array_equal(arg, prev):
            break
        prev = arg
        for k in range(K):
            m = arg == k
            cnt = int(m.sum())
            if cnt:
                C[k] = X[m].sum(axis=0) / cnt
    _, best = _assign(X, C)
    mse = float(np.cumsum(best)[-1]) / X.size
    return C, mse, it


def generate_multid_codebook(g: int) -> dict:
    """Run the full 2-D / 4-D codebook recipe (slow: about a minute).

    MULTID_RESTARTS k-means++ restarts (seed SEED + 2000 + 100 g + r), each
    refined by Lloyd iterations; the restart with the lowest distortion wins
    (first on ties); its codewords are sorted lexicographically and rounded
    to binary16.
    """
    X = multid_samples(g)
    best = None
    for r in range(MULTID_RESTARTS):
        C0 = _kmeans_pp_init(X, 16, SEED + 2000 + 100 * g + r)
        C, mse, iters = kmeans_lloyd(X, C0, MULTID_MAX_ITERS)
        if best is None or mse < best[1]:
            best = (C, mse, r, iters)
    C = best[0]
    order = np.lexsort(tuple(C[:, j] for j in reversed(range(g))))
    C = C[order]
    return {
        "g": g,
        "K": 16,
        "float64": C.tolist(),
        "f16": round_to_f16(C).tolist(),
        "mse_per_dim_samples": best[1],
        "restart": best[2],
        "iterations": best[3],
    }


@functools.lru_cache(maxsize=None)
def multid_codebook(g: int) -> np.ndarray:
    """Stored 16 x g codebook (binary16-rounded, lexicographic order).

    Written by ``oracle/gen_codebooks.py``, which calls only this module.
    """
    with open(_MULTID_FILE) as f:
        data = json.load(f)
    return np.array(data[str(g)]["f16"], dtype=np.float64)


# ------------------------------------------------------------------ codebooks
class Codebook:
    """A K-entry, g-dimensional codebook (Sec. 3.2, Table of codecs).

    ``C`` is K x g (float64 values).  For g == 1, ``thresholds`` are the K-1
    decision thresholds (midpoints of adjacent levels); a value u maps to
    the number of thresholds <= u (u exactly on a threshold goes up).
    For g > 1 a group maps to the nearest codeword, ties to the lowest index.
    """

    def __init__(self, C: np.ndarray, name: str):
        self.C = np.asarray(C, dtype=np.float64)
        self.K, self.g = self.C.shape
        self.name = name
        if self.g == 1:
            lv = self.C[:, 0]
            assert np.all(np.diff(lv) > 0)
            self.thresholds = 0.5 * (lv[1:] + lv[:-1])
        else:
            self.thresholds = None

    def assign(self, U: np.ndarray) -> np.ndarray:
        """Codes of groups U (..., g) -> (...,) int64."""
        if self.g == 1:
            return np.searchsorted(self.thresholds, U[..., 0], side="right").astype(np.int64)
        flat = U.reshape(-1, self.g)
        arg, _ = _assign(flat, self.C)
        return arg.reshape(U.shape[:-1])


@functools.lru_cache(maxsize=None)
def codebook(bits: int) -> Codebook:
    """The RSLM codebook for ``bits`` per dimension (Sec. 3.2).

    b=1: 4-D, K=16; b=2: 2-D, K=16; b=3: 1-D, K=8; b=4: 1-D, K=16.
    """
    if bits == 4:
        return Codebook(round_to_f16(lloyd_max_gaussian(16))[:, None], "1D-K16")
    if bits == 3:
        return Codebook(round_to_f16(lloyd_max_gaussian(8))[:, None], "1D-K8")
    if bits == 2:
        return Codebook(multid_codebook(2), "2D-K16")
    if bits == 1:
        return Codebook(multid_codebook(4), "4D-K16")
    raise ValueError(f"unsupported bits {bits}")


def group_size(bits: int) -> int:
    """Coordinates per code: 4 for b=1, 2 for b=2, 1 for b=3 and b=4."""
    return {1: 4, 2: 2, 3: 1, 4: 1}[bits]


def highres_codebook(bits: int) -> Codebook:
    """A 1-D, 2^bits-level Gaussian quantizer at high resolution (test use).

    For large K the Lloyd fixed point converges too slowly; the
    asymptotically optimal (Panter-Dite) point density proportional to
    pdf^(1/3), i.e. levels at the N(0, 3) quantiles (i + 1/2)/K, stands in.
    Used only to check that the search reduces to exact MIPS as the
    quantization error vanishes.
    """
    K = 1 << bits
    p = (np.arange(K) + 0.5) / K
    lv = math.sqrt(3.0) * math.sqrt(2.0) * special.erfinv(2.0 * p - 1.0)
    return Codebook(lv[:, None], f"1D-K{K}-highres")


# ------------------------------------------------------------------- E_max(D)
@functools.lru_cache(maxsize=None)
def e_max(D: int) -> float:
    """E[max_i |Z_i|], Z ~ N(0, I_D): integral of 1 - erf(t/sqrt2)^D."""
    # 1 - erf^D written as -expm1(D log1p(-erfc)) to keep the tail accurate;
    # beyond t = 40 the integrand is below 1e-300.
    f = lambda t: -math.expm1(D * math.log1p(-special.erfc(t / math.sqrt(2.0))))  # noqa: E731
    val, _ = integrate.quad(f, 0.0, 40.0, epsabs=1e-13, epsrel=1e-13, limit=1000)
    return float(val)


# -------------------------------------------------------------- scale formats
class UEFormat:
    """Unsigned float with ``ebits`` exponent and ``mbits`` mantissa bits.

    Value of code u = (e << mbits) | m: 0 if e == 0, else
    2^(e - bias) * (1 + m / 2^mbits); bias = 2^(ebits-1) - 1.
    """

    def __init__(self, ebits: int, mbits: int):
        self.ebits, self.mbits = ebits, mbits
        self.bias = (1 << (ebits - 1)) - 1
        self.emax = (1 << ebits) - 1

    def decode(self, u) -> np.ndarray:
        u = np.asarray(u, dtype=np.int64)
        e = u >> self.mbits
        m = u & ((1 << self.mbits) - 1)
        val = np.ldexp(1.0 + m / float(1 << self.mbits), (e - self.bias).astype(np.int32))
        return np.where(e == 0, 0.0, val)

    def encode_one(self, v: float) -> int:
        v = float(v)
        if not v > 0.0:
            return 0
        f, k = math.frexp(v)  # v = f * 2^k, f in [0.5, 1)
        e = k - 1
        frac = 2.0 * f - 1.0  # in [0, 1), exact
        m = round(frac * (1 << self.mbits))  # Python round: half to even
        if m == (1 << self.mbits):
            m = 0
            e += 1
        be = e + self.bias
        if be <= 0:
            return 0
        if be > self.emax:
            return (self.emax << self.mbits) | ((1 << self.mbits) - 1)
        return (be << self.mbits) | m

    def encode(self, v) -> np.ndarray:
        v = np.asarray(v, dtype=np.float64)
        return np.array([self.encode_one(x) for x in v.reshape(-1)], dtype=np.int64).reshape(v.shape)


UE7M9 = UEFormat(7, 9)
UE4M12 = UEFormat(4, 12)
