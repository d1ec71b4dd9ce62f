"""Seeded synthetic workloads (inputs only; none of the codec arithmetic).

These generators stand in for the paper's datasets (glove D=100, bigann
D=128, openai D=1536, wiki D=3072/384; Sec. 4.2, Table "Overview of
Evaluated Datasets"), which are not available: Gaussian-mixture vectors with
the same dimensionalities and scale of N, optionally unit-normalised (like
the text-embedding sets) or with log-normal norms (non-normalised MIPS).

Every random stream is a numpy PCG64 generator seeded by
``SeedSequence(seed, spawn_key=(stream, chunk))`` so that any chunk of rows
can be regenerated on its own.  Streams: 0 mixture centers, 1 component ids,
2 noise, 3 norms (database rows); 5, 6, 7 the same for queries.

Recipe of a row: component k ~ uniform{0..P-1}; y = center_k + sigma * eps,
eps ~ N(0, I); then y / ||y|| when ``normalize``; rho * y / ||y|| with
rho ~ LogNormal(0, lognormal_sigma) when ``lognormal_sigma`` is set.  The
IVF assignment of a row is its generating component.  Centroids are either
the true centers or the member means of the generated rows.
"""

from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

CHUNK = 1 << 16  # rows per independently seeded chunk


@dataclass(frozen=True)
class Workload:
    name: str
    N: int
    D: int
    P: int                    # mixture components = IVF partitions
    sigma: float
    normalize: bool
    lognormal_sigma: float | None
    centroids: str            # 'true' or 'mean'
    nq: int
    bits: int
    rescore_bits: int
    nprobe: int
    k: int                    # stage-1 top-K
    k_final: int              # final top-k (== k without rescoring)
    seed: int = 0
    description: str = ""

    def scaled(self, **kw) -> "Workload":
        """A copy with some fields replaced (smaller parity cases)."""
        return replace(self, **kw)


WORKLOADS = {
    "C1": Workload("C1", 10_000, 128, 16, 0.3, False, None, "true", 100, 4, 0, 4, 10, 10,
                   description="N=1e4 d=128 16-Gaussian mixture sigma=0.3, IVF16 true centers, "
                               "4-bit codes, 100 queries, nprobe=4, top-10"),
    "C2": Workload("C2", 1_000_000, 96, 1024, 0.5, False, None, "true", 10_000, 2, 4, 32, 100, 10,
                   description="N=1e6 d=96 1024-Gaussian mixture sigma=0.5, IVF1024 true centers, "
                               "2-bit scoring + 4-bit rescoring, 1e4 queries, nprobe=32, "
                               "top-100 -> top-10"),
    "C3": Workload("C3", 1_000_000, 768, 2048, 0.5, True, None, "mean", 10_000, 1, 4, 64, 100, 10,
                   description="N=1e6 d=768 unit-normalised 2048-Gaussian mixture, IVF2048 "
                               "member means, 1-bit scoring + 4-bit rescoring, 1e4 queries, "
                               "nprobe=64, top-100 -> top-10"),
    "C4": Workload("C4", 10_000_000, 128, 8192, 0.5, False, 0.5, "mean", 100_000, 4, 0, 64, 10, 10,
                   description="N=1e7 d=128 8192-Gaussian mixture with log-normal(0, 0.5) norms, "
                               "IVF8192 member means, 4-bit codes, 1e5 queries, nprobe=64, top-10"),
    "C5": Workload("C5", 5_000_000, 1536, 4096, 0.5, True, None, "mean", 50_000, 2, 4, 128, 200, 10,
                   description="N=5e6 d=1536 unit-normalised 4096-Gaussian mixture, IVF4096 member "
                               "means, 2-bit scoring + 4-bit rescoring, 5e4 queries, nprobe=128, "
                               "top-200 -> top-10"),
}


def _rng(seed: int, stream: int, chunk: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed, spawn_key=(stream, chunk))))


def centers(w: Workload) -> np.ndarray:
    """Mixture centers, P x D float32, ~ N(0, I)."""
    return _rng(w.seed, 0).standard_normal((w.P, w.D), dtype=np.float32)


def _rows(w: Workload, ctr: np.ndarray, n: int, base: int, chunk: int, out: np.ndarray | None = None):
    comp = _rng(w.seed, base + 1, chunk).integers(0, w.P, size=n, dtype=np.int64)
    y = out if out is not None else np.empty((n, w.D), dtype=np.float32)
    _rng(w.seed, base + 2, chunk).standard_normal((n, w.D), dtype=np.float32, out=y)
    rho = None
    if w.lognormal_sigma is not None:
        rho = _rng(w.seed, base + 3, chunk).lognormal(0.0, w.lognormal_sigma, size=n)
    step = max(1, (1 << 18) // w.D)  # small temporaries: about 1 MB per sub-block
    for lo in range(0, n, step):
        yb = y[lo:lo + step]
        yb *= np.float32(w.sigma)
        yb += ctr[comp[lo:lo + step]]
        if w.normalize or rho is not None:
            nrm = np.sqrt(np.einsum("ij,ij->i", yb, yb, dtype=np.float64))
            scale = 1.0 / np.where(nrm > 0, nrm, 1.0)
            if rho is not None:
                scale = scale * rho[lo:lo + step]
            yb *= scale.astype(np.float32)[:, None]
    return y, comp.astype(np.int32)


def workers() -> int:
    try:
        n = len(os.sched_getaffinity(0))
    except AttributeError:
        n = os.cpu_count() or 1
    return max(1, min(16, n))


def chunk_rows(w: Workload, chunk: int, ctr: np.ndarray | None = None):
    """Rows [chunk*CHUNK, min(N, (chunk+1)*CHUNK)) and their components."""
    ctr = centers(w) if ctr is None else ctr
    lo = chunk * CHUNK
    n = max(0, min(w.N, lo + CHUNK) - lo)
    return _rows(w, ctr, n, 0, chunk)


def n_chunks(w: Workload) -> int:
    return math.ceil(w.N / CHUNK)


def rows(w: Workload, ids, ctr: np.ndarray | None = None):
    """Rows with the given ids (regenerating only the chunks they live in, in threads)."""
    ids = np.asarray(ids, dtype=np.int64)
    ctr = centers(w) if ctr is None else ctr
    X = np.zeros((ids.size, w.D), dtype=np.float32)
    A = np.zeros(ids.size, dtype=np.int32)

    def one(c):
        sel = np.nonzero(ids // CHUNK == c)[0]
        Xc, Ac = chunk_rows(w, int(c), ctr)
        X[sel] = Xc[ids[sel] - c * CHUNK]
        A[sel] = Ac[ids[sel] - c * CHUNK]

    with ThreadPoolExecutor(workers()) as ex:
        list(ex.map(one, np.unique(ids // CHUNK).tolist()))
    return X, A


def row_blocks(w: Workload, block: int, ctr: np.ndarray | None = None):
    """Yield (first row, rows) for consecutive blocks of `block` rows (a
    multiple of the generation chunk), each generated in threads."""
    assert block % CHUNK == 0
    ctr = centers(w) if ctr is None else ctr
    per = block // CHUNK
    with ThreadPoolExecutor(workers()) as ex:
        for c0 in range(0, n_chunks(w), per):
            parts = list(ex.map(lambda c: chunk_rows(w, c, ctr)[0], range(c0, min(n_chunks(w), c0 + per))))
            yield c0 * CHUNK, np.concatenate(parts)


def database(w: Workload):
    """All N rows (float32) and their components (int32), chunks generated in threads."""
    ctr = centers(w)
    X = np.empty((w.N, w.D), dtype=np.float32)
    A = np.empty(w.N, dtype=np.int32)

    def one(c):
        lo = c * CHUNK
        n = min(w.N, lo + CHUNK) - lo
        _, a = _rows(w, ctr, n, 0, c, out=X[lo:lo + n])
        A[lo:lo + n] = a

    with ThreadPoolExecutor(workers()) as ex:
        list(ex.map(one, range(n_chunks(w))))
    return X, A


def member_means(w: Workload, X: np.ndarray, A: np.ndarray, ctr: np.ndarray) -> np.ndarray:
    """Per-component mean of the rows (float32); empty components keep the center.

    Each row block of 2^16 is summed by a sparse one-hot product (float32,
    about 8 rows per partition); block sums are added in float64 in block
    order so the result does not depend on thread scheduling.
    """
    from scipy import sparse
    cnt = np.bincount(A, minlength=w.P)
    block = 1 << 16
    bounds = list(range(0, X.shape[0], block)) + [X.shape[0]]

    def part(i):
        lo, hi = bounds[i], bounds[i + 1]
        m = sparse.csr_matrix((np.ones(hi - lo, dtype=np.float32), (A[lo:hi], np.arange(hi - lo))),
                              shape=(w.P, hi - lo))
        return m @ X[lo:hi]

    sums = np.zeros((w.P, w.D))
    with ThreadPoolExecutor(workers()) as ex:
        for p in ex.map(part, range(len(bounds) - 1)):
            sums += p
    out = ctr.astype(np.float64).copy()
    nz = cnt > 0
    out[nz] = sums[nz] / cnt[nz, None]
    return out.astype(np.float32)


def assignment(w: Workload) -> np.ndarray:
    """Component (= IVF partition) of every row, without generating the rows."""
    A = np.empty(w.N, dtype=np.int32)
    for c in range(n_chunks(w)):
        lo = c * CHUNK
        n = min(w.N, lo + CHUNK) - lo
        A[lo:lo + n] = _rng(w.seed, 1, c).integers(0, w.P, size=n, dtype=np.int64)
    return A


def member_means_streamed(w: Workload, ctr: np.ndarray | None = None) -> np.ndarray:
    """``member_means`` computed chunk by chunk (same blocks, same order, same
    result) without holding the N x D database in memory."""
    from scipy import sparse
    ctr = centers(w) if ctr is None else ctr

    def part(c):
        X, A = chunk_rows(w, c, ctr)
        m = sparse.csr_matrix((np.ones(A.size, dtype=np.float32), (A, np.arange(A.size))),
                              shape=(w.P, A.size))
        return m @ X, np.bincount(A, minlength=w.P)

    sums = np.zeros((w.P, w.D))
    cnt = np.zeros(w.P, dtype=np.int64)
    with ThreadPoolExecutor(workers()) as ex:
        for ps, pc in ex.map(part, range(n_chunks(w))):
            sums += ps
            cnt += pc
    out = ctr.astype(np.float64).copy()
    nz = cnt > 0
    out[nz] = sums[nz] / cnt[nz, None]
    return out.astype(np.float32)


def ivf_centroids(w: Workload, X: np.ndarray | None = None, A: np.ndarray | None = None) -> np.ndarray:
    """IVF centroids: the true centers, or the member means of the data."""
    ctr = centers(w)
    if w.centroids == "true":
        return ctr
    if X is None:
        return member_means_streamed(w, ctr)
    return member_means(w, X, A, ctr)


def queries(w: Workload, nq: int | None = None) -> np.ndarray:
    """The first ``nq`` (default all) queries, drawn from the same mixture."""
    nq = w.nq if nq is None else nq
    ctr = centers(w)
    out = np.empty((nq, w.D), dtype=np.float32)
    for c in range(math.ceil(nq / CHUNK)):
        lo = c * CHUNK
        n = min(nq, lo + CHUNK) - lo
        out[lo:lo + n] = _rows(w, ctr, n, 4, c)[0]
    return out
