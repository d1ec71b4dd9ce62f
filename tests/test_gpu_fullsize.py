"""GPU path vs the float64 oracle at the full sizes of workloads C2-C5, on
sampled outputs (C1 runs in full in test_gpu_parity).

Each index is built the way bench.py builds it (true-center or member-mean
centroids, rows encoded in 2^20-row calls) and searched with the whole query
batch in one call, the launch configuration bench.py times (C3 also at its
batches of 1, 64 and 1024 queries).  Checked, with the tolerances of
test_gpu_parity:

* encode parity of row blocks spread over the database (the first rows, a
  middle block, the ragged end), both stages;
* the probe lists of sampled queries against exact float64 <q, c_p>;
* the results of sampled queries against the oracle's scores computed from
  the GPU's exported codes (sample-verified by the encode check): the
  stage-1 score of every candidate of the probed partitions
  (Sec. 3.5: G (<q, c> + L <R q, uhat>)), the stage-2 rescoring of the
  survivors, and the top-k rule of lib_util.check_topk.
"""

import math

import numpy as np
import pytest

from oracle import codec, constants as K
from oracle.rotation import rotation_matrix, rotation_mode
from paper_2608_30384_gb300 import workloads as W
from tests.gpu_cases import check_stage
from tests.lib_util import check_topk, ensure_library, kth_of, score_tol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ENCODE_ROWS = 1 << 20   # rows per rslm_encode call, as in bench.py
BLOCK = 384             # rows per encode-parity block
N_SAMPLED = {"C2": 16, "C3": 6, "C4": 16, "C5": 4}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_library()


def _unpack(packed: np.ndarray, ngroups: int) -> np.ndarray:
    """Canonical nibble rows -> (n, ngroups) uint8 codes (even group = low nibble)."""
    out = np.empty((packed.shape[0], 2 * packed.shape[1]), dtype=np.uint8)
    out[:, 0::2] = packed & 15
    out[:, 1::2] = packed >> 4
    return out[:, :ngroups]


class Codes:
    """Exported codes and scales of the rows of a set of partitions."""

    def __init__(self, rows, packed, L, G):
        self.rows = rows            # original row ids, ascending
        self.packed = packed
        self.L = K.UE7M9.decode(L.astype(np.int64))
        self.G = K.UE4M12.decode(G.astype(np.int64))

    def dots(self, qrot_padded, bits, sel):
        """<R q, uhat> of rows sel through per-group codeword tables."""
        cb = K.codebook(bits)
        ng = qrot_padded.size // cb.g
        lut = qrot_padded.reshape(ng, cb.g) @ cb.C.T      # (ngroups, 16)
        out = np.empty(sel.size)
        for lo in range(0, sel.size, 1 << 15):
            s = sel[lo:lo + (1 << 15)]
            codes = _unpack(self.packed[s], ng)
            out[lo:lo + s.size] = lut[np.arange(ng)[None, :], codes].sum(1)
        return out


class Full:
    """A full-size workload: GPU index, sampled rows and host-side references."""

    def __init__(self, name: str):
        from paper_2608_30384_gb300 import Index
        w = self.w = W.WORKLOADS[name]
        ctr = W.centers(w)
        self.C = W.ivf_centroids(w) if w.centroids == "mean" else ctr
        self.A = W.assignment(w)
        self.Q = W.queries(w)
        self.ix = Index(torch.from_numpy(self.C).cuda(), w.bits, w.rescore_bits)
        self.ix.reserve(torch.from_numpy(self.A).cuda())
        mid = (w.N // 2) // BLOCK * BLOCK
        self.blocks = [0, mid, w.N - BLOCK]          # the last block ends at the ragged end
        self.Xb = {b: np.zeros((BLOCK, w.D), dtype=np.float32) for b in self.blocks}
        self.xnorm = np.empty(w.N)  # ||x|| of every row (the score tolerance's floor)
        nch = W.n_chunks(w)
        per = ENCODE_ROWS // W.CHUNK
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(W.workers()) as ex:
            for c0 in range(0, nch, per):
                parts = list(ex.map(lambda c: W.chunk_rows(w, c, ctr)[0], range(c0, min(nch, c0 + per))))
                X = np.concatenate(parts)
                del parts
                lo, hi = c0 * W.CHUNK, c0 * W.CHUNK + X.shape[0]
                self.xnorm[lo:hi] = np.sqrt(np.einsum("ij,ij->i", X, X, dtype=np.float64))
                for b in self.blocks:
                    a0, a1 = max(lo, b), min(hi, b + BLOCK)
                    if a0 < a1:
                        self.Xb[b][a0 - b:a1 - b] = X[a0 - lo:a1 - lo]
                self.ix.encode(torch.from_numpy(X).cuda(), lo)
                del X
        self.ix.sync()
        self._rot = {}

    def rot(self, bits):
        if bits not in self._rot:
            self._rot[bits] = rotation_matrix(self.w.D, rotation_mode(bits, self.w.D))
        return self._rot[bits]

    def qrot(self, q, bits):
        g = K.group_size(bits)
        out = np.zeros(g * math.ceil(self.w.D / g))
        out[:self.w.D] = self.rot(bits) @ q.astype(np.float64)
        return out

    def export(self, which, parts):
        """Codes of the rows of the given partitions, exported in 2^20-row calls."""
        want = np.isin(self.A, np.asarray(sorted(parts)))
        rows, pk, Ls, Gs = [], [], [], []
        for lo in range(0, self.w.N, ENCODE_ROWS):
            n = min(self.w.N, lo + ENCODE_ROWS) - lo
            m = want[lo:lo + n]
            if not m.any():
                continue
            c, L, G = (t.cpu().numpy() for t in self.ix.export_codes(which, lo, n))
            rows.append(np.nonzero(m)[0] + lo)
            pk.append(c[m])
            Ls.append(L[m])
            Gs.append(G[m])
        return Codes(np.concatenate(rows), np.concatenate(pk), np.concatenate(Ls), np.concatenate(Gs))


def _encode_blocks(F: Full):
    w = F.w
    for b in F.blocks:
        X = F.Xb[b]
        A1 = F.C[F.A[b:b + BLOCK]].astype(np.float64)
        st1 = codec.encode(X, A1, w.bits)
        c1, L1, G1 = (t.cpu().numpy() for t in F.ix.export_codes(1, b, BLOCK))
        ok = check_stage(c1, L1, G1, st1, X, A1, w.bits, True, f"block {b} stage 1")
        if w.rescore_bits:
            sel = np.nonzero(ok)[0]
            st2 = codec.encode(X[sel], st1.recon[sel], w.rescore_bits)
            c2, L2, G2 = (t.cpu().numpy() for t in F.ix.export_codes(2, b, BLOCK))
            check_stage(c2[sel], L2[sel], G2[sel], st2, X[sel], st1.recon[sel], w.rescore_bits, True,
                        f"block {b} stage 2")


def _search_check(F: Full, nq: int, sampled):
    """Search the first nq queries in one call; check the sampled ones."""
    w = F.w
    Qt = torch.from_numpy(F.Q[:nq]).cuda()
    ids, sc = F.ix.search(Qt, w.nprobe, w.k, k_final=w.k_final)
    gp, gcs = F.ix.probe(Qt, w.nprobe)  # same call shape as the search's own probe step
    F.ix.sync()
    ids, sc, gp, gcs = ids.cpu().numpy(), sc.cpu().numpy(), gp.cpu().numpy(), gcs.cpu().numpy()
    parts = set(gp[sampled].reshape(-1).tolist())
    s1c = F.export(1, parts)
    s2c = F.export(2, parts) if w.rescore_bits else None
    cmax = np.linalg.norm(F.C.astype(np.float64), axis=1).max()
    for i in sampled:
        q = F.Q[i].astype(np.float64)
        qn = float(np.linalg.norm(q))
        cs = F.C.astype(np.float64) @ q
        # probe: the nprobe largest <q, c_p> up to near-ties
        kth_p = np.sort(cs)[::-1][w.nprobe - 1]
        probs = check_topk(gp[i], gcs[i], lambda j: cs[j], kth_p, lambda s, j=None: 1e-5 * qn * cmax)
        assert not probs, (i, "probe", probs[:3])
        # stage 1 over every candidate of the GPU's probe lists
        sel = np.nonzero(np.isin(F.A[s1c.rows], gp[i]))[0]
        cand = s1c.rows[sel]
        s1 = s1c.G[sel] * (cs[F.A[cand]] + s1c.L[sel] * s1c.dots(F.qrot(q, w.bits), w.bits, sel))
        tol = lambda s, j=None: float(score_tol(s, qn, F.xnorm[j] if j is not None else F.xnorm.max()))  # noqa: E731
        order = np.lexsort((cand, -s1))
        if not w.rescore_bits:
            ref = dict(zip(cand.tolist(), s1.tolist()))
            kth = s1[order[w.k - 1]] if cand.size >= w.k else -np.inf
            kid = int(cand[order[w.k - 1]]) if cand.size >= w.k else None
        else:
            # stage 2 (reading B): G2 (s1 + L2 <R2 q, uhat2>) of the oracle's
            # survivors and of every id the GPU returned
            surv = order[:w.k]
            extra = np.nonzero(np.isin(cand, ids[i][ids[i] >= 0]))[0]
            need = np.union1d(surv, extra)
            pos2 = np.searchsorted(s2c.rows, cand[need])
            s2 = s2c.G[pos2] * (s1[need] + s2c.L[pos2] * s2c.dots(F.qrot(q, w.rescore_bits),
                                                                 w.rescore_bits, pos2))
            ref = dict(zip(cand[need].tolist(), s2.tolist()))
            kth, kid = kth_of({c: ref[c] for c in cand[surv].tolist()}, w.k_final)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, tol, allowed_ids=ref, kth_id=kid)
        assert not probs, (i, "results", probs[:3])
        assert (ids[i] >= 0).sum() == min(w.k_final, cand.size)


def _sampled(n_total: int, n: int):
    return np.unique(np.linspace(0, n_total - 1, n).astype(np.int64))


@pytest.mark.parametrize("name", ["C2", "C3", "C4", "C5"])
def test_fullsize(name):
    F = Full(name)
    try:
        _encode_blocks(F)
        w = F.w
        batches = [1, 64, 1024, w.nq] if name == "C3" else [w.nq]
        for nq in batches:
            _search_check(F, nq, _sampled(nq, min(nq, N_SAMPLED[name])))
    finally:
        del F.ix
        torch.cuda.empty_cache()
