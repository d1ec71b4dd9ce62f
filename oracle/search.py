"""IVF probe, brute-force scoring and rescoring in float64.

Test infrastructure only: see ``oracle/__init__.py``.

Follows the end-to-end pipeline of Sec. 5.5.1 (partitioning, residual
quantization against the assigned centroid, query routing by the dot product
to the centroids, scan of the quantized residuals of the probed partitions
for the top-k) with the score identities of Sec. 3.5:

* Sec. 3.5.1: <q, a + rt> = <q, a> + <q, rt>, and <q, rt> = Lhat <R q, uhat>
  because R is orthogonal (Sec. 5.4: scoring happens in the rotated space,
  the query being rotated once).
* Sec. 3.5.2: with the global scale the score is Ghat (<q, a> + <q, rt>).
* Rescoring (Sec. 2.1 and Sec. 5.2): the survivors of the first stage are
  rescored from higher-bit codes of the second residual x - a2, where the
  approximation a2 is the full first-stage reconstruction, so <q, a2> is the
  first-stage score itself ("reading B", the default).  Reading A: a2 is the
  first stage's own approximation (the centroid), so the second stage is an
  independent, finer code of the same residual and its score is
  Ghat2 (<q, c> + Lhat2 <R2 q, uhat2>).
* Full-vector quantization (Sec. 3.5, first paragraph: the codec applied to
  x itself): the approximation is 0, the partitions only route the probe,
  and a score is Ghat Lhat <R q, uhat>.

Orders: probes by (<q, c_p> descending, p ascending); candidates by (score
descending, id ascending).  Missing results are id -1 with score -inf.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from oracle.codec import Encoded, encode, encode_lite
from oracle.rotation import rotation_matrix, rotation_mode


@dataclass
class OracleIndex:
    """Encoded rows of a (sub)set of the database, grouped by partition."""

    D: int
    bits: int
    rescore_bits: int
    global_scale: bool
    centroids: np.ndarray          # (P, D)
    ids: np.ndarray                # (n,) original row ids
    assign: np.ndarray             # (n,) partition of each row
    stage1: Encoded
    stage2: Encoded | None
    members: dict = field(default_factory=dict)  # partition -> row positions
    reading: str = "B"             # rescoring approximation: "B" stage-1 reconstruction, "A" centroid
    full_vector: bool = False      # the approximation is 0 (no residual)

    def rows_of(self, p: int) -> np.ndarray:
        return self.members.get(int(p), np.zeros(0, dtype=np.int64))


def build_index(X, ids, assign, centroids, bits: int, rescore_bits: int = 0,
                global_scale: bool = True, lite: bool = False, reading: str = "B",
                full_vector: bool = False) -> OracleIndex:
    """Encode rows X (ids, partition ``assign``) against their centroids.

    Stage 1 quantizes r = x - c_p with ``bits`` per dimension (``lite``:
    Rslm4Lite, bits must be 4).  With ``rescore_bits`` > 0, stage 2
    quantizes x - a2 with a2 the stage-1 reconstruction, using
    ``rescore_bits`` per dimension.
    """
    X = np.asarray(X, dtype=np.float64)
    C = np.asarray(centroids, dtype=np.float64)
    assign = np.asarray(assign, dtype=np.int64)
    A1 = C[assign]
    if lite and bits != 4:
        raise ValueError("Rslm4Lite is a 4-bit codec")
    if reading not in ("A", "B"):
        raise ValueError("reading is 'A' or 'B'")
    if full_vector:
        A1 = np.zeros_like(A1)
    st1 = encode_lite(X, A1, global_scale) if lite else encode(X, A1, bits, global_scale=global_scale)
    st2 = None
    if rescore_bits:
        st2 = encode(X, st1.recon if reading == "B" else A1, rescore_bits, global_scale=global_scale)
    members = {}
    for p in np.unique(assign):
        members[int(p)] = np.nonzero(assign == p)[0]
    return OracleIndex(X.shape[1], bits, rescore_bits, global_scale, C,
                       np.asarray(ids, dtype=np.int64), assign, st1, st2, members, reading, full_vector)


def order_desc(scores: np.ndarray, ids: np.ndarray) -> np.ndarray:
    """Permutation sorting by (score descending, id ascending)."""
    return np.lexsort((ids, -scores))


def take_top(scores: np.ndarray, ids: np.ndarray, k: int):
    """First k of the full sort, padded with (-1, -inf)."""
    o = order_desc(scores, ids)[:k]
    out_ids = np.full(k, -1, dtype=np.int64)
    out_sc = np.full(k, -np.inf)
    out_ids[:len(o)] = ids[o]
    out_sc[:len(o)] = scores[o]
    return out_ids, out_sc


def probe(Q, centroids, nprobe: int):
    """Partitions with the largest <q, c_p> (ties: lower p) and those scores."""
    Q = np.atleast_2d(np.asarray(Q, dtype=np.float64))
    C = np.asarray(centroids, dtype=np.float64)
    cs = Q @ C.T
    P = C.shape[0]
    pid = np.arange(P)
    out = np.zeros((Q.shape[0], nprobe), dtype=np.int64)
    out_cs = np.zeros((Q.shape[0], nprobe))
    for i in range(Q.shape[0]):
        o = order_desc(cs[i], pid)[:nprobe]
        out[i] = o
        out_cs[i] = cs[i, o]
    return out, out_cs, cs


def rotate_query(q, bits: int) -> np.ndarray:
    """R_b q for the rotation used by the ``bits`` codec (Sec. 5.4)."""
    q = np.asarray(q, dtype=np.float64)
    return rotation_matrix(q.shape[-1], rotation_mode(bits, q.shape[-1])) @ q


def stage1_scores(index: OracleIndex, q, probes, cs):
    """Scores Ghat (cs_p + Lhat <R q, uhat>) of every row of the probed lists."""
    qb = rotate_query(q, index.bits)
    rows, sc = [], []
    st = index.stage1
    for p, c in zip(probes, cs):
        r = index.rows_of(p)
        if r.size == 0:
            continue
        dot = st.uhat[r] @ qb
        a_term = 0.0 if index.full_vector else c
        sc.append(st.Ghat[r] * (a_term + st.Lhat[r] * dot))
        rows.append(r)
    if not rows:
        return np.zeros(0, dtype=np.int64), np.zeros(0)
    return np.concatenate(rows), np.concatenate(sc)


def scan(index: OracleIndex, q, probes, cs, k: int):
    """Top-k (row ids, scores) over all rows of the probed partitions."""
    rows, sc = stage1_scores(index, q, probes, cs)
    ids, scores = take_top(sc, index.ids[rows], k)
    return ids, scores


def rescore(index: OracleIndex, q, cand_ids, cand_scores, k_final: int):
    """Stage-2 scores Ghat2 (<q, a2> + Lhat2 <R2 q, uhat2>) and their top k_final.

    <q, a2> is the stage-1 score s1 (reading B), or <q, c> of the row's
    partition (reading A; 0 for full-vector codes).
    """
    st = index.stage2
    qb = rotate_query(q, index.rescore_bits)
    pos_of = {int(i): j for j, i in enumerate(index.ids)}
    valid = np.asarray(cand_ids) >= 0
    cid = np.asarray(cand_ids)[valid]
    s1 = np.asarray(cand_scores, dtype=np.float64)[valid]
    r = np.array([pos_of[int(i)] for i in cid], dtype=np.int64)
    if r.size == 0:
        return take_top(np.zeros(0), np.zeros(0, dtype=np.int64), k_final) + (np.zeros(0),)
    if index.reading == "B":
        a_term = s1
    elif index.full_vector:
        a_term = np.zeros(r.size)
    else:
        a_term = index.centroids[index.assign[r]] @ np.asarray(q, dtype=np.float64)
    s2 = st.Ghat[r] * (a_term + st.Lhat[r] * (st.uhat[r] @ qb))
    ids, scores = take_top(s2, cid, k_final)
    return ids, scores, s2


def search(index: OracleIndex, Q, nprobe: int, k: int, k_final: int | None = None,
           rescore_stage: bool | None = None, probes=None, probe_cs=None):
    """Full search of every query row of Q.

    Returns a dict with probes, cs, stage-1 (ids, scores) and, when the index
    has rescoring codes and ``rescore_stage`` is not False, the final
    (ids, scores).  ``probes`` / ``probe_cs`` may fix the probe lists (used
    when another valid probe set is to be followed).
    """
    Q = np.atleast_2d(np.asarray(Q, dtype=np.float64))
    nq = Q.shape[0]
    if probes is None:
        probes, probe_cs, _ = probe(Q, index.centroids, nprobe)
    do_rescore = index.stage2 is not None if rescore_stage is None else rescore_stage
    s1_ids = np.zeros((nq, k), dtype=np.int64)
    s1_sc = np.zeros((nq, k))
    kf = k_final if k_final is not None else k
    f_ids = np.zeros((nq, kf), dtype=np.int64)
    f_sc = np.zeros((nq, kf))
    for i in range(nq):
        s1_ids[i], s1_sc[i] = scan(index, Q[i], probes[i], probe_cs[i], k)
        if do_rescore:
            f_ids[i], f_sc[i], _ = rescore(index, Q[i], s1_ids[i], s1_sc[i], kf)
        else:
            f_ids[i], f_sc[i] = s1_ids[i][:kf], s1_sc[i][:kf]
    return {"probes": probes, "cs": probe_cs, "s1_ids": s1_ids, "s1_scores": s1_sc,
            "ids": f_ids, "scores": f_sc}
