"""Helpers shared by the tests (library build, tolerant comparisons)."""

import os
import threading

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
_lock = threading.Lock()


def ensure_library():
    """Build librslm.so in-tree if it is missing (nvcc is needed, not a GPU)."""
    from paper_2608_30384_gb300 import build
    with _lock:
        if not os.path.exists(build.LIB):
            build.build_library()
    return build.LIB


def score_tol(scores, qnorm, xnorm, rel=1e-4):
    """Tolerance of a score: rel * max(|s|, 0.01 ||q|| ||x||), ||x|| the row's own norm.

    The floor keeps the relative bound meaningful for scores near zero: a
    float32 dot product of cancelling terms has absolute error proportional
    to ||q|| ||x||, not to the (possibly cancelled) result.
    """
    return rel * np.maximum(np.abs(scores), 0.01 * qnorm * xnorm)


def kth_of(ref: dict, k: int):
    """(k-th best score, its id) of {id: score} by (score desc, id asc); (-inf, None) if fewer than k."""
    if len(ref) < k:
        return -np.inf, None
    items = sorted(ref.items(), key=lambda t: (-t[1], t[0]))
    return items[k - 1][1], items[k - 1][0]


def check_topk(gpu_ids, gpu_scores, ref_score_of, ref_kth, tol_of, allowed_ids=None, kth_id=None):
    """Top-k parity rule (ties / near-ties may swap).

    * returned ids are distinct and (if given) members of ``allowed_ids``;
    * each returned score matches the reference score of that id within tol;
    * each returned id's reference score is >= the reference k-th score minus
      the two rows' tolerances;
    * scores are non-increasing;
    * a -1 id only where the reference list also ran out.
    ``tol_of(score, id)`` is the tolerance of a score of row ``id`` (``id`` is
    ``kth_id`` for the k-th score, possibly None).  Returns a list of problems
    (empty when the list is accepted).
    """
    problems = []
    ids = [int(i) for i in gpu_ids if i >= 0]
    if len(set(ids)) != len(ids):
        problems.append("duplicate ids")
    for i, s in zip(gpu_ids, gpu_scores):
        if i < 0:
            if np.isfinite(ref_kth):
                problems.append("missing entries")
            continue
        if allowed_ids is not None and int(i) not in allowed_ids:
            problems.append(f"id {i} not a candidate")
            continue
        r = ref_score_of(int(i))
        t = tol_of(r, int(i))
        if abs(float(s) - r) > t:
            problems.append(f"id {i}: score {s} vs reference {r} (tol {t})")
        if np.isfinite(ref_kth) and r < ref_kth - tol_of(ref_kth, kth_id) - t:
            problems.append(f"id {i}: reference score {r} below k-th {ref_kth}")
    fin = np.asarray([s for i, s in zip(gpu_ids, gpu_scores) if i >= 0], dtype=np.float64)
    if fin.size > 1 and np.any(np.diff(fin) > 0):
        problems.append("scores not sorted")
    return problems
