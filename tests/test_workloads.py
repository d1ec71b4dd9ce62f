"""Seeded synthetic workloads: determinism and the streamed helpers (CPU)."""

import numpy as np

from paper_2608_30384_gb300 import workloads as W

# several generation chunks and a ragged last one
SMALL = W.Workload("wl", 3 * W.CHUNK + 1234, 16, 50, 0.5, False, 0.5, "mean", 7, 4, 0, 3, 10, 10, seed=3)
UNIT = W.Workload("wu", W.CHUNK + 10, 24, 9, 0.5, True, None, "mean", 5, 2, 4, 2, 10, 5, seed=4)


def test_database_is_deterministic_and_chunked():
    X1, A1 = W.database(SMALL)
    X2, A2 = W.database(SMALL)
    assert np.array_equal(X1, X2) and np.array_equal(A1, A2)
    assert X1.shape == (SMALL.N, SMALL.D) and X1.dtype == np.float32
    ids = np.array([0, W.CHUNK - 1, W.CHUNK, 2 * W.CHUNK + 5, SMALL.N - 1])
    Xr, Ar = W.rows(SMALL, ids)
    assert np.array_equal(Xr, X1[ids]) and np.array_equal(Ar, A1[ids])


def test_assignment_matches_generated_components():
    _, A = W.database(SMALL)
    assert np.array_equal(W.assignment(SMALL), A)
    assert A.min() >= 0 and A.max() < SMALL.P


def test_member_means_streamed_matches_in_memory():
    X, A = W.database(SMALL)
    ctr = W.centers(SMALL)
    assert np.array_equal(W.member_means_streamed(SMALL, ctr), W.member_means(SMALL, X, A, ctr))
    # they are the partition means (float32 rounding of a float64 mean)
    ref = np.stack([X[A == p].astype(np.float64).mean(0) for p in range(SMALL.P)])
    assert np.allclose(W.member_means(SMALL, X, A, ctr), ref, rtol=0, atol=1e-5)


def test_generator_shapes_the_norms():
    X, _ = W.database(UNIT)
    assert np.allclose(np.linalg.norm(X.astype(np.float64), axis=1), 1.0, atol=1e-5)
    X, _ = W.database(SMALL)
    # log-normal(0, 0.5) norms: log-norm mean ~0, sd ~0.5
    ln = np.log(np.linalg.norm(X.astype(np.float64), axis=1))
    assert abs(ln.mean()) < 0.01 and abs(ln.std() - 0.5) < 0.01


def test_queries_are_a_prefix_of_the_query_stream():
    Q = W.queries(SMALL)
    assert Q.shape == (SMALL.nq, SMALL.D)
    assert np.array_equal(W.queries(SMALL, 3), Q[:3])


def test_row_blocks_cover_the_database_in_order():
    X, _ = W.database(SMALL)
    got = list(W.row_blocks(SMALL, 2 * W.CHUNK))
    assert [lo for lo, _ in got] == [0, 2 * W.CHUNK]
    assert np.array_equal(np.concatenate([b for _, b in got]), X)
