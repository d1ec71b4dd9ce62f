"""rslm_probe_noalloc, the probe step for callers that cannot allocate device memory.

Programs whose device memory is owned by another allocator, and serving loops
that must not call cudaMalloc / cudaFree (those calls can synchronize the
device), probe through this entry point: its scratch is a fixed array inside
the library.  These tests call it through the C ABI, twice in a row, and
compare each result with rslm_probe's within the probe tolerance the other
GPU tests use (1e-5 ||q|| max||c|| on a <q, centroid> score; ids may differ
only between near-equal scores).  This file is collected last on purpose.
"""

import numpy as np
import pytest

from tests.lib_util import ensure_library

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_library()


def _compare(p, c, p_ref, c_ref, exact, tol):
    """Same probe lists up to near-ties; matching scores within tol."""
    for i in range(p.shape[0]):
        a, b = p[i].tolist(), p_ref[i].tolist()
        assert np.all(np.abs(c[i] - exact[i, p[i]]) <= tol[i])
        if a == b:
            assert np.all(np.abs(c[i] - c_ref[i]) <= tol[i])
            continue
        kth = exact[i, p_ref[i]].min()
        for j in set(a) ^ set(b):  # only near-ties at the nprobe boundary may swap
            assert abs(exact[i, j] - kth) <= 2 * tol[i], (i, j)


def test_probe_noalloc_matches_probe_twice():
    from paper_2608_30384_gb300 import Index, binding as B
    rng = np.random.default_rng(2024)
    nlist, D, nq, nprobe = 4096, 128, 2500, 32  # 1024 queries per scratch chunk: 3 chunks
    C = rng.standard_normal((nlist, D)).astype(np.float32)
    Q = rng.standard_normal((nq, D)).astype(np.float32)
    Ct, Qt = torch.from_numpy(C).cuda(), torch.from_numpy(Q).cuda()
    ix = Index(Ct, 4)
    p_ref, c_ref = ix.probe(Qt, nprobe)
    exact = Q.astype(np.float64) @ C.astype(np.float64).T
    tol = 1e-5 * np.linalg.norm(Q, axis=1) * np.linalg.norm(C, axis=1).max()
    p_ref, c_ref = p_ref.cpu().numpy(), c_ref.cpu().numpy()
    for _ in range(2):
        p = torch.full((nq, nprobe), -7, dtype=torch.int32, device="cuda")
        c = torch.full((nq, nprobe), float("nan"), device="cuda")
        B.rslm_probe_noalloc(ix.handle, Qt, nprobe, p, c)
        ix.sync()
        _compare(p.cpu().numpy(), c.cpu().numpy(), p_ref, c_ref, exact, tol)


def test_probe_noalloc_rejects_nlist_beyond_scratch():
    from paper_2608_30384_gb300 import Index, RslmError, binding as B
    nlist = (4 << 20) + 1  # one query's scores no longer fit the fixed scratch
    ix = Index(torch.zeros((nlist, 1), device="cuda"), 4)
    q = torch.zeros((1, 1), device="cuda")
    p = torch.empty((1, 1), dtype=torch.int32, device="cuda")
    c = torch.empty((1, 1), device="cuda")
    with pytest.raises(RslmError) as ei:
        B.rslm_probe_noalloc(ix.handle, q, 1, p, c)
    assert ei.value.status == 1 and "scratch" in str(ei.value)
