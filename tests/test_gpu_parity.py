"""GPU path vs the float64 oracle, element by element, through the C ABI.

Tolerances (the contract): codes bit-exact except groups decided within 1e-5
of a decision boundary (at most 1e-4 of all groups); scale codes exact
except where the exact value lies at a rounding tie; scores within 1e-4
relative (floor 0.01 ||q|| ||x|| of the row, see lib_util.score_tol); top-k lists
equal up to swaps of near-equal scores (lib_util.check_topk).
"""

import numpy as np
import pytest

from oracle import codec, constants as K, search
from oracle.rotation import rotation_matrix, rotation_mode
from paper_2608_30384_gb300 import workloads as W
from tests.gpu_cases import Case, check_lite_stage, check_stage
from tests.lib_util import check_topk, ensure_library, kth_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

Wl = W.Workload
CASES = {
    # the small configuration, in full
    "C1": W.WORKLOADS["C1"],
    # reduced copies of the larger configurations: several tiles per partition and a ragged tail
    "C2s": Wl("C2s", 30_000, 96, 64, 0.5, False, None, "true", 40, 2, 4, 8, 100, 10, seed=1),
    "C3s": Wl("C3s", 12_000, 768, 24, 0.5, True, None, "mean", 12, 1, 4, 6, 100, 10, seed=2),
    "C4s": Wl("C4s", 40_000, 128, 64, 0.5, False, 0.5, "mean", 40, 4, 0, 16, 10, 10, seed=3),
    "C5s": Wl("C5s", 6_000, 1536, 12, 0.5, True, None, "mean", 6, 2, 4, 4, 200, 10, seed=4),
    # zero padding of the last group (D not a multiple of g), odd group counts
    "pad1": Wl("pad1", 5_000, 100, 8, 0.5, False, None, "true", 20, 1, 4, 3, 50, 5, seed=5),
    "pad2": Wl("pad2", 5_000, 99, 8, 0.5, False, None, "true", 20, 2, 0, 3, 20, 20, seed=6),
    # tiny dimensions: block size shrinks to 1, 2, 4 (Sec. 3.1.1)
    "D1": Wl("D1", 2_000, 1, 4, 0.5, False, None, "true", 20, 4, 0, 2, 8, 8, seed=7),
    "D5": Wl("D5", 2_000, 5, 4, 0.5, False, None, "true", 20, 2, 4, 2, 16, 4, seed=8),
    "D300": Wl("D300", 4_000, 300, 8, 0.5, True, None, "mean", 10, 4, 0, 3, 30, 30, seed=9),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_library()


@pytest.fixture(scope="module", params=list(CASES))
def case(request):
    return Case(CASES[request.param])


@pytest.fixture(scope="module")
def local_case():
    return Case(Wl("loc", 6_000, 64, 8, 0.5, False, 0.5, "mean", 20, 4, 4, 3, 40, 10, seed=10),
                global_scale=False)


# ------------------------------------------------------------------ rotation
@pytest.mark.parametrize("D", [1, 2, 3, 5, 64, 96, 100, 127, 128, 129, 200, 256, 300, 768, 1536, 2049])
@pytest.mark.parametrize("bits", [1, 4])
def test_query_rotation(D, bits):
    from paper_2608_30384_gb300 import Index
    C = torch.zeros((1, D), device="cuda")
    ix = Index(C, bits)
    q = np.random.default_rng(D).standard_normal((37, D)).astype(np.float32)
    out = ix.rotate(torch.from_numpy(q).cuda()).cpu().numpy()
    R = rotation_matrix(D, rotation_mode(bits, D))
    ref = q.astype(np.float64) @ R.T
    g = K.group_size(bits)
    Dp = g * -(-D // g)
    assert out.shape == (37, Dp)
    assert np.all(out[:, D:] == 0)
    err = np.abs(out[:, :D] - ref).max(1) / np.linalg.norm(q, axis=1)
    assert err.max() < 2e-6


# -------------------------------------------------------------------- encode
def _encode_check(case):
    ix = case.gpu_index()
    w = case.w
    c1, L1, G1 = (t.cpu().numpy() for t in ix.export_codes(1))
    A1, A2 = case.approximations()
    ok = check_stage(c1, L1, G1, case.oracle.stage1, case.X, A1, w.bits, case.global_scale, "stage 1")
    if w.rescore_bits:
        c2, L2, G2 = (t.cpu().numpy() for t in ix.export_codes(2))
        st2 = case.oracle.stage2
        sel = np.nonzero(ok)[0]
        sub = codec.Encoded(st2.bits, st2.mode, st2.D, st2.g, st2.codes[sel], st2.L_u16[sel],
                            st2.G_u16[sel], st2.Lhat[sel], st2.Ghat[sel], st2.uhat[sel], st2.u[sel],
                            st2.recon[sel], st2.L_exact[sel], st2.G_exact[sel])
        check_stage(c2[sel], L2[sel], G2[sel], sub, case.X[sel], A2[sel],
                     w.rescore_bits, case.global_scale, "stage 2")
    return ix


def test_encode_parity(case):
    _encode_check(case)


def test_encode_parity_local_scale(local_case):
    _encode_check(local_case)


def test_chunked_encode_matches_single_pass():
    """Encoding in several chunks, out of order, gives the same index."""
    case = Case(CASES["C4s"])
    a = case.gpu_index()
    b = case.gpu_index(encode=False)
    X = torch.from_numpy(case.X).cuda()
    for lo in (30_000, 0, 10_000, 20_000):
        b.encode(X[lo:lo + 10_000], lo)
    for which in (1,):
        for u, v in zip(a.export_codes(which), b.export_codes(which)):
            assert torch.equal(u, v)


def test_encode_all_matches_the_three_calls():
    """rslm_encode_all (create + reserve + encode in one call) builds the same
    index as the three calls: identical codes and scales of both stages."""
    from paper_2608_30384_gb300 import binding as B
    case = Case(CASES["C2s"])
    a = case.gpu_index()
    h = B.rslm_encode_all(torch.from_numpy(case.X).cuda(), torch.from_numpy(case.A).cuda(),
                          torch.from_numpy(case.C).cuda(), case.w.bits, case.w.rescore_bits)
    B.rslm_sync(h)
    assert B.rslm_index_describe(h)["n_rows"] == case.w.N
    for which in (1, 2):
        d = a.desc
        nb = d["code_bytes"] if which == 1 else d["rescore_code_bytes"]
        got = (torch.empty((case.w.N, nb), dtype=torch.uint8, device="cuda"),
               torch.empty(case.w.N, dtype=torch.uint16, device="cuda"),
               torch.empty(case.w.N, dtype=torch.uint16, device="cuda"))
        B.rslm_export_codes(h, which, 0, case.w.N, *got)
        for u, v in zip(a.export_codes(which), got):
            assert torch.equal(u, v)


# ------------------------------------------------------------------- search
def _oracle_stage1(case, i, probes, cs):
    rows, s1 = search.stage1_scores(case.oracle, case.Q[i], probes, cs)
    return dict(zip(case.oracle.ids[rows].tolist(), s1.tolist())), s1


def _kth(values, k):
    v = np.sort(np.asarray(values))[::-1]
    return v[k - 1] if len(v) >= k else -np.inf


def test_probe_parity(case):
    ix = case.gpu_index(encode=False)
    w = case.w
    p, cs = (t.cpu().numpy() for t in ix.probe(torch.from_numpy(case.Q).cuda(), w.nprobe))
    full = case.Q.astype(np.float64) @ case.C.astype(np.float64).T
    cn = np.linalg.norm(case.C, axis=1).max()
    for i in range(len(case.Q)):
        tol = lambda s, j=None: 1e-5 * case.qnorm(i) * cn  # noqa: E731
        probs = check_topk(p[i], cs[i], lambda j: full[i, j], _kth(full[i], w.nprobe), tol)
        assert not probs, (i, probs[:3])


@pytest.mark.parametrize("nlist,nprobe,layout,D", [
    (1001, 1, "random", 32), (1001, 64, "random", 32), (8192, 64, "random", 32),
    (8192, 256, "random", 32), (777, 200, "random", 32), (4099, 300, "random", 32),
    (3000, 64, "sorted", 32), (2048, 100, "tied", 32), (513, 513, "random", 32), (6, 5, "random", 32),
    # tensor-core probe (D <= 128, nlist >= 32 nprobe): ragged nlist and D, sorted
    # scores, ties everywhere (list overflow: every centroid is rescored)
    (8192, 64, "random", 128), (1000, 31, "random", 100), (4100, 128, "sorted", 96),
    (4096, 64, "tied", 128), (2500, 77, "random", 5), (300, 9, "random", 128),
])
def test_probe_selection_paths(nlist, nprobe, layout, D):
    """Top-nprobe of <q, c> on layouts that steer the selection kernels: random
    order (the warp kernel's bound leaves about nprobe candidates), scores
    sorted along the centroid index, all centroids equal (every element ties
    at the bound, so rows go to the block kernel), nprobe above 256 (block
    kernel only), and nlist not a multiple of 4."""
    rng = np.random.default_rng(nlist * 7 + nprobe + D)
    nq = 300
    Q = rng.standard_normal((nq, D)).astype(np.float32)
    if layout == "tied":
        C = np.repeat(rng.standard_normal((1, D)), nlist, axis=0).astype(np.float32)
    else:
        C = rng.standard_normal((nlist, D)).astype(np.float32)
    if layout == "sorted":
        # same direction, decreasing norm: <q, c_j> is monotone in j for every q
        C = (np.linspace(2.0, 1.0, nlist)[:, None] * C[:1]).astype(np.float32)
    from paper_2608_30384_gb300 import Index
    ix = Index(torch.from_numpy(C).cuda(), 4)
    p, cs = (t.cpu().numpy() for t in ix.probe(torch.from_numpy(Q).cuda(), nprobe))
    full = Q.astype(np.float64) @ C.astype(np.float64).T
    cn = np.linalg.norm(C, axis=1).max()
    for i in range(nq):
        tol = lambda s, j=None: 1e-5 * np.linalg.norm(Q[i]) * cn  # noqa: E731
        probs = check_topk(p[i], cs[i], lambda j: full[i, j], _kth(full[i], nprobe), tol)
        assert not probs, (i, probs[:3])
        if layout == "tied":
            # equal scores are ordered by centroid index
            np.testing.assert_array_equal(p[i], np.arange(nprobe))


def _scan_inputs(case):
    probes, cs, _ = search.probe(case.Q, case.C, case.w.nprobe)
    return probes, cs


def test_scan_parity_on_oracle_codes(case):
    """rslm_scan with the oracle's probes, on the oracle's imported codes."""
    w = case.w
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    probes, cs = _scan_inputs(case)
    qrot = ix.rotate(torch.from_numpy(case.Q).cuda())
    ids, sc = ix.scan(qrot, torch.from_numpy(probes.astype(np.int32)).cuda(),
                      torch.from_numpy(cs.astype(np.float32)).cuda(), w.k)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    for i in range(len(case.Q)):
        ref, s1 = _oracle_stage1(case, i, probes[i], cs[i])
        kth, kid = kth_of(ref, w.k)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, case.score_tol_of(i), allowed_ids=ref,
                           kth_id=kid)
        assert not probs, (i, probs[:3])
        assert (ids[i] >= 0).sum() == min(w.k, len(s1))


# Single-query scan of 4-bit codes of one coordinate (padded D <= 128): one
# unit per query (batches of >= 4 units per SM), units split over probe
# ranges (small batches), partitions shorter than half a tile and an empty
# one, chunk columns past the row's codes (D = 96, 33), large k near the
# shared-memory limit, k = 256 (falls back to the table scan) and
# nprobe = nlist.
SINGLE = {
    "one_unit": Wl("sq1", 20_000, 128, 64, 0.5, False, 0.5, "mean", 700, 4, 0, 4, 10, 10, seed=21),
    "split_units": Wl("sq2", 20_000, 128, 64, 0.5, False, 0.5, "mean", 3, 4, 0, 16, 10, 10, seed=22),
    "short_lists": Wl("sq3", 3_000, 128, 64, 0.5, False, None, "true", 40, 4, 0, 8, 10, 10, seed=23),
    "D96": Wl("sq4", 8_000, 96, 16, 0.5, False, None, "true", 40, 4, 0, 4, 10, 10, seed=24),
    "D33": Wl("sq5", 8_000, 33, 16, 0.5, False, None, "true", 40, 4, 0, 4, 10, 10, seed=25),
    "k200": Wl("sq6", 20_000, 128, 32, 0.5, False, None, "mean", 30, 4, 0, 8, 200, 200, seed=26),
    "k256": Wl("sq7", 20_000, 128, 32, 0.5, False, None, "mean", 30, 4, 0, 8, 256, 256, seed=27),
    "all_probes": Wl("sq8", 6_000, 128, 16, 0.5, False, None, "true", 20, 4, 0, 16, 20, 20, seed=28),
}


@pytest.mark.parametrize("name", sorted(SINGLE))
def test_single_query_scan_paths(name):
    """rslm_scan on 4-bit codes of one coordinate, at the edges of its launch plan."""
    case = Case(SINGLE[name])
    if name == "short_lists":
        A = case.A.copy()
        A[A == 5] = 6  # partition 5 left empty
        case.A = A
        case.oracle = search.build_index(case.X, np.arange(case.w.N), A, case.C, 4, 0)
    w = case.w
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    probes, cs = _scan_inputs(case)
    qrot = ix.rotate(torch.from_numpy(case.Q).cuda())
    ids, sc = ix.scan(qrot, torch.from_numpy(probes.astype(np.int32)).cuda(),
                      torch.from_numpy(cs.astype(np.float32)).cuda(), w.k)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    for i in range(len(case.Q)):
        ref, s1 = _oracle_stage1(case, i, probes[i], cs[i])
        kth, kid = kth_of(ref, w.k)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, case.score_tol_of(i), allowed_ids=ref,
                           kth_id=kid)
        assert not probs, (i, probs[:3])
        assert (ids[i] >= 0).sum() == min(w.k, len(s1))
        assert np.all(np.isneginf(sc[i][ids[i] < 0]))


def _scan_parity(case, batched: bool):
    w = case.w
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    probes, cs = _scan_inputs(case)
    qrot = ix.rotate(torch.from_numpy(case.Q).cuda())
    fn = ix.scan_batched if batched else ix.scan
    ids, sc = fn(qrot, torch.from_numpy(probes.astype(np.int32)).cuda(),
                 torch.from_numpy(cs.astype(np.float32)).cuda(), w.k)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    for i in range(len(case.Q)):
        ref, s1 = _oracle_stage1(case, i, probes[i], cs[i])
        kth, kid = kth_of(ref, w.k)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, case.score_tol_of(i), allowed_ids=ref,
                           kth_id=kid)
        assert not probs, (i, probs[:3])
        assert (ids[i] >= 0).sum() == min(w.k, len(s1))
    # the two passes of the batched scan agree: no query needed the exact re-scan for a short list
    assert ix.counters()["batched_short_rescans"] == 0
    return ix, (qrot, probes, cs), (ids, sc)


def test_batched_scan_parity_on_oracle_codes(case):
    """rslm_scan_batched (tensor cores, partition-major) with the oracle's probes."""
    _scan_parity(case, batched=True)


def test_batched_scan_overflow_fallback():
    """Partitions smaller than k give no threshold: every candidate is kept,
    the per-query buffer overflows and the single-query kernel re-scans."""
    _scan_parity(Case(Wl("ovf", 20_000, 64, 256, 0.5, False, None, "true", 24, 4, 0, 128, 100, 100,
                         seed=12)), batched=True)


def test_batched_scan_many_partitions():
    """More partitions (25000) than the shared-memory histograms of the
    probe-list inversion hold (24576): the global-atomic inversion path."""
    _scan_parity(Case(Wl("np", 60_000, 16, 25_000, 0.5, False, 0.5, "true", 200, 4, 0, 16, 10, 10,
                         seed=21)), batched=True)


@pytest.mark.parametrize("bits,D", [(4, 128), (2, 96), (1, 128), (4, 256), (1, 768), (2, 300),
                                    (1, 256), (2, 768), (4, 768), (1, 384), (3, 128), (3, 300)])
def test_batched_scan_many_queries_per_partition(bits, D):
    """About 225 queries per partition: two work items per partition (N = 128
    and a partial N), about 20 row tiles each, so the pipelined kernels'
    slot, slab and accumulator rings wrap many times; D > 128 runs several
    K chunks (D = 300: a partial last chunk)."""
    _scan_parity(Case(Wl(f"mq{bits}", 20_000, D, 8, 0.5, False, 0.5, "mean", 600, bits, 0, 3, 10, 10,
                         seed=13 + bits)), batched=True)


@pytest.mark.parametrize("bits,D,N", [(4, 256, 20_000), (4, 768, 20_000), (2, 1536, 8_000)])
def test_batched_scan_repeatable(bits, D, N):
    """The tensor-core scan with several K chunks, run 20 times in one
    process on the same inputs: the first result passes the top-k rule, and
    every repeat returns bit-identical ids and scores without any query
    falling back to the exact re-scan.  (The per-partition query lists are
    built with atomics, so every run places the queries in other MMA
    columns and the warps' timing differs: a synchronisation fault shows up
    as a differing repeat.)"""
    case = Case(Wl(f"rp{bits}", N, D, 8, 0.5, False, 0.5, "mean", 600, bits, 0, 3, 10, 10, seed=31 + bits))
    ix, (qrot, probes, cs), (ids0, sc0) = _scan_parity(case, batched=True)
    P = torch.from_numpy(probes.astype(np.int32)).cuda()
    CS = torch.from_numpy(cs.astype(np.float32)).cuda()
    for rep in range(19):
        ids, sc = ix.scan_batched(qrot, P, CS, case.w.k)
        ix.sync()
        ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
        bad = (ids != ids0).any(1) | (sc != sc0).any(1)
        assert not bad.any(), (rep, int(bad.sum()), "queries differ from the first run; largest score change",
                               float(np.abs(sc - sc0).max()), "first", int(np.nonzero(bad)[0][0]))
    assert ix.counters()["batched_short_rescans"] == 0


# ------------------------------------------------------------ decompress
def _decompress_check(case):
    """rslm_decompress of both stages against the oracle's decode of the
    GPU's own exported codes and scales (Sec. 4): equal up to the float32
    rounding of the output."""
    w = case.w
    ix = case.gpu_index()
    A1, _ = case.approximations()
    c1, L1, G1 = (t.cpu().numpy().astype(np.int64) for t in ix.export_codes(1))
    ng1 = case.oracle.stage1.codes.shape[1]
    if case.lite:
        ref1 = codec.decode_lite(A1, codec.unpack_nibbles(c1, w.D), w.D, case.global_scale)
    else:
        unpack = codec.unpack_bits3 if w.bits == 3 else codec.unpack_nibbles
        ref1 = codec.decode(A1, unpack(c1, ng1), L1, G1, w.bits, w.D)
    tol = 1e-6 * float(np.abs(case.X).max()) + 1e-6
    got1 = ix.decompress(1).cpu().numpy()
    assert np.allclose(got1, ref1, rtol=1e-6, atol=tol), np.abs(got1 - ref1).max()
    if w.rescore_bits:
        c2, L2, G2 = (t.cpu().numpy().astype(np.int64) for t in ix.export_codes(2))
        A2 = A1 if case.reading == "A" else ref1
        ref2 = codec.decode(A2, codec.unpack_nibbles(c2, case.oracle.stage2.codes.shape[1]), L2, G2,
                            w.rescore_bits, w.D)
        got2 = ix.decompress(2).cpu().numpy()
        assert np.allclose(got2, ref2, rtol=1e-6, atol=tol), np.abs(got2 - ref2).max()
        # the rescoring reconstruction is closer to x than the scoring one
        e1 = np.linalg.norm(got1 - case.X, axis=1).mean()
        e2 = np.linalg.norm(got2 - case.X, axis=1).mean()
        assert e2 < e1


def test_decompress_parity(case):
    _decompress_check(case)


@pytest.mark.parametrize("kind", ["lite", "reading_a", "full_vector"])
def test_decompress_parity_variants(kind):
    if kind == "lite":
        case = Case(Wl("dl", 6_000, 128, 8, 0.5, False, 0.5, "mean", 8, 4, 0, 3, 10, 10, seed=51), lite=True)
    else:
        case = Case(Wl("dv", 6_000, 96, 8, 0.5, False, 0.5, "mean", 8, 2, 4, 3, 40, 10, seed=52),
                    reading="A" if kind == "reading_a" else "B", full_vector=kind == "full_vector")
    _decompress_check(case)


# ----------------------------------------------------------------- Rslm3
# Sec. 3.4: 3 bits per dimension on the K = 8 levels, eight codes in 3 bytes.
# D = 100: a partial last 32-code group (and 4-bit rescoring on top);
# D = 768: many groups.
R3 = {
    "r3a": Wl("r3a", 20_000, 128, 16, 0.5, False, 0.5, "mean", 40, 3, 0, 4, 10, 10, seed=61),
    "r3b": Wl("r3b", 15_000, 100, 12, 0.5, True, None, "mean", 40, 3, 4, 4, 60, 10, seed=62),
    "r3c": Wl("r3c", 6_000, 768, 8, 0.5, True, None, "mean", 24, 3, 0, 3, 10, 10, seed=63),
}


@pytest.mark.parametrize("name", sorted(R3))
def test_rslm3_encode_and_decompress_parity(name):
    case = Case(R3[name])
    ix = _encode_check(case)
    assert ix.desc["code_bytes"] == (3 * case.w.D + 7) // 8
    _decompress_check(case)


@pytest.mark.parametrize("name", sorted(R3))
@pytest.mark.parametrize("batched", [False, True])
def test_rslm3_scan_parity(name, batched):
    """Both scan forms on 3-bit rows: the single-query kernel's shift /
    funnel-shift extraction and the tensor-core decode of 6-bit code pairs
    (D = 768: six K chunks)."""
    _scan_parity(Case(R3[name]), batched=batched)


def test_rslm3_search_end_to_end_batched():
    """rslm_search on 3-bit scoring codes with enough queries per probed
    list for the tensor-core regime, then 4-bit rescoring."""
    case = Case(Wl("r3e", 20_000, 128, 8, 0.5, True, None, "mean", 200, 3, 4, 3, 40, 10, seed=64))
    assert case.w.nq * case.w.nprobe >= 16 * case.w.P
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    _end_to_end(case, ix)


# ---------------------------------------------- relative-mode variants
# Rescoring reading A (codes of x - c, scored with <q, c>) and full-vector
# codes (approximation 0), Sec. 3.5 / Sec. 5.2.  C2-like: 2-bit scoring,
# 4-bit rescoring, D = 96 (two FWHT blocks).
REL = Wl("rel", 20_000, 96, 16, 0.5, False, 0.5, "mean", 40, 2, 4, 4, 60, 10, seed=41)


@pytest.mark.parametrize("reading,full_vector", [("A", False), ("B", True), ("A", True)])
def test_relative_variants_encode_parity(reading, full_vector):
    _encode_check(Case(REL, reading=reading, full_vector=full_vector))


@pytest.mark.parametrize("reading,full_vector", [("A", False), ("B", True), ("A", True)])
@pytest.mark.parametrize("batched", [False, True])
def test_relative_variants_scan_and_rescore_parity(reading, full_vector, batched):
    """Stage 1 ignores <q, c> for full-vector codes; rescoring reading A
    adds <q, c> of the row's partition (from the rotated centroids)."""
    case = Case(REL, reading=reading, full_vector=full_vector)
    _scan_parity(case, batched=batched)
    test_rescore_parity_on_oracle_codes(case)


# ------------------------------------------------------------- Rslm4Lite
# Sec. 3.4: the scale codes ride in the top bits of the first 16 (32 with the
# global scale) codes, which take the K = 8 levels.  D = 100 exercises 4-byte
# code chunks and a partial last group; D = 768 the several-K-chunk kernel.
LITE = {
    "l128": Wl("l128", 30_000, 128, 24, 0.5, False, 0.5, "mean", 48, 4, 0, 6, 10, 10, seed=31),
    "l100": Wl("l100", 20_000, 100, 16, 0.5, True, None, "mean", 48, 4, 0, 4, 10, 10, seed=32),
    "l768": Wl("l768", 8_000, 768, 8, 0.5, True, None, "mean", 48, 4, 0, 3, 10, 10, seed=33),
}


@pytest.mark.parametrize("name", sorted(LITE))
@pytest.mark.parametrize("gs", [True, False])
def test_lite_encode_parity(name, gs):
    case = Case(LITE[name], global_scale=gs, lite=True)
    ix = case.gpu_index()
    c1, L1, G1 = (t.cpu().numpy() for t in ix.export_codes(1))
    assert c1.shape[1] == (case.w.D + 1) // 2
    check_lite_stage(c1, L1, G1, case.oracle.stage1, case.X, case.C[case.A].astype(np.float64), gs, name)


@pytest.mark.parametrize("name", sorted(LITE))
@pytest.mark.parametrize("gs", [True, False])
@pytest.mark.parametrize("batched", [False, True])
def test_lite_scan_parity(name, gs, batched):
    """Scan of imported oracle Rslm4Lite codes: the single-query kernel reads
    the scales from the codes' top bits, the tensor-core kernels decode the
    head through the K = 8 table."""
    _scan_parity(Case(LITE[name], global_scale=gs, lite=True), batched=batched)


def test_rescore_parity_on_oracle_codes(case):
    w = case.w
    if not w.rescore_bits:
        pytest.skip("no rescoring codes")
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    res = search.search(case.oracle, case.Q, w.nprobe, w.k, w.k_final)
    q2 = ix.rotate(torch.from_numpy(case.Q).cuda(), which=2)
    ids, sc = ix.rescore(q2, torch.from_numpy(res["s1_ids"]).cuda(),
                         torch.from_numpy(res["s1_scores"].astype(np.float32)).cuda(), w.k_final)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    for i in range(len(case.Q)):
        _, _, s2 = search.rescore(case.oracle, case.Q[i], res["s1_ids"][i], res["s1_scores"][i], w.k)
        cid = res["s1_ids"][i][res["s1_ids"][i] >= 0]
        ref = dict(zip(cid.tolist(), s2.tolist()))
        kth, kid = kth_of(ref, w.k_final)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, case.score_tol_of(i), allowed_ids=ref,
                           kth_id=kid)
        assert not probs, (i, probs[:3])


# (case, stage-1 k, k_final, share of candidate slots set to -1): the
# largest k, a ragged k returned whole, holes in the lists, D = 1536
RESCORE_PATHS = {
    "k256": ("C2s", 256, 10, 0.0),
    "ragged_all": ("C2s", 45, 45, 0.0),
    "holes": ("C2s", 100, 10, 0.3),
    "D1536_holes": ("C5s", 200, 20, 0.1),
}


@pytest.mark.parametrize("name", sorted(RESCORE_PATHS))
def test_rescore_paths(name):
    cname, k, kf, holes = RESCORE_PATHS[name]
    case = Case(CASES[cname])
    w = case.w
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    res = search.search(case.oracle, case.Q, w.nprobe, k, kf)
    s1_ids, s1_sc = res["s1_ids"].copy(), res["s1_scores"].copy()
    if holes:
        s1_ids[np.random.default_rng(11).random(s1_ids.shape) < holes] = -1
    q2 = ix.rotate(torch.from_numpy(case.Q).cuda(), which=2)
    ids, sc = ix.rescore(q2, torch.from_numpy(s1_ids).cuda(), torch.from_numpy(s1_sc.astype(np.float32)).cuda(), kf)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    assert ids.shape == (len(case.Q), kf)
    for i in range(len(case.Q)):
        _, _, s2 = search.rescore(case.oracle, case.Q[i], s1_ids[i], s1_sc[i], k)
        cid = s1_ids[i][s1_ids[i] >= 0]
        ref = dict(zip(cid.tolist(), s2.tolist()))
        kth, kid = kth_of(ref, kf)
        probs = check_topk(ids[i], sc[i], lambda j: ref[j], kth, case.score_tol_of(i), allowed_ids=ref,
                           kth_id=kid)
        assert not probs, (i, probs[:3])


def _end_to_end(case, ix, code_ok=None):
    w = case.w
    Qt = torch.from_numpy(case.Q).cuda()
    ids, sc = ix.search(Qt, w.nprobe, w.k, k_final=w.k_final)
    gp, _ = ix.probe(Qt, w.nprobe)
    ix.sync()
    ids, sc, gp = ids.cpu().numpy(), sc.cpu().numpy(), gp.cpu().numpy()
    oprobes, ocs = _scan_inputs(case)
    for i in range(len(case.Q)):
        probes, cs = oprobes[i], ocs[i]
        if set(gp[i].tolist()) != set(probes.tolist()):
            # a near-tie at the nprobe boundary (validated by test_probe_parity): follow the GPU's set
            probes = gp[i].astype(np.int64)
            cs = case.Q[i].astype(np.float64) @ case.C[probes].astype(np.float64).T
        ref1, s1 = _oracle_stage1(case, i, probes, cs)
        if w.rescore_bits:
            cid = np.array(list(ref1), dtype=np.int64)
            cs1 = np.array([ref1[j] for j in cid])
            _, _, s2 = search.rescore(case.oracle, case.Q[i], cid, cs1, len(cid))
            ref = dict(zip(cid.tolist(), s2.tolist()))
            surv, _ = search.take_top(cs1, cid, w.k)
            kth, kid = kth_of({j: ref[j] for j in surv if j >= 0}, w.k_final)
        else:
            ref = ref1
            kth, kid = kth_of(ref1, w.k_final)
        gpu_score = dict(zip(ids[i].tolist(), sc[i].tolist()))
        # rows whose GPU codes sit on the other side of a decision boundary score differently
        score_of = lambda j: gpu_score[j] if (code_ok is not None and not code_ok[j]) else ref[j]  # noqa: E731
        probs = check_topk(ids[i], sc[i], score_of, kth, case.score_tol_of(i), allowed_ids=ref, kth_id=kid)
        assert not probs, (i, probs[:3])
    assert ix.counters()["batched_short_rescans"] == 0


def test_search_end_to_end_on_oracle_codes(case):
    ix = case.gpu_index(encode=False)
    case.import_oracle_codes(ix)
    _end_to_end(case, ix)


def test_search_end_to_end_gpu_encoded(case):
    """GPU encode + GPU search vs oracle encode + oracle search."""
    ix = case.gpu_index()
    c1, _, _ = ix.export_codes(1)
    got = codec.unpack_nibbles(c1.cpu().numpy(), case.oracle.stage1.codes.shape[1])
    code_ok = (got == case.oracle.stage1.codes).all(1)
    if case.w.rescore_bits:
        c2, _, _ = ix.export_codes(2)
        got2 = codec.unpack_nibbles(c2.cpu().numpy(), case.oracle.stage2.codes.shape[1])
        code_ok &= (got2 == case.oracle.stage2.codes).all(1)
    _end_to_end(case, ix, code_ok)


# --------------------------------------------------------------- edge cases
def test_edge_cases():
    from paper_2608_30384_gb300 import RslmError, rslm_scan
    case = Case(Wl("edge", 700, 32, 6, 0.5, False, None, "true", 5, 4, 0, 6, 256, 256, seed=11))
    A = case.A.copy()
    A[A == 2] = 3  # partition 2 left empty
    case.A = A
    case.oracle = search.build_index(case.X, np.arange(700), A, case.C, 4, 0)
    ix = case.gpu_index()
    Q = torch.from_numpy(case.Q).cuda()
    # nq = 0 is a no-op
    e_ids = torch.empty((0, 4), dtype=torch.int64, device="cuda")
    e_sc = torch.empty((0, 4), dtype=torch.float32, device="cuda")
    ix.search(Q[:0], 2, 4, out=(e_ids, e_sc))
    # nprobe = nlist, k = 256 > rows of the probed lists: tail is -1 / -inf
    ids, sc = ix.search(Q, 6, 256)
    ix.sync()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    assert np.all((ids >= 0).sum(1) == 256)  # 700 rows, k = 256
    ids1, sc1 = ix.search(Q, 1, 256)
    ix.sync()
    n1 = (ids1.cpu().numpy() >= 0).sum(1)
    probes, _ = ix.probe(Q, 1)
    sizes = np.bincount(A, minlength=6)[probes.cpu().numpy()[:, 0]]
    assert np.array_equal(n1, np.minimum(sizes, 256))
    tail = ids1.cpu().numpy() < 0
    assert np.all(np.isneginf(sc1.cpu().numpy()[tail]))
    # k = 1
    i1, _ = ix.search(Q, 3, 1)
    i10, _ = ix.search(Q, 3, 10)
    assert torch.equal(i1[:, 0], i10[:, 0])
    # an out-of-range probe id sets the sticky device error, reported by rslm_sync
    qrot = ix.rotate(Q)
    bad = torch.full((Q.shape[0], 2), 1, dtype=torch.int32, device="cuda")
    bad[:, 1] = 99
    cs = torch.zeros((Q.shape[0], 2), device="cuda")
    out_i = torch.empty((Q.shape[0], 4), dtype=torch.int64, device="cuda")
    out_s = torch.empty((Q.shape[0], 4), dtype=torch.float32, device="cuda")
    rslm_scan(ix.handle, qrot, bad, cs, 4, out_i, out_s)
    with pytest.raises(RslmError) as ei:
        ix.sync()
    assert ei.value.status == 6
    ix.sync()  # cleared
    # argument errors are reported synchronously
    with pytest.raises(RslmError) as ei:
        ix.search(Q, 7, 4)
    assert ei.value.status == 1
    with pytest.raises(RslmError):
        ix.search(Q, 2, 300)
    # a row range whose end overflows int64 is rejected before any launch
    from paper_2608_30384_gb300 import binding as Bnd
    small = torch.empty((1, 32), device="cuda")
    lib, h, buf = Bnd.lib(), Bnd._ptr(ix.handle), small.data_ptr()
    assert lib.rslm_decompress(h, 1, 2 ** 62, 2 ** 62, buf, None) == 1
    assert lib.rslm_export_codes(h, 1, 2 ** 62, 2 ** 62, buf, buf, buf, None) == 1
    assert lib.rslm_import_codes(h, 1, 2 ** 62, 2 ** 62, buf, buf, buf, None) == 1
    assert lib.rslm_encode(h, buf, 2 ** 62, 2 ** 62, None) == 1


def test_state_errors():
    from paper_2608_30384_gb300 import Index, RslmError
    C = torch.zeros((4, 16), device="cuda")
    ix = Index(C, 4)
    with pytest.raises(RslmError) as ei:
        ix.encode(torch.zeros((3, 16), device="cuda"), 0)
    assert ei.value.status == 5
    with pytest.raises(RslmError) as ei:
        ix.reserve(torch.tensor([0, 1, 9], dtype=torch.int32, device="cuda"))
    assert ei.value.status == 1
    ix.reserve(torch.tensor([0, 1, 3], dtype=torch.int32, device="cuda"))
    with pytest.raises(RslmError) as ei:
        ix.reserve(torch.tensor([0, 1, 3], dtype=torch.int32, device="cuda"))
    assert ei.value.status == 5
    with pytest.raises(RslmError):
        ix.encode(torch.zeros((3, 16), device="cuda"), 1)  # rows 1..3 exceed n = 3
