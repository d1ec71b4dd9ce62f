"""Shared builders for the GPU parity tests: one synthetic case on both sides."""

from __future__ import annotations

import numpy as np

from oracle import codec, constants as K, search
from oracle.rotation import rotation_matrix, rotation_mode
from paper_2608_30384_gb300 import workloads as W


def ue_near_tie(v, fmt: K.UEFormat, rel: float = 1e-9) -> np.ndarray:
    """Exact scale values within ``rel`` of a mantissa rounding tie."""
    v = np.asarray(v, dtype=np.float64)
    out = np.zeros(v.shape, dtype=bool)
    for i, x in enumerate(v.reshape(-1)):
        if not x > 0:
            continue
        f, e = np.frexp(x)
        m = (2 * f - 1) * (1 << fmt.mbits)
        frac = m - np.floor(m)
        out.reshape(-1)[i] = abs(frac - 0.5) < rel * (1 << fmt.mbits) * 2
    return out


class Case:
    """A workload, its oracle index and (lazily) its GPU index."""

    def __init__(self, w: W.Workload, nq: int | None = None, global_scale: bool = True, lite: bool = False,
                 reading: str = "B", full_vector: bool = False):
        self.w = w
        self.X, self.A = W.database(w)
        self.C = W.ivf_centroids(w, self.X, self.A)
        self.Q = W.queries(w, nq)
        self.global_scale = global_scale
        self.lite = lite
        self.reading = reading
        self.full_vector = full_vector
        self.oracle = search.build_index(self.X, np.arange(w.N), self.A, self.C, w.bits,
                                         w.rescore_bits, global_scale=global_scale, lite=lite,
                                         reading=reading, full_vector=full_vector)
        self._gpu = None

    def gpu_index(self, encode: bool = True):
        import torch
        from paper_2608_30384_gb300 import Index
        ix = Index(torch.from_numpy(self.C).cuda(), self.w.bits, self.w.rescore_bits, self.global_scale,
                   lite=self.lite, reading=self.reading, full_vector=self.full_vector)
        ix.reserve(torch.from_numpy(self.A).cuda())
        if encode:
            ix.encode(torch.from_numpy(self.X).cuda(), 0)
        torch.cuda.synchronize()
        return ix

    def import_oracle_codes(self, ix):
        import torch
        st = self.oracle.stage1
        pack = codec.pack_bits3 if self.w.bits == 3 else codec.pack_nibbles
        ix.import_codes(1, 0, torch.from_numpy(pack(st.codes)).cuda(),
                        torch.from_numpy(st.L_u16.astype(np.uint16)).cuda(),
                        torch.from_numpy(st.G_u16.astype(np.uint16)).cuda())
        if self.oracle.stage2 is not None:
            s2 = self.oracle.stage2
            ix.import_codes(2, 0, torch.from_numpy(codec.pack_nibbles(s2.codes)).cuda(),
                            torch.from_numpy(s2.L_u16.astype(np.uint16)).cuda(),
                            torch.from_numpy(s2.G_u16.astype(np.uint16)).cuda())
        torch.cuda.synchronize()

    def approximations(self):
        """The stage-1 and stage-2 approximations of every row (float64)."""
        A1 = self.C[self.A].astype(np.float64)
        if self.full_vector:
            A1 = np.zeros_like(A1)
        A2 = A1 if self.reading == "A" else self.oracle.stage1.recon
        return A1, A2

    # ---------------------------------------------------------- references
    def qnorm(self, i):
        return float(np.linalg.norm(self.Q[i]))

    def xnorm_max(self):
        return float(self.xnorm().max())

    def xnorm(self):
        """||x|| of every row (row ids are row indices)."""
        if not hasattr(self, "_xn"):
            self._xn = np.linalg.norm(self.X.astype(np.float64), axis=1)
        return self._xn

    def score_tol_of(self, i):
        """tol(score, row id) for query i: 1e-4 relative with the floor
        0.01 ||q|| ||x|| of that row (the largest ||x|| when the row is not known)."""
        from tests.lib_util import score_tol
        xn, qn = self.xnorm(), self.qnorm(i)
        return lambda s, j=None: float(score_tol(s, qn, xn[j] if j is not None else xn.max()))


def check_stage(gpu_codes, gpu_L, gpu_G, enc, X, A, bits, global_scale, name):
    """Encode parity of one stage (tolerance rules in test_gpu_parity's header):
    codes bit-exact except near a decision boundary (at most 1e-4 of them),
    scale codes exact except at rounding ties, and on rows with a boundary
    flip the scales the GPU's own codes imply.  Returns the rows without a
    code flip."""
    ng = enc.codes.shape[1]
    got = codec.unpack_bits3(gpu_codes, ng) if bits == 3 else codec.unpack_nibbles(gpu_codes, ng)
    mism = got != enc.codes
    near = codec.near_threshold(enc.u, bits, 1e-5)
    assert np.all(near[mism]), f"{name}: code mismatch away from a decision boundary"
    assert mism.sum() <= max(1, 1e-4 * mism.size), f"{name}: {mism.sum()} mismatched codes"
    ok = ~mism.any(1)
    for gv, ov, ex, fmt in ((gpu_L, enc.L_u16, enc.L_exact, K.UE7M9), (gpu_G, enc.G_u16, enc.G_exact, K.UE4M12)):
        bad = ok & (gv.astype(np.int64) != ov)
        if bad.any():
            tie = ue_near_tie(ex[bad], fmt)
            assert np.all(tie) and np.all(np.abs(gv[bad].astype(np.int64) - ov[bad]) <= 1), \
                f"{name}: {bad.sum()} scale codes differ away from rounding ties"
    # rows with a boundary code flip: the GPU's scales must be those its codes imply
    for r in np.nonzero(~ok)[0]:
        Lu, Gu, Le, Ge = codec.scales_from_codes(X[r:r + 1], A[r:r + 1], bits, got[r:r + 1], global_scale)
        assert abs(int(gpu_L[r]) - int(Lu[0])) <= (1 if ue_near_tie(Le, K.UE7M9)[0] else 0)
        assert abs(int(gpu_G[r]) - int(Gu[0])) <= (1 if ue_near_tie(Ge, K.UE4M12)[0] else 0)
    return ok


def check_lite_stage(gpu_codes, gpu_L, gpu_G, enc, X, A, global_scale, name):
    """Encode parity of Rslm4Lite scoring codes, with the rules of
    ``check_stage``: the level codes (K = 8 head, K = 16 tail) bit-exact
    except near their decision boundaries, the scale codes embedded in the
    head's top bits equal to the decoded pair the index keeps, and both equal
    to the oracle's except at rounding ties (or, on a row with a boundary
    flip, to the scales the GPU's own levels imply)."""
    D = enc.D
    H = codec.lite_head(global_scale)
    got = codec.unpack_nibbles(gpu_codes, D)
    lv, eL, eG = codec.unpack_lite(got, global_scale)
    assert np.array_equal(eL, gpu_L.astype(np.int64)), f"{name}: embedded UE7M9 code != kept scale"
    if global_scale:
        assert np.array_equal(eG, gpu_G.astype(np.int64)), f"{name}: embedded UE4M12 code != kept scale"
    olv, _, _ = codec.unpack_lite(enc.codes, global_scale)
    mism = lv != olv
    near = np.zeros_like(mism)
    for lo, hi, cb in ((0, H, K.codebook(3)), (H, D, K.codebook(4))):
        d = np.abs(enc.u[:, lo:hi, None] - cb.thresholds[None, None, :])
        near[:, lo:hi] = d.min(axis=-1) < 1e-5
    assert np.all(near[mism]), f"{name}: level mismatch away from a decision boundary"
    assert mism.sum() <= max(1, 1e-4 * mism.size), f"{name}: {mism.sum()} mismatched codes"
    ok = ~mism.any(1)
    for gv, ov, ex, fmt in ((gpu_L, enc.L_u16, enc.L_exact, K.UE7M9), (gpu_G, enc.G_u16, enc.G_exact, K.UE4M12)):
        bad = ok & (gv.astype(np.int64) != ov)
        if bad.any():
            tie = ue_near_tie(ex[bad], fmt)
            assert np.all(tie) and np.all(np.abs(gv[bad].astype(np.int64) - ov[bad]) <= 1), \
                f"{name}: {bad.sum()} scale codes differ away from rounding ties"
    for r in np.nonzero(~ok)[0]:
        # the scales the GPU's levels imply: steps 4-6 with those codewords
        uhat = np.empty(D)
        uhat[:H] = K.codebook(3).C[lv[r, :H], 0]
        uhat[H:] = K.codebook(4).C[lv[r, H:], 0]
        Rm = rotation_matrix(D, rotation_mode(4, D))
        rr = np.asarray(X[r], dtype=np.float64) - A[r]
        L = np.linalg.norm(rr) / np.linalg.norm(uhat)
        Lu = int(K.UE7M9.encode(np.array([L]))[0])
        assert abs(int(gpu_L[r]) - Lu) <= (1 if ue_near_tie(np.array([L]), K.UE7M9)[0] else 0)
        if global_scale:
            rt = K.UE7M9.decode(np.array([Lu]))[0] * (uhat @ Rm)
            G = np.linalg.norm(X[r]) / np.linalg.norm(A[r] + rt)
            Gu = int(K.UE4M12.encode(np.array([G]))[0])
            assert abs(int(gpu_G[r]) - Gu) <= (1 if ue_near_tie(np.array([G]), K.UE4M12)[0] else 0)
    return ok
