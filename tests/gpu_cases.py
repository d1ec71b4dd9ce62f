"""Shared builders for the GPU parity tests: one synthetic case on both sides."""

from __future__ import annotations

import numpy as np

from oracle import codec, constants as K, search
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

    def __init__(self, w: W.Workload, nq: int | None = None, global_scale: bool = True):
        self.w = w
        self.X, self.A = W.database(w)
        self.C = W.ivf_centroids(w, self.X, self.A)
        self.Q = W.queries(w, nq)
        self.global_scale = global_scale
        self.oracle = search.build_index(self.X, np.arange(w.N), self.A, self.C, w.bits,
                                         w.rescore_bits, global_scale=global_scale)
        self._gpu = None

    def gpu_index(self, encode: bool = True):
        import torch
        from paper_2608_30384_gb300 import Index
        ix = Index(torch.from_numpy(self.C).cuda(), self.w.bits, self.w.rescore_bits, self.global_scale)
        ix.reserve(torch.from_numpy(self.A).cuda())
        if encode:
            ix.encode(torch.from_numpy(self.X).cuda(), 0)
        torch.cuda.synchronize()
        return ix

    def import_oracle_codes(self, ix):
        import torch
        st = self.oracle.stage1
        ix.import_codes(1, 0, torch.from_numpy(codec.pack_nibbles(st.codes)).cuda(),
                        torch.from_numpy(st.L_u16.astype(np.uint16)).cuda(),
                        torch.from_numpy(st.G_u16.astype(np.uint16)).cuda())
        if self.oracle.stage2 is not None:
            s2 = self.oracle.stage2
            ix.import_codes(2, 0, torch.from_numpy(codec.pack_nibbles(s2.codes)).cuda(),
                            torch.from_numpy(s2.L_u16.astype(np.uint16)).cuda(),
                            torch.from_numpy(s2.G_u16.astype(np.uint16)).cuda())
        torch.cuda.synchronize()

    # ---------------------------------------------------------- references
    def qnorm(self, i):
        return float(np.linalg.norm(self.Q[i]))

    def xnorm_max(self):
        return float(np.linalg.norm(self.X.astype(np.float64), axis=1).max())
