"""One RSLM index on the GPU: the C-ABI calls of ``binding`` bound to a handle."""

from __future__ import annotations

from . import binding as B


class Index:
    """IVF index with RSLM residual codes (create, reserve, encode, search).

    ``centroids`` is a CUDA float32 tensor [nlist, dim]; outputs are allocated
    on the centroids' device.
    """

    def __init__(self, centroids, score_bits: int, rescore_bits: int = 0, global_scale: bool = True,
                 stream=None, lite: bool = False, reading: str = "B", full_vector: bool = False):
        nlist, dim = centroids.shape
        self.device = centroids.device
        if reading not in ("A", "B"):
            raise ValueError("reading is 'A' or 'B'")
        flags = ((B.RSLM_GLOBAL_SCALE if global_scale else 0) | (B.RSLM_LITE if lite else 0)
                 | (B.RSLM_RESCORE_READING_A if reading == "A" else 0)
                 | (B.RSLM_FULL_VECTOR if full_vector else 0))
        self.handle = B.rslm_index_create(dim, nlist, centroids.contiguous(), score_bits, rescore_bits,
                                          flags, stream)

    @property
    def desc(self) -> dict:
        return B.rslm_index_describe(self.handle)

    def reserve(self, assignment, stream=None):
        B.rslm_index_reserve(self.handle, assignment.contiguous(), stream)

    def encode(self, vectors, row_begin: int = 0, stream=None):
        B.rslm_encode(self.handle, vectors.contiguous(), row_begin, vectors.shape[0], stream)

    def search(self, queries, nprobe: int, k: int, rescore: bool | None = None,
               k_final: int | None = None, out=None, stream=None):
        import torch
        d = self.desc
        rescore = bool(d["rescore_bits"]) if rescore is None else rescore
        k_final = k if k_final is None else k_final
        nq = queries.shape[0]
        if out is None:
            out = (torch.empty((nq, k_final), dtype=torch.int64, device=queries.device),
                   torch.empty((nq, k_final), dtype=torch.float32, device=queries.device))
        B.rslm_search(self.handle, queries, nprobe, k, rescore, k_final, out[0], out[1], stream)
        return out

    def probe(self, queries, nprobe: int, stream=None):
        import torch
        nq = queries.shape[0]
        p = torch.empty((nq, nprobe), dtype=torch.int32, device=queries.device)
        c = torch.empty((nq, nprobe), dtype=torch.float32, device=queries.device)
        B.rslm_probe(self.handle, queries, nprobe, p, c, stream)
        return p, c

    def rotate(self, queries, which: int = 1, stream=None):
        import torch
        d = self.desc
        width = d["padded_dim"] if which == 1 else d["rescore_padded_dim"]
        out = torch.empty((queries.shape[0], width), dtype=torch.float32, device=queries.device)
        B.rslm_rotate_queries(self.handle, which, queries, out, stream)
        return out

    def scan(self, qrot, probes, cs, k: int, stream=None):
        import torch
        nq = probes.shape[0]
        ids = torch.empty((nq, k), dtype=torch.int64, device=probes.device)
        sc = torch.empty((nq, k), dtype=torch.float32, device=probes.device)
        B.rslm_scan(self.handle, qrot, probes, cs, k, ids, sc, stream)
        return ids, sc

    def scan_batched(self, qrot, probes, cs, k: int, stream=None):
        import torch
        nq = probes.shape[0]
        ids = torch.empty((nq, k), dtype=torch.int64, device=probes.device)
        sc = torch.empty((nq, k), dtype=torch.float32, device=probes.device)
        B.rslm_scan_batched(self.handle, qrot, probes, cs, k, ids, sc, stream)
        return ids, sc

    def rescore(self, qrot2, cand_ids, cand_scores, k_final: int, stream=None):
        import torch
        nq = cand_ids.shape[0]
        ids = torch.empty((nq, k_final), dtype=torch.int64, device=cand_ids.device)
        sc = torch.empty((nq, k_final), dtype=torch.float32, device=cand_ids.device)
        B.rslm_rescore(self.handle, qrot2, cand_ids, cand_scores, k_final, ids, sc, stream)
        return ids, sc

    def export_codes(self, which: int = 1, row_begin: int = 0, rows: int | None = None, stream=None):
        import torch
        d = self.desc
        rows = d["n_rows"] - row_begin if rows is None else rows
        nb = d["code_bytes"] if which == 1 else d["rescore_code_bytes"]
        codes = torch.empty((rows, nb), dtype=torch.uint8, device=self.device)
        L = torch.empty(rows, dtype=torch.uint16, device=self.device)
        G = torch.empty(rows, dtype=torch.uint16, device=self.device)
        B.rslm_export_codes(self.handle, which, row_begin, rows, codes, L, G, stream)
        return codes, L, G

    def decompress(self, which: int = 1, row_begin: int = 0, rows: int | None = None, stream=None):
        """Reconstructed vectors [rows, dim] of stage ``which`` (float32)."""
        import torch
        d = self.desc
        rows = d["n_rows"] - row_begin if rows is None else rows
        out = torch.empty((rows, d["dim"]), dtype=torch.float32, device=self.device)
        B.rslm_decompress(self.handle, which, row_begin, rows, out, stream)
        return out

    def import_codes(self, which, row_begin, codes, L, G, stream=None):
        B.rslm_import_codes(self.handle, which, row_begin, codes.shape[0], codes.contiguous(),
                            L.contiguous(), G.contiguous(), stream)

    def sync(self, stream=None):
        B.rslm_sync(self.handle, stream)

    def counters(self) -> dict:
        return B.rslm_counters(self.handle)
