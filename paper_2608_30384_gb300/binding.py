"""Thin ctypes binding of librslm (include/rslm.h), same names as the C ABI.

Argument marshalling only: every step runs in the library's CUDA kernels.
Device arrays are torch CUDA tensors (contiguous, the dtype the header
states); ``stream`` defaults to torch's current stream.  A failing call
raises ``RslmError`` with the library's message.  There is no fallback: if
``librslm.so`` is missing the first call raises.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librslm.so")

RSLM_GLOBAL_SCALE = 1
RSLM_LITE = 2
RSLM_RESCORE_READING_A = 4
RSLM_FULL_VECTOR = 8
STATUS = {0: "RSLM_OK", 1: "RSLM_ERR_INVALID_ARG", 2: "RSLM_ERR_OUT_OF_MEMORY", 3: "RSLM_ERR_CUDA",
          4: "RSLM_ERR_TIMEOUT", 5: "RSLM_ERR_STATE", 6: "RSLM_ERR_DEVICE", 7: "RSLM_ERR_INTERNAL"}

# Every symbol of include/rslm.h with (restype, argtypes).
_P = ctypes.c_void_p
_I32, _I64, _U32, _D = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32, ctypes.c_double
SIGNATURES = {
    "rslm_index_create": (ctypes.c_int, [_I32, _I32, _P, _I32, _I32, _U32, _P, ctypes.POINTER(_P)]),
    "rslm_index_describe": (ctypes.c_int, [_P, _P]),
    "rslm_index_reserve": (ctypes.c_int, [_P, _P, _I64, _P]),
    "rslm_encode": (ctypes.c_int, [_P, _P, _I64, _I64, _P]),
    "rslm_encode_all": (ctypes.c_int, [_P, _P, _I64, _I32, _I32, _P, _I32, _I32, _U32, _P, ctypes.POINTER(_P)]),
    "rslm_rotate_queries": (ctypes.c_int, [_P, _I32, _P, _I64, _P, _P]),
    "rslm_probe": (ctypes.c_int, [_P, _P, _I64, _I32, _P, _P, _P]),
    "rslm_probe_noalloc": (ctypes.c_int, [_P, _P, _I64, _I32, _P, _P, _P]),
    "rslm_scan": (ctypes.c_int, [_P, _P, _I64, _P, _P, _I32, _I32, _P, _P, _P]),
    "rslm_scan_batched": (ctypes.c_int, [_P, _P, _I64, _P, _P, _I32, _I32, _P, _P, _P]),
    "rslm_rescore": (ctypes.c_int, [_P, _P, _I64, _P, _P, _I32, _I32, _P, _P, _P]),
    "rslm_search": (ctypes.c_int, [_P, _P, _I64, _I32, _I32, _I32, _I32, _P, _P, _P]),
    "rslm_export_codes": (ctypes.c_int, [_P, _I32, _I64, _I64, _P, _P, _P, _P]),
    "rslm_import_codes": (ctypes.c_int, [_P, _I32, _I64, _I64, _P, _P, _P, _P]),
    "rslm_codebook": (ctypes.c_int, [_I32, _P, _P, _P]),
    "rslm_rotation_tables": (ctypes.c_int, [_P, _P]),
    "rslm_e_max": (ctypes.c_int, [_I32, ctypes.POINTER(_D)]),
    "rslm_profile_enable": (ctypes.c_int, [_P, _I32]),
    "rslm_profile_read": (ctypes.c_int, [_P, ctypes.POINTER(_D), ctypes.POINTER(_I64), _P, _I32]),
    "rslm_decompress": (ctypes.c_int, [_P, _I32, _I64, _I64, _P, _P]),
    "rslm_sync": (ctypes.c_int, [_P, _P]),
    "rslm_counters": (ctypes.c_int, [_P, ctypes.POINTER(_I64), _I32]),
    "rslm_last_error": (ctypes.c_char_p, []),
    "rslm_index_destroy": (None, [_P]),
}


class RslmError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


class _Desc(ctypes.Structure):
    _fields_ = [(n, _I32) for n in (
        "dim", "nlist", "score_bits", "rescore_bits", "group", "padded_dim", "code_bytes",
        "rescore_group", "rescore_padded_dim", "rescore_code_bytes", "rotation_passes",
        "rescore_rotation_passes")] + [("n_rows", _I64), ("n_slots", _I64), ("device_bytes", _I64),
                                       ("flags", _U32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded librslm.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int):
    if status != 0:
        raise RslmError(status, lib().rslm_last_error().decode())


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def _dev(t, dtype, name, numel=None):
    """Device pointer of a contiguous CUDA tensor of the stated dtype (or None)."""
    if t is None:
        return None
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, needs {numel}")
    return t.data_ptr()


class IndexHandle:
    """Owner of an rslm_index*; destroyed with the object."""

    def __init__(self, ptr: int):
        self.ptr = ptr

    def __del__(self):
        if getattr(self, "ptr", None):
            try:
                lib().rslm_index_destroy(self.ptr)
            except Exception:
                pass
            self.ptr = None


def _ptr(index) -> int:
    return index.ptr if isinstance(index, IndexHandle) else index


def rslm_index_create(dim, nlist, centroids, score_bits, rescore_bits=0,
                      flags=RSLM_GLOBAL_SCALE, stream=None) -> IndexHandle:
    import torch
    out = _P()
    _check(lib().rslm_index_create(dim, nlist, _dev(centroids, torch.float32, "centroids", nlist * dim),
                                   score_bits, rescore_bits, flags, _stream(stream), ctypes.byref(out)))
    return IndexHandle(out.value)


def rslm_index_describe(index) -> dict:
    d = _Desc()
    _check(lib().rslm_index_describe(_ptr(index), ctypes.byref(d)))
    return {name: getattr(d, name) for name, _ in _Desc._fields_}


def rslm_index_reserve(index, assignment, stream=None):
    import torch
    _check(lib().rslm_index_reserve(_ptr(index), _dev(assignment, torch.int32, "assignment"),
                                    assignment.numel(), _stream(stream)))


def rslm_encode(index, vectors, row_begin, rows=None, stream=None):
    import torch
    rows = vectors.shape[0] if rows is None else rows
    _check(lib().rslm_encode(_ptr(index), _dev(vectors, torch.float32, "vectors"), row_begin, rows,
                             _stream(stream)))


def rslm_encode_all(vectors, assignment, centroids, score_bits, rescore_bits=0, flags=RSLM_GLOBAL_SCALE,
                    stream=None) -> IndexHandle:
    """Create, reserve and encode an index from vectors [n, dim] in one call."""
    import torch
    n, dim = vectors.shape
    nlist = centroids.shape[0]
    out = _P()
    _check(lib().rslm_encode_all(_dev(vectors, torch.float32, "vectors", n * dim),
                                 _dev(assignment, torch.int32, "assignment", n), n, dim, nlist,
                                 _dev(centroids, torch.float32, "centroids", nlist * dim), score_bits,
                                 rescore_bits, flags, _stream(stream), ctypes.byref(out)))
    return IndexHandle(out.value)


def rslm_rotate_queries(index, which, queries, out, stream=None):
    import torch
    _check(lib().rslm_rotate_queries(_ptr(index), which, _dev(queries, torch.float32, "queries"),
                                     queries.shape[0], _dev(out, torch.float32, "out"), _stream(stream)))


def rslm_probe(index, queries, nprobe, out_probes, out_cs, stream=None):
    import torch
    nq = queries.shape[0]
    _check(lib().rslm_probe(_ptr(index), _dev(queries, torch.float32, "queries"), nq, nprobe,
                            _dev(out_probes, torch.int32, "out_probes", nq * nprobe),
                            _dev(out_cs, torch.float32, "out_cs", nq * nprobe), _stream(stream)))


def rslm_probe_noalloc(index, queries, nprobe, out_probes, out_cs, stream=None):
    """rslm_probe with its scratch in the library's fixed device array (no allocation)."""
    import torch
    nq = queries.shape[0]
    _check(lib().rslm_probe_noalloc(_ptr(index), _dev(queries, torch.float32, "queries"), nq, nprobe,
                                    _dev(out_probes, torch.int32, "out_probes", nq * nprobe),
                                    _dev(out_cs, torch.float32, "out_cs", nq * nprobe),
                                    _stream(stream)))


def rslm_scan(index, qrot, probes, cs, k, out_ids, out_scores, stream=None):
    import torch
    nq, nprobe = probes.shape
    _check(lib().rslm_scan(_ptr(index), _dev(qrot, torch.float32, "qrot"), nq,
                           _dev(probes, torch.int32, "probes"), _dev(cs, torch.float32, "cs"), nprobe, k,
                           _dev(out_ids, torch.int64, "out_ids", nq * k),
                           _dev(out_scores, torch.float32, "out_scores", nq * k), _stream(stream)))


def rslm_scan_batched(index, qrot, probes, cs, k, out_ids, out_scores, stream=None):
    import torch
    nq, nprobe = probes.shape
    _check(lib().rslm_scan_batched(_ptr(index), _dev(qrot, torch.float32, "qrot"), nq,
                                   _dev(probes, torch.int32, "probes"), _dev(cs, torch.float32, "cs"),
                                   nprobe, k, _dev(out_ids, torch.int64, "out_ids", nq * k),
                                   _dev(out_scores, torch.float32, "out_scores", nq * k),
                                   _stream(stream)))


def rslm_rescore(index, qrot2, cand_ids, cand_scores, k_final, out_ids, out_scores, stream=None):
    import torch
    nq, k = cand_ids.shape
    _check(lib().rslm_rescore(_ptr(index), _dev(qrot2, torch.float32, "qrot2"), nq,
                              _dev(cand_ids, torch.int64, "cand_ids"),
                              _dev(cand_scores, torch.float32, "cand_scores"), k, k_final,
                              _dev(out_ids, torch.int64, "out_ids", nq * k_final),
                              _dev(out_scores, torch.float32, "out_scores", nq * k_final),
                              _stream(stream)))


def rslm_search(index, queries, nprobe, k, rescore, k_final, out_ids, out_scores, stream=None):
    import torch
    nq = queries.shape[0]
    _check(lib().rslm_search(_ptr(index), _dev(queries, torch.float32, "queries"), nq, nprobe, k,
                             int(bool(rescore)), k_final,
                             _dev(out_ids, torch.int64, "out_ids", nq * k_final),
                             _dev(out_scores, torch.float32, "out_scores", nq * k_final),
                             _stream(stream)))


def rslm_export_codes(index, which, row_begin, rows, codes, local_scale, global_scale, stream=None):
    import torch
    _check(lib().rslm_export_codes(_ptr(index), which, row_begin, rows,
                                   _dev(codes, torch.uint8, "codes"),
                                   _dev(local_scale, torch.uint16, "local_scale", rows),
                                   _dev(global_scale, torch.uint16, "global_scale", rows),
                                   _stream(stream)))


def rslm_import_codes(index, which, row_begin, rows, codes, local_scale, global_scale, stream=None):
    import torch
    _check(lib().rslm_import_codes(_ptr(index), which, row_begin, rows,
                                   _dev(codes, torch.uint8, "codes"),
                                   _dev(local_scale, torch.uint16, "local_scale", rows),
                                   _dev(global_scale, torch.uint16, "global_scale", rows),
                                   _stream(stream)))


def rslm_codebook(bits) -> np.ndarray:
    out = np.zeros(64, dtype=np.float32)
    K, g = ctypes.c_int32(), ctypes.c_int32()
    _check(lib().rslm_codebook(bits, out.ctypes.data, ctypes.byref(K), ctypes.byref(g)))
    return out[:K.value * g.value].reshape(K.value, g.value)


def rslm_rotation_tables():
    s1 = np.zeros(256, dtype=np.int8)
    perm = np.zeros(128, dtype=np.int32)
    _check(lib().rslm_rotation_tables(s1.ctypes.data, perm.ctypes.data))
    return s1, perm


def rslm_e_max(dim) -> float:
    v = ctypes.c_double()
    _check(lib().rslm_e_max(dim, ctypes.byref(v)))
    return v.value


def rslm_profile_enable(index, on=True):
    _check(lib().rslm_profile_enable(_ptr(index), int(bool(on))))


def rslm_decompress(index, which, row_begin, rows, out, stream=None):
    """Reconstructions of rows [row_begin, row_begin + rows) of stage ``which`` into out [rows, dim]."""
    import torch
    dim = rslm_index_describe(index)["dim"]
    _check(lib().rslm_decompress(_ptr(index), which, row_begin, rows,
                                 _dev(out, torch.float32, "out", rows * dim), _stream(stream)))


def rslm_profile_read(index):
    """(total kernel ms, launches, kernel name) recorded since enable / last read."""
    ms, n = ctypes.c_double(), ctypes.c_int64()
    name = ctypes.create_string_buffer(64)
    _check(lib().rslm_profile_read(_ptr(index), ctypes.byref(ms), ctypes.byref(n), name, 64))
    return ms.value, n.value, name.value.decode()


def rslm_sync(index, stream=None):
    _check(lib().rslm_sync(_ptr(index), _stream(stream)))


COUNTERS = ("batched_short_rescans", "batched_overflow_rescans", "probe_exact_fallbacks", "hi_exact_rescores")


def rslm_counters(index) -> dict:
    """Event counters of the index since creation (waits for the device)."""
    out = (_I64 * 4)()
    _check(lib().rslm_counters(_ptr(index), out, 4))
    return dict(zip(COUNTERS, (int(v) for v in out)))


def rslm_last_error() -> str:
    return lib().rslm_last_error().decode()
