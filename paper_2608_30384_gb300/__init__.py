"""GB300-native RSLM residual-code IVF search (CUDA sm_103a, C ABI + ctypes).

The compute lives in ``librslm.so`` (sources in ``csrc/``, interface in
``include/rslm.h``); ``binding`` marshals torch tensors into its calls and
``index.Index`` bundles them for one index.  ``workloads`` generates the
seeded synthetic inputs.
"""

from .binding import (RSLM_GLOBAL_SCALE, RslmError, lib, rslm_codebook, rslm_e_max, rslm_encode,
                      rslm_export_codes, rslm_import_codes, rslm_index_create, rslm_index_describe,
                      rslm_index_reserve, rslm_last_error, rslm_probe, rslm_rescore,
                      rslm_rotate_queries, rslm_rotation_tables, rslm_scan, rslm_scan_batched, rslm_search,
                      rslm_sync)
from .index import Index

__all__ = [
    "RSLM_GLOBAL_SCALE", "RslmError", "Index", "lib", "rslm_codebook", "rslm_e_max", "rslm_encode",
    "rslm_export_codes", "rslm_import_codes", "rslm_index_create", "rslm_index_describe",
    "rslm_index_reserve", "rslm_last_error", "rslm_probe", "rslm_rescore", "rslm_rotate_queries",
    "rslm_rotation_tables", "rslm_scan", "rslm_scan_batched", "rslm_search", "rslm_sync",
]
