"""librslm.so on the CPU: symbols, host-side tables, argument checks (no GPU calls).

The library's tables are computed by its own C++ code; the oracle's by
NumPy.  Agreement here means two independent implementations of the same
definitions produce the same bits.
"""

import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from oracle import constants as K
from tests.lib_util import ROOT, ensure_library


@pytest.fixture(scope="module")
def L():
    ensure_library()
    from paper_2608_30384_gb300 import binding
    return binding


def _declared_symbols():
    txt = open(os.path.join(ROOT, "include", "rslm.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(rslm_[a-z_0-9]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(L):
    names = _declared_symbols()
    assert len(names) >= 15
    lib = L.lib()
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(L.SIGNATURES)


def test_codebooks_match_oracle_bit_for_bit(L):
    for bits in (1, 2, 3, 4):
        cb = L.rslm_codebook(bits)
        ref = K.codebook(bits).C
        assert cb.shape == ref.shape
        assert np.array_equal(cb.astype(np.float64), ref), bits


def test_rotation_tables_match_oracle(L):
    s1, perm = L.rslm_rotation_tables()
    assert np.array_equal(s1.astype(np.float64), K.sign_table_s1())
    assert tuple(perm.tolist()) == K.perm_p128()


@pytest.mark.parametrize("D", [1, 2, 96, 100, 128, 768, 1536, 4096])
def test_e_max_matches_oracle(L, D):
    assert abs(L.rslm_e_max(D) - K.e_max(D)) < 1e-12


def test_argument_checks_need_no_gpu(L):
    lib = L.lib()
    out = ctypes.c_void_p()
    dummy = ctypes.c_void_p(16)
    # bad dim, nlist, bits, rescore bits; an unknown flag; RSLM_LITE below
    # D = 64 or with 2-bit codes; RSLM_RESCORE_READING_A without rescoring codes
    cases = [(0, 4, 4, 0, 1), (4097, 4, 4, 0, 1), (64, 0, 4, 0, 1), (64, 4, 5, 0, 1), (64, 4, 3, 0, 2),
             (64, 4, 4, 2, 1), (64, 4, 4, 0, 16), (48, 4, 4, 0, 2), (64, 4, 2, 0, 2), (64, 4, 4, 0, 4)]
    for dim, nlist, bits, rb, flags in cases:
        st = lib.rslm_index_create(dim, nlist, dummy, bits, rb, flags, None, ctypes.byref(out))
        assert st == 1, (dim, nlist, bits, rb, flags)
        assert out.value is None
        assert L.rslm_last_error()
    st = lib.rslm_index_create(64, 4, None, 4, 0, 1, None, ctypes.byref(out))
    assert st == 1 and "centroids" in L.rslm_last_error()
    # the one-shot encode checks its arguments before any device work
    st = lib.rslm_encode_all(dummy, dummy, 10, 64, 4, dummy, 4, 0, 1, None, None)
    assert st == 1 and "out" in L.rslm_last_error()
    st = lib.rslm_encode_all(None, dummy, 10, 64, 4, dummy, 4, 0, 1, None, ctypes.byref(out))
    assert st == 1 and "vectors" in L.rslm_last_error() and out.value is None
    st = lib.rslm_encode_all(dummy, dummy, 10, 0, 4, dummy, 4, 0, 1, None, ctypes.byref(out))
    assert st == 1 and out.value is None
    assert lib.rslm_e_max(0, ctypes.byref(ctypes.c_double())) == 1
    with pytest.raises(L.RslmError):
        L.rslm_codebook(5)


def test_generated_codebook_header_is_reproducible(tmp_path):
    """The committed codebooks_multid.inc is what gen_codebooks.cpp writes."""
    src = os.path.join(ROOT, "paper_2608_30384_gb300", "csrc", "gen_codebooks.cpp")
    exe = tmp_path / "gen"
    subprocess.run(["g++", "-O2", "-std=c++17", src, "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    committed = open(os.path.join(ROOT, "paper_2608_30384_gb300", "csrc", "codebooks_multid.inc")).read()
    assert out == committed
