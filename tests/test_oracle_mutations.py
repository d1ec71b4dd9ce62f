"""The oracle's pins catch plausible mistakes (CPU).

Each case plants one mistake in the oracle (a dropped term, a wrong sign,
index or offset, a transposed operand, a wrong rounding or tie rule, a
wrong bit order) through monkeypatch, and requires at least one of the
existing pin tests to fail on the mutated oracle.  The mistakes live only
in this process for the duration of one test; the oracle's caches are
cleared before and after so no mutated table leaks into another test.
"""

import math

import numpy as np
import pytest

import tests.test_oracle_codec as TC
import tests.test_oracle_constants as TK
import tests.test_oracle_lite as TL
import tests.test_oracle_relative as TRel
import tests.test_oracle_rotation as TR
from oracle import codec, constants as K, rotation, search


def _clear_caches():
    for fn in (rotation.rotation_matrix, rotation.hadamard_unnormalized, K.sign_table_s1, K.sign_table_s2,
               K.codebook, K.e_max):
        if hasattr(fn, "cache_clear"):
            fn.cache_clear()


@pytest.fixture
def mutate(monkeypatch):
    _clear_caches()
    yield monkeypatch
    monkeypatch.undo()
    _clear_caches()


def _caught(*calls):
    """True when at least one pin test fails on the mutated oracle."""
    for fn, args in calls:
        try:
            fn(*args)
        except AssertionError:
            return True
    return False


def test_pins_pass_on_the_unmutated_oracle(mutate):
    assert not _caught((TC.test_evt_normalisation_and_nearest_codeword, (4, 128)),
                       (TC.test_norm_correction_invariants, (4, 128)),
                       (TC.test_score_identity_equals_explicit_reconstruction, ()),
                       (TC.test_rslm3_packing_by_hand_and_round_trip, ()),
                       (TC.test_probe_order_and_padding, ()),
                       (TK.test_ue7m9_and_ue4m12_formats, ()),
                       (TK.test_1d_assignment_tie_goes_up, ()),
                       (TR.test_matches_factor_product, (300, "two")),
                       (TL.test_scale_bits_in_the_top_bits, (True,)),
                       (TRel.test_reading_a_codes_are_the_finer_codec_of_x_minus_c, ()),
                       (TRel.test_rescore_score_identity, ("B",)),
                       (TRel.test_full_vector_codes_encode_x_itself, ()),
                       (TR.test_mode_rule, ()),
                       (TR.test_orthogonal_and_inverse, (96, "single")),
                       (TR.test_overlap_block_is_applied_last, ()))


def test_transposed_rotation_in_the_codec(mutate):
    orig = codec.rotation_matrix
    mutate.setattr(codec, "rotation_matrix", lambda D, mode: orig(D, mode).T)
    assert _caught((TC.test_evt_normalisation_and_nearest_codeword, (4, 128)),
                   (TC.test_norm_correction_invariants, (4, 128)))


def test_dropped_global_scale_term(mutate):
    orig = codec.encode

    def no_global(X, A, bits, global_scale=True, **kw):
        return orig(X, A, bits, global_scale=False, **kw)

    mutate.setattr(codec, "encode", no_global)
    assert _caught((TC.test_norm_correction_invariants, (4, 128)))


def test_evt_scale_for_the_wrong_dimension(mutate):
    orig = codec.e_max
    mutate.setattr(codec, "e_max", lambda D: orig(D + 1))
    assert _caught((TC.test_evt_normalisation_and_nearest_codeword, (4, 128)))


def test_scale_codes_rounded_down(mutate):
    def floor_one(self, v):
        v = float(v)
        if not v > 0.0:
            return 0
        f, k = math.frexp(v)
        m = int(math.floor((2.0 * f - 1.0) * (1 << self.mbits)))
        be = k - 1 + self.bias
        if be <= 0:
            return 0
        if be > self.emax:
            return (self.emax << self.mbits) | ((1 << self.mbits) - 1)
        return (be << self.mbits) | m

    mutate.setattr(K.UEFormat, "encode_one", floor_one)
    assert _caught((TK.test_ue7m9_and_ue4m12_formats, ()))


def test_threshold_ties_go_down(mutate):
    orig = K.Codebook.assign

    def assign_left(self, U):
        if self.g == 1:
            return np.searchsorted(self.thresholds, U[..., 0], side="left").astype(np.int64)
        return orig(self, U)

    mutate.setattr(K.Codebook, "assign", assign_left)
    assert _caught((TK.test_1d_assignment_tie_goes_up, ()))


def test_stage1_score_without_the_centroid_term(mutate):
    def no_cq(index, q, probes, cs):
        return orig(index, q, probes, np.zeros_like(np.asarray(cs, dtype=np.float64)))

    orig = search.stage1_scores
    mutate.setattr(search, "stage1_scores", no_cq)
    assert _caught((TC.test_score_identity_equals_explicit_reconstruction, ()))


def test_rslm3_bits_most_significant_first(mutate):
    def pack_msb(codes):
        codes = np.asarray(codes, dtype=np.int64)
        n, ng = codes.shape
        nb = (3 * ng + 7) // 8
        out = np.zeros((n, nb), dtype=np.uint8)
        for i in range(ng):
            for b in range(3):
                bit = 3 * i + b
                out[:, bit // 8] |= (((codes[:, i] >> (2 - b)) & 1) << (bit % 8)).astype(np.uint8)
        return out

    mutate.setattr(codec, "pack_bits3", pack_msb)
    assert _caught((TC.test_rslm3_packing_by_hand_and_round_trip, ()))


def test_second_sign_table_offset_by_128(mutate):
    mutate.setattr(rotation, "sign_table_s2", lambda: np.roll(K.sign_table_s1(), -128))
    assert _caught((TR.test_matches_factor_product, (300, "two")),
                   (TR.test_matches_factor_product, (1536, "two")))


def test_ties_ordered_by_descending_id(mutate):
    mutate.setattr(search, "order_desc", lambda scores, ids: np.lexsort((-ids, -scores)))
    assert _caught((TC.test_probe_order_and_padding, ()),
                   (TC.test_empty_partition_and_fewer_candidates_than_k, ()))


def test_lite_scale_bits_one_code_late(mutate):
    orig = codec.encode_lite

    def shifted(X, A, global_scale=True):
        enc = orig(X, A, global_scale)
        codes = enc.codes.copy()
        top = (codes[:, :16] >> 3) & 1
        codes[:, :16] = (codes[:, :16] & 7) | (np.roll(top, 1, axis=1) << 3)
        enc.codes = codes
        return enc

    mutate.setattr(codec, "encode_lite", shifted)
    assert _caught((TL.test_scale_bits_in_the_top_bits, (True,)))


def test_reading_a_built_as_reading_b(mutate):
    orig = search.build_index

    def always_b(*args, **kw):
        kw["reading"] = "B"
        return orig(*args, **kw)

    mutate.setattr(search, "build_index", always_b)
    assert _caught((TRel.test_reading_a_codes_are_the_finer_codec_of_x_minus_c, ()))


def test_rescoring_without_its_global_scale(mutate):
    orig = search.rescore

    def no_g2(index, *args):
        st = index.stage2
        saved = st.Ghat
        st.Ghat = np.ones_like(saved)
        try:
            return orig(index, *args)
        finally:
            st.Ghat = saved

    mutate.setattr(search, "rescore", no_g2)
    assert _caught((TRel.test_rescore_score_identity, ("B",)), (TRel.test_rescore_score_identity, ("A",)))


def test_full_vector_scores_keep_the_centroid_term(mutate):
    orig = search.stage1_scores

    def with_cq(index, *args):
        saved = index.full_vector
        index.full_vector = False
        try:
            return orig(index, *args)
        finally:
            index.full_vector = saved

    mutate.setattr(search, "stage1_scores", with_cq)
    assert _caught((TRel.test_full_vector_codes_encode_x_itself, ()))


def test_rotation_mode_rule_flipped(mutate):
    mutate.setattr(rotation, "rotation_mode", lambda bits, D: "two" if bits == 4 else "single")
    assert _caught((TR.test_mode_rule, ()))


def test_hadamard_left_unnormalised(mutate):
    mutate.setattr(rotation, "hadamard", rotation.hadamard_unnormalized)
    assert _caught((TR.test_orthogonal_and_inverse, (96, "single")))


def test_overlapping_block_applied_first(mutate):
    orig = rotation.block_starts

    def overlap_first(D):
        s = orig(D)
        return s[-1:] + s[:-1] if D % rotation.block_size(D) else s

    mutate.setattr(rotation, "block_starts", overlap_first)
    assert _caught((TR.test_overlap_block_is_applied_last, ()))
