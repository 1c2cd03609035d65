"""The comparisons the GPU parity tests make (tests/harness.py) reject what
they must: results outside the stated tolerances, NaN, and shape mismatches.
A comparator that let such results through would make every parity test
vacuous, so it is checked here on the CPU with planted errors."""

import numpy as np
import pytest

from harness import ATTN_MAX_ABS, ATTN_REL_L2, FEAT_FLOOR, FEAT_RTOL, check_attention, close_rel


def test_attention_check_bounds():
    rng = np.random.default_rng(0)
    ref = rng.standard_normal((4, 128)) * 0.1
    check_attention(ref.copy(), ref, "equal")
    one = ref.copy()
    one[2, 7] += 0.9 * ATTN_MAX_ABS            # inside both bounds
    check_attention(one, ref, "one entry inside")
    one[2, 7] = ref[2, 7] + 1.1 * ATTN_MAX_ABS  # one entry past max-abs (rel-L2 still small)
    assert np.linalg.norm(one - ref) / np.linalg.norm(ref) < ATTN_REL_L2
    with pytest.raises(AssertionError, match="max-abs"):
        check_attention(one, ref, "one entry outside")
    scaled = ref * (1 + 1.2 * ATTN_REL_L2)        # rel-L2 past its bound, max-abs far inside
    assert np.max(np.abs(scaled - ref)) < ATTN_MAX_ABS
    with pytest.raises(AssertionError, match="rel-L2"):
        check_attention(scaled, ref, "scaled")
    nan = ref.copy()
    nan[0, 0] = np.nan
    with pytest.raises(AssertionError):
        check_attention(nan, ref, "nan")
    with pytest.raises(AssertionError):
        check_attention(ref[0], ref, "broadcast")


def test_feature_check_bounds():
    rng = np.random.default_rng(1)
    ref = rng.uniform(1.0, 2.0, 300)
    close_rel(ref * (1 + 0.9 * FEAT_RTOL), ref, FEAT_RTOL, FEAT_FLOOR, "inside")
    with pytest.raises(AssertionError, match="1/300"):
        bad = ref.copy()
        bad[17] *= 1 + 3 * FEAT_RTOL                 # past rtol + floor (floor <= 2e-3 here)
        close_rel(bad, ref, FEAT_RTOL, FEAT_FLOOR, "one outside")
    # near-zero values are held to the floor: 1e-3 x the column's RMS
    tiny = np.concatenate([ref, [0.0]])
    rms = np.sqrt(np.mean(tiny ** 2))
    close_rel(np.concatenate([ref, [0.5 * FEAT_FLOOR * rms]]), tiny, FEAT_RTOL, FEAT_FLOOR, "zero inside floor")
    with pytest.raises(AssertionError):
        close_rel(np.concatenate([ref, [2.0 * FEAT_FLOOR * rms]]), tiny, FEAT_RTOL, FEAT_FLOOR, "zero past floor")
    with pytest.raises(AssertionError):
        close_rel(np.where(np.arange(300) == 5, np.nan, ref), ref, FEAT_RTOL, FEAT_FLOOR, "nan")
    with pytest.raises(AssertionError):
        close_rel(ref[:-1], ref, FEAT_RTOL, FEAT_FLOOR, "shape")
