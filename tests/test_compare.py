"""CPU checks of the parity tests' comparison helpers (no GPU): the per-row
check catches a wrong low-magnitude row that the infinity-norm bound alone
passes, and the tile-coverage count is right on a hand-built permutation."""
import numpy as np
import pytest

import oracle
from gpu_helpers import assert_close, error_report, rel_err, tiles_covered


def test_per_row_check_fails_a_wrong_small_row():
    rng = np.random.default_rng(1)
    ref = rng.standard_normal((64, 256))
    ref[7] *= 0.01  # a small row
    got = ref.copy()
    got[7] = -got[7]  # that row wrong (sign flipped)
    assert rel_err(got, ref) <= 2e-2  # the infinity-norm bound alone passes it
    rep = error_report(got, ref)
    assert rep["worst_rows"][0][0] == 7 and rep["row_max"] > 2e-2
    with pytest.raises(AssertionError):
        assert_close(got, ref, 2e-2)
    assert_close(ref * (1 + 1e-3), ref, 2e-2)  # a uniformly close answer passes


def test_tiles_covered_counts_expert_tiles():
    # 3 tokens x 2 slots; expert 0 gets 4 pairs, expert 2 gets 2 (tile height 2)
    ids = np.array([[0, 2], [0, 0], [2, 0]], np.int32)
    counts, offsets, sp, _ = oracle.permute(ids, 3)
    assert tiles_covered(ids, np.arange(3), counts, sp, offsets, bm=2) == (3, 3)
    # token 2 alone: pairs 4 (expert 2) and 5 (expert 0, its second tile)
    assert tiles_covered(ids, np.array([2]), counts, sp, offsets, bm=2) == (2, 3)
