"""Host checks of the parity harness's own helpers (no GPU): the pooled oracle top-K returns
what the oracle returns row by row, and the near-tie neighbours of a residual draw are the ids
with residual mass on either side."""
import numpy as np

from oracle import brisk_oracle as O

import oracle_pool
from parity import residual_neighbours


def test_pooled_topk_equals_the_oracle_row_by_row():
    rng = np.random.default_rng(3)
    rows = rng.normal(size=(70, 997)).astype(np.float32)
    rows[5, :] = 1.0                      # all ties
    rows[9, ::2] = -np.inf
    ids, lp, lse = oracle_pool.topk_all_rows(rows, 8, workers=2)
    for j in range(rows.shape[0]):
        o_ids, o_lp, o_lse = O.topk_candidates(rows[j].astype(np.float64), 8)
        np.testing.assert_array_equal(ids[j], o_ids)
        np.testing.assert_array_equal(lp[j], o_lp)
        assert lse[j] == o_lse


def test_residual_neighbours_skip_ids_without_mass():
    row = np.log(np.array([0.1, 0.2, 0.05, 0.3, 0.35]))
    # the proposal puts more mass than p on ids 1 and 3: their residual is 0
    below, above = residual_neighbours(row, [1, 3], [0.5, 0.5], 2)
    assert (below, above) == (0, 4)
    assert residual_neighbours(row, [1, 3], [0.5, 0.5], 0) == (None, 2)
    assert residual_neighbours(row, [1, 3], [0.5, 0.5], 4) == (2, None)
