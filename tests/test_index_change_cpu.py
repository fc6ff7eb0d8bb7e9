"""The level-index statistics of the reconstruction loop (the paper's Table 2:
shares of weights whose level index moves by 0, 1, 2 and more than 2),
computed on torch tensors by recon.level_ranks / index_change_shares, against
the oracle's sorted level order (oracle.sorted_levels: ascending, equal levels
in code-word order).  Runs on CPU tensors."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300.recon import index_change_shares, level_ranks

F32 = np.float32


@pytest.mark.parametrize("q,g", [(1, 32), (2, 64), (3, 128), (4, 32)])
def test_level_ranks_match_the_oracle_order(q, g):
    rng = np.random.default_rng(q * 10 + g)
    out, n_in = 5, 4 * g
    Gr = n_in // g
    alpha = rng.uniform(0.2, 1.2, (out, Gr, q)).astype(F32)
    alpha[0, :, :] = np.float32(0.5)                  # every alpha equal: many equal levels
    if q >= 2:
        alpha[1, :, 1] = alpha[1, :, 0]               # alpha_1 = alpha_2: pairs of equal levels
        alpha[2, :, q - 1] *= -1                      # a negative alpha reorders the levels
    zb = rng.uniform(-1, 1, (out, Gr)).astype(F32)
    codes = rng.integers(0, 256, (out, n_in)).astype(np.uint8)   # high bits must be ignored
    r = level_ranks(torch.from_numpy(alpha), torch.from_numpy(zb), torch.from_numpy(codes), g).numpy()
    _, _, rank_of_code = O.sorted_levels(O.levels(alpha, zb))
    want = np.take_along_axis(rank_of_code, (codes.reshape(out, Gr, g) & ((1 << q) - 1)).astype(np.int64),
                              axis=-1).reshape(out, n_in)
    assert np.array_equal(r, want)


def test_index_change_shares_bins():
    a = torch.tensor([0, 1, 2, 3, 7, 5, 0, 15], dtype=torch.uint8)
    b = torch.tensor([0, 2, 0, 7, 7, 4, 3, 0], dtype=torch.uint8)
    # |a - b| = 0, 1, 2, 4, 0, 1, 3, 15
    assert index_change_shares(a, b) == [2 / 8, 2 / 8, 1 / 8, 3 / 8]
    assert sum(index_change_shares(a, a)) == 1.0 and index_change_shares(a, a)[0] == 1.0
