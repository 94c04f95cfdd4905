"""GPU acceptance counts (Sec. 3.2: the profile is estimated from how far verification reached)
against the oracle, bit for bit."""
import numpy as np
import pytest
import torch

from oracle import acceptance as A

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


@pytest.mark.parametrize("Bn,L", [(1, 1), (5, 4), (128, 32), (1000, 64), (70000, 8)])
def test_counts_match_oracle_over_several_steps(B, Bn, L):
    rng = np.random.default_rng(Bn + L)
    counts = torch.zeros(2 * L, dtype=torch.int64, device="cuda")
    all_lens = []
    for step in range(3):
        lens = rng.integers(0, L + 1, Bn).astype(np.int32)
        all_lens.append(lens)
        B.acceptance_counts(torch.from_numpy(lens).cuda(), L, counts)
    torch.cuda.synchronize()
    reach, accept = A.accept_counts(np.concatenate(all_lens), L)
    got = counts.cpu().numpy()
    assert got[:L].tolist() == reach.tolist()
    assert got[L:].tolist() == accept.tolist()


def test_out_of_range_lengths_are_clamped_and_empty_batch_is_a_no_op(B):
    L = 6
    counts = torch.zeros(2 * L, dtype=torch.int64, device="cuda")
    B.acceptance_counts(torch.tensor([-3, 9, 2], dtype=torch.int32, device="cuda"), L, counts)
    B.acceptance_counts(torch.zeros(0, dtype=torch.int32, device="cuda"), L, counts)
    torch.cuda.synchronize()
    reach, accept = A.accept_counts([0, 6, 2], L)
    got = counts.cpu().numpy()
    assert got[:L].tolist() == reach.tolist() and got[L:].tolist() == accept.tolist()
