"""Pins of the acceptance-profile oracle (Sec. 2.2; Sec. 3.2 Eqs. 2-3) against values the paper
prints and identities that hold independently of the implementation."""
import os

import numpy as np
import pytest

from oracle import acceptance as A

HERE = os.path.dirname(os.path.abspath(__file__))


def _golden():
    rows = []
    with open(os.path.join(HERE, "golden", "tpf_isd_n8.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                n, r, t = line.split()
                rows.append((int(n), float(r), float(t)))
    return rows


@pytest.mark.parametrize("N,r,t", _golden())
def test_isd_tpf_matches_printed_values(N, r, t):
    assert abs(A.tpf_isd(N, r) - t) <= 0.005


def test_length_law_is_a_distribution_and_mean_is_survival_sum():
    rng = np.random.default_rng(1)
    for M in (1, 3, 7, 32):
        a = rng.uniform(0.2, 0.99, M)
        pr = A.length_law(a)
        assert abs(pr.sum() - 1.0) < 1e-12
        assert np.all(pr >= 0)
        # E[L] = sum_k A_k (Sec. 2.2)
        assert abs(np.dot(np.arange(M + 1), pr) - A.survival(a)[1:].sum()) < 1e-12


def test_unit_cost_tpf_reduces_to_one_plus_survival_sum():
    a = np.array([0.95, 0.9, 0.8, 0.85, 0.7, 0.6, 0.9])
    g, c = A.unit_costs(len(a))
    # brute force over the 2^M accept/reject patterns: L = first rejection
    M = len(a)
    total = 0.0
    for bits in range(1 << M):
        p = 1.0
        for i in range(M):
            acc = (bits >> i) & 1
            p *= a[i] if acc else 1.0 - a[i]
        L = next((i for i in range(M) if not (bits >> i) & 1), M)
        total += p * (L + 1)
    assert abs(A.tpf(a, g, c) - total) < 1e-12
    assert abs(A.tpf(a, g, c) - (1.0 + np.cumprod(a).sum())) < 1e-12


def test_weights_match_finite_differences_of_fpt_in_log_odds():
    rng = np.random.default_rng(2)
    M = 7
    a = rng.uniform(0.3, 0.97, M)
    g = np.arange(M + 1) + 1.0 + rng.uniform(0, 0.5, M + 1)   # arbitrary gains and costs
    c = 1.0 + rng.uniform(0, 1.0, M + 1)
    w_raw, _ = A.weights(a, g, c)
    z = np.log(a / (1 - a))
    h = 1e-6
    for i in range(M):
        zp, zm = z.copy(), z.copy()
        zp[i] += h
        zm[i] -= h
        ap, am = 1 / (1 + np.exp(-zp)), 1 / (1 + np.exp(-zm))
        fd = -(A.fpt(ap, g, c) - A.fpt(am, g, c)) / (2 * h)
        assert abs(fd - w_raw[i]) < 1e-7 * max(1.0, abs(fd))


def test_weights_are_mean_one_and_favour_early_positions_at_constant_acceptance():
    M = 7
    a = np.full(M, 0.8)
    g, c = A.unit_costs(M)
    w_raw, w_bar = A.weights(a, g, c, eps=0.0)
    assert abs(w_bar.mean() - 1.0) < 1e-12
    # with equal a_i an early rejection truncates more of the block
    assert np.all(np.diff(w_raw) < 0)


def test_counts_and_profile_on_a_hand_example():
    # accepted lengths of 5 blocks of M = 4
    lens = [0, 4, 2, 2, 1]
    reach, accept = A.accept_counts(lens, 4)
    assert reach.tolist() == [5, 4, 3, 1]
    assert accept.tolist() == [4, 3, 1, 1]
    a = A.profile(reach, accept)
    assert np.allclose(a, [0.8, 0.75, 1 / 3, 1.0])


def test_profile_recovers_a_known_law_statistically():
    rng = np.random.default_rng(3)
    a_true = np.array([0.95, 0.9, 0.85, 0.8, 0.75, 0.7, 0.65, 0.6])
    pr = A.length_law(a_true)
    lens = rng.choice(len(pr), size=200000, p=pr)
    reach, accept = A.accept_counts(lens, len(a_true))
    a = A.profile(reach, accept)
    se = np.sqrt(a_true * (1 - a_true) / reach)
    assert np.all(np.abs(a - a_true) < 5 * se)


def test_isd_instantiation_equals_renewal_reward_with_its_costs():
    """Eq. 8's closed form against Eq. 2 evaluated with the gains and costs the paper states for
    it (two independent formulas)."""
    rng = np.random.default_rng(5)
    for M in (1, 2, 3, 7, 15, 31):
        for _ in range(5):
            a = rng.uniform(0.0, 1.0, M)
            g, c = A.isd_costs(M)
            assert abs(A.tpf(a, g, c) - A.tpf_isd_profile(a)) < 1e-12 * A.tpf_isd_profile(a)


@pytest.mark.parametrize("N,r,t", _golden())
def test_isd_instantiation_at_constant_profile_gives_printed_values(N, r, t):
    """At a_i = 1 - r (M = N - 1 positions) Eq. 8 is the Sec. 2.2 rule: the printed TPF_8."""
    a = np.full(N - 1, 1.0 - r)
    assert abs(A.tpf_isd_profile(a) - A.tpf_isd(N, r)) < 1e-12
    assert abs(A.tpf_isd_profile(a) - t) <= 0.005


def test_isd_weights_match_finite_differences():
    rng = np.random.default_rng(6)
    M = 7
    a = rng.uniform(0.3, 0.97, M)
    g, c = A.isd_costs(M)
    w_raw, w_bar = A.weights(a, g, c)
    z = np.log(a / (1 - a))
    h = 1e-6
    for i in range(M):
        zp, zm = z.copy(), z.copy()
        zp[i] += h
        zm[i] -= h
        fp = 1.0 / A.tpf_isd_profile(1 / (1 + np.exp(-zp)))
        fm = 1.0 / A.tpf_isd_profile(1 / (1 + np.exp(-zm)))
        fd = -(fp - fm) / (2 * h)
        assert abs(fd - w_raw[i]) < 1e-7 * max(1.0, abs(fd))
    assert abs(w_bar.mean() - 1.0) < 1e-6
