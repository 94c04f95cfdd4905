"""The library's host-side acceptance functions (Sec. 2.2; Sec. 3.2 Eqs. 2-3) against the
oracle. No GPU needed: these entry points do no device work."""
import numpy as np
import pytest

from oracle import acceptance as A


@pytest.fixture(scope="module")
def B():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


@pytest.mark.parametrize("M", [1, 2, 7, 32, 64])
def test_weights_and_tpf_match_oracle(B, M):
    rng = np.random.default_rng(M)
    a = rng.uniform(0.05, 0.995, M)
    for with_gc in (False, True):
        if with_gc:
            g = np.arange(M + 1) + 1.0 + rng.uniform(0, 0.5, M + 1)
            c = 1.0 + rng.uniform(0, 1.0, M + 1)
        else:
            g, c = A.unit_costs(M)
        tpf, w_raw, w_bar = B.acceptance_weights(a, g if with_gc else None, c if with_gc else None,
                                                 eps=1e-8)
        ow_raw, ow_bar = A.weights(a, g, c, eps=1e-8)
        assert abs(tpf - A.tpf(a, g, c)) <= 1e-12 * abs(tpf)
        np.testing.assert_allclose(w_raw, ow_raw, rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(w_bar, ow_bar, rtol=1e-10, atol=1e-15)


def test_edge_profiles(B):
    # a_i = 1 everywhere: the block always survives; a_i = 0 at the front: nothing survives
    for a in (np.ones(5), np.zeros(5), np.array([1.0, 0.0, 1.0, 0.5, 0.25])):
        g, c = A.unit_costs(len(a))
        tpf, w_raw, w_bar = B.acceptance_weights(a, eps=1e-8)
        ow_raw, ow_bar = A.weights(a, g, c, eps=1e-8)
        assert abs(tpf - A.tpf(a, g, c)) < 1e-12
        np.testing.assert_allclose(w_raw, ow_raw, atol=1e-15)
        np.testing.assert_allclose(w_bar, ow_bar, atol=1e-12)


def test_isd_tpf_matches_oracle(B):
    for N in (2, 3, 8, 16):
        for r in (0.0, 0.05, 0.1, 0.15, 0.2, 0.5, 1.0):
            assert abs(B.tpf_isd(N, r) - A.tpf_isd(N, r)) <= 1e-12 * A.tpf_isd(N, r)
    assert np.isnan(B.tpf_isd(1, 0.1)) and np.isnan(B.tpf_isd(8, 1.5))


def test_invalid_profiles_rejected(B):
    with pytest.raises(B.BriskError):
        B.acceptance_weights(np.array([0.5, 1.2]))
    with pytest.raises(B.BriskError):
        B.acceptance_weights(np.array([np.nan]))
    with pytest.raises(B.BriskError):
        B.acceptance_weights(np.full(65, 0.5))


@pytest.mark.parametrize("M", [1, 2, 7, 64])
def test_isd_costs_and_weights_match_oracle(B, M):
    g, c = B.isd_costs(M)
    og, oc = A.isd_costs(M)
    np.testing.assert_array_equal(g, og)
    np.testing.assert_array_equal(c, oc)
    a = np.random.default_rng(10 + M).uniform(0.2, 0.99, M)
    tpf, w_raw, w_bar = B.acceptance_weights(a, g, c, eps=1e-8)
    assert abs(tpf - A.tpf_isd_profile(a)) <= 1e-12 * tpf
    ow_raw, ow_bar = A.weights(a, og, oc, eps=1e-8)
    np.testing.assert_allclose(w_raw, ow_raw, rtol=1e-10, atol=1e-15)
    np.testing.assert_allclose(w_bar, ow_bar, rtol=1e-10, atol=1e-15)
    with pytest.raises(B.BriskError):
        B.isd_costs(0)
