"""Pins of the same-state replay diagnostics oracle (App. B, "Same-state replay", Eq. 6)."""
import numpy as np
import pytest
import scipy.special

from oracle import brisk_oracle as O
from tests.test_oracle_pins import _random_params

RNG = np.random.default_rng(77)


def _setup(L, r, d, V, K, seed, alpha=0.0, scale=0.3, same_p=False):
    g = np.random.default_rng(seed)
    p = _random_params(L, r, d, V, scale=scale, alpha=alpha, seed=seed)
    lq = g.normal(scale=1.5, size=(L, V))
    lp = lq.copy() if same_p else lq + g.normal(scale=1.0, size=(L, V))
    cand = np.zeros((L, K), np.int64)
    clp = np.zeros((L, K))
    top4 = np.zeros((L, 4), np.int64)
    for i in range(L):
        cand[i], clp[i], _ = O.topk_candidates(lq[i], K)
        top4[i] = O.ranked_ids(lq[i])[:4]
    hidden, h_c = g.normal(size=(L, d)), g.normal(size=d)
    return p, lq, lp, cand, clp, top4, hidden, h_c


def _replay(p, lq, lp, cand, clp, top4, hidden, h_c, u, mode=O.GREEDY, u_sel=None):
    return O.replay_sequence(p, lambda i: lq[i], lambda i: lp[i], hidden, h_c, 3, cand, clp, top4,
                             u, mode, u_sel)


def _alpha_brute(lq, lp, i, tok):
    return min(1.0, scipy.special.softmax(lp[i])[tok] / scipy.special.softmax(lq[i])[tok])


@pytest.mark.parametrize("mode", [O.GREEDY, O.SAMPLE])
def test_closed_gate_means_no_intervention_rescue_or_regression(mode):
    L, r, d, V, K = 8, 8, 16, 60, 6
    p, lq, lp, cand, clp, top4, hidden, h_c = _setup(L, r, d, V, K, 1, alpha=-np.inf)
    u_sel = RNG.random(L)
    for trial in range(5):
        u = RNG.random(L)
        res = _replay(p, lq, lp, cand, clp, top4, hidden, h_c, u, mode, u_sel)
        assert not res.intervention.any() and not res.rescue.any() and not res.regression.any()
        base_tok = cand[np.arange(L), res.base_rank]
        jb = [u[i] < _alpha_brute(lq, lp, i, base_tok[i]) for i in range(L)]
        assert res.first_breaker == next((i for i in range(L) if not jb[i]), L)


def test_identical_distributions_never_break():
    L, r, d, V, K = 8, 8, 16, 60, 6
    p, lq, lp, cand, clp, top4, hidden, h_c = _setup(L, r, d, V, K, 2, scale=1.0, same_p=True)
    res = _replay(p, lq, lp, cand, clp, top4, hidden, h_c, RNG.random(L))
    assert res.first_breaker == L
    assert np.all(res.alpha_base == 1.0) and np.all(res.alpha_head == 1.0)
    assert not res.rescue.any() and not res.regression.any()


def test_alpha_matches_brute_force_and_head_stays_in_candidates():
    L, r, d, V, K = 6, 8, 16, 40, 5
    p, lq, lp, cand, clp, top4, hidden, h_c = _setup(L, r, d, V, K, 3, scale=1.0)
    res = _replay(p, lq, lp, cand, clp, top4, hidden, h_c, RNG.random(L))
    for i in range(L):
        assert abs(res.alpha_base[i] - _alpha_brute(lq, lp, i, cand[i][res.base_rank[i]])) < 1e-12
        assert abs(res.alpha_head[i] - _alpha_brute(lq, lp, i, cand[i][res.head_rank[i]])) < 1e-12


def test_constructed_rescue_and_regression():
    # find a state where the head changes the token at position 0, then place the draw between
    # the two acceptance probabilities
    L, r, d, V, K = 4, 8, 16, 50, 6
    for seed in range(200):
        p, lq, lp, cand, clp, top4, hidden, h_c = _setup(L, r, d, V, K, seed, scale=1.5)
        res = _replay(p, lq, lp, cand, clp, top4, hidden, h_c, np.zeros(L))
        if res.head_rank[0] != res.base_rank[0] and res.alpha_head[0] != res.alpha_base[0]:
            break
    else:
        pytest.skip("no intervention found")
    lo, hi = sorted((res.alpha_base[0], res.alpha_head[0]))
    u = np.zeros(L)
    u[0] = 0.5 * (lo + hi)
    res2 = _replay(p, lq, lp, cand, clp, top4, hidden, h_c, u)
    if res.alpha_head[0] > res.alpha_base[0]:
        # the base token is rejected at 0 (a first breaker) and the head token accepted: rescue
        assert res2.first_breaker == 0 and res2.rescue[0] and res2.intervention[0]
        assert not res2.regression.any()
    else:
        # the base token is accepted at 0 and the head token rejected: regression at 0
        assert res2.first_breaker > 0 and res2.regression[0] and not res2.rescue[0]


def test_forced_prefix_equal_to_own_selection_reproduces_the_corrector():
    L, r, d, V, K = 6, 8, 16, 40, 5
    p, lq, lp, cand, clp, top4, hidden, h_c = _setup(L, r, d, V, K, 5, scale=1.0)
    own = O.corrector_sequence(p, hidden, h_c, 3, lambda i: lq[i], cand, clp, top4)
    forced = O.corrector_sequence(p, hidden, h_c, 3, lambda i: lq[i], cand, clp, top4,
                                  prefix_ranks=own.sel_rank)
    np.testing.assert_array_equal(own.refined, forced.refined)
