"""Pins of the CPU oracle against facts fixed outside it.

Each test checks the oracle against something it does not compute itself:
brute force on tiny vocabularies, closed forms derived by hand for special
parameter settings, a worked example of the confidence features, the
speculative-sampling theorem by exact enumeration of the uniforms, and the
accepted-prefix law E[L] = sum_k prod_{i<=k} a_i (Sec. 2.2).
"""
import math
import zlib

import numpy as np
import pytest
import scipy.special
import torch

from oracle import brisk_oracle as O

RNG = np.random.default_rng(1234)


# ---------------------------------------------------------------------------
# Step 1: top-K and the log-partition
# ---------------------------------------------------------------------------

def _topk_by_repeated_argmax(row, K):
    """Independent of any sort: K times pick the largest remaining value, lowest id on ties."""
    alive = list(range(len(row)))
    out = []
    for _ in range(K):
        best = alive[0]
        for v in alive[1:]:
            if row[v] > row[best]:
                best = v
        out.append(best)
        alive.remove(best)
    return out


@pytest.mark.parametrize("V,K", [(8, 1), (8, 4), (17, 8), (64, 16), (33, 32), (64, 64)])
def test_topk_matches_brute_force(V, K):
    for trial in range(20):
        if trial % 2:
            row = RNG.integers(-3, 4, size=V).astype(np.float64)   # many exact ties
        else:
            row = RNG.normal(size=V)
        ids, lp, lse = O.topk_candidates(row, K)
        assert list(ids) == _topk_by_repeated_argmax(row, K)
        assert np.all(np.diff(lp) <= 0)
        np.testing.assert_allclose(lse, scipy.special.logsumexp(row), rtol=0, atol=1e-12)


def test_logprob_normalises_over_the_whole_vocabulary():
    for V in (5, 100, 4096):
        row = RNG.normal(scale=3.0, size=V)
        _, lp, lse = O.topk_candidates(row, V)
        assert abs(np.exp(lp).sum() - 1.0) < 1e-12
        assert abs(np.exp(row - lse).sum() - 1.0) < 1e-12


def test_all_equal_row_gives_lowest_ids_and_uniform_logprob():
    V, K = 50, 8
    ids, lp, lse = O.topk_candidates(np.full(V, 0.75), K)
    assert list(ids) == list(range(K))
    np.testing.assert_allclose(lp, -math.log(V), atol=1e-15)
    assert abs(lse - (0.75 + math.log(V))) < 1e-14


def test_minus_infinity_entries_and_single_finite_value():
    row = np.full(10, -np.inf)
    row[7] = 2.5
    ids, lp, lse = O.topk_candidates(row, 3)
    assert ids[0] == 7 and lse == 2.5 and lp[0] == 0.0
    assert np.isneginf(lp[1]) and list(ids[1:]) == [0, 1]
    with pytest.raises(O.OracleError):
        O.log_partition(np.full(4, -np.inf))
    with pytest.raises(O.OracleError):
        O.log_partition(np.array([0.0, np.nan]))


def test_topk_values_agree_with_torch():
    row = RNG.normal(size=1000)
    ids, lp, lse = O.topk_candidates(row, 16)
    t = torch.topk(torch.tensor(row), 16)
    np.testing.assert_array_equal(row[ids], t.values.numpy())
    assert abs(lse - torch.logsumexp(torch.tensor(row), 0).item()) < 1e-12


def test_verifier_argmax_lowest_id_on_ties():
    row = np.array([1.0, 3.0, 0.0, 3.0, 3.0])
    assert O.verifier_argmax(row) == 1


# ---------------------------------------------------------------------------
# Confidence features: a worked example from the definitions in App. C.3
# ---------------------------------------------------------------------------

def test_features_worked_example():
    #        id: 0    1    2     3    4    5    6    7
    row = np.array([0.5, 3.0, -1.0, 2.0, 2.5, 1.0, 1.0, -2.0])
    top4 = O.ranked_ids(row)[:4]
    assert list(top4) == [1, 4, 3, 5]           # 3.0, 2.5, 2.0, then 1.0 (id 5 before id 6)
    # prev = 3: not top-1, inside top-4, gap 3.0 - 2.0
    np.testing.assert_array_equal(O.confidence_features(row, top4, 3), [0.5, 2.0, 0.0, 1.0, 1.0])
    # prev = 1 is the top-1 token
    np.testing.assert_array_equal(O.confidence_features(row, top4, 1), [0.5, 2.0, 1.0, 1.0, 0.0])
    # prev = 6 ties with rank 4 in value but sits outside the top-4 ids
    np.testing.assert_array_equal(O.confidence_features(row, top4, 6), [0.5, 2.0, 0.0, 0.0, 2.0])
    # prev = 7: far below
    np.testing.assert_array_equal(O.confidence_features(row, top4, 7), [0.5, 2.0, 0.0, 0.0, 5.0])


# ---------------------------------------------------------------------------
# Corrector: special cases with closed forms
# ---------------------------------------------------------------------------

def _random_params(L, r, d, V, scale=0.3, alpha=0.0, b_g=0.0, seed=0):
    g = np.random.default_rng(seed)
    S = 2 * r
    return O.Params(
        P_h=g.normal(scale=scale, size=(r, d)), P_e=g.normal(scale=scale, size=(r, d)),
        P_phi=g.normal(scale=scale, size=(16, 5)), pos=g.normal(scale=scale, size=(L, 16)),
        W0=g.normal(scale=scale, size=(S, 2 * r)), Wz=g.normal(scale=scale, size=(S, 2 * r + 32)),
        Wh=g.normal(scale=scale, size=(S, 2 * r + 32)), W_s=g.normal(scale=scale, size=(r, S)),
        W_c=g.normal(scale=scale, size=(r, d)), w_g=g.normal(scale=scale, size=S + 5),
        b_g=b_g, alpha=alpha, E_in=g.normal(size=(V, d)), E_out=g.normal(size=(V, d)))


def _run(p, lq, hidden, h_c, x0, K, mode=O.GREEDY, u_sel=None):
    L = lq.shape[0]
    cand = np.zeros((L, K), np.int64)
    lp = np.zeros((L, K))
    top4 = np.zeros((L, 4), np.int64)
    for i in range(L):
        cand[i], lp[i], _ = O.topk_candidates(lq[i], K)
        top4[i] = O.ranked_ids(lq[i])[:4]
    tr = O.corrector_sequence(p, hidden, h_c, x0, lambda i: lq[i], cand, lp, top4, mode, u_sel)
    return cand, lp, tr


def test_gate_closed_gives_base_ranking():
    L, r, d, V, K = 6, 8, 16, 40, 5
    p = _random_params(L, r, d, V, alpha=-np.inf)
    lq = RNG.normal(size=(L, V))
    cand, lp, tr = _run(p, lq, RNG.normal(size=(L, d)), RNG.normal(size=d), 3, K)
    np.testing.assert_array_equal(tr.refined, lp)
    np.testing.assert_array_equal(tr.sel_tokens, cand[:, 0])
    assert np.all(tr.gamma == 0.0)


def test_single_candidate_selects_top1_and_selection_stays_in_candidates():
    L, r, d, V = 5, 8, 16, 30
    p = _random_params(L, r, d, V, scale=1.0)
    lq = RNG.normal(size=(L, V))
    cand, _, tr = _run(p, lq, RNG.normal(size=(L, d)), RNG.normal(size=d), 0, 1)
    np.testing.assert_array_equal(tr.sel_tokens, cand[:, 0])
    for K in (4, 8):
        for mode, u in ((O.GREEDY, None), (O.SAMPLE, RNG.random(L))):
            cand, _, tr = _run(p, lq, RNG.normal(size=(L, d)), RNG.normal(size=d), 7, K, mode, u)
            for i in range(L):
                assert tr.sel_tokens[i] in cand[i]
                assert tr.refined[i].shape == (K,)


def _probe_params(L, r, V, *, z_logit, path, shift=2, init=None, w_g_feature=None):
    """One-hot 'linear probe' parameters (d = 2r, S = 2r).

    E_in(v) = e_{v mod r}, E_out(v) = e_{(v+1) mod r} (in R^d); P_e = P_h = [I_r | 0];
    W_s reads state dims cyclically shifted by ``shift``; W_c = [I_r | 0]. W_z only sees the
    position block, whose rows are one-hot, so z = sigmoid(z_logit) in every state dim. W_h
    routes one block of the GRU input (``path``) into the first state dims. With
    alpha = b_g = +inf the gate is exactly 1 (or sigmoid(phi_f) with ``w_g_feature`` = f).
    Hence d_{i,k} = s_i[(c_{i,k} + 1 + shift) mod r].
    """
    d, S = 2 * r, 2 * r
    I = np.eye(r)
    Pr = np.hstack([I, np.zeros((r, d - r))])
    E_in = np.zeros((V, d))
    E_out = np.zeros((V, d))
    for v in range(V):
        E_in[v, v % r] = 1.0
        E_out[v, (v + 1) % r] = 1.0
    Wz = np.zeros((S, 2 * r + 32))
    Wz[:, 2 * r:2 * r + 16] = z_logit
    Wh = np.zeros((S, 2 * r + 32))
    blk = {"hidden": 0, "token": r, "pos": 2 * r, "phi": 2 * r + 16}[path]
    width = {"hidden": r, "token": r, "pos": 16, "phi": 16}[path]
    for j in range(min(width, r)):
        Wh[j, blk + j] = 1.0
    W0 = np.zeros((S, 2 * r))
    if init == "token":
        W0[:r, r:2 * r] = I
    elif init == "hidden":
        W0[:r, :r] = I
    W_s = np.zeros((r, S))
    for j in range(r):
        W_s[j, (j + shift) % r] = 1.0
    pos = np.zeros((L, 16))
    pos[np.arange(L), np.arange(L) % 16] = 1.0
    P_phi = np.zeros((16, 5))
    P_phi[:5, :5] = np.eye(5)
    w_g = np.zeros(S + 5)
    b_g = np.inf
    if w_g_feature is not None:
        w_g[S + w_g_feature] = 1.0
        b_g = 0.0
    return O.Params(P_h=Pr, P_e=Pr.copy(), P_phi=P_phi, pos=pos, W0=W0, Wz=Wz, Wh=Wh, W_s=W_s,
                    W_c=Pr.copy(), w_g=w_g, b_g=b_g, alpha=np.inf, E_in=E_in, E_out=E_out)


def _designed_rows(L, V, K, g):
    """Rows whose top-K logits are close together, so a bonus in [0, 1] reorders them."""
    lq = g.normal(scale=0.3, size=(L, V)) - 6.0
    for i in range(L):
        ids = g.permutation(V)[:K]
        lq[i, ids] = g.uniform(0.0, 0.6, size=K)
    return lq


@pytest.mark.parametrize("path,init,z_logit", [
    ("token", None, 0.0), ("token", None, math.log(3.0)), ("token", "token", -0.7),
    ("hidden", "hidden", 0.4), ("pos", None, 1.1), ("phi", "token", 0.0)])
def test_probe_closed_form(path, init, z_logit):
    """s_i = (1-z) s_{i-1} + z h~_i with u_0 = tanh(one-hot), evaluated by hand."""
    L, r, V, K = 7, 8, 24, 4
    shift = 2
    g = np.random.default_rng(zlib.crc32(f"{path}/{init}".encode()))   # stable across runs
    p = _probe_params(L, r, V, z_logit=z_logit, path=path, shift=shift, init=init)
    lq = _designed_rows(L, V, K, g)
    d = 2 * r
    hid_tok = g.integers(0, r, size=L)
    hidden = np.zeros((L, d))
    hidden[np.arange(L), hid_tok] = 1.0
    hc_tok = 5
    h_c = np.zeros(d)
    h_c[hc_tok] = 1.0
    x0 = 13
    cand, lp, tr = _run(p, lq, hidden, h_c, x0, K)

    z = 1.0 / (1.0 + math.exp(-z_logit))
    state = np.zeros(r)
    if init == "token":
        state[x0 % r] = math.tanh(1.0)
    elif init == "hidden":
        state[hc_tok] = math.tanh(1.0)
    prev = x0
    for i in range(L):
        row = lq[i]
        order = sorted(range(V), key=lambda v: (-row[v], v))
        t4 = order[:4]
        phi = [row[t4[0]] - row[t4[1]], row[t4[0]] - row[t4[3]], float(prev == t4[0]),
               float(prev in t4), row[t4[0]] - row[prev]]
        inject = np.zeros(r)
        if path == "token":
            inject[prev % r] = 1.0
        elif path == "hidden":
            inject[hid_tok[i]] = 1.0
        elif path == "pos":
            inject[i % 16 % r] = 1.0 if i % 16 < r else 0.0
        else:
            inject[:5] = phi
        state = (1.0 - z) * state + z * inject
        bonus = np.array([state[(int(c) + 1 + shift) % r] for c in cand[i]])
        expect = lp[i] + bonus
        np.testing.assert_allclose(tr.refined[i], expect, rtol=0, atol=1e-12)
        k = int(np.argmax(expect))
        assert tr.sel_tokens[i] == cand[i][k]
        prev = int(cand[i][k])
    # the probe really reorders candidates somewhere, so a wrong index would show
    if path == "token":
        assert np.any(tr.sel_tokens != cand[:, 0])


@pytest.mark.parametrize("f", range(5))
def test_gate_reads_raw_features(f):
    """w_g = e_{S+f}, b_g = 0, alpha = +inf: gamma_i = sigmoid(phi_{i,f}) exactly."""
    L, r, V, K = 6, 8, 24, 4
    g = np.random.default_rng(77 + f)
    p = _probe_params(L, r, V, z_logit=0.0, path="token", w_g_feature=f)
    lq = _designed_rows(L, V, K, g)
    x0 = 2
    cand, lp, tr = _run(p, lq, np.zeros((L, 2 * r)), np.zeros(2 * r), x0, K)
    prev = x0
    for i in range(L):
        row = lq[i]
        order = sorted(range(V), key=lambda v: (-row[v], v))
        t4 = order[:4]
        phi = [row[t4[0]] - row[t4[1]], row[t4[0]] - row[t4[3]], float(prev == t4[0]),
               float(prev in t4), row[t4[0]] - row[prev]]
        assert abs(tr.gamma[i] - 1.0 / (1.0 + math.exp(-phi[f]))) < 1e-15
        prev = int(tr.sel_tokens[i])


# ---------------------------------------------------------------------------
# Verification
# ---------------------------------------------------------------------------

def test_identical_distributions_greedy_corrector_off_accepts_whole_block():
    L, r, d, V, K = 8, 8, 16, 50, 4
    p = _random_params(L, r, d, V, alpha=-np.inf)
    lq = RNG.normal(size=(L, V))
    cand, lp, tr = _run(p, lq, RNG.normal(size=(L, d)), RNG.normal(size=d), 1, K)
    vr = O.verify_sequence(lambda i: lq[i], tr.sel_tokens, cand, tr.refined)
    assert vr.accepted_len == L and vr.correction == -1
    np.testing.assert_array_equal(vr.out_tokens, tr.sel_tokens)


def test_first_position_rejected_gives_verifier_argmax():
    L, V, K = 5, 30, 4
    lq = RNG.normal(size=(L, V))
    lpv = lq.copy()
    cand = np.array([O.ranked_ids(lq[i])[:K] for i in range(L)])
    outside = [v for v in range(V) if v not in cand[0]][0]
    lpv[0, outside] = 50.0
    sel = cand[:, 0]
    vr = O.verify_sequence(lambda i: lpv[i], sel, cand, np.zeros((L, K)))
    assert vr.accepted_len == 0 and vr.correction == outside
    assert vr.out_tokens[0] == outside and np.all(vr.out_tokens[1:] == -1)


def test_rejection_in_the_middle_truncates():
    L, V, K = 6, 30, 4
    lq = RNG.normal(size=(L, V))
    cand = np.array([O.ranked_ids(lq[i])[:K] for i in range(L)])
    sel = cand[:, 0].copy()
    lpv = np.zeros((L, V))
    for i in range(L):
        lpv[i, sel[i]] = 10.0
    lpv[3, sel[3]] = 0.0
    lpv[3, cand[3, 2]] = 10.0
    vr = O.verify_sequence(lambda i: lpv[i], sel, cand, np.zeros((L, K)))
    assert vr.accepted_len == 3 and vr.correction == cand[3, 2]
    np.testing.assert_array_equal(vr.out_tokens, list(sel[:3]) + [cand[3, 2], -1, -1])


def _first_at_least(f, k, lo=0.0, hi=1.0, iters=60):
    """inf{u in [lo, hi): f(u) >= k} for a non-decreasing integer step function f."""
    if f(lo) >= k:
        return lo
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if f(mid) >= k:
            hi = mid
        else:
            lo = mid
    return hi


def _step_measure(f, values):
    """Lebesgue measure on [0, 1) of {u : f(u) = v} for each v, f non-decreasing."""
    values = sorted(values)
    bounds = [_first_at_least(f, v) for v in values] + [1.0]
    out = {}
    for j, v in enumerate(values):
        nxt = min([b for b in bounds[j + 1:]] + [1.0])
        out[v] = max(0.0, nxt - bounds[j])
    return out


@pytest.mark.parametrize("select_mode,seed", [(O.SAMPLE, 0), (O.SAMPLE, 1), (O.GREEDY, 2),
                                              (O.SAMPLE, 3)])
def test_speculative_sampling_commits_verifier_distribution_exactly(select_mode, seed):
    """L = 1, tiny V: integrate the committed token over (u_sel, u_acc, u_res) exactly.
    The theorem of speculative sampling (Sec. 3.3) says the result is p itself, and the
    acceptance probability is sum_v min(pi(v), p(v))."""
    g = np.random.default_rng(seed)
    V, K, r, d = 6, 4, 4, 8
    p_ = _random_params(1, r, d, V, scale=0.8, seed=seed)
    lq = g.normal(size=(1, V))
    lpv = g.normal(scale=1.5, size=(1, V))
    hidden = g.normal(size=(1, d))
    h_c = g.normal(size=d)
    cand = O.ranked_ids(lq[0])[:K][None, :]
    lp = (lq[0][cand[0]] - O.log_partition(lq[0]))[None, :]
    top4 = O.ranked_ids(lq[0])[:4][None, :]

    def trace(u_sel):
        return O.corrector_sequence(p_, hidden, h_c, 0, lambda i: lq[i], cand, lp, top4,
                                    select_mode, np.array([u_sel]))

    if select_mode == O.SAMPLE:
        sel_meas = _step_measure(lambda u: int(trace(u).sel_rank[0]), range(K))
    else:
        sel_meas = {int(trace(0.5).sel_rank[0]): 1.0}
    p_true = scipy.special.softmax(lpv[0])
    commit = np.zeros(V)
    acc_total = 0.0
    for k, mk in sel_meas.items():
        if mk == 0.0:
            continue
        tr = trace(0.5) if select_mode == O.GREEDY else None
        if tr is None:
            # a u_sel inside the interval of rank k
            lo = _first_at_least(lambda u: int(trace(u).sel_rank[0]), k)
            tr = trace(lo + 0.5 * mk)
        assert tr.sel_rank[0] == k

        def res(u_acc, u_res):
            return O.verify_sequence(lambda i: lpv[i], tr.sel_tokens, cand, tr.refined,
                                     select_mode, O.STOCHASTIC, np.array([u_acc]),
                                     np.array([u_res]))
        # acceptance region is [0, alpha)
        a = _first_at_least(lambda u: 0 if res(u, 0.5).accepted_len == 1 else 1, 1)
        commit[int(tr.sel_tokens[0])] += mk * a
        acc_total += mk * a
        if a < 1.0:
            u_rej = 0.5 * (a + 1.0)
            meas = _step_measure(lambda u: int(res(u_rej, u).correction), range(V))
            for v, mv in meas.items():
                commit[v] += mk * (1.0 - a) * mv
    np.testing.assert_allclose(commit, p_true, rtol=0, atol=1e-9)
    # acceptance probability = sum_v min(pi(v), p(v))
    pi = np.zeros(V)
    for k, mk in sel_meas.items():
        pi[cand[0][k]] += mk
    assert abs(acc_total - np.minimum(pi, p_true).sum()) < 1e-9


def test_residual_walks_ids_in_ascending_order():
    row = np.log(np.array([0.1, 0.2, 0.3, 0.4]))
    # pi puts 0.4 on id 3 and 0.6 on id 2: residual = [0.1, 0.2, 0, 0] / 0.3
    v, _ = O.residual_sample(row, [3, 2], [0.4, 0.6], 0.0)
    assert v == 0
    v, _ = O.residual_sample(row, [3, 2], [0.4, 0.6], 0.34)
    assert v == 1
    v, _ = O.residual_sample(row, [3, 2], [0.4, 0.6], 0.999)
    assert v == 1
    # Z = 0: proposal equals the verifier, fall back to the verifier argmax
    v, _ = O.residual_sample(row, [0, 1, 2, 3], [0.1, 0.2, 0.3, 0.4], 0.5)
    assert v == 3


def test_mean_accepted_prefix_follows_survival_law():
    """Corrector off, greedy: accepted length L has E[L] = sum_k prod_{i<=k} a_i (Sec. 2.2).
    The generator plants the verifier argmax at the proposal top-1 with probability a_i,
    otherwise elsewhere (a random id collides with the top-1 with probability 1/V)."""
    from paper_2609_33390_gb300 import synth
    n, L, V = 1200, 8, 256
    wl = synth.Workload("pin", B=n, L=L, V=V, d=16, K=4, r=8, logits_dtype=torch.float32,
                        hidden_dtype=torch.float32, agree0=0.9, agree_decay=0.95)
    blk = synth.make_block(wl, "cpu")
    lq = blk["logits_q"].double().numpy()
    lpv = blk["logits_p"].double().numpy()
    lens = []
    for b in range(n):
        sel = np.array([O.verifier_argmax(lq[b, i]) for i in range(L)])
        cand = sel[:, None]
        vr = O.verify_sequence(lambda i: lpv[b, i], sel, cand, np.zeros((L, 1)))
        lens.append(vr.accepted_len)
    lens = np.array(lens)
    a = 0.9 * 0.95 ** np.arange(L)
    acc = a + (1 - a) * (1 - wl.rescue_frac) / V
    expect = np.cumprod(acc).sum()
    se = lens.std() / math.sqrt(n)
    assert abs(lens.mean() - expect) < 4.5 * se, (lens.mean(), expect, se)


# ---------------------------------------------------------------------------
# Commit step (Algorithm 1(b)): the anchor of the next block
# ---------------------------------------------------------------------------

def test_next_anchor_is_the_last_committed_token():
    """The next block's anchor is the last token this block commits: the correction when a
    position is rejected, the last selection when the whole block is accepted. Checked against
    the out_tokens row read independently (its last entry >= 0) over random stochastic blocks
    whose rejections fall at every position."""
    L, V, K = 6, 12, 4
    rng = np.random.default_rng(77)
    seen = set()
    for _ in range(300):
        lq = rng.normal(size=(L, V)) * 2.0
        lpv = lq + rng.normal(size=(L, V)) * rng.uniform(0.0, 3.0)
        cand = np.array([O.ranked_ids(lq[i])[:K] for i in range(L)])
        refined = np.array([lq[i][cand[i]] for i in range(L)]) + rng.normal(size=(L, K))
        ranks = rng.integers(0, K, size=L)
        sel = cand[np.arange(L), ranks]
        vr = O.verify_sequence(lambda i: lpv[i], sel, cand, refined, O.SAMPLE, O.STOCHASTIC,
                               rng.uniform(size=L), rng.uniform(size=L))
        committed = [int(t) for t in vr.out_tokens if t >= 0]
        assert len(committed) == min(vr.accepted_len + 1, L)
        assert O.next_anchor(vr, sel) == committed[-1]
        seen.add(vr.accepted_len)
    assert seen == set(range(L + 1))   # every rejection position and the full block


def test_next_anchor_closed_cases():
    L, V, K = 5, 30, 4
    lq = RNG.normal(size=(L, V))
    cand = np.array([O.ranked_ids(lq[i])[:K] for i in range(L)])
    sel = cand[:, 0]
    # identical distributions, greedy, the base ranking: the whole block, anchor = last token
    vr = O.verify_sequence(lambda i: lq[i], sel, cand, np.zeros((L, K)))
    assert vr.accepted_len == L and O.next_anchor(vr, sel) == sel[-1]
    # the verifier's argmax at position 0 outside the candidates: anchor = that argmax
    lpv = lq.copy()
    outside = [v for v in range(V) if v not in cand[0]][0]
    lpv[0, outside] = 50.0
    vr = O.verify_sequence(lambda i: lpv[i], sel, cand, np.zeros((L, K)))
    assert vr.accepted_len == 0 and O.next_anchor(vr, sel) == outside


def test_residual_mass_is_one_minus_the_acceptance_rate():
    """sum_v [p(v) - pi(v)]_+ = 1 - sum_v min(p(v), pi(v)) for a proposal law pi on the
    candidates: the residual's mass is the rejection probability (Sec. 3.3)."""
    rng = np.random.default_rng(5)
    for _ in range(50):
        V, K = 40, 6
        row = rng.normal(size=V) * 2
        p = scipy.special.softmax(row)
        ids = rng.choice(V, size=K, replace=False)
        pi = scipy.special.softmax(rng.normal(size=K))
        R = O.residual_mass(row, ids, pi)
        assert np.all(R >= 0)
        pim = np.zeros(V)
        pim[ids] = pi
        assert abs(R.sum() - (1.0 - np.minimum(p, pim).sum())) < 1e-12
