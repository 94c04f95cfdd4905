"""Plain CPU oracle of the acceptance profile and the risk-reward position weights (float64).

TEST INFRASTRUCTURE ONLY: the literal statement of these formulas, to check the library's
versions against. Only the tests may import it. It shares no code with the library.

What it follows (paper "From Position Risks to Block Survival: Faster Generation for Diffusion
Language Models"):

* Sec. 2.2 ("Rejection Severely Limits Effective Throughput"): a_i = probability that position i
  is accepted given the prefix before it; survival A_k = prod_{i<=k} a_i; expected accepted
  prefix E[L] = sum_k A_k; and the ISD stride-N rule with constant rejection r,
  TPF_N(r) = (2 + sum_{i=1}^{N-2} (1-r)^i) / (2 - (1-r)^{N-1}).
* Sec. 3.2, Eq. 2 (non-uniform TPF): Pr(L = k) = A_k (1 - a_{k+1}) for k < M and A_M for k = M;
  TPF(a) = sum_k Pr(L=k) g_k / sum_k Pr(L=k) c_k; FPT = 1 / TPF; with unit cost and one
  guaranteed token, TPF = 1 + sum_{k=1}^M A_k. The profile a_i is estimated as one minus the
  rejection rate at position i among the blocks whose verification reached i.
* Sec. 3.2, Eq. 3 (risk-reward weights): w_i^raw = -dFPT/dz_i = -dFPT/da_i * a_i (1 - a_i) with
  z_i = log(a_i / (1 - a_i)); w_bar_i = M w_i^raw / (sum_j w_j^raw + eps).
* App. C.1, Eq. 8 (the instantiation for ISD verification, which the paper uses for
  its FPT and weights): TPF(a) = (2 + sum_{k=1}^{M-1} A_k) / (2 - A_M) with M = N - 1; the same
  as Eq. 2 with gains g_k = 2 + min(k, M - 1) and costs c_k = 2 (k < M), c_M = 1.

Positions are 0-based here (position i of the paper is index i-1); A has M+1 entries with
A[0] = 1. Parity pins: the paper's printed TPF_8 values, the unit-cost identity, the length
law summing to one, E[L] = sum A_k, the weights against finite differences of FPT, Eq. 8
against Eq. 2 with its stated costs and, at a constant profile, against the Sec. 2.2 rule and
the printed TPF_8 values.
"""
from __future__ import annotations

import numpy as np


def accept_counts(accepted_len, M: int):
    """Per position i: how many blocks reached it (accepted_len >= i) and how many accepted it
    (accepted_len >= i + 1)."""
    lens = np.asarray(accepted_len, dtype=np.int64).ravel()
    reach = np.array([(lens >= i).sum() for i in range(M)], dtype=np.int64)
    accept = np.array([(lens >= i + 1).sum() for i in range(M)], dtype=np.int64)
    return reach, accept


def profile(reach, accept):
    """a_i = accepted / reached at position i (NaN where no block reached it)."""
    reach = np.asarray(reach, dtype=np.float64)
    accept = np.asarray(accept, dtype=np.float64)
    out = np.full(reach.shape, np.nan)
    ok = reach > 0
    out[ok] = accept[ok] / reach[ok]
    return out


def survival(a):
    """A_0 = 1, A_k = prod_{i<k} a_i (0-based a), k = 0..M."""
    a = np.asarray(a, dtype=np.float64)
    A = np.ones(len(a) + 1)
    for k in range(1, len(a) + 1):
        A[k] = A[k - 1] * a[k - 1]
    return A


def length_law(a):
    """Pr(L = k), k = 0..M (Eq. 2)."""
    a = np.asarray(a, dtype=np.float64)
    M = len(a)
    A = survival(a)
    pr = np.empty(M + 1)
    for k in range(M):
        pr[k] = A[k] * (1.0 - a[k])
    pr[M] = A[M]
    return pr


def tpf(a, g, c):
    pr = length_law(a)
    return float(np.dot(pr, g) / np.dot(pr, c))


def fpt(a, g, c):
    return 1.0 / tpf(a, g, c)


def unit_costs(M: int):
    """g_k = k + 1 committed tokens (the accepted prefix plus one), c_k = 1 forward pass."""
    return np.arange(M + 1, dtype=np.float64) + 1.0, np.ones(M + 1)


def isd_costs(M: int):
    """Eq. 8's gains and costs for Eq. 2: g_k = 2 + min(k, M - 1); c_k = 2 for k < M, c_M = 1."""
    g = np.array([2.0 + min(k, M - 1) for k in range(M + 1)])
    c = np.array([2.0] * M + [1.0])
    return g, c


def tpf_isd_profile(a) -> float:
    """Eq. 8: TPF(a) = (2 + sum_{k=1}^{M-1} A_k) / (2 - A_M) for a profile of M positions."""
    a = np.asarray(a, dtype=np.float64)
    M = len(a)
    A = survival(a)
    return float((2.0 + sum(A[k] for k in range(1, M))) / (2.0 - A[M]))


def tpf_isd(N: int, r: float) -> float:
    """Sec. 2.2: tokens per forward of the ISD stride-N rule at constant rejection r."""
    q = 1.0 - r
    num = 2.0 + sum(q ** i for i in range(1, N - 1))
    return num / (2.0 - q ** (N - 1))


def _dlaw_da(a):
    """J[k, i] = dPr(L = k) / da_i, from products that leave a_i out (no division)."""
    a = np.asarray(a, dtype=np.float64)
    M = len(a)
    J = np.zeros((M + 1, M))
    for k in range(M + 1):
        for i in range(M):
            if i < k:   # A_k contains a_i
                d_Ak = np.prod([a[j] for j in range(k) if j != i])
                J[k, i] += d_Ak * ((1.0 - a[k]) if k < M else 1.0)
            if k < M and i == k:   # the factor (1 - a_k)
                J[k, i] -= np.prod(a[:k])
    return J


def weights(a, g, c, eps: float = 1e-8):
    """w_raw_i = -dFPT/dz_i and the mean-one normalised w_bar (Eq. 3)."""
    a = np.asarray(a, dtype=np.float64)
    M = len(a)
    pr = length_law(a)
    G = float(np.dot(pr, g))
    C = float(np.dot(pr, c))
    J = _dlaw_da(a)
    dG = J.T @ np.asarray(g, dtype=np.float64)
    dC = J.T @ np.asarray(c, dtype=np.float64)
    # FPT = C / G  ->  dFPT/da = (dC G - C dG) / G^2
    dfpt_da = (dC * G - C * dG) / (G * G)
    w_raw = -dfpt_da * a * (1.0 - a)
    w_bar = M * w_raw / (w_raw.sum() + eps)
    return w_raw, w_bar
