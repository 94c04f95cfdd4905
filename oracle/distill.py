"""Plain CPU oracle of the corrector's distillation loss and its gradient (float64).

TEST INFRASTRUCTURE ONLY: the literal statement of the training objective of the refinement
head, to check the library's kernel against. Only the tests may import it. It shares no code
with the library.

What it follows (paper "From Position Risks to Block Survival", App. C.3, Eq. 10 "head training
loss" and the paragraph before it): at every reached position j of a block (the accepted prefix
and the first rejected position; every position of an all-pass block) the target is the
verifier distribution restricted to the candidate set S_j and renormalised, p_S; the base
distribution restricted to S_j is q_S; the refined distribution is r = softmax(refined scores).
The per-position loss is CE(p_S, r) + beta KL(q_S || r), beta = 0.01, and the objective is one
mean over all reached positions of the batch.

Readings: positions are 0-based, so a block with accepted length a reaches positions
0..min(a, L-1); p_S uses the verifier logits at the candidate ids (exp-normalised over the K
candidates); q_S uses the candidates' log-probabilities of the proposal (the same as its raw
logits after renormalisation). Gradient with respect to the refined scores of a reached
position: ((r - p_S) + beta (r - q_S)) / (number of reached positions).
"""
from __future__ import annotations

import numpy as np

BETA = 0.01


def _softmax(x):
    x = np.asarray(x, dtype=np.float64)
    m = np.max(x)
    if not np.isfinite(m):
        raise ValueError("no finite entry")
    e = np.exp(x - m)
    return e / e.sum()


def _log_softmax(x):
    x = np.asarray(x, dtype=np.float64)
    m = np.max(x)
    return x - (m + np.log(np.exp(x - m).sum()))


def reached_mask(accepted_len, L: int):
    """m[b, j] = 1 for j <= min(accepted_len[b], L - 1); lengths outside 0..L are clamped
    (an accepted length is at least 0, so position 0 is always reached)."""
    a = np.clip(np.asarray(accepted_len, dtype=np.int64), 0, L)
    j = np.arange(L)
    return (j[None, :] <= np.minimum(a, L - 1)[:, None]).astype(np.float64)


def position_loss(p_logits_at_cands, cand_logprob, refined, beta: float = BETA):
    """CE(p_S, r) + beta KL(q_S || r) for one position, and its gradient in the refined scores."""
    p = _softmax(p_logits_at_cands)
    q = _softmax(cand_logprob)
    log_r = _log_softmax(refined)
    r = np.exp(log_r)
    ce = -np.sum(p * log_r)
    kl = np.sum(np.where(q > 0, q * (np.log(np.where(q > 0, q, 1.0)) - log_r), 0.0))
    loss = ce + beta * kl
    grad = (r - p) + beta * (r - q)
    return loss, grad


def distill_loss(p_logits_at_cands, cand_logprob, refined, accepted_len, beta: float = BETA):
    """Mean loss over the reached positions of a batch [B, L, K] and its gradient."""
    P = np.asarray(p_logits_at_cands, dtype=np.float64)
    Q = np.asarray(cand_logprob, dtype=np.float64)
    R = np.asarray(refined, dtype=np.float64)
    B, L, K = R.shape
    mask = reached_mask(accepted_len, L)
    n = mask.sum()
    total = 0.0
    grad = np.zeros_like(R)
    for b in range(B):
        for j in range(L):
            if mask[b, j] == 0:
                continue
            l, g = position_loss(P[b, j], Q[b, j], R[b, j], beta)
            total += l
            grad[b, j] = g
    if n == 0:
        return 0.0, grad
    return total / n, grad / n
