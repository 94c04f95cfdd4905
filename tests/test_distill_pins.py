"""Pins of the distillation-loss oracle (App. C.3, Eq. 10) against closed forms, invariances,
finite differences and float64 autograd."""
import numpy as np
import pytest
import torch

from oracle import distill as D


def _batch(seed, B=3, L=5, K=6):
    rng = np.random.default_rng(seed)
    P = rng.normal(0, 2, (B, L, K))
    Q = rng.normal(0, 2, (B, L, K))
    Q = Q - np.log(np.exp(Q).sum(-1, keepdims=True)) - rng.uniform(0, 3, (B, L, 1))  # log-probs
    R = rng.normal(0, 2, (B, L, K))
    acc = rng.integers(0, L + 1, B)
    return P, Q, R, acc


def test_gradient_matches_finite_differences():
    P, Q, R, acc = _batch(1)
    loss, grad = D.distill_loss(P, Q, R, acc)
    h = 1e-6
    for idx in [(0, 0, 0), (1, 2, 3), (2, 4, 5), (0, 1, 2)]:
        Rp, Rm = R.copy(), R.copy()
        Rp[idx] += h
        Rm[idx] -= h
        fd = (D.distill_loss(P, Q, Rp, acc)[0] - D.distill_loss(P, Q, Rm, acc)[0]) / (2 * h)
        assert abs(fd - grad[idx]) < 1e-8


def test_loss_and_gradient_match_float64_autograd():
    P, Q, R, acc = _batch(2)
    B, L, K = R.shape
    Rt = torch.tensor(R, dtype=torch.float64, requires_grad=True)
    p = torch.softmax(torch.tensor(P, dtype=torch.float64), -1)
    q = torch.softmax(torch.tensor(Q, dtype=torch.float64), -1)
    logr = torch.log_softmax(Rt, -1)
    per = -(p * logr).sum(-1) + 0.01 * (q * (torch.log(q) - logr)).sum(-1)
    mask = torch.tensor([[1.0 if j <= min(a, L - 1) else 0.0 for j in range(L)] for a in acc],
                        dtype=torch.float64)
    tot = (per * mask).sum() / mask.sum()
    tot.backward()
    loss, grad = D.distill_loss(P, Q, R, acc)
    assert abs(loss - tot.item()) < 1e-12
    np.testing.assert_allclose(grad, Rt.grad.numpy(), atol=1e-14)


def test_matching_distributions_give_entropy_and_zero_gradient():
    rng = np.random.default_rng(3)
    x = rng.normal(0, 1.5, 7)
    loss, grad = D.position_loss(x + 4.0, x - 2.0, x)     # p_S = q_S = r (shift invariance)
    p = np.exp(x - x.max()); p /= p.sum()
    assert abs(loss - (-(p * np.log(p)).sum())) < 1e-12
    assert np.abs(grad).max() < 1e-15


def test_single_candidate_has_no_loss():
    loss, grad = D.position_loss([3.0], [-0.1], [9.0])
    assert loss == 0.0 and grad.tolist() == [0.0]


def test_one_hot_verifier_gives_cross_entropy_of_that_candidate():
    R = np.array([1.0, 2.0, 0.5, -1.0])
    Q = np.log(np.array([0.4, 0.3, 0.2, 0.1]))
    P = np.array([-60.0, -60.0, 60.0, -60.0])
    loss, _ = D.position_loss(P, Q, R, beta=0.0)
    logr = R - (R.max() + np.log(np.exp(R - R.max()).sum()))
    assert abs(loss - (-logr[2])) < 1e-12


def test_unreached_positions_do_not_count():
    P, Q, R, acc = _batch(4, B=4, L=6)
    acc = np.array([0, 2, 6, 3])
    loss, grad = D.distill_loss(P, Q, R, acc)
    R2 = R.copy()
    for b, a in enumerate(acc):
        R2[b, min(a, 5) + 1:] = np.random.default_rng(b).normal(0, 5, R2[b, min(a, 5) + 1:].shape)
    loss2, grad2 = D.distill_loss(P, Q, R2, acc)
    assert loss == loss2
    for b, a in enumerate(acc):
        assert np.all(grad[b, min(a, 5) + 1:] == 0)
    assert D.reached_mask(acc, 6).sum() == 1 + 3 + 6 + 4
