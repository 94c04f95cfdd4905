"""GPU same-state replay diagnostics (App. B, Eq. 6) against the oracle."""
import numpy as np
import pytest
import torch

from oracle import brisk_oracle as O
from paper_2609_33390_gb300 import synth
from tests.parity import TIE_TOL, np64, oracle_params

pytestmark = pytest.mark.gpu

F32 = torch.float32


@pytest.fixture(scope="module")
def brisk():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


def _to(d, device):
    return {k: (v.to(device) if torch.is_tensor(v) else v) for k, v in d.items()}


CASES = [
    ("bf16_greedy", dict(B=3, L=8, V=5003, d=64, K=8, r=16)),
    ("bf16_sample", dict(B=2, L=12, V=4096, d=128, K=8, r=64, select_mode="sample")),
    ("f32_k16", dict(B=2, L=6, V=3001, d=48, K=16, r=32, logits_dtype=F32, hidden_dtype=F32)),
    ("long_block", dict(B=1, L=64, V=1500, d=32, K=4, r=16)),
]


def _oracle_replay(params, block, b, K, mode):
    lq, lp = np64(block["logits_q"][b]), np64(block["logits_p"][b])
    L = lq.shape[0]
    cand = np.zeros((L, K), np.int64)
    clp = np.zeros((L, K))
    top4 = np.zeros((L, 4), np.int64)
    for i in range(L):
        cand[i], clp[i], _ = O.topk_candidates(lq[i], K)
        top4[i] = O.ranked_ids(lq[i])[:4]
    u_sel = block["u_sel"][b].cpu().numpy().astype(np.float64)
    u_acc = block["u_acc"][b].cpu().numpy().astype(np.float64)
    res = O.replay_sequence(params, lambda i: lq[i], lambda i: lp[i], np64(block["hidden"][b]),
                            np64(block["h_c"][b]), int(block["x0"][b]), cand, clp, top4, u_acc,
                            mode, u_sel)
    return cand, res, u_acc


@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
def test_replay_matches_oracle(brisk, name, kw):
    base = dict(agree0=0.9, agree_decay=0.97, weight_std=0.2)
    base.update(kw)
    wl = synth.Workload(name, **base)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    tail = brisk.DecodeTail.for_workload(wl, weights)
    tail.prepare()
    sm, _ = brisk.mode_ids(wl.select_mode, "greedy")
    out = tail.replay(block, sm)
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    head = out["head_tokens"].cpu().numpy()
    flags = out["flags"].cpu().numpy()
    fb_gpu = out["first_breaker"].cpu().numpy()
    params = oracle_params(weights)
    mode = O.SAMPLE if wl.select_mode == "sample" else O.GREEDY
    compared = 0
    for b in range(wl.B):
        cand, res, u = _oracle_replay(params, block, b, wl.K, mode)
        # compare up to the first near-tie of a decision (head selection or a draw vs alpha)
        stop = wl.L
        for i in range(wl.L):
            if (res.trace.margin[i] < TIE_TOL or abs(u[i] - res.alpha_base[i]) < 1e-5
                    or abs(u[i] - res.alpha_head[i]) < 1e-5):
                stop = i
                break
        for i in range(stop):
            assert head[b, i] == cand[i][res.head_rank[i]], (b, i)
            f = flags[b, i]
            jb, jh = bool(f & 1), bool(f & 2)
            assert jb == (u[i] < res.alpha_base[i]) and jh == (u[i] < res.alpha_head[i]), (b, i)
            assert bool(f & 8) == bool(res.intervention[i])
            if stop == wl.L or i < stop:
                assert bool(f & 32) == bool(res.regression[i])
            compared += 1
        if stop == wl.L:
            assert fb_gpu[b] == res.first_breaker
            for i in range(wl.L):
                assert bool(flags[b, i] & 4) == (i == res.first_breaker)
                assert bool(flags[b, i] & 16) == bool(res.rescue[i])
    assert compared > 0


def test_closed_gate_never_intervenes(brisk):
    wl = synth.Workload("off", B=4, L=16, V=3000, d=32, K=8, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    weights["alpha"] = float("-inf")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    tail = brisk.DecodeTail.for_workload(wl, weights)
    tail.prepare()
    out = tail.replay(block)
    torch.cuda.synchronize()
    flags = out["flags"]
    assert not torch.any(flags & (8 | 16 | 32))
