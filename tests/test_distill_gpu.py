"""GPU distillation loss (App. C.3, Eq. 10) and its gradient against the float64 oracle."""
import numpy as np
import pytest
import torch

from oracle import distill as D

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


def _tail(B, Bn, L, V, K, ldt):
    from paper_2609_33390_gb300 import synth
    wl = synth.Workload("distill", B=Bn, L=L, V=V, d=64, K=K, r=16, logits_dtype=ldt,
                        hidden_dtype=torch.bfloat16, agree0=0.8)
    w = {k: v for k, v in synth.make_weights(wl, "cuda").items()}
    tail = B.DecodeTail.for_workload(wl, w, torch.device("cuda"))
    return tail


def _check(B, tail, logits_p, ids, lp, ref, acc, beta=0.01):
    out = tail.distill_loss(logits_p, ids, lp, ref, acc, beta)
    torch.cuda.synchronize()
    assert tail.device_status() == B.OK
    P = np.take_along_axis(logits_p.float().cpu().numpy(), ids.long().cpu().numpy(), axis=-1)
    loss, grad = D.distill_loss(P, lp.cpu().numpy(), ref.cpu().numpy(), acc.cpu().numpy(), beta)
    got_loss = float(out["loss"].item())
    assert abs(got_loss - loss) <= 2e-5 * max(1.0, abs(loss))
    np.testing.assert_allclose(out["grad"].cpu().numpy(), grad, rtol=1e-4, atol=2e-7)
    return got_loss


@pytest.mark.parametrize("ldt", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("Bn,L,K", [(1, 1, 4), (3, 8, 8), (17, 33, 32), (64, 64, 16)])
def test_random_inputs_match_oracle(B, ldt, Bn, L, K):
    V = 701
    tail = _tail(B, Bn, L, V, K, ldt)
    g = torch.Generator(device="cpu").manual_seed(Bn * 100 + L + K)
    logits_p = (torch.randn(Bn, L, V, generator=g) * 2).to(ldt).cuda()
    ids = torch.stack([torch.randperm(V, generator=g)[:K] for _ in range(Bn * L)]).view(Bn, L, K)
    ids = ids.int().cuda()
    lp = torch.log_softmax(torch.randn(Bn, L, V, generator=g) * 2, -1)
    lp = torch.gather(lp, -1, ids.long().cpu()).float().cuda()
    ref = (lp.cpu() + torch.randn(Bn, L, K, generator=g)).float().cuda()
    acc = torch.randint(-1, L + 2, (Bn,), generator=g).int().cuda()
    _check(B, tail, logits_p, ids, lp, ref, acc)


def test_on_decode_tail_outputs_and_deterministic(B):
    from paper_2609_33390_gb300 import synth
    wl = synth.WORKLOADS["tiny"]
    w = synth.make_weights(wl, "cuda")
    tail = B.DecodeTail.for_workload(wl, w, torch.device("cuda"))
    tail.prepare()
    blk = synth.make_block(wl, "cuda")
    sm, vm = B.mode_ids(wl.select_mode, wl.verify_mode)
    out = tail.tail(blk, sm, vm)
    torch.cuda.synchronize()
    l1 = _check(B, tail, blk["logits_p"], out["cand_ids"], out["cand_logprob"], out["refined"],
                out["accepted_len"])
    l2 = _check(B, tail, blk["logits_p"], out["cand_ids"], out["cand_logprob"], out["refined"],
                out["accepted_len"])
    assert l1 == l2
    no_grad = tail.distill_loss(blk["logits_p"], out["cand_ids"], out["cand_logprob"],
                                out["refined"], out["accepted_len"], with_grad=False)
    assert float(no_grad["loss"].item()) == l1
