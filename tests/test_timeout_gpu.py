"""A bounded device-side wait that runs out (failure detection without a GPU fault).

The tensor-core products wait on mbarriers for their TMA loads and tensor-core operations; each
wait gives up after a limit of SM cycles. A limit of one cycle makes the first wait whose data is
still arriving give up (a TMA load from memory takes far longer): the call must report
BRISK_ERR_TIMEOUT through the device status, drain what it started, leave the context usable,
and the next call with the default limit must return the same results as before."""
import pytest
import torch

from paper_2609_33390_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def brisk():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


def test_expired_wait_reports_timeout_and_the_next_call_is_correct(brisk):
    wl = synth.Workload("timeout", B=2, L=16, V=2048, d=4096, K=8, r=64, agree0=0.9,
                        agree_decay=0.97)
    w = synth.make_weights(wl, "cuda")
    blk = synth.make_block(wl, "cuda")
    tail = brisk.DecodeTail.for_workload(wl, w)
    tail.prepare()
    c = tail.topk(blk["logits_q"])
    args = (blk["hidden"], blk["h_c"], blk["x0"], blk["logits_q"], c["cand_ids"],
            c["cand_logprob"])
    ref = tail.select(*args)
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    prev = brisk.set_wait_limit(1)
    try:
        tail.select(*args)
        torch.cuda.synchronize()
        assert tail.device_status() == brisk.ERR_TIMEOUT
    finally:
        brisk.set_wait_limit(prev)
    again = tail.select(*args)
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    assert torch.equal(again["sel_tokens"], ref["sel_tokens"])
    assert torch.equal(again["refined"], ref["refined"])
