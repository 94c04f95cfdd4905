"""The fused decode tail on logits in page-locked host memory, read in place by the kernels.

The results must be those of the same call on device-resident logits, bit for bit, and those
of the oracle. Cases: a fused small-batch call (both tensors in one sweep launch, the corrector
verifying in its CTA) under stochastic verification, and an overlapping-schedule call (one task
per proposal row, verifier sweep on the low-priority stream).
"""
import numpy as np
import pytest
import torch

from paper_2609_33390_gb300 import synth

from parity import Report, check_sequence, oracle_params, to_numpy

pytestmark = pytest.mark.gpu

CASES = [
    ("fused_stochastic", dict(B=2, L=8, V=20011, d=64, K=8, r=32, select_mode="sample",
                              verify_mode="stochastic")),
    ("overlap_greedy", dict(B=80, L=32, V=4096, d=64, K=8, r=32)),
]


@pytest.fixture(scope="module")
def brisk():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
def test_host_logits_match_device_logits_and_oracle(brisk, name, kw):
    base = dict(agree0=0.9, agree_decay=0.97, weight_std=0.1)
    base.update(kw)
    wl = synth.Workload(name, **base)
    dev = torch.device("cuda")
    weights = {k: (v.to(dev) if torch.is_tensor(v) else v)
               for k, v in synth.make_weights(wl, "cpu").items()}
    cpu_block = synth.make_block(wl, "cpu")
    block = {k: (v.to(dev) if torch.is_tensor(v) else v) for k, v in cpu_block.items()}
    host_block = dict(block)
    host_block["logits_q"] = cpu_block["logits_q"].pin_memory()
    host_block["logits_p"] = cpu_block["logits_p"].pin_memory()
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    tail = brisk.DecodeTail.for_workload(wl, weights, dev)
    tail.prepare()
    out_dev = tail.tail(block, sm, vm)
    out_host = tail.tail(host_block, sm, vm)
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    g_dev, g_host = to_numpy(out_dev), to_numpy(out_host)
    for k in g_dev:
        np.testing.assert_array_equal(g_host[k], g_dev[k], err_msg=k)
    params = oracle_params(weights)
    rep = Report()
    seqs = range(wl.B) if wl.B <= 4 else (0, 1, wl.B // 2, wl.B - 1)
    for b in seqs:
        check_sequence(b, block, params, wl.K, g_host, wl.select_mode, wl.verify_mode, rep)
    assert rep.sequences == len(seqs)
