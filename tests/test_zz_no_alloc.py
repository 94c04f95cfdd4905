"""The no-allocation candidate entry point, for callers that cannot give the library a workspace
(a plug-in handed only its input and output buffers, an engine whose memory manager owns all of
HBM, a decode loop that must not allocate). It must agree with brisk_topk_candidates, which
uses a caller workspace, on two calls in a row: the second call reuses the library's fixed
scratch array that the first call left behind. Both calls are also checked against the oracle's
candidates row by row."""
import ctypes

import numpy as np
import pytest
import torch

from oracle import brisk_oracle as O
from paper_2609_33390_gb300 import synth

ATOL = 1e-3


@pytest.fixture(scope="module")
def B():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk
    return brisk


def test_noalloc_rejects_problems_larger_than_its_array(B):
    d = B.make_dims(B=4096, L=64, V=151936, d=64, K=32, r=16, logits_dtype=torch.bfloat16,
                    hidden_dtype=torch.bfloat16)
    fake = ctypes.c_void_p(256)   # never used: the size check comes first
    assert B.lib().brisk_topk_candidates_noalloc(ctypes.byref(d), fake, fake, fake, fake,
                                                 None) == B.ERR_UNSUPPORTED
    bad = B.make_dims(B=1, L=1, V=100, d=64, K=3, r=16, logits_dtype=torch.bfloat16,
                      hidden_dtype=torch.bfloat16)
    assert B.lib().brisk_topk_candidates_noalloc(ctypes.byref(bad), fake, fake, fake, fake,
                                                 None) == B.ERR_INVALID_ARG


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_twice(B):
    dev = torch.device("cuda")
    wl = synth.Workload("noalloc", B=6, L=16, V=40003, d=32, K=16, r=16, agree0=0.9,
                        agree_decay=0.97)
    weights = {k: (v.to(dev) if torch.is_tensor(v) else v)
               for k, v in synth.make_weights(wl.with_(V=64), "cpu").items()}
    tail = B.DecodeTail(wl.B, wl.L, wl.V, wl.d, wl.K, wl.r, wl.logits_dtype, wl.hidden_dtype,
                        weights, dev)
    for call, block_id in enumerate((0, 1)):
        lq = synth.make_block(wl, "cpu", block=block_id)["logits_q"].to(dev)
        ref = tail.topk(lq)
        ids = torch.full((wl.B, wl.L, wl.K), -7, dtype=torch.int32, device=dev)
        lp = torch.full((wl.B, wl.L, wl.K), float("nan"), device=dev)
        lse = torch.full((wl.B, wl.L), float("nan"), device=dev)
        st = B.topk_candidates_noalloc(tail.dims, lq, ids, lp, lse)
        assert st == B.OK, B.status_string(st)
        torch.cuda.synchronize()
        assert torch.equal(ids, ref["cand_ids"]), f"call {call}"
        np.testing.assert_allclose(lp.cpu().numpy(), ref["cand_logprob"].cpu().numpy(), rtol=0,
                                   atol=ATOL, err_msg=f"call {call}")
        np.testing.assert_allclose(lse.cpu().numpy(), ref["lse_q"].cpu().numpy(), rtol=0,
                                   atol=ATOL, err_msg=f"call {call}")
        # and against the oracle's candidates, row by row
        rows = lq.float().reshape(-1, wl.V).cpu().numpy().astype(np.float64)
        ids_h = ids.reshape(-1, wl.K).cpu().numpy()
        lp_h = lp.reshape(-1, wl.K).cpu().numpy()
        lse_h = lse.reshape(-1).cpu().numpy()
        for j in range(rows.shape[0]):
            o_ids, o_lp, o_lse = O.topk_candidates(rows[j], wl.K)
            np.testing.assert_array_equal(ids_h[j], o_ids, err_msg=f"call {call} row {j}")
            assert np.abs(lp_h[j] - o_lp).max() <= ATOL and abs(lse_h[j] - o_lse) <= ATOL
