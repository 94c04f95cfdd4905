"""The decode tail captured into a CUDA graph (App. F) replays exactly what direct calls
compute, block after block with the anchor chained on the device."""
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


@pytest.mark.parametrize("kw", [dict(B=2, L=8, V=4099, d=64, K=8, r=32),
                                dict(B=3, L=12, V=5003, d=64, K=4, r=16, select_mode="sample",
                                     verify_mode="stochastic"),
                                # 2560 rows: the overlapping schedule (three side streams)
                                dict(B=80, L=32, V=4096, d=512, K=8, r=256)])
def test_graph_replays_match_direct_calls(brisk, kw):
    wl = synth.Workload("graph", agree0=0.9, agree_decay=0.97, weight_std=0.2, **kw)
    w = synth.make_weights(wl, "cuda")
    blk = synth.make_block(wl, "cuda")
    tail = brisk.DecodeTail.for_workload(wl, w)
    tail.prepare()
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    steps = 4
    # direct calls, anchor chained by hand
    direct = []
    x0 = blk["x0"].clone()
    for _ in range(steps):
        out = tail.tail(blk, sm, vm, x0=x0)
        torch.cuda.synchronize()
        direct.append({k: v.clone() for k, v in out.items()})
        x0 = out["next_anchor"].clone()
    # the same blocks through one captured graph
    stream = torch.cuda.Stream()
    g = tail.graph(blk, sm, vm, stream=stream)
    for s in range(steps):
        out = g.launch()
        stream.synchronize()
        for k in ("accepted_len", "out_tokens", "correction", "sel_tokens", "refined", "cand_ids",
                  "cand_logprob"):
            assert torch.equal(out[k], direct[s][k]), (s, k)
        assert torch.equal(g.anchor, direct[s]["next_anchor"])
    g.close()
    assert tail.device_status() == brisk.OK


def test_double_buffered_graph_loop_matches_direct_calls(brisk):
    """Two captured graphs over two input buffer sets, the next block copied in on a second
    stream while the current one runs, the anchor chained on the device: the same results as
    direct calls on the same sequence of blocks."""
    from paper_2609_33390_gb300.loop import graph_loop_double_buffered
    wl = synth.Workload("graphloop", B=2, L=8, V=4099, d=64, K=8, r=32, agree0=0.9,
                        agree_decay=0.97, weight_std=0.2)
    w = synth.make_weights(wl, "cuda")
    pool = [synth.make_block(wl, "cuda", block=j) for j in range(3)]
    tail = brisk.DecodeTail.for_workload(wl, w)
    tail.prepare()
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    blocks = 7
    direct = []
    x0 = pool[0]["x0"].clone()
    for t in range(blocks):
        out = tail.tail(pool[t % len(pool)], sm, vm, x0=x0)
        torch.cuda.synchronize()
        direct.append({k: v.clone() for k, v in out.items()})
        x0 = out["next_anchor"].clone()
    stream = torch.cuda.Stream()
    ms, nbytes, outs = graph_loop_double_buffered(tail, pool, sm, vm, stream, blocks, keep=True)
    assert ms > 0 and nbytes > 0 and len(outs) == blocks
    for t in range(blocks):
        for k in ("accepted_len", "out_tokens", "correction", "sel_tokens", "refined",
                  "cand_ids", "next_anchor"):
            assert torch.equal(outs[t][k], direct[t][k]), (t, k)
    assert tail.device_status() == brisk.OK
