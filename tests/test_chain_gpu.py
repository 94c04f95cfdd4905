"""Consecutive blocks of a decode stream against the oracle (Algorithm 1(b), commit step; App. F
CUDA Graph replay of the fused head).

The anchor of block t+1 is the last token block t commits: the correction when a position is
rejected, the last selection when the whole block is accepted. On the GPU the anchor chains on
the device (the fused call's next_anchor output feeds the next call's x0); the oracle chains its
own anchors from its own results, block by block, and every block of every checked sequence is
compared element by element (candidates, log-probabilities, selections, refined scores, accepted
length, committed tokens, correction and next anchor). Rejected blocks are asserted to occur, so
the anchor after a rejection is checked as well as the one after a fully accepted block.
"""
import numpy as np
import pytest
import torch

from oracle import brisk_oracle as O
from paper_2609_33390_gb300 import synth

from parity import Report, check_sequence, oracle_params, to_numpy

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def brisk():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


def _direct_chain(tail, pool, sm, vm, blocks):
    """`blocks` fused calls, block t on pool[t % len(pool)], the anchor chained on the device."""
    outs = []
    x0 = pool[0]["x0"].clone()
    for t in range(blocks):
        out = tail.tail(pool[t % len(pool)], sm, vm, x0=x0)
        x0 = out["next_anchor"]
        outs.append(out)
    torch.cuda.synchronize()
    return [to_numpy(o) for o in outs]


def _oracle_chain(wl, weights, pool, gpu_outs, seqs):
    """Checks every block of the sequences `seqs` against the oracle with its own chained
    anchors; returns the report and the number of (sequence, block) pairs with a rejection."""
    params = oracle_params(weights)
    rep = Report()
    anchors = {b: int(pool[0]["x0"][b]) for b in seqs}
    rejected = 0
    for t, g in enumerate(gpu_outs):
        blk = pool[t % len(pool)]
        for b in seqs:
            tr, vr = check_sequence(b, blk, params, wl.K, g, wl.select_mode, wl.verify_mode, rep,
                                    x0=anchors[b])
            anchors[b] = O.next_anchor(vr, tr.sel_tokens)
            rejected += int(vr.accepted_len < wl.L)
    return rep, rejected


SMALL = [
    dict(B=3, L=8, V=4099, d=64, K=8, r=32),
    dict(B=3, L=12, V=5003, d=64, K=4, r=16, select_mode="sample", verify_mode="stochastic"),
    dict(B=2, L=6, V=3001, d=48, K=16, r=32, logits_dtype=torch.float32,
         hidden_dtype=torch.float32),
]


@pytest.mark.parametrize("kw", SMALL, ids=["greedy_bf16", "stochastic_bf16", "greedy_f32"])
def test_chained_blocks_direct_and_graph_loop_match_oracle(brisk, kw):
    wl = synth.Workload("chain", agree0=0.9, agree_decay=0.97, weight_std=0.2, **kw)
    w = synth.make_weights(wl, "cuda")
    pool = [synth.make_block(wl, "cuda", block=j) for j in range(3)]
    tail = brisk.DecodeTail.for_workload(wl, w)
    tail.prepare()
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    blocks = 6
    direct = _direct_chain(tail, pool, sm, vm, blocks)
    assert tail.device_status() == brisk.OK
    rep, rejected = _oracle_chain(wl, w, pool, direct, range(wl.B))
    assert rep.sequences == wl.B * blocks
    assert rejected > 0
    # the same stream of blocks through the double-buffered graph loop
    from paper_2609_33390_gb300.loop import graph_loop_double_buffered
    stream = torch.cuda.Stream()
    _, _, outs = graph_loop_double_buffered(tail, pool, sm, vm, stream, blocks, keep=True)
    assert tail.device_status() == brisk.OK
    rep2, _ = _oracle_chain(wl, w, pool, [to_numpy(o) for o in outs], range(wl.B))
    assert rep2.sequences == wl.B * blocks


@pytest.mark.parametrize("name,seqs", [("decode_stream", [0, 1, 64, 127]),
                                       ("batched_stochastic", [0, 5, 10, 15])])
def test_chained_blocks_full_size_match_oracle(brisk, name, seqs):
    """Three consecutive blocks at full size (each block's inputs regenerated from the seed and
    the (sequence, block) pair, the anchor chained), direct calls and the double-buffered graph
    loop, sampled sequences against the chained oracle."""
    wl = synth.WORKLOADS[name]
    w = synth.make_weights(wl, "cuda")
    pool = [synth.make_block(wl, "cuda", block=j) for j in range(3)]
    tail = brisk.DecodeTail.for_workload(wl, w)
    tail.prepare()
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    direct = _direct_chain(tail, pool, sm, vm, 3)
    assert tail.device_status() == brisk.OK
    rep, rejected = _oracle_chain(wl, w, pool, direct, seqs)
    assert rep.sequences == 3 * len(seqs) and rejected > 0
    assert rep.near_ties <= 2, rep.notes
    from paper_2609_33390_gb300.loop import graph_loop_double_buffered
    stream = torch.cuda.Stream()
    _, _, outs = graph_loop_double_buffered(tail, pool, sm, vm, stream, 3, keep=True)
    assert tail.device_status() == brisk.OK
    for t in range(3):
        for k in ("accepted_len", "out_tokens", "correction", "sel_tokens", "refined",
                  "cand_ids", "next_anchor"):
            np.testing.assert_array_equal(outs[t][k].cpu().numpy(), direct[t][k],
                                          err_msg=f"block {t} {k}")
