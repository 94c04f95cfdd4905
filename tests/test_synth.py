"""The seeded generator: published known-answer values and recipe properties."""
import numpy as np
import torch

from paper_2609_33390_gb300 import synth


def _philox(ctr, key):
    out = synth.philox4x32_10(tuple(torch.tensor([c], dtype=torch.int64) for c in ctr), key)
    return [int(o) for o in out]


def test_philox4x32_10_known_answers():
    # Known-answer vectors published with Random123 (Salmon et al., SC'11).
    assert _philox([0, 0, 0, 0], (0, 0)) == [0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8]
    m = 0xFFFFFFFF
    assert _philox([m, m, m, m], (m, m)) == [0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD]
    assert _philox([0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344], (0xA4093822, 0x299F31D0)) \
        == [0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1]


def test_splitmix64_reference_sequence():
    # Vigna's splitmix64 from state 0 yields these two words first.
    assert synth.splitmix64(0) == 0xE220A8397B1DCDAF
    assert synth.splitmix64(0x9E3779B97F4A7C15) == 0x6E789E6AA1B965F4


def test_words_are_position_independent():
    keys = [synth.sequence_key(0, 3, 1), synth.sequence_key(0, 4, 1)]
    full = synth.philox_words(keys, 7, 0, 50, "cpu")
    part = synth.philox_words(keys, 7, 13, 20, "cpu")
    assert torch.equal(full[:, 13:33], part)


def test_distributions_roughly_right():
    keys = [synth.sequence_key(5, 0)]
    z = synth.normal(keys, 1, 200000, "cpu")[0].numpy()
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1) < 0.01
    u = synth.uniform_f32(keys, 2, 100000, "cpu")[0].numpy()
    assert u.min() >= 0 and u.max() < 1 and abs(u.mean() - 0.5) < 0.005
    e = synth.exponential(keys, 3, 100000, 3.0, "cpu")[0].numpy()
    assert abs(e.mean() - 3.0) < 0.05


def test_planted_head_is_the_proposal_argmax_and_blocks_are_deterministic():
    wl = synth.Workload("t", B=3, L=5, V=300, d=16, K=4, r=8, agree0=0.9, agree_decay=0.97)
    a = synth.make_block(wl, "cpu")
    b = synth.make_block(wl, "cpu")
    for k in a:
        assert torch.equal(a[k], b[k]), k
    lq = a["logits_q"].float()
    top2 = torch.topk(lq, 2, dim=-1).values
    assert torch.all(top2[..., 0] >= top2[..., 1])
    assert a["logits_q"].dtype == torch.bfloat16 and a["x0"].dtype == torch.int32
    c = synth.make_block(wl, "cpu", block=1)
    assert not torch.equal(a["logits_q"], c["logits_q"])


def test_zipf_recipe_and_weights_shapes():
    wl = synth.Workload("z", B=2, L=3, V=500, d=32, K=16, r=16, recipe="zipf", agree0=0.9,
                        agree_decay=0.98)
    blk = synth.make_block(wl, "cpu")
    lq = blk["logits_q"].float()
    assert lq.shape == (2, 3, 500)
    # the same id is near the top in every row of a sequence (one permutation per sequence)
    top = lq.argmax(-1)
    assert (top[0] == top[0, 0]).float().mean() > 0.3
    w = synth.make_weights(wl, "cpu")
    for k, shape in synth.weight_shapes(wl).items():
        assert tuple(w[k].shape) == shape
    assert w["E_in"].shape == (500, 32) and w["E_out"].shape == (500, 32)


def test_decode_stream_agreement_is_per_sequence():
    wl = synth.WORKLOADS["decode_stream"].with_(V=100, d=8, r=8)
    a = synth.agreement(wl, [0, 1, 2], "cpu")
    assert a.shape == (3, wl.L)
    assert torch.all(a[:, :1] == a)
    assert torch.all((a >= 0.6) & (a <= 0.98))
