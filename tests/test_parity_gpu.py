"""GPU parity: the CUDA decode tail, called through the C ABI, against the CPU oracle.

Small cases (the oracle runs every sequence) span several chunks, ragged
vocabularies, both dtypes, every K class and both mode pairs; the five
workload configurations run at full size with a sample of sequences checked.
"""
import numpy as np
import pytest
import torch

from oracle import brisk_oracle as O
from paper_2609_33390_gb300 import synth

from parity import Report, check_sequence, oracle_params, to_numpy

pytestmark = pytest.mark.gpu

BF16, F32 = torch.bfloat16, torch.float32


@pytest.fixture(scope="module")
def brisk():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk as B
    return B


def _to(d, device):
    return {k: (v.to(device) if torch.is_tensor(v) else v) for k, v in d.items()}


def _run_and_check(B, wl, weights, block, seqs=None, unfused=True, status=None):
    dev = torch.device("cuda")
    sm, vm = B.mode_ids(wl.select_mode, wl.verify_mode)
    tail = B.DecodeTail.for_workload(wl, weights, dev, B=block["logits_q"].shape[0])
    tail.prepare()
    out = tail.tail(block, sm, vm)
    torch.cuda.synchronize()
    assert tail.device_status() == (B.OK if status is None else status)
    g = to_numpy(out)
    if unfused:
        c = tail.topk(block["logits_q"])
        s = tail.select(block["hidden"], block["h_c"], block["x0"], block["logits_q"],
                        c["cand_ids"], c["cand_logprob"], sm, block["u_sel"])
        v = tail.verify(block["logits_p"], s["sel_tokens"], c["cand_ids"], s["refined"], sm, vm,
                        block["u_acc"], block["u_res"])
        torch.cuda.synchronize()
        u = to_numpy({**c, **s, **v})
        for k in u:   # the fused path is the unfused path, bit for bit
            np.testing.assert_array_equal(u[k], g[k], err_msg=k)
    params = oracle_params(weights)
    rep = Report()
    n = block["logits_q"].shape[0]
    for b in (range(n) if seqs is None else seqs):
        check_sequence(b, block, params, wl.K, g, wl.select_mode, wl.verify_mode, rep)
    return rep, g


SMALL = [
    # name, shape overrides
    ("bf16_k4_ragged", dict(B=3, L=8, V=5003, d=64, K=4, r=16)),
    ("bf16_k8_sample", dict(B=2, L=12, V=4096, d=128, K=8, r=64, select_mode="sample",
                            verify_mode="stochastic")),
    ("f32_k16", dict(B=2, L=6, V=3001, d=48, K=16, r=32, logits_dtype=F32, hidden_dtype=F32)),
    ("f32_logits_bf16_hidden", dict(B=2, L=7, V=2048, d=64, K=8, r=16, logits_dtype=F32)),
    ("bf16_k32_stoch_greedy_select", dict(B=2, L=9, V=6007, d=32, K=32, r=48,
                                          verify_mode="stochastic")),
    ("zipf_ties", dict(B=2, L=10, V=20000, d=64, K=16, r=32, recipe="zipf", agree0=0.9,
                       agree_decay=0.98)),
    ("one_position", dict(B=5, L=1, V=999, d=16, K=4, r=16)),
    ("k_equals_v", dict(B=2, L=4, V=8, d=16, K=8, r=16, select_mode="sample",
                        verify_mode="stochastic")),
    ("long_block", dict(B=1, L=64, V=1500, d=32, K=8, r=16)),
    # states wider than 512 (eight warps a sequence), every K class of that kernel; weights of
    # std 0.06 keep the refined scores O(10) as in the workloads (at 0.2 they reach ~2800, where
    # fp32 rounding alone is ~1e-5 relative, beyond the 1e-3 absolute bound)
    ("wide_state_k8_sample", dict(B=2, L=5, V=2000, d=64, K=8, r=512, select_mode="sample",
                                  verify_mode="stochastic", weight_std=0.06)),
    ("wide_state_k16", dict(B=2, L=7, V=2500, d=64, K=16, r=384, weight_std=0.06)),
    ("wide_state_k32", dict(B=2, L=6, V=3000, d=64, K=32, r=512, weight_std=0.06)),
    # 2-element chunks: four warps (S = 192, chunks ending inside the third warp; S = 256) and
    # eight warps (S = 512) in the K classes the workloads do not reach
    ("state192_k16", dict(B=2, L=6, V=2200, d=64, K=16, r=96, weight_std=0.1)),
    ("state256_k32_sample", dict(B=2, L=5, V=2600, d=64, K=32, r=128, select_mode="sample",
                                 verify_mode="stochastic", weight_std=0.1)),
    ("state512_k16", dict(B=2, L=6, V=2400, d=64, K=16, r=256, weight_std=0.06)),
    ("state512_k32", dict(B=2, L=5, V=3100, d=64, K=32, r=256, weight_std=0.06)),
]


@pytest.mark.parametrize("name,kw", SMALL, ids=[s[0] for s in SMALL])
def test_small_parity(brisk, name, kw):
    base = dict(agree0=0.9, agree_decay=0.97, weight_std=0.2)
    base.update(kw)
    wl = synth.Workload(name, **base)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    rep, g = _run_and_check(brisk, wl, weights, block)
    assert rep.sequences == wl.B
    # the corrector really acts on these inputs
    if wl.K > 1 and name not in ("one_position",):
        assert rep.max_ref_err <= 1e-3


def test_corrector_off_identical_distributions_accept_all(brisk):
    wl = synth.Workload("off", B=3, L=16, V=3000, d=32, K=8, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    weights["alpha"] = float("-inf")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    block["logits_p"] = block["logits_q"].clone()
    tail = brisk.DecodeTail.for_workload(wl, weights)
    tail.prepare()
    out = tail.tail(block)
    torch.cuda.synchronize()
    assert torch.all(out["accepted_len"] == wl.L)
    assert torch.equal(out["sel_tokens"], out["cand_ids"][..., 0])
    assert torch.all(out["correction"] == -1)
    assert torch.equal(out["next_anchor"], out["sel_tokens"][:, -1])


def test_ties_and_minus_infinity(brisk):
    wl = synth.Workload("ties", B=2, L=4, V=1000, d=32, K=8, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    lq = block["logits_q"]
    lq[0, 0] = 1.0                             # all equal: ids 0..K-1
    lq[0, 1, ::3] = float("-inf")              # -inf entries
    lq[1, 2] = torch.round(lq[1, 2].float() * 2).to(lq.dtype)   # many exact ties
    lq[1, 3, :] = float("-inf")
    lq[1, 3, 500:503] = 2.0                    # three finite values, the rest -inf
    # the last row's top1-top4 gap is +inf, so its gate and refined scores are NaN: reported
    rep, g = _run_and_check(brisk, wl, weights, block, status=brisk.ERR_NUMERIC)
    assert np.isnan(g["refined"][1, 3]).all() and np.isfinite(g["refined"][:, :3]).all()
    assert list(g["cand_ids"][0, 0]) == list(range(wl.K))
    assert list(g["cand_ids"][1, 3, :3]) == [500, 501, 502]


def test_unaligned_rows_and_base(brisk):
    """Rows whose start is not 16-byte aligned take the scalar head/tail path."""
    wl = synth.Workload("unal", B=2, L=5, V=2053, d=32, K=8, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    for key in ("logits_q", "logits_p"):
        t = block[key]
        buf = torch.empty(t.numel() + 1, dtype=t.dtype, device=t.device)
        buf[1:] = t.reshape(-1)
        block[key] = buf[1:].view(t.shape)
    _run_and_check(brisk, wl, weights, block)


def test_overlap_schedule_matches_unfused(brisk):
    """At least 2432 rows (one proposal-sweep task per row) take the overlapping schedule: the
    verifier sweep from the start, the products in that schedule's tiles (2-stage, in the
    sweep's carveout for this state width). Bit for bit the same as the three separate calls
    (4-stage tiles, serial), and parity with the oracle."""
    wl = synth.Workload("overlap", B=80, L=32, V=4096, d=512, K=8, r=256)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    rep, g = _run_and_check(brisk, wl, weights, block, seqs=[0, 1, 40, 79], unfused=True)
    assert rep.sequences == 4


def test_separate_schedule_matches_unfused(brisk):
    """Chunked proposal rows with both logit tensors above 64 MB take the separate small-batch
    schedule (the verifier sweep beside the corrector, six launches): bit for bit the same as
    the three separate calls, and parity with the oracle."""
    wl = synth.Workload("separate", B=4, L=32, V=140000, d=64, K=8, r=16, agree0=0.9,
                        agree_decay=0.97, weight_std=0.2)
    dims = brisk.make_dims(wl.B, wl.L, wl.V, wl.d, wl.K, wl.r, wl.logits_dtype, wl.hidden_dtype)
    assert brisk.kernels_per_tail(dims) == 6
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    rep, g = _run_and_check(brisk, wl, weights, block, unfused=True)
    assert rep.sequences == wl.B


@pytest.mark.parametrize("modes", [("sample", "stochastic"), ("greedy", "stochastic"),
                                   ("greedy", "greedy")])
def test_fused_schedule_matches_unfused(brisk, modes):
    """Chunked proposal rows with both logit tensors within 64 MB take the fused small-batch
    schedule (one sweep of both tensors, the corrector verifying in the same CTA, four launches),
    in every mode pair: bit for bit the same as the three separate calls, and parity with the
    oracle."""
    sm_, vm_ = modes
    wl = synth.Workload("fused", B=3, L=8, V=65536, d=64, K=8, r=16, select_mode=sm_,
                        verify_mode=vm_, agree0=0.8, agree_decay=0.9, weight_std=0.2)
    dims = brisk.make_dims(wl.B, wl.L, wl.V, wl.d, wl.K, wl.r, wl.logits_dtype, wl.hidden_dtype)
    assert brisk.kernels_per_tail(dims) == 4
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    rep, g = _run_and_check(brisk, wl, weights, block, unfused=True)
    assert rep.sequences == wl.B


def test_non_finite_row_sets_numeric_status(brisk):
    wl = synth.Workload("nan", B=1, L=3, V=512, d=16, K=4, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    block["logits_q"][0, 1] = float("-inf")
    tail = brisk.DecodeTail.for_workload(wl, weights)
    tail.prepare()
    c = tail.topk(block["logits_q"])
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.ERR_NUMERIC
    assert tail.device_status() == brisk.OK   # cleared by the first read


@pytest.mark.parametrize("mode", ["greedy", "sample"])
def test_nan_scores_still_select_a_candidate(brisk, mode):
    """NaN candidate log-probabilities (caller data, or a row with no finite logit) give NaN
    refined scores: Select ranks them below every number, every selection is still one of the
    position's candidates and the device status reports the numeric problem."""
    wl = synth.Workload("nansel", B=3, L=6, V=1024, d=32, K=8, r=16)
    weights = _to(synth.make_weights(wl, "cpu"), "cuda")
    block = _to(synth.make_block(wl, "cpu"), "cuda")
    tail = brisk.DecodeTail.for_workload(wl, weights)
    tail.prepare()
    c = tail.topk(block["logits_q"])
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    lp = c["cand_logprob"].clone()
    lp[0, 2, :] = float("nan")          # a whole position
    lp[1, :, 0] = float("nan")          # rank 0 everywhere
    lp[2, 4, 3:] = float("nan")         # part of a position
    sm = brisk.SELECT_SAMPLE if mode == "sample" else brisk.SELECT_GREEDY
    s = tail.select(block["hidden"], block["h_c"], block["x0"], block["logits_q"], c["cand_ids"],
                    lp, sm, u_sel=block["u_sel"])
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.ERR_NUMERIC
    sel = s["sel_tokens"].cpu()
    ids = c["cand_ids"].cpu()
    assert bool((sel[..., None] == ids).any(-1).all())
    if mode == "greedy":
        # rows without NaN keep the argmax of the finite scores
        ref = s["refined"].cpu()
        for b, i in ((1, 0), (2, 4)):
            r = ref[b, i].clone()
            r[torch.isnan(r)] = float("-inf")
            assert int(sel[b, i]) == int(ids[b, i, int(torch.argmax(r))])
    v = tail.verify(block["logits_p"], s["sel_tokens"], c["cand_ids"], s["refined"], sm,
                    brisk.VERIFY_GREEDY)
    torch.cuda.synchronize()
    assert tail.device_status() == brisk.OK
    a = v["accepted_len"].cpu()
    assert bool(((a >= 0) & (a <= wl.L)).all())


def test_generator_same_on_cpu_and_gpu():
    wl = synth.Workload("gen", B=2, L=3, V=700, d=16, K=4, r=16, agree0=0.9, agree_decay=0.9)
    a = synth.make_block(wl, "cpu")
    b = synth.make_block(wl, "cuda")
    for k in a:
        if k in ("logits_q", "logits_p", "hidden", "h_c"):
            # transcendental functions may differ by an ulp between devices before rounding
            assert (a[k].float() - b[k].cpu().float()).abs().max() < 1e-2, k
        else:
            assert torch.equal(a[k], b[k].cpu()), k


FULL = ["tiny", "single", "batched_stochastic", "large_vocab", "decode_stream"]


@pytest.mark.parametrize("name", FULL)
def test_workload_parity_full_size(brisk, name):
    wl = synth.WORKLOADS[name]
    weights = synth.make_weights(wl, "cuda")
    block = synth.make_block(wl, "cuda")
    B = wl.B
    seqs = list(range(B)) if B <= 16 else [0, 1, B // 2, B - 1]
    rep, g = _run_and_check(brisk, wl, weights, block, seqs=seqs, unfused=(name == "single"))
    assert rep.sequences == len(seqs)
    assert rep.near_ties <= max(1, len(seqs) * wl.L // 50), rep.notes
    # step 1 of every row against the oracle (the rows of the sequences not checked above too)
    if B > 16:
        import oracle_pool
        BL = B * wl.L
        rows = block["logits_q"].float().reshape(BL, wl.V).cpu().numpy()
        ids, lp, lse = oracle_pool.topk_all_rows(rows, wl.K)
        np.testing.assert_array_equal(g["cand_ids"].reshape(BL, wl.K), ids)
        e = np.abs(g["cand_logprob"].reshape(BL, wl.K) - lp)
        assert np.where(np.isfinite(lp), e, 0.0).max() <= 1e-3
        assert np.abs(g["lse_q"].reshape(BL) - lse).max() <= 1e-3
    # every sequence's invariants, checked or not
    a = g["accepted_len"]
    assert np.all((a >= 0) & (a <= wl.L))
    for b in range(B):
        assert np.all(g["out_tokens"][b, :a[b]] == g["sel_tokens"][b, :a[b]])
        for i in range(wl.L):
            assert g["sel_tokens"][b, i] in g["cand_ids"][b, i]
