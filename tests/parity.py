"""Parity harness: the CUDA decode tail against the CPU oracle on the same inputs.

Ids, selected tokens, accepted lengths, output tokens and corrections must be
identical; log-probabilities, log-partitions and refined scores must agree to
ATOL. Where the oracle's own decision is a near-tie (two refined scores, a
uniform and an acceptance probability, or a uniform and an inverse-CDF
boundary closer than TIE_TOL), both outcomes are correct: the GPU's choice is
accepted, the oracle is re-run from that choice for the rest of the block,
and the event is counted.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from oracle import brisk_oracle as O

ATOL = 1e-3          # fp32 log-probs and corrector scores (absolute)
TIE_TOL = 1e-4       # decision margins below this count as near-ties


class LazyRows:
    """Row provider over a (possibly CUDA) [V, d] tensor: rows come back as float64 numpy."""

    def __init__(self, t: torch.Tensor):
        self.t = t
        self.cache = {}

    def __getitem__(self, v):
        v = int(v)
        if v not in self.cache:
            self.cache[v] = self.t[v].to(torch.float64).cpu().numpy()
        return self.cache[v]


def oracle_params(weights: dict) -> O.Params:
    arr = {}
    for k in ("P_h", "P_e", "P_phi", "pos", "W0", "Wz", "Wh", "W_s", "W_c", "w_g"):
        arr[k] = weights[k].to(torch.float64).cpu().numpy()
    arr["E_in"] = LazyRows(weights["E_in"])
    arr["E_out"] = LazyRows(weights["E_out"])
    arr["b_g"] = weights["b_g"]
    arr["alpha"] = weights["alpha"]
    return O.params_from_arrays(arr)


def np64(t: torch.Tensor) -> np.ndarray:
    return t.to(torch.float64).cpu().numpy()


@dataclass
class Report:
    sequences: int = 0
    near_ties: int = 0
    max_lp_err: float = 0.0
    max_lse_err: float = 0.0
    max_ref_err: float = 0.0
    notes: list = field(default_factory=list)


def residual_neighbours(row_p: np.ndarray, pi_ids, pi_mass, v: int):
    """The ids on either side of v with positive residual [p - pi]_+ (the only other outcomes
    an inverse-CDF draw that lands near one of v's boundaries can give); None where none."""
    R = O.residual_mass(row_p, pi_ids, pi_mass)
    pos = np.nonzero(R > 0)[0]
    below = pos[pos < v]
    above = pos[pos > v]
    return (int(below[-1]) if below.size else None, int(above[0]) if above.size else None)


def check_sequence(b: int, block: dict, params: O.Params, K: int, gpu: dict, select_mode: str,
                   verify_mode: str, rep: Report, x0=None):
    """Compare sequence b of the GPU outputs `gpu` (numpy) with the oracle; x0 overrides the
    block's anchor (a chained block starts from the previous block's last committed token).
    Returns the oracle's (corrector trace, verify result) of the accepted run."""
    lq = np64(block["logits_q"][b])
    lpv = np64(block["logits_p"][b])
    hidden = np64(block["hidden"][b])
    h_c = np64(block["h_c"][b])
    x0 = int(block["x0"][b]) if x0 is None else int(x0)
    L = lq.shape[0]
    u_sel = block["u_sel"][b].cpu().numpy().astype(np.float64)
    u_acc = block["u_acc"][b].cpu().numpy().astype(np.float64)
    u_res = block["u_res"][b].cpu().numpy().astype(np.float64)
    force_sel, force_acc, force_corr = {}, {}, None
    for _attempt in range(2 * L + 2):
        cand, lp, lse, tr, vr = O.decode_tail_sequence(
            params, lambda i: lq[i], lambda i: lpv[i], hidden, h_c, x0, K, select_mode, verify_mode,
            u_sel, u_acc, u_res, force_sel, force_acc, force_corr)
        # step 1: candidates (no near-ties possible: exact comparisons of exact values)
        np.testing.assert_array_equal(gpu["cand_ids"][b], cand, err_msg=f"cand_ids seq {b}")
        fin = np.isfinite(lp)   # a candidate of zero mass (K > support) is -inf on both sides
        np.testing.assert_array_equal(gpu["cand_logprob"][b][~fin], lp[~fin],
                                      err_msg=f"cand_logprob seq {b}")
        e = np.where(fin, np.abs(gpu["cand_logprob"][b] - np.where(fin, lp, 0.0)), 0.0)
        rep.max_lp_err = max(rep.max_lp_err, float(e.max()))
        assert e.max() <= ATOL, f"cand_logprob seq {b}: {e.max()}"
        el = float(np.abs(gpu["lse_q"][b] - lse).max())
        rep.max_lse_err = max(rep.max_lse_err, el)
        assert el <= ATOL, f"lse_q seq {b}: {el}"
        # step 2: selections, walking positions in order
        g_sel = gpu["sel_tokens"][b]
        mism = np.nonzero(g_sel != tr.sel_tokens)[0]
        if mism.size:
            i = int(mism[0])
            if tr.margin[i] < TIE_TOL and g_sel[i] in cand[i]:
                force_sel[i] = int(np.nonzero(cand[i] == g_sel[i])[0][0])
                rep.near_ties += 1
                rep.notes.append(f"seq {b} pos {i}: select near-tie ({tr.margin[i]:.2e})")
                continue
            raise AssertionError(f"sel_tokens seq {b} pos {i}: gpu {g_sel[i]} oracle "
                                 f"{tr.sel_tokens[i]} margin {tr.margin[i]:.3e}\n"
                                 f"gpu refined {gpu['refined'][b][i]}\noracle {tr.refined[i]}")
        er = np.abs(gpu["refined"][b] - tr.refined)
        er = np.where(np.isfinite(tr.refined), er, 0.0)
        rep.max_ref_err = max(rep.max_ref_err, float(er.max()))
        assert er.max() <= ATOL, f"refined seq {b}: {er.max()}"
        # step 3: verification
        ga = int(gpu["accepted_len"][b])
        if ga != vr.accepted_len and verify_mode == O.STOCHASTIC:
            j = min(ga, vr.accepted_len)
            if vr.accept_margins[j] < TIE_TOL and j not in force_acc:
                force_acc[j] = ga > j
                rep.near_ties += 1
                rep.notes.append(f"seq {b} pos {j}: accept near-tie")
                continue
        assert ga == vr.accepted_len, f"accepted_len seq {b}: gpu {ga} oracle {vr.accepted_len}"
        gc = int(gpu["correction"][b])
        if gc != vr.correction and verify_mode == O.STOCHASTIC and force_corr is None \
                and vr.resample_margin < TIE_TOL:
            # only the neighbouring id with residual mass across the boundary is also correct
            j = vr.accepted_len
            rank = int(np.nonzero(cand[j] == tr.sel_tokens[j])[0][0])
            pi = O.proposal_law(tr.refined[j], select_mode, rank)
            assert gc in residual_neighbours(lpv[j], cand[j], pi, vr.correction), \
                f"correction seq {b}: gpu {gc} is not a neighbour of the oracle's {vr.correction}"
            force_corr = gc
            rep.near_ties += 1
            rep.notes.append(f"seq {b}: residual near-tie")
            continue
        assert gc == vr.correction, f"correction seq {b}: gpu {gc} oracle {vr.correction}"
        np.testing.assert_array_equal(gpu["out_tokens"][b], vr.out_tokens,
                                      err_msg=f"out_tokens seq {b}")
        if "next_anchor" in gpu:
            na = O.next_anchor(vr, tr.sel_tokens)
            assert int(gpu["next_anchor"][b]) == na, \
                f"next_anchor seq {b}: gpu {int(gpu['next_anchor'][b])} oracle {na}"
        rep.sequences += 1
        return tr, vr
    raise AssertionError(f"seq {b}: too many near-tie re-runs")


def to_numpy(out: dict) -> dict:
    return {k: v.cpu().numpy() for k, v in out.items()}
