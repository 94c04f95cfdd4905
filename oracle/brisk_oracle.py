"""Plain CPU oracle of the BRISK-DLM per-block decode tail (float64, numpy).

TEST INFRASTRUCTURE ONLY. This module is the slow, literal statement of what
the decode tail computes; it exists to check the CUDA library against. Only
the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it. It shares no code with the CUDA path and imports
nothing from the package.

What it follows (section / equation of the paper, "From Position Risks to
Block Survival: Faster Generation for Diffusion Language Models"):

1. Candidates (Sec. 3.3, "C_i = TopK(q_i, K)" on the normalised proposal
   q_i; App. C.3, the ordered candidate set S_j that the head never expands):
   log-partition LSE = m + log sum exp(l - m); the K ids of largest logit,
   ordered by (logit descending, id ascending); cand_logprob = l - LSE.
2. Corrector (Sec. 3.3, Eq. 4 recurrent state and Eq. 5 candidate residual;
   App. C.3 head details and Eq. 9 residual logits; Algorithm 1(b)):
   u_0 = Init(h_c, E(x_0)); per position i the minimal GRU reads the
   concatenation [P_h m_i ; P_e E_in(x_{i-1}) ; pos_i ; P_phi phi_i],
   d_{i,k} = <W_s s_i, W_c E_out(c_{i,k})>,
   gamma_i = sigmoid(alpha) * sigmoid(w_g^T [s_i ; phi_i] + b_g),
   refined_{i,k} = log q_i(c_{i,k}) + gamma_i d_{i,k}, then Select.
3. Verification (Sec. 3.1, accept-prefix semantics; Sec. 3.3, standard
   speculative sampling with acceptance min{1, p/pi} and resampling from the
   normalised [p - pi]_+; App. B, Eq. 6, strict u < alpha): left to right up
   to the first rejection.

Readings taken where the paper is silent or ambiguous (each is listed in the
design notes): minimal GRU = input-only gates, z = sigmoid(W_z in),
h~ = W_h in, s = (1-z) s + z h~, no biases; Init = tanh(W_0 [P_h h_c ; P_e E_in(x_0)]);
h_c enters only Init; widths rank = hidden/token projection = r, state S = 2r,
position and feature projections 16; features phi_i come from the proposal row
i itself (top-1/top-2 gap, top-1/top-4 gap, [x_{i-1} = top-1],
[x_{i-1} in top-4], top-1 logit minus the logit of x_{i-1}), with x_{-1} = x_0;
the gate sees the raw 5 features; refined scores are on the log q basis;
greedy Select = argmax with the lowest rank on ties; sample Select walks the
candidate ranks; greedy verify accepts iff x_i is the verifier argmax (lowest
id) and the correction is that argmax; stochastic residual sampling walks ids
in ascending order and falls back to the verifier argmax when Z <= 1e-6 (a
rejection then has probability Z itself, and Z is below what an fp32 sum resolves);
a fully accepted block has no bonus token (correction -1).

Arrays: logits rows are float64 views of the exact bf16/fp32 inputs; ids are
int64. Nothing here is blocked, fused or reordered beyond the definitions.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, Dict, Optional, Sequence

import numpy as np

GREEDY = "greedy"
SAMPLE = "sample"
STOCHASTIC = "stochastic"
Z_FLOOR = 1e-6
NEG_INF = float("-inf")


class OracleError(ValueError):
    """Raised for rows the method leaves undefined (all -inf, NaN)."""


# ---------------------------------------------------------------------------
# Step 1: log-partition and Top-K (Sec. 3.3, App. C.3)
# ---------------------------------------------------------------------------

def log_partition(row: np.ndarray) -> float:
    """LSE of one logit row: m + log(sum(exp(l - m))), m = max l."""
    row = np.asarray(row, dtype=np.float64)
    if np.isnan(row).any():
        raise OracleError("NaN logit")
    m = row.max()
    if m == NEG_INF:
        raise OracleError("all logits are -inf")
    return float(m + np.log(np.sum(np.exp(row - m))))


def ranked_ids(row: np.ndarray) -> np.ndarray:
    """All ids ordered by (logit descending, id ascending): a full stable sort."""
    row = np.asarray(row, dtype=np.float64)
    return np.argsort(-row, kind="stable")


def topk_candidates(row: np.ndarray, K: int):
    """C_i = TopK(q_i, K): (ids[K], log q_i(ids)[K], LSE). Ordering of ranked_ids."""
    row = np.asarray(row, dtype=np.float64)
    lse = log_partition(row)
    ids = ranked_ids(row)[:K]
    return ids, row[ids] - lse, lse


def verifier_argmax(row: np.ndarray) -> int:
    """argmax_v p_i(v), lowest id on ties."""
    return int(ranked_ids(row)[0])


# ---------------------------------------------------------------------------
# Step 2: the prefix-conditioned corrector (Sec. 3.3 Eqs. 4-5, App. C.3 Eq. 9)
# ---------------------------------------------------------------------------

def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-np.asarray(x, dtype=np.float64)))


def confidence_features(row: np.ndarray, top4: Sequence[int], prev: int) -> np.ndarray:
    """phi_i (App. C.3): top1-top2 gap, top1-top4 gap, [prev = top1], [prev in top4],
    top1 minus the logit of the previous token, all on position i's own proposal row."""
    t1, t2, t4 = int(top4[0]), int(top4[1]), int(top4[3])
    return np.array([
        row[t1] - row[t2],
        row[t1] - row[t4],
        1.0 if prev == t1 else 0.0,
        1.0 if prev in [int(t) for t in top4] else 0.0,
        row[t1] - row[prev],
    ], dtype=np.float64)


@dataclass
class Params:
    """Corrector parameters psi and the frozen vocabulary rows, float64.

    P_h, P_e: [r, d]; P_phi: [16, 5]; pos: [L, 16]; W0: [S, 2r];
    Wz, Wh: [S, 2r + 32]; W_s: [r, S]; W_c: [r, d]; w_g: [S + 5]; b_g, alpha: scalars.
    E_in, E_out: anything indexable by an id that yields a [d] row.
    """
    P_h: np.ndarray
    P_e: np.ndarray
    P_phi: np.ndarray
    pos: np.ndarray
    W0: np.ndarray
    Wz: np.ndarray
    Wh: np.ndarray
    W_s: np.ndarray
    W_c: np.ndarray
    w_g: np.ndarray
    b_g: float
    alpha: float
    E_in: object
    E_out: object


def params_from_arrays(a: dict) -> Params:
    """Params from a dict of array-likes (converted to float64); E_in / E_out kept as given
    when they are not plain arrays (row providers for large vocabularies)."""
    f = {k: np.asarray(a[k], dtype=np.float64) for k in
         ("P_h", "P_e", "P_phi", "pos", "W0", "Wz", "Wh", "W_s", "W_c", "w_g")}
    emb = {k: (np.asarray(a[k], dtype=np.float64) if isinstance(a[k], np.ndarray) else a[k])
           for k in ("E_in", "E_out")}
    return Params(b_g=float(a["b_g"]), alpha=float(a["alpha"]), **f, **emb)


def init_state(p: Params, h_c: np.ndarray, x0: int) -> np.ndarray:
    """u_0 = Init(h_c, E(x_0)) = tanh(W_0 [P_h h_c ; P_e E_in(x_0)])."""
    return np.tanh(p.W0 @ np.concatenate([p.P_h @ h_c, p.P_e @ _row(p.E_in, x0)]))


def proposal_law(refined: np.ndarray, mode: str, sel_rank: int) -> np.ndarray:
    """pi_i over the K candidates induced by the selection rule (App. C.3): softmax of
    the refined scores for sampling; greedy selection puts all mass on the selected rank."""
    if mode == SAMPLE:
        m = np.max(refined)
        e = np.exp(refined - m)
        return e / e.sum()
    out = np.zeros_like(refined)
    out[sel_rank] = 1.0
    return out


def greedy_pick(refined: np.ndarray) -> int:
    """argmax_k refined_k, the lowest k (higher base rank) on ties."""
    return int(np.argmax(refined))


def sample_pick(refined: np.ndarray, u: float):
    """Inverse-CDF draw from softmax(refined) over ranks 0..K-1 with one uniform u:
    the first k whose cumulative mass exceeds u * total; the last k with mass if none.
    Returns (k, distance of u*total to the nearest cumulative boundary)."""
    m = np.max(refined)
    w = np.exp(refined - m)
    target = float(u) * w.sum()
    cum = np.cumsum(w)
    hit = np.nonzero(cum > target)[0]
    k = int(hit[0]) if hit.size else int(np.nonzero(w > 0)[0][-1])
    bounds = np.concatenate([[0.0], cum]) / w.sum()
    margin = float(np.min(np.abs(bounds - float(u))))
    return k, margin


@dataclass
class CorrectorTrace:
    sel_rank: np.ndarray          # [L]
    sel_tokens: np.ndarray        # [L]
    refined: np.ndarray           # [L, K]
    gamma: np.ndarray             # [L]
    features: np.ndarray          # [L, 5]
    margin: np.ndarray            # [L] decision margin of Select (score gap or CDF distance)


def corrector_sequence(p: Params, hidden: np.ndarray, h_c: np.ndarray, x0: int,
                       rows_q: Callable[[int], np.ndarray], cand_ids: np.ndarray,
                       cand_logprob: np.ndarray, top4: np.ndarray, mode: str = GREEDY,
                       u_sel: Optional[np.ndarray] = None,
                       force: Optional[Dict[int, int]] = None,
                       prefix_ranks: Optional[np.ndarray] = None) -> CorrectorTrace:
    """The corrector loop of Algorithm 1(b) over i = 1..M for one sequence (0-based i here).

    hidden: [L, d] MASK hidden states m_i; h_c: [d]; x0: anchor token;
    rows_q(i): proposal logit row i; cand_ids/cand_logprob: [L, K] from step 1;
    top4: [L, 4] the row's four highest ids (for phi); force: {i: rank} overrides
    Select at position i (used where two choices are equally correct);
    prefix_ranks: [L] candidate ranks of a fixed prefix; when given, the token before
    position i + 1 is cand_ids[i][prefix_ranks[i]] instead of the selection at i (the
    same-state replay of App. B conditions the head on the factual base prefix).
    """
    L, K = cand_ids.shape
    s = init_state(p, h_c, x0)                          # s_{-1} = u_0
    prev = int(x0)                                      # x_{-1} = x_0
    out = CorrectorTrace(np.zeros(L, np.int64), np.zeros(L, np.int64), np.zeros((L, K)),
                         np.zeros(L), np.zeros((L, 5)), np.zeros(L))
    for i in range(L):
        row = np.asarray(rows_q(i), dtype=np.float64)
        phi = confidence_features(row, top4[i], prev)
        inp = np.concatenate([p.P_h @ hidden[i], p.P_e @ _row(p.E_in, prev), p.pos[i],
                              p.P_phi @ phi])
        z = sigmoid(p.Wz @ inp)
        h_tilde = p.Wh @ inp
        s = (1.0 - z) * s + z * h_tilde
        ws = p.W_s @ s
        d = np.array([ws @ (p.W_c @ _row(p.E_out, int(c))) for c in cand_ids[i]])
        gamma = float(sigmoid(p.alpha) * sigmoid(p.w_g @ np.concatenate([s, phi]) + p.b_g))
        refined = cand_logprob[i] + gamma * d
        if mode == SAMPLE:
            k, margin = sample_pick(refined, float(u_sel[i]))
        else:
            k = greedy_pick(refined)
            others = np.delete(refined, k)
            margin = float(refined[k] - others.max()) if others.size else np.inf
        if force and i in force:
            k = int(force[i])
        out.sel_rank[i] = k
        out.sel_tokens[i] = int(cand_ids[i][k])
        out.refined[i] = refined
        out.gamma[i] = gamma
        out.features[i] = phi
        out.margin[i] = margin
        prev = int(cand_ids[i][k if prefix_ranks is None else int(prefix_ranks[i])])
    return out


# ---------------------------------------------------------------------------
# Same-state replay diagnostics (App. B, "Same-state replay", Eq. 6)
# ---------------------------------------------------------------------------

def base_ranks(cand_logprob: np.ndarray, mode: str = GREEDY,
               u_sel: Optional[np.ndarray] = None) -> np.ndarray:
    """The head-off (factual base) selection: the Select rule applied to the base scores
    log q (rank 0 under greedy; the inverse-CDF draw from the base law under sampling)."""
    L = cand_logprob.shape[0]
    if mode == SAMPLE:
        return np.array([sample_pick(cand_logprob[i], float(u_sel[i]))[0] for i in range(L)])
    return np.array([greedy_pick(cand_logprob[i]) for i in range(L)])


@dataclass
class ReplayResult:
    base_rank: np.ndarray       # [L]
    head_rank: np.ndarray       # [L] the head's selection on the factual base prefix
    alpha_base: np.ndarray      # [L] min(1, p/q) at the base token
    alpha_head: np.ndarray      # [L]
    first_breaker: int          # first position whose base token the draw rejects (L if none)
    intervention: np.ndarray    # [L] bool: head token != base token
    rescue: np.ndarray          # [L] bool: at the first breaker, the draw accepts the head token
    regression: np.ndarray      # [L] bool: before the first breaker, the draw rejects the head
    trace: CorrectorTrace


def replay_sequence(p: Params, rows_q, rows_p, hidden, h_c, x0, cand_ids, cand_logprob, top4,
                    u_acc, mode: str = GREEDY, u_sel=None) -> ReplayResult:
    """Same-state replay: with the factual base prefix, the base q_i (normalised over the full
    vocabulary), the verifier p_i and the draw u_i fixed, only the token at each position
    changes: alpha_i(x) = min(1, p_i(x) / q_i(x)), J_i(x) = [u_i < alpha_i(x)] (App. B, Eq. 6).
    A rescue is J(x_base) = 0 and J(x_head) = 1 at the factual first breaker; a regression is
    J(x_base) = 1 and J(x_head) = 0 at a factual accepted position (one before the breaker)."""
    L, K = cand_ids.shape
    b = base_ranks(cand_logprob, mode, u_sel)
    tr = corrector_sequence(p, hidden, h_c, int(x0), rows_q, cand_ids, cand_logprob, top4, mode,
                            u_sel, prefix_ranks=b)
    h = tr.sel_rank.copy()

    def alpha(i, k):
        row = np.asarray(rows_p(i), dtype=np.float64)
        lp = float(row[int(cand_ids[i][k])]) - log_partition(row)
        return min(1.0, float(np.exp(lp - cand_logprob[i][k])))

    ab = np.array([alpha(i, b[i]) for i in range(L)])
    ah = np.array([alpha(i, h[i]) for i in range(L)])
    jb = np.asarray(u_acc, dtype=np.float64) < ab
    jh = np.asarray(u_acc, dtype=np.float64) < ah
    fb = next((i for i in range(L) if not jb[i]), L)
    pos = np.arange(L)
    return ReplayResult(b, h, ab, ah, fb, h != b, (pos == fb) & jh, (pos < fb) & ~jh, tr)


# ---------------------------------------------------------------------------
# Step 3: verification through the first rejection (Sec. 3.1, 3.3; App. B Eq. 6)
# ---------------------------------------------------------------------------

@dataclass
class VerifyResult:
    accepted_len: int
    out_tokens: np.ndarray        # [L]: accepted prefix, correction, then -1
    correction: int               # -1 when the whole block is accepted
    accept_margin: float = np.inf  # min |u_acc - alpha| over decided positions
    resample_margin: float = np.inf
    accept_margins: Optional[np.ndarray] = None  # [L] |u_acc - alpha| per decided position


def residual_mass(row_p: np.ndarray, pi_ids: Sequence[int], pi_mass: Sequence[float]) -> np.ndarray:
    """The unnormalised residual R(v) = max(0, p(v) - pi(v)) over the whole vocabulary
    (Sec. 3.3, speculative sampling), with pi(v) = 0 outside the candidate ids."""
    lse = log_partition(row_p)
    p = np.exp(np.asarray(row_p, dtype=np.float64) - lse)
    R = p.copy()
    for v, m in zip(pi_ids, pi_mass):
        R[int(v)] = max(0.0, p[int(v)] - float(m))
    return R


def residual_sample(row_p: np.ndarray, pi_ids: Sequence[int], pi_mass: Sequence[float], u: float):
    """Draw from the normalised positive part [p - pi]_+ with one uniform u, walking ids
    in ascending order; Z <= Z_FLOOR falls back to argmax p. Returns (id, margin)."""
    R = residual_mass(row_p, pi_ids, pi_mass)
    Z = R.sum()
    if Z <= Z_FLOOR:
        return verifier_argmax(row_p), np.inf
    target = float(u) * Z
    cum = np.cumsum(R)
    hit = np.nonzero(cum > target)[0]
    v = int(hit[0]) if hit.size else int(np.nonzero(R > 0)[0][-1])
    lo = cum[v - 1] if v > 0 else 0.0
    margin = min(abs(target - lo), abs(cum[v] - target)) / Z
    return v, float(margin)


def verify_sequence(rows_p: Callable[[int], np.ndarray], sel_tokens: np.ndarray,
                    cand_ids: np.ndarray, refined: np.ndarray, select_mode: str = GREEDY,
                    verify_mode: str = GREEDY, u_acc: Optional[np.ndarray] = None,
                    u_res: Optional[np.ndarray] = None,
                    force_accept: Optional[Dict[int, bool]] = None,
                    force_correction: Optional[int] = None) -> VerifyResult:
    """Left-to-right verification of x_{1:M} against p_i with proposal law pi_i."""
    L = len(sel_tokens)
    out = np.full(L, -1, dtype=np.int64)
    acc_margin = np.inf
    margins = np.full(L, np.inf)
    for i in range(L):
        row = np.asarray(rows_p(i), dtype=np.float64)
        x = int(sel_tokens[i])
        if verify_mode == GREEDY:
            t = verifier_argmax(row)
            ok = (x == t)
        else:
            rank = int(np.nonzero(np.asarray(cand_ids[i]) == x)[0][0])
            pi = proposal_law(refined[i], select_mode, rank)
            p_x = np.exp(row[x] - log_partition(row))
            alpha = min(1.0, p_x / pi[rank])
            ok = float(u_acc[i]) < alpha
            margins[i] = abs(float(u_acc[i]) - alpha)
            acc_margin = min(acc_margin, margins[i])
        if force_accept and i in force_accept:
            ok = bool(force_accept[i])
        if ok:
            out[i] = x
            continue
        res_margin = np.inf
        if verify_mode == GREEDY:
            corr = verifier_argmax(row)
        else:
            corr, res_margin = residual_sample(row, cand_ids[i], pi, float(u_res[i]))
        if force_correction is not None:
            corr = int(force_correction)
        out[i] = corr
        return VerifyResult(i, out, int(corr), acc_margin, res_margin, margins)
    return VerifyResult(L, out, -1, acc_margin, np.inf, margins)


def next_anchor(vr: VerifyResult, sel_tokens: Sequence[int]) -> int:
    """The anchor of the next block (Algorithm 1(b), commit step): the last token this block
    commits, which is the correction at the first rejection, or the last selected token when
    the whole block is accepted (no bonus token is drawn, see the verification readings)."""
    L = len(sel_tokens)
    return int(vr.correction) if vr.accepted_len < L else int(sel_tokens[L - 1])


# ---------------------------------------------------------------------------
# The whole tail for one block
# ---------------------------------------------------------------------------

def _row(table, v: int) -> np.ndarray:
    return np.asarray(table[int(v)], dtype=np.float64)


@dataclass
class TailResult:
    cand_ids: np.ndarray          # [B, L, K]
    cand_logprob: np.ndarray      # [B, L, K]
    lse_q: np.ndarray             # [B, L]
    argmax_p: np.ndarray          # [B, L]
    lse_p: np.ndarray             # [B, L]
    sel_tokens: np.ndarray        # [B, L]
    refined: np.ndarray           # [B, L, K]
    accepted_len: np.ndarray      # [B]
    out_tokens: np.ndarray        # [B, L]
    correction: np.ndarray        # [B]
    traces: list = field(default_factory=list)
    verifies: list = field(default_factory=list)


def decode_tail_sequence(p: Params, rows_q, rows_p, hidden, h_c, x0, K, select_mode=GREEDY,
                         verify_mode=GREEDY, u_sel=None, u_acc=None, u_res=None,
                         force_sel=None, force_accept=None, force_correction=None):
    """Steps 1-3 for one sequence; rows_q(i) / rows_p(i) return logit rows."""
    L = hidden.shape[0]
    cand = np.zeros((L, K), np.int64)
    lp = np.zeros((L, K))
    lse = np.zeros(L)
    top4 = np.zeros((L, 4), np.int64)
    for i in range(L):
        row = np.asarray(rows_q(i), dtype=np.float64)
        cand[i], lp[i], lse[i] = topk_candidates(row, K)
        top4[i] = ranked_ids(row)[:4]
    tr = corrector_sequence(p, hidden, h_c, int(x0), rows_q, cand, lp, top4, select_mode,
                            u_sel, force_sel)
    vr = verify_sequence(rows_p, tr.sel_tokens, cand, tr.refined, select_mode, verify_mode,
                         u_acc, u_res, force_accept, force_correction)
    return cand, lp, lse, tr, vr


def decode_tail(p: Params, logits_q, logits_p, hidden, h_c, x0, K, select_mode=GREEDY,
                verify_mode=GREEDY, u_sel=None, u_acc=None, u_res=None) -> TailResult:
    """The decode tail for a whole block: logits [B, L, V], hidden [B, L, d], h_c [B, d], x0 [B]."""
    logits_q = np.asarray(logits_q, dtype=np.float64)
    logits_p = np.asarray(logits_p, dtype=np.float64)
    hidden = np.asarray(hidden, dtype=np.float64)
    h_c = np.asarray(h_c, dtype=np.float64)
    B, L, V = logits_q.shape
    res = TailResult(np.zeros((B, L, K), np.int64), np.zeros((B, L, K)), np.zeros((B, L)),
                     np.zeros((B, L), np.int64), np.zeros((B, L)), np.zeros((B, L), np.int64),
                     np.zeros((B, L, K)), np.zeros(B, np.int64), np.zeros((B, L), np.int64),
                     np.zeros(B, np.int64))
    for b in range(B):
        cand, lp, lse, tr, vr = decode_tail_sequence(
            p, lambda i: logits_q[b, i], lambda i: logits_p[b, i], hidden[b], h_c[b], x0[b], K,
            select_mode, verify_mode,
            None if u_sel is None else u_sel[b], None if u_acc is None else u_acc[b],
            None if u_res is None else u_res[b])
        res.cand_ids[b], res.cand_logprob[b], res.lse_q[b] = cand, lp, lse
        for i in range(L):
            res.argmax_p[b, i] = verifier_argmax(logits_p[b, i])
            res.lse_p[b, i] = log_partition(logits_p[b, i])
        res.sel_tokens[b] = tr.sel_tokens
        res.refined[b] = tr.refined
        res.accepted_len[b] = vr.accepted_len
        res.out_tokens[b] = vr.out_tokens
        res.correction[b] = vr.correction
        res.traces.append(tr)
        res.verifies.append(vr)
    return res
