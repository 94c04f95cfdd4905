"""Seeded synthetic inputs for the BRISK-DLM per-block decode tail.

This module only draws random numbers and lays them out as the backbone's
outputs would be laid out: proposal logits, verifier logits, MASK hidden
states, the context hidden state, the anchor token, the frozen embedding
rows, the corrector parameters and the uniforms that the stochastic rules
consume. It computes nothing that the decode tail computes; the decode tail
runs in the CUDA library and, for testing, in the CPU oracle, and both read
the buffers built here.

Random numbers come from one counter-based generator, Philox4x32-10
(Salmon, Moraes, Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3",
SC'11), written with int64 torch ops so that CPU and GPU produce the same
words. Keys per sequence and block come from splitmix64 (Steele, Lea and
Flood, OOPSLA'14). Normals use Box-Muller, exponentials use -mu*log(1-u).

Workload recipes (the paper's workloads are GSM8K / MATH-500 / HumanEval
prompts on I-DLM-8B/32B; none of those datasets or checkpoints is used, these
recipes stand in for their shapes):

* ``planted``: proposal logits N(0, q_std) with one planted head token whose
  margin over the rest is Exp(head_margin). Verifier logits are the proposal
  plus N(0, p_noise). With an agreement law a_i, the verifier's argmax is then
  planted (margin Exp(verify_margin)) at the proposal's top-1 with probability
  a_i, else at a uniformly chosen proposal rank 1..K-1 with probability
  ``rescue_frac``, else at a uniformly random id.
* ``zipf``: per sequence a seeded permutation of the vocabulary; the id at
  rank rho gets -zipf_scale*ln(rho+1) + N(0, zipf_noise). Verifier as above.

The one ordering the generator uses (a stable descending sort, to find which
id holds proposal rank rho when planting the verifier's argmax) only decides
where to plant a value; no expected output is ever taken from this module.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace
from typing import Iterable, Optional, Sequence

import torch

MASK32 = 0xFFFFFFFF
MASK64 = 0xFFFFFFFFFFFFFFFF

# Philox4x32 round multipliers and Weyl key increments (Salmon et al., SC'11).
_PH_M0, _PH_M1 = 0xD2511F53, 0xCD9E8D57
_PH_W0, _PH_W1 = 0x9E3779B9, 0xBB67AE85

# Stream ids: every drawn quantity has its own counter space.
S_Q, S_HEAD, S_HMARG, S_P, S_AGREE, S_RESCUE, S_PICK, S_VMARG = 0, 1, 2, 3, 4, 5, 6, 7
S_HID, S_HC, S_X0, S_USEL, S_UACC, S_URES, S_PERM, S_RHO = 8, 9, 10, 11, 12, 13, 14, 15
S_W = 32  # weights use S_W + index
S_EIN, S_EOUT = 64, 65

_WEIGHT_KEY_SALT = 0x5745494748545321
_RHO_KEY_SALT = 0x52484F5F53455153


def splitmix64(x: int) -> int:
    """One splitmix64 output for state ``x`` (Steele, Lea and Flood, 2014)."""
    x = (x + 0x9E3779B97F4A7C15) & MASK64
    z = x
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def sequence_key(seed: int, seq: int, block: int = 0) -> int:
    """Key of sequence ``seq`` in block ``block``: splitmix64(seed ^ (seq<<32 | block))."""
    return splitmix64((seed ^ (((seq & MASK32) << 32) | (block & MASK32))) & MASK64)


def _mulhilo32(a: int, b: torch.Tensor):
    """High and low 32-bit words of a*b for a < 2^32 and an int64 tensor b < 2^32.

    Split into 16-bit halves so that no intermediate product leaves int64.
    """
    al, ah = a & 0xFFFF, a >> 16
    bl, bh = b & 0xFFFF, b >> 16
    ll = bl * al
    mid = bh * al + bl * ah + (ll >> 16)
    lo = ((mid & 0xFFFF) << 16) | (ll & 0xFFFF)
    hi = bh * ah + (mid >> 16)
    return hi, lo


def philox4x32_10(ctr, key):
    """Philox4x32 with 10 rounds. ``ctr`` is 4 int64 tensors, ``key`` 2 ints or tensors,
    all holding 32-bit values; returns 4 int64 tensors of 32-bit words."""
    c0, c1, c2, c3 = ctr
    k0, k1 = key
    for rnd in range(10):
        if rnd:
            k0 = (k0 + _PH_W0) & MASK32
            k1 = (k1 + _PH_W1) & MASK32
        hi0, lo0 = _mulhilo32(_PH_M0, c0)
        hi1, lo1 = _mulhilo32(_PH_M1, c2)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def _key_tensors(keys: Sequence[int], device) -> tuple:
    lo = torch.tensor([int(x) & MASK32 for x in keys], dtype=torch.int64, device=device)
    hi = torch.tensor([(int(x) >> 32) & MASK32 for x in keys], dtype=torch.int64, device=device)
    return lo.view(-1, 1), hi.view(-1, 1)


def philox_words(keys: Sequence[int], stream: int, start: int, count: int, device) -> torch.Tensor:
    """Words ``start .. start+count-1`` of ``stream`` for each key: int64 [len(keys), count].

    Word n sits in lane n % 4 of the Philox block with counter (n//4 low, n//4 high, stream, 0).
    """
    k0, k1 = _key_tensors(keys, device)
    first = start // 4
    last = (start + count + 3) // 4
    idx = torch.arange(first, last, device=device, dtype=torch.int64)
    c0 = (idx & MASK32).view(1, -1)
    c1 = (idx >> 32).view(1, -1)
    c2 = torch.full_like(c0, stream & MASK32)
    c3 = torch.zeros_like(c0)
    out = philox4x32_10((c0, c1, c2, c3), (k0, k1))
    out = [o.expand(len(keys), -1) for o in out]
    words = torch.stack(out, dim=-1).reshape(len(keys), -1)
    off = start - first * 4
    return words[:, off:off + count]


def _chunk_words(device) -> int:
    """Philox words generated per slab: bounded host memory, fewer launches on a GPU."""
    return (1 << 26) if torch.device(device).type == "cuda" else (1 << 22)


def _draw(keys, stream, count, device, fn, out_dtype=torch.float64, words_per_item=1):
    """Apply ``fn`` to consecutive word groups in bounded chunks; returns [len(keys), count]."""
    out = torch.empty((len(keys), count), dtype=out_dtype, device=device)
    per = max(1, _chunk_words(device) // max(1, len(keys)) // words_per_item)
    for s in range(0, count, per):
        n = min(per, count - s)
        w = philox_words(keys, stream, s * words_per_item, n * words_per_item, device)
        out[:, s:s + n] = fn(w.view(len(keys), n, words_per_item))
    return out


def _open01(w):
    return ((w >> 8).to(torch.float64) + 0.5) * (1.0 / 16777216.0)


def uniform_open(keys, stream, count, device) -> torch.Tensor:
    """float64 uniforms in (0, 1), 24-bit resolution: [len(keys), count]."""
    return _draw(keys, stream, count, device, lambda w: _open01(w[..., 0]))


def uniform_f32(keys, stream, count, device) -> torch.Tensor:
    """fp32 uniforms in [0, 1) with 24-bit resolution (exact in fp32): [len(keys), count]."""
    return _draw(keys, stream, count, device,
                 lambda w: (w[..., 0] >> 8).to(torch.float32) * (1.0 / 16777216.0),
                 out_dtype=torch.float32)


def normal(keys, stream, count, device) -> torch.Tensor:
    """float64 standard normals by Box-Muller from two open uniforms: [len(keys), count]."""
    def bm(w):
        u1 = _open01(w[..., 0])
        u2 = _open01(w[..., 1])
        return torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2)
    return _draw(keys, stream, count, device, bm, words_per_item=2)


def exponential(keys, stream, count, mean, device) -> torch.Tensor:
    """float64 Exp(mean) draws, -mean*log(1-u): [len(keys), count]."""
    return -mean * torch.log1p(-uniform_open(keys, stream, count, device))


def uniform_int(keys, stream, count, n, device) -> torch.Tensor:
    """int64 draws uniform on [0, n): floor(u*n): [len(keys), count]."""
    u = uniform_open(keys, stream, count, device)
    return torch.clamp((u * n).floor().to(torch.int64), 0, n - 1)


@dataclass(frozen=True)
class Workload:
    """Shapes and recipe of one synthetic decode-tail workload."""
    name: str
    B: int
    L: int
    V: int
    d: int
    K: int
    r: int
    logits_dtype: torch.dtype = torch.bfloat16
    hidden_dtype: torch.dtype = torch.bfloat16
    select_mode: str = "greedy"        # "greedy" | "sample"
    verify_mode: str = "greedy"        # "greedy" | "stochastic"
    recipe: str = "planted"            # "planted" | "zipf"
    q_std: float = 1.5
    head_margin: float = 3.0
    p_noise: float = 0.5
    agree0: Optional[float] = None     # a_i = agree0 * agree_decay**i
    agree_decay: float = 1.0
    agree_per_seq: Optional[tuple] = None  # (lo, hi): a_i = rho_s ~ U(lo, hi), constant in i
    rescue_frac: float = 0.9
    verify_margin: float = 3.0
    zipf_scale: float = 1.1
    zipf_noise: float = 0.3
    weight_std: float = 0.02
    emb_std: float = 1.0
    hidden_std: float = 1.0
    n_seqs: int = 0                    # decode stream: total sequences (0 = B)
    n_blocks: int = 1                  # decode stream: blocks per sequence
    seed: int = 0

    @property
    def S(self) -> int:
        return 2 * self.r

    @property
    def logit_bytes(self) -> int:
        return torch.empty((), dtype=self.logits_dtype).element_size()

    @property
    def hidden_bytes(self) -> int:
        return torch.empty((), dtype=self.hidden_dtype).element_size()

    def sweep_bytes(self) -> int:
        """Algorithmic bytes of the vocabulary sweep: both logit tensors read once."""
        return 2 * self.B * self.L * self.V * self.logit_bytes

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    "tiny": Workload("tiny", B=1, L=8, V=32000, d=512, K=4, r=64,
                     logits_dtype=torch.float32, hidden_dtype=torch.float32,
                     q_std=1.0, head_margin=2.0, p_noise=0.5),
    "single": Workload("single", B=1, L=32, V=126464, d=4096, K=8, r=256,
                       agree0=0.95, agree_decay=0.97),
    "batched_stochastic": Workload("batched_stochastic", B=16, L=32, V=126464, d=4096, K=8,
                                   r=256, select_mode="sample", verify_mode="stochastic",
                                   agree0=0.95, agree_decay=0.97),
    "large_vocab": Workload("large_vocab", B=64, L=64, V=151936, d=3584, K=16, r=512,
                            recipe="zipf", agree0=0.9, agree_decay=0.98),
    "decode_stream": Workload("decode_stream", B=128, L=32, V=126464, d=4096, K=8, r=256,
                              agree_per_seq=(0.6, 0.98), n_seqs=1024, n_blocks=32),
}


def weight_shapes(wl: Workload) -> dict:
    """Corrector parameter shapes (row-major) under the width mapping
    rank = hidden projection = token projection = r, state S = 2r, position and
    feature projections 16 (App. C.3, head configuration table)."""
    r, S, d = wl.r, wl.S, wl.d
    return {
        "P_h": (r, d), "P_e": (r, d), "P_phi": (16, 5), "pos": (wl.L, 16),
        "W0": (S, 2 * r), "Wz": (S, 2 * r + 32), "Wh": (S, 2 * r + 32),
        "W_s": (r, S), "W_c": (r, d), "w_g": (S + 5,),
    }


def make_corrector_weights(wl: Workload, device="cpu", seed: Optional[int] = None) -> dict:
    """The corrector parameters alone, N(0, weight_std), in ``wl.hidden_dtype``."""
    seed = wl.seed if seed is None else seed
    key = [splitmix64(seed ^ _WEIGHT_KEY_SALT)]
    out = {}
    for j, (name, shape) in enumerate(weight_shapes(wl).items()):
        n = math.prod(shape)
        w = normal(key, S_W + j, n, device).view(shape) * wl.weight_std
        out[name] = w.to(wl.hidden_dtype)
    return out


def make_weights(wl: Workload, device="cpu", seed: Optional[int] = None) -> dict:
    """Corrector parameters N(0, weight_std), frozen embedding rows E_in, E_out N(0, emb_std),
    gate bias b_g = 0 and gate scale alpha = 0. Tensors are in ``wl.hidden_dtype``."""
    seed = wl.seed if seed is None else seed
    key = [splitmix64(seed ^ _WEIGHT_KEY_SALT)]
    out = make_corrector_weights(wl, device, seed)
    for name, stream in (("E_in", S_EIN), ("E_out", S_EOUT)):
        e = torch.empty((wl.V, wl.d), dtype=wl.hidden_dtype, device=device)
        rows = max(1, _chunk_words(device) // (2 * wl.d))
        for v0 in range(0, wl.V, rows):
            nv = min(rows, wl.V - v0)
            z = _normal_range(key, stream, v0 * wl.d, nv * wl.d, device)
            e[v0:v0 + nv] = (z.view(nv, wl.d) * wl.emb_std).to(wl.hidden_dtype)
        out[name] = e
    out["b_g"] = 0.0
    out["alpha"] = 0.0
    return out


class EmbeddingRows:
    """Rows of E_in / E_out generated on demand, identical to ``make_weights``'s tensors
    (for consumers that need a few rows of a large vocabulary table)."""

    def __init__(self, wl: Workload, which: str, seed: Optional[int] = None):
        seed = wl.seed if seed is None else seed
        self.key = [splitmix64(seed ^ _WEIGHT_KEY_SALT)]
        self.stream = S_EIN if which == "E_in" else S_EOUT
        self.wl = wl
        self.cache = {}

    def row(self, v: int) -> torch.Tensor:
        v = int(v)
        if v not in self.cache:
            d = self.wl.d
            z = _normal_range(self.key, self.stream, v * d, d, "cpu") * self.wl.emb_std
            self.cache[v] = z.to(self.wl.hidden_dtype)
        return self.cache[v]

    def __getitem__(self, v):
        return self.row(v)


def _normal_range(keys, stream, start, count, device):
    """Normals number ``start .. start+count-1`` of ``stream`` (same numbering as ``normal``)."""
    w = philox_words(keys, stream, 2 * start, 2 * count, device).view(len(keys), count, 2)
    u1 = _open01(w[..., 0])
    u2 = _open01(w[..., 1])
    return (torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2))[0]


def agreement(wl: Workload, seqs: Sequence[int], device) -> torch.Tensor:
    """Per-(sequence, position) verifier agreement probabilities a_i: float64 [n, L]."""
    i = torch.arange(wl.L, dtype=torch.float64, device=device)
    if wl.agree_per_seq is not None:
        lo, hi = wl.agree_per_seq
        keys = [splitmix64((wl.seed ^ _RHO_KEY_SALT ^ (s << 20)) & MASK64) for s in seqs]
        rho = lo + (hi - lo) * uniform_open(keys, S_RHO, 1, device)
        return rho.expand(len(seqs), wl.L).clone()
    if wl.agree0 is None:
        return None
    return (wl.agree0 * wl.agree_decay ** i).expand(len(seqs), wl.L).clone()


def _plant(values: torch.Tensor, ids: torch.Tensor, margin: torch.Tensor) -> None:
    """Set values[..., ids] = (max over the other ids) + margin, in place (float64)."""
    others = values.scatter(-1, ids.unsqueeze(-1), float("-inf")).amax(-1)
    values.scatter_(-1, ids.unsqueeze(-1), (others + margin).unsqueeze(-1))


def _logits_for(wl: Workload, keys: list, agree: Optional[torch.Tensor], device):
    n, L, V, K = len(keys), wl.L, wl.V, wl.K
    if wl.recipe == "planted":
        q = normal(keys, S_Q, L * V, device).view(n, L, V) * wl.q_std
        head = uniform_int(keys, S_HEAD, L, V, device)
        _plant(q, head, exponential(keys, S_HMARG, L, wl.head_margin, device))
    elif wl.recipe == "zipf":
        perm = torch.argsort(uniform_open(keys, S_PERM, V, device), dim=-1)   # perm[b, rho] = id
        rho = torch.arange(V, dtype=torch.float64, device=device)
        by_rank = -wl.zipf_scale * torch.log1p(rho) + \
            normal(keys, S_Q, L * V, device).view(n, L, V) * wl.zipf_noise
        q = torch.empty_like(by_rank)
        q.scatter_(-1, perm.unsqueeze(1).expand(n, L, V), by_rank)
    else:
        raise ValueError(wl.recipe)
    lq = q.to(wl.logits_dtype)
    del q
    p = lq.to(torch.float64) + normal(keys, S_P, L * V, device).view(n, L, V) * wl.p_noise
    if agree is not None:
        order = torch.sort(lq.to(torch.float64), dim=-1, descending=True, stable=True).indices
        top = order[..., :K]
        del order
        ua = uniform_open(keys, S_AGREE, L, device)
        ur = uniform_open(keys, S_RESCUE, L, device)
        upick = uniform_open(keys, S_PICK, L, device)
        rank_pick = torch.clamp(1 + (upick * (K - 1)).floor().to(torch.int64), 1, max(1, K - 1))
        rand_id = torch.clamp((upick * V).floor().to(torch.int64), 0, V - 1)
        rescue = top.gather(-1, rank_pick.unsqueeze(-1)).squeeze(-1)
        target = torch.where(ua < agree, top[..., 0], torch.where(ur < wl.rescue_frac, rescue, rand_id))
        _plant(p, target, exponential(keys, S_VMARG, L, wl.verify_margin, device))
    lp = p.to(wl.logits_dtype)
    return lq, lp


def make_block(wl: Workload, device="cpu", seqs: Optional[Iterable[int]] = None, block: int = 0,
               seed: Optional[int] = None, chunk: int = 0) -> dict:
    """Backbone outputs for one block of ``len(seqs)`` sequences (default 0..B-1).

    Returns logits_q, logits_p [n, L, V] (logits dtype); hidden [n, L, d], h_c [n, d]
    (hidden dtype); x0 [n] int32; u_sel, u_acc, u_res [n, L] fp32 uniforms in [0, 1).
    """
    seed = wl.seed if seed is None else seed
    seqs = list(range(wl.B)) if seqs is None else list(seqs)
    wl_s = wl.with_(seed=seed)
    n = len(seqs)
    keys = [sequence_key(seed, s, block) for s in seqs]
    agree = agreement(wl_s, seqs, device)
    if chunk <= 0:
        chunk = max(1, (_chunk_words(device) // 4) // max(1, wl.L * wl.V))
    lq = torch.empty((n, wl.L, wl.V), dtype=wl.logits_dtype, device=device)
    lp = torch.empty_like(lq)
    for c in range(0, n, chunk):
        kk = keys[c:c + chunk]
        a = None if agree is None else agree[c:c + chunk]
        q, p = _logits_for(wl, kk, a, device)
        lq[c:c + len(kk)] = q
        lp[c:c + len(kk)] = p
    hidden = (normal(keys, S_HID, wl.L * wl.d, device) * wl.hidden_std).view(n, wl.L, wl.d)
    h_c = normal(keys, S_HC, wl.d, device) * wl.hidden_std
    x0 = uniform_int(keys, S_X0, 1, wl.V, device).view(n).to(torch.int32)
    return {
        "logits_q": lq, "logits_p": lp,
        "hidden": hidden.to(wl.hidden_dtype), "h_c": h_c.to(wl.hidden_dtype), "x0": x0,
        "u_sel": uniform_f32(keys, S_USEL, wl.L, device),
        "u_acc": uniform_f32(keys, S_UACC, wl.L, device),
        "u_res": uniform_f32(keys, S_URES, wl.L, device),
    }
