"""ctypes binding of ``libbrisk.so`` (the C ABI in ``include/brisk.h``).

Argument marshalling only: every step of the decode tail runs in the CUDA
library. Tensors are torch CUDA tensors; their data pointers and the current
torch stream are handed to the library. Loading fails loudly when the library
has not been built; nothing here falls back to another implementation.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Dict, Optional

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libbrisk.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_TIMEOUT, ERR_NUMERIC = range(6)
DT_F32, DT_BF16 = 0, 1
SELECT_GREEDY, SELECT_SAMPLE = 0, 1
VERIFY_GREEDY, VERIFY_STOCHASTIC = 0, 1

_vp = ctypes.c_void_p


class Dims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("B", "L", "V", "d", "K", "r", "logits_dtype", "hidden_dtype")]


class Params(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("E_in", "E_out", "P_h", "P_e", "P_phi", "pos", "W0", "Wz", "Wh",
                                   "W_s", "W_c", "w_g")] + [("b_g", ctypes.c_float),
                                                           ("alpha", ctypes.c_float)]


class TailIO(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("logits_q", "logits_p", "hidden", "h_ctx", "x0", "u_sel", "u_acc",
                                   "u_res", "cand_ids", "cand_logprob", "lse_q", "sel_tokens",
                                   "refined", "accepted_len", "out_tokens", "correction",
                                   "next_anchor")]


class Events(ctypes.Structure):
    _fields_ = [("sweep_q_begin", _vp), ("sweep_q_end", _vp), ("sweep_p_begin", _vp),
                ("sweep_p_end", _vp)]


class BriskError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)}")


_lib = None

# (name, restype, argtypes) of every exported entry point
_SIGS = [
    ("brisk_workspace_bytes", ctypes.c_size_t, [ctypes.POINTER(Dims)]),
    ("brisk_tables_bytes", ctypes.c_size_t, [ctypes.POINTER(Dims)]),
    ("brisk_corrector_prepare", ctypes.c_int, [ctypes.POINTER(Dims), ctypes.POINTER(Params), _vp, _vp]),
    ("brisk_topk_candidates", ctypes.c_int, [ctypes.POINTER(Dims), _vp, _vp, _vp, _vp, _vp, _vp]),
    ("brisk_corrector_select", ctypes.c_int,
     [ctypes.POINTER(Dims), ctypes.POINTER(Params), _vp, _vp, _vp, _vp, _vp, _vp, _vp,
      ctypes.c_int32, _vp, _vp, _vp, _vp, _vp]),
    ("brisk_verify_block", ctypes.c_int,
     [ctypes.POINTER(Dims), _vp, _vp, _vp, _vp, ctypes.c_int32, ctypes.c_int32, _vp, _vp, _vp, _vp,
      _vp, _vp, _vp]),
    ("brisk_decode_tail", ctypes.c_int,
     [ctypes.POINTER(Dims), ctypes.POINTER(Params), _vp, ctypes.POINTER(TailIO), ctypes.c_int32,
      ctypes.c_int32, _vp, ctypes.POINTER(Events), _vp]),
    ("brisk_topk_candidates_noalloc", ctypes.c_int,
     [ctypes.POINTER(Dims), _vp, _vp, _vp, _vp, _vp]),
    ("brisk_kernels_per_tail", ctypes.c_int32, [ctypes.POINTER(Dims)]),
    ("brisk_last_device_status", ctypes.c_int, [_vp, ctypes.c_int32, _vp]),
    ("brisk_status_string", ctypes.c_char_p, [ctypes.c_int]),
    ("brisk_set_wait_limit", ctypes.c_int64, [ctypes.c_int64]),
    ("brisk_acceptance_counts", ctypes.c_int, [_vp, ctypes.c_int32, ctypes.c_int32, _vp, _vp]),
    ("brisk_acceptance_weights", ctypes.c_int,
     [ctypes.c_int32, _vp, _vp, _vp, ctypes.c_double, _vp, _vp, _vp]),
    ("brisk_tpf_isd", ctypes.c_double, [ctypes.c_int32, ctypes.c_double]),
    ("brisk_isd_costs", ctypes.c_int, [ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]),
    ("brisk_tail_graph_create", ctypes.c_int,
     [ctypes.POINTER(Dims), ctypes.POINTER(Params), _vp, ctypes.POINTER(TailIO), ctypes.c_int32,
      ctypes.c_int32, _vp, _vp, ctypes.POINTER(_vp)]),
    ("brisk_tail_graph_launch", ctypes.c_int, [_vp, _vp]),
    ("brisk_tail_graph_destroy", None, [_vp]),
    ("brisk_replay_diagnostics", ctypes.c_int,
     [ctypes.POINTER(Dims), ctypes.POINTER(Params), _vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_int32,
      _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    ("brisk_distill_loss", ctypes.c_int,
     [ctypes.POINTER(Dims), _vp, _vp, _vp, _vp, _vp, ctypes.c_float, _vp, _vp, _vp, _vp]),
]


def lib():
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        h = ctypes.CDLL(LIB_PATH)
        for name, res, args in _SIGS:
            f = getattr(h, name)
            f.restype = res
            f.argtypes = args
        _lib = h
    return _lib


def set_wait_limit(cycles: int) -> int:
    """Limit (SM cycles) of the library's bounded device-side waits; <= 0 restores the default.
    Returns the previous limit."""
    return int(lib().brisk_set_wait_limit(int(cycles)))


def status_string(s: int) -> str:
    return lib().brisk_status_string(int(s)).decode()


def _check(s: int, where: str) -> None:
    if s != OK:
        raise BriskError(s, where)


def _dt(t: torch.dtype) -> int:
    if t == torch.bfloat16:
        return DT_BF16
    if t == torch.float32:
        return DT_F32
    raise ValueError(f"unsupported dtype {t}")


def _p(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return _vp(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return _vp(s.cuda_stream)


def make_dims(B, L, V, d, K, r, logits_dtype, hidden_dtype) -> Dims:
    return Dims(B, L, V, d, K, r, _dt(logits_dtype), _dt(hidden_dtype))


def workspace_bytes(dims: Dims) -> int:
    return int(lib().brisk_workspace_bytes(ctypes.byref(dims)))


def tables_bytes(dims: Dims) -> int:
    return int(lib().brisk_tables_bytes(ctypes.byref(dims)))


def kernels_per_tail(dims: Dims) -> int:
    return int(lib().brisk_kernels_per_tail(ctypes.byref(dims)))


def topk_candidates_noalloc(dims: Dims, logits_q, cand_ids, cand_logprob, lse_q, stream=None) -> int:
    """Step 1 without a workspace, for callers that cannot allocate device memory; the
    library's own fixed scratch array is used instead. Returns the status code."""
    return int(lib().brisk_topk_candidates_noalloc(ctypes.byref(dims), _p(logits_q), _p(cand_ids),
                                                   _p(cand_logprob), _p(lse_q), _stream(stream)))


def make_params(w: Dict[str, object]) -> Params:
    names = ("E_in", "E_out", "P_h", "P_e", "P_phi", "pos", "W0", "Wz", "Wh", "W_s", "W_c", "w_g")
    return Params(*[_p(w[n]) for n in names], float(w["b_g"]), float(w["alpha"]))


class DecodeTail:
    """Device buffers and calls of the decode tail for one problem size and weight set.

    ``weights`` holds the corrector parameters and E_in / E_out as CUDA tensors in the hidden
    dtype (see ``synth.make_weights``). The workspace and the folded tables are allocated once
    here with torch; the library itself never allocates.
    """

    def __init__(self, B, L, V, d, K, r, logits_dtype, hidden_dtype, weights, device="cuda"):
        self.dims = make_dims(B, L, V, d, K, r, logits_dtype, hidden_dtype)
        self.B, self.L, self.V, self.d, self.K, self.r = B, L, V, d, K, r
        self.device = torch.device(device)
        ws = workspace_bytes(self.dims)
        tb = tables_bytes(self.dims)
        if ws == 0 or tb == 0:
            raise BriskError(ERR_INVALID_ARG, "dims")
        self.workspace = torch.zeros(ws, dtype=torch.uint8, device=self.device)
        self.tables = torch.empty(tb, dtype=torch.uint8, device=self.device)
        self.weights = weights
        self.params = make_params(weights)
        self.prepared = False

    @classmethod
    def for_workload(cls, wl, weights, device="cuda", B=None):
        return cls(wl.B if B is None else B, wl.L, wl.V, wl.d, wl.K, wl.r, wl.logits_dtype,
                   wl.hidden_dtype, weights, device)

    def prepare(self, stream=None):
        _check(lib().brisk_corrector_prepare(ctypes.byref(self.dims), ctypes.byref(self.params),
                                             _p(self.tables), _stream(stream)), "prepare")
        self.prepared = True

    def _i32(self, *shape):
        return torch.empty(shape, dtype=torch.int32, device=self.device)

    def _f32(self, *shape):
        return torch.empty(shape, dtype=torch.float32, device=self.device)

    def topk(self, logits_q, stream=None):
        B, L, K = self.B, self.L, self.K
        ids, lp, lse = self._i32(B, L, K), self._f32(B, L, K), self._f32(B, L)
        _check(lib().brisk_topk_candidates(ctypes.byref(self.dims), _p(logits_q), _p(ids), _p(lp),
                                           _p(lse), _p(self.workspace), _stream(stream)), "topk")
        return {"cand_ids": ids, "cand_logprob": lp, "lse_q": lse}

    def select(self, hidden, h_ctx, x0, logits_q, cand_ids, cand_logprob, select_mode=SELECT_GREEDY,
               u_sel=None, stream=None):
        B, L, K = self.B, self.L, self.K
        sel, ref = self._i32(B, L), self._f32(B, L, K)
        _check(lib().brisk_corrector_select(
            ctypes.byref(self.dims), ctypes.byref(self.params), _p(self.tables), _p(hidden), _p(h_ctx),
            _p(x0), _p(logits_q), _p(cand_ids), _p(cand_logprob), int(select_mode), _p(u_sel),
            _p(sel), _p(ref), _p(self.workspace), _stream(stream)), "select")
        return {"sel_tokens": sel, "refined": ref}

    def verify(self, logits_p, sel_tokens, cand_ids, refined, select_mode=SELECT_GREEDY,
               verify_mode=VERIFY_GREEDY, u_acc=None, u_res=None, stream=None):
        B, L = self.B, self.L
        a, out, corr = self._i32(B), self._i32(B, L), self._i32(B)
        _check(lib().brisk_verify_block(
            ctypes.byref(self.dims), _p(logits_p), _p(sel_tokens), _p(cand_ids), _p(refined),
            int(select_mode), int(verify_mode), _p(u_acc), _p(u_res), _p(a), _p(out), _p(corr),
            _p(self.workspace), _stream(stream)), "verify")
        return {"accepted_len": a, "out_tokens": out, "correction": corr}

    def replay(self, block, select_mode=SELECT_GREEDY, stream=None):
        """Same-state replay diagnostics (App. B, Eq. 6) of one block (see synth.make_block)."""
        B, L, K = self.B, self.L, self.K
        head, flags, fb, ref = self._i32(B, L), self._i32(B, L), self._i32(B), self._f32(B, L, K)
        _check(lib().brisk_replay_diagnostics(
            ctypes.byref(self.dims), ctypes.byref(self.params), _p(self.tables),
            _p(block["hidden"]), _p(block["h_c"]), _p(block["x0"]), _p(block["logits_q"]),
            _p(block["logits_p"]), int(select_mode), _p(block["u_sel"]), _p(block["u_acc"]),
            _p(head), _p(flags), _p(fb), _p(ref), _p(self.workspace), _stream(stream)),
            "replay_diagnostics")
        return {"head_tokens": head, "flags": flags, "first_breaker": fb, "refined": ref}

    def distill_loss(self, logits_p, cand_ids, cand_logprob, refined, accepted_len, beta=0.01,
                     with_grad=True, stream=None):
        """Distillation loss of the refinement head (App. C.3, Eq. 10) and its gradient in the
        refined scores."""
        loss = self._f32(1)
        grad = self._f32(self.B, self.L, self.K) if with_grad else None
        _check(lib().brisk_distill_loss(
            ctypes.byref(self.dims), _p(logits_p), _p(cand_ids), _p(cand_logprob), _p(refined),
            _p(accepted_len), float(beta), _p(loss), _p(grad), _p(self.workspace),
            _stream(stream)), "distill_loss")
        return {"loss": loss, "grad": grad}

    def alloc_outputs(self, full=True):
        B, L, K = self.B, self.L, self.K
        o = {"accepted_len": self._i32(B), "out_tokens": self._i32(B, L), "correction": self._i32(B),
             "next_anchor": self._i32(B)}
        if full:
            o.update(cand_ids=self._i32(B, L, K), cand_logprob=self._f32(B, L, K),
                     lse_q=self._f32(B, L), sel_tokens=self._i32(B, L), refined=self._f32(B, L, K))
        return o

    @staticmethod
    def _io(block, out, x0):
        return TailIO(_p(block["logits_q"]), _p(block["logits_p"]), _p(block["hidden"]),
                      _p(block["h_c"]), _p(block["x0"] if x0 is None else x0), _p(block.get("u_sel")),
                      _p(block.get("u_acc")), _p(block.get("u_res")), _p(out.get("cand_ids")),
                      _p(out.get("cand_logprob")), _p(out.get("lse_q")), _p(out.get("sel_tokens")),
                      _p(out.get("refined")), _p(out["accepted_len"]), _p(out["out_tokens"]),
                      _p(out["correction"]), _p(out.get("next_anchor")))

    def tail(self, block, select_mode=SELECT_GREEDY, verify_mode=VERIFY_GREEDY, out=None, x0=None,
             events=None, stream=None):
        """One fused decode-tail call on the tensors of ``block`` (see ``synth.make_block``)."""
        if out is None:
            out = self.alloc_outputs()
        io = self._io(block, out, x0)
        ev = None
        if events is not None:
            ev = ctypes.byref(Events(*[_vp(e.cuda_event) for e in events]))
        _check(lib().brisk_decode_tail(ctypes.byref(self.dims), ctypes.byref(self.params),
                                       _p(self.tables), ctypes.byref(io), int(select_mode),
                                       int(verify_mode), _p(self.workspace), ev, _stream(stream)),
               "decode_tail")
        return out

    def graph(self, block, select_mode=SELECT_GREEDY, verify_mode=VERIFY_GREEDY, out=None,
              chain_anchor=True, stream=None):
        """The decode tail on these buffers captured into a replayable CUDA graph (App. F). With
        chain_anchor the anchor buffer is also the next-anchor output, so replays chain blocks."""
        return TailGraph(self, block, select_mode, verify_mode, out, chain_anchor, stream)

    def device_status(self, clear=True, stream=None) -> int:
        return int(lib().brisk_last_device_status(_p(self.workspace), int(clear), _stream(stream)))


class TailGraph:
    """A captured decode tail (see brisk_tail_graph_create); launch() replays it."""

    def __init__(self, tail, block, select_mode, verify_mode, out, chain_anchor, stream):
        if stream is None:
            raise ValueError("capture needs a non-default stream")
        self.tail = tail
        self.block = block
        self.out = tail.alloc_outputs() if out is None else out
        if chain_anchor:
            self.anchor = block["x0"].clone()
            self.out["next_anchor"] = self.anchor
        else:
            self.anchor = block["x0"]
        self.stream = stream
        self._iob = tail._io(block, self.out, self.anchor)
        saved = self.anchor.clone()
        torch.cuda.synchronize()
        h = _vp()
        _check(lib().brisk_tail_graph_create(ctypes.byref(tail.dims), ctypes.byref(tail.params),
                                             _p(tail.tables), ctypes.byref(self._iob),
                                             int(select_mode), int(verify_mode),
                                             _p(tail.workspace), _stream(stream), ctypes.byref(h)),
               "tail_graph_create")
        self.handle = h
        # the direct call inside create advanced a chained anchor: start the replays from x0
        with torch.cuda.stream(stream):
            self.anchor.copy_(saved)
        stream.synchronize()

    def launch(self):
        _check(lib().brisk_tail_graph_launch(self.handle, _stream(self.stream)), "tail_graph_launch")
        return self.out

    def close(self):
        if self.handle:
            lib().brisk_tail_graph_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def mode_ids(select_mode: str, verify_mode: str):
    return (SELECT_SAMPLE if select_mode == "sample" else SELECT_GREEDY,
            VERIFY_STOCHASTIC if verify_mode == "stochastic" else VERIFY_GREEDY)


# ---------------------------------------------------------------- acceptance profile

def acceptance_counts(accepted_len: torch.Tensor, L: int, counts: torch.Tensor, stream=None) -> None:
    """Adds one step's accepted lengths ([B] int32, device) to running per-position counts
    (counts: [2L] int64 device tensor used as uint64; reached first, then accepted)."""
    if accepted_len.dtype != torch.int32 or counts.dtype != torch.int64 or counts.numel() != 2 * L:
        raise ValueError("accepted_len int32 [B], counts int64 [2L]")
    _check(lib().brisk_acceptance_counts(_p(accepted_len), int(accepted_len.numel()), int(L),
                                         _p(counts), _stream(stream)), "acceptance_counts")


def acceptance_weights(a, g=None, c=None, eps: float = 1e-8):
    """TPF, w_raw and the mean-one w_bar of a profile a[0..M-1] (host, float64)."""
    import numpy as np
    a = np.ascontiguousarray(a, dtype=np.float64)
    M = a.size
    gg = None if g is None else np.ascontiguousarray(g, dtype=np.float64)
    cc = None if c is None else np.ascontiguousarray(c, dtype=np.float64)
    if (gg is not None and gg.size != M + 1) or (cc is not None and cc.size != M + 1):
        raise ValueError("g and c need M + 1 entries")
    tpf = ctypes.c_double()
    w_raw = np.empty(M)
    w_bar = np.empty(M)
    vp = lambda x: None if x is None else x.ctypes.data_as(ctypes.c_void_p)
    _check(lib().brisk_acceptance_weights(M, vp(a), vp(gg), vp(cc), float(eps), ctypes.byref(tpf),
                                          vp(w_raw), vp(w_bar)), "acceptance_weights")
    return tpf.value, w_raw, w_bar


def isd_costs(M: int):
    """Gains g[0..M] and costs c[0..M] of the ISD instantiation (App. C.1, Eq. 8)."""
    import numpy as np
    g = np.zeros(int(M) + 1, dtype=np.float64)
    c = np.zeros(int(M) + 1, dtype=np.float64)
    _check(lib().brisk_isd_costs(int(M), g.ctypes.data_as(ctypes.c_void_p),
                                 c.ctypes.data_as(ctypes.c_void_p)), "isd_costs")
    return g, c


def tpf_isd(N: int, r: float) -> float:
    return float(lib().brisk_tpf_isd(int(N), float(r)))
