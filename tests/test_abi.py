"""The C ABI without a GPU: the library loads, exports every entry point that
include/brisk.h declares, and rejects bad arguments on the host before any
CUDA call."""
import ctypes
import os
import re

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "brisk.h")


@pytest.fixture(scope="session")
def B():
    from paper_2609_33390_gb300 import build
    build.build()
    from paper_2609_33390_gb300 import brisk
    return brisk


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(brisk_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_four_paper_entry_points():
    names = declared_functions()
    for n in ("brisk_topk_candidates", "brisk_corrector_select", "brisk_verify_block",
              "brisk_decode_tail"):
        assert n in names


def test_every_declared_symbol_is_exported(B):
    lib = B.lib()
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def _dims(lib_mod, **kw):
    d = dict(B=2, L=8, V=1000, d=64, K=4, r=16, logits_dtype=torch.bfloat16,
             hidden_dtype=torch.bfloat16)
    d.update(kw)
    return lib_mod.make_dims(**d)


def test_sizes_for_valid_and_invalid_dims(B):
    ok = _dims(B)
    assert B.workspace_bytes(ok) > 0 and B.workspace_bytes(ok) % 256 == 0
    assert B.tables_bytes(ok) > 0 and B.tables_bytes(ok) % 256 == 0
    for bad in (dict(K=3), dict(K=33), dict(L=0), dict(L=65), dict(V=3), dict(r=8), dict(r=24),
                dict(r=1024), dict(d=12)):
        assert B.workspace_bytes(_dims(B, **bad)) == 0, bad
        assert B.tables_bytes(_dims(B, **bad)) == 0, bad
    d = _dims(B)
    d.B = 0
    assert B.workspace_bytes(d) == 0
    d = _dims(B)
    d.logits_dtype = 7
    assert B.workspace_bytes(d) == 0


def test_null_pointers_and_bad_modes_rejected_on_host(B):
    lib = B.lib()
    d = _dims(B)
    dp = ctypes.byref(d)
    fake = ctypes.c_void_p(256)  # never dereferenced: validation fails first
    assert lib.brisk_topk_candidates(dp, None, fake, fake, fake, fake, None) == B.ERR_INVALID_ARG
    assert lib.brisk_topk_candidates(None, fake, fake, fake, fake, fake, None) == B.ERR_INVALID_ARG
    # misaligned workspace
    assert lib.brisk_topk_candidates(dp, fake, fake, fake, fake, ctypes.c_void_p(258),
                                     None) == B.ERR_INVALID_ARG
    p = B.Params()
    assert lib.brisk_corrector_prepare(dp, ctypes.byref(p), fake, None) == B.ERR_INVALID_ARG
    assert lib.brisk_verify_block(dp, fake, fake, fake, fake, 0, 7, None, None, fake, fake, fake,
                                  fake, None) == B.ERR_INVALID_ARG
    # stochastic verify needs its uniforms
    assert lib.brisk_verify_block(dp, fake, fake, fake, fake, 0, 1, None, None, fake, fake, fake,
                                  fake, None) == B.ERR_INVALID_ARG
    io = B.TailIO()
    ev = B.Events()
    assert lib.brisk_decode_tail(dp, ctypes.byref(p), fake, ctypes.byref(io), 0, 0, fake,
                                 ctypes.byref(ev), None) == B.ERR_INVALID_ARG
    assert lib.brisk_last_device_status(None, 0, None) == B.ERR_INVALID_ARG


def test_status_strings(B):
    assert B.status_string(B.OK) == "BRISK_OK"
    assert B.status_string(B.ERR_NUMERIC) == "BRISK_ERR_NUMERIC"
    assert B.status_string(99) == "BRISK_ERR_UNKNOWN"


def test_binding_refuses_to_run_without_the_library(tmp_path, monkeypatch):
    from paper_2609_33390_gb300 import brisk
    monkeypatch.setattr(brisk, "_lib", None)
    monkeypatch.setattr(brisk, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError):
        brisk.lib()


def test_wait_limit_setter_returns_the_previous_limit(B):
    default = 4000000000
    prev = B.set_wait_limit(1234)
    try:
        assert prev == default
        assert B.set_wait_limit(0) == 1234          # 0 restores the default
        assert B.set_wait_limit(-5) == default
        assert B.set_wait_limit(99) == default
    finally:
        B.set_wait_limit(0)


def test_kernels_per_tail_follows_the_schedule(B):
    """Four launches in the fused small-batch schedule (one sweep of both tensors, two tensor-core
    products, the corrector that verifies), six otherwise; four SIMT products with fp32 weights."""
    fused = _dims(B, B=2, L=8, V=65536, d=64, K=8, r=16)          # chunked rows, 4 MB of logits
    separate = _dims(B, B=4, L=32, V=140000, d=64, K=8, r=16)     # chunked rows, 72 MB
    overlap = _dims(B, B=128, L=32, V=126464, d=4096, K=8, r=256)  # one task a row (many rows)
    short_rows = _dims(B, B=2, L=8, V=4096, d=64, K=8, r=16)      # one task a row (rows too short)
    assert B.kernels_per_tail(fused) == 4
    assert B.kernels_per_tail(separate) == 6
    assert B.kernels_per_tail(overlap) == 6
    assert B.kernels_per_tail(short_rows) == 6
    assert B.kernels_per_tail(_dims(B, B=2, L=8, V=65536, d=64, K=8, r=16,
                                    hidden_dtype=torch.float32)) == 6
    assert B.kernels_per_tail(_dims(B, B=2, L=8, V=4096, d=64, K=8, r=16,
                                    hidden_dtype=torch.float32)) == 8
    bad = _dims(B, K=3)
    assert B.kernels_per_tail(bad) == 0
