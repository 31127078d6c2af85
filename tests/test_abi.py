"""The C-ABI library on the host: it loads, exports every entry point the
header declares, and rejects bad arguments with the documented status before
touching the GPU (so these run without a device)."""

import ctypes
import os
import re
import subprocess
import sys

import numpy as np
import pytest

from paper_2608_22883_gb300 import fovea

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fovea.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"FOVEA_API\s+[^;(]*?\b(fovea_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(fovea.LIB_PATH):
        from paper_2608_22883_gb300 import _build
        _build.build()
    return fovea.lib()


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("fovea_build_memory", "fovea_retrieve_fuse", "fovea_memory_destroy",
                 "fovea_last_error"):
        assert name in syms
    assert set(syms) == set(fovea.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    out = subprocess.run(["nm", "-D", "--defined-only", fovea.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (fovea_\w+)", out))
    missing = set(declared_symbols()) - exported
    assert not missing, f"not exported: {missing}"
    for name in declared_symbols():
        assert hasattr(L, name)
    assert L.fovea_version() == 200


def dummy_params(d=256, H=512, D=6, dtype=fovea.BF16, ptr=0x10000):
    c = fovea.CParams()
    c.d_model, c.mlp_hidden, c.max_depth, c.dtype = d, H, D, dtype
    c.ln_eps, c.rms_eps = 1e-5, 1e-6
    for n in fovea.PARAM_NAMES:
        setattr(c, n, ptr)      # never dereferenced: every call below fails its checks first
    return c


def call_step(L, c, *, rho=0.9, k_min=1, k_max=16, l_max=6, mem=None, h=0x10000, ws=0x10000):
    offs = (ctypes.c_int32 * 2)(0, 4)
    return L.fovea_retrieve_fuse(ctypes.byref(c) if c is not None else None, mem, h, 0x10000, offs,
                                 None, rho, k_min, k_max, l_max, 0x10000, None, None, None, None,
                                 ws, 1 << 20, None)


@pytest.mark.parametrize("kw,status", [
    (dict(rho=0.0), fovea.ERR_INVALID_ARG),
    (dict(rho=1.5), fovea.ERR_INVALID_ARG),
    (dict(rho=float("nan")), fovea.ERR_INVALID_ARG),
    (dict(k_min=0), fovea.ERR_INVALID_ARG),
    (dict(k_min=20, k_max=16), fovea.ERR_INVALID_ARG),
    (dict(k_max=2048), fovea.ERR_UNSUPPORTED),
    (dict(), fovea.ERR_INVALID_ARG),               # memory is NULL
])
def test_step_argument_checks(L, kw, status):
    assert call_step(L, dummy_params(), **kw) == status
    assert fovea.last_error() != ""


@pytest.mark.parametrize("mutate,status", [
    (lambda c: setattr(c, "d_model", 100), fovea.ERR_INVALID_ARG),
    (lambda c: setattr(c, "d_model", 16384), fovea.ERR_UNSUPPORTED),
    (lambda c: setattr(c, "mlp_hidden", 96), fovea.ERR_INVALID_ARG),
    (lambda c: setattr(c, "mlp_hidden", 8192), fovea.ERR_UNSUPPORTED),
    (lambda c: setattr(c, "max_depth", -1), fovea.ERR_INVALID_ARG),
    (lambda c: setattr(c, "dtype", 7), fovea.ERR_INVALID_ARG),
    (lambda c: setattr(c, "W_Q", None), fovea.ERR_INVALID_ARG),
    (lambda c: setattr(c, "W_f2", 0x10004), fovea.ERR_INVALID_ARG),   # misaligned
    (lambda c: setattr(c, "rms_eps", 0.0), fovea.ERR_INVALID_ARG),
])
def test_param_checks(L, mutate, status):
    c = dummy_params()
    mutate(c)
    assert call_step(L, c) == status
    assert L.fovea_retrieve_fuse(None, None, None, None, None, None, 0.9, 1, 4, 6, None, None,
                                 None, None, None, None, 0, None) == fovea.ERR_INVALID_ARG


def test_build_argument_checks(L):
    out = ctypes.c_void_p()
    c = dummy_params()
    assert L.fovea_build_memory(None, 0x10000, None, 1, 8, None, ctypes.byref(out)) == fovea.ERR_INVALID_ARG
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 0, 8, None, ctypes.byref(out)) == fovea.ERR_INVALID_ARG
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 1, -1, None, ctypes.byref(out)) == fovea.ERR_INVALID_ARG
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 600, 8, None, ctypes.byref(out)) == fovea.ERR_UNSUPPORTED
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 1, 40000, None, ctypes.byref(out)) == fovea.ERR_UNSUPPORTED
    assert L.fovea_build_memory(ctypes.byref(c), None, None, 1, 8, None, ctypes.byref(out)) == fovea.ERR_INVALID_ARG
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 1, 8, None, None) == fovea.ERR_INVALID_ARG
    c.W_U = None
    assert L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 1, 8, None, ctypes.byref(out)) == fovea.ERR_INVALID_ARG
    assert out.value is None


def test_injected_allocation_failure():
    # A fresh process so the environment variable is read by the library.
    code = (
        "import ctypes, sys; sys.path.insert(0, %r)\n"
        "from paper_2608_22883_gb300 import fovea\n"
        "from tests.test_abi import dummy_params\n"
        "L = fovea.lib(); out = ctypes.c_void_p(); c = dummy_params()\n"
        "st = L.fovea_build_memory(ctypes.byref(c), 0x10000, None, 1, 8, None, ctypes.byref(out))\n"
        "print(st, fovea.last_error()); sys.exit(0 if st == fovea.ERR_OOM and out.value is None else 1)\n"
    ) % ROOT
    env = dict(os.environ, FOVEA_FAULT_ALLOC="1")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, cwd=ROOT)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "FOVEA_FAULT_ALLOC" in r.stdout


def test_memory_queries_reject_null(L):
    assert L.fovea_memory_info(None, None, None, None) == fovea.ERR_INVALID_ARG
    assert L.fovea_memory_tensors(None, None, None, None, None) == fovea.ERR_INVALID_ARG
    f = ctypes.c_void_p()
    assert L.fovea_memory_folded_keys(None, None, ctypes.byref(f)) == fovea.ERR_INVALID_ARG
    n = ctypes.c_size_t()
    c = dummy_params()
    assert L.fovea_workspace_size(ctypes.byref(c), None, None, 16, ctypes.byref(n)) == fovea.ERR_INVALID_ARG
    assert L.fovea_workspace_init(None, 1024, None) == fovea.ERR_INVALID_ARG
    assert L.fovea_sync_errors(None, None) == fovea.ERR_INVALID_ARG
    L.fovea_memory_destroy(None)      # ignored


def test_debug_wait_limit_is_a_host_setting(L):
    # process-wide; takes effect at the next tensor-core launch (none here)
    assert L.fovea_debug_wait_limit(1000) == fovea.OK
    assert L.fovea_debug_wait_limit(0) == fovea.OK       # back to the default


def test_product_path_fails_loudly_without_library(tmp_path, monkeypatch):
    monkeypatch.setattr(fovea, "_lib", None)
    monkeypatch.setattr(fovea, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        fovea.lib()


def call_lm_head(L, *, W=0x10000, V=1000, d=256, dtype=fovea.BF16, h=0x10000, N=4, k_c=6,
                 logits=0x10000, idx=0x10000, ws=0x10000, ws_bytes=1 << 20):
    return L.fovea_lm_head_topk(W, V, d, dtype, h, N, k_c, logits, idx, None, ws, ws_bytes, None)


@pytest.mark.parametrize("kw,status", [
    (dict(k_c=0), fovea.ERR_INVALID_ARG),
    (dict(k_c=33), fovea.ERR_INVALID_ARG),
    (dict(V=5), fovea.ERR_INVALID_ARG),              # vocab < k_c
    (dict(d=100), fovea.ERR_INVALID_ARG),
    (dict(N=-1), fovea.ERR_INVALID_ARG),
    (dict(W=None), fovea.ERR_INVALID_ARG),
    (dict(h=0x10004), fovea.ERR_INVALID_ARG),        # misaligned
    (dict(idx=None), fovea.ERR_INVALID_ARG),
    (dict(ws=0x10010), fovea.ERR_INVALID_ARG),       # not 256-byte aligned
    (dict(ws_bytes=1024), fovea.ERR_INVALID_ARG),
    (dict(dtype=7), fovea.ERR_INVALID_ARG),
    (dict(dtype=fovea.FP32), fovea.ERR_UNSUPPORTED),
])
def test_lm_head_argument_checks(L, kw, status):
    assert call_lm_head(L, **kw) == status
    assert fovea.last_error() != ""
