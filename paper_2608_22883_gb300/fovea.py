"""Thin ctypes binding of libfovea (include/fovea.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch provides device memory (tensors, workspaces) and streams.
If the library has not been built this module raises at first use: there is
no CPU fallback.
"""

from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libfovea.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_OOM, ERR_TIMEOUT = range(6)
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "OOM", 5: "TIMEOUT"}
BF16, FP32 = 0, 1
MAX_D, MAX_H, MAX_K, MAX_ENTRIES, MAX_SEQ = 8192, 4096, 1024, 32768, 512

# Field order of fovea_params after the scalar header (C struct order).
PARAM_NAMES = (
    "ln_v_gamma", "ln_v_beta", "W_K", "W_U",
    "ln_h_gamma", "ln_h_beta", "E_dep", "W_Q",
    "W_f1", "b_f1", "W_f2", "b_f2",
    "W_g1", "b_g1", "w_g2", "b_g2",
    "rms_gamma",
)

EXPORTS = (
    "fovea_build_memory", "fovea_memory_destroy", "fovea_memory_info", "fovea_memory_tensors",
    "fovea_workspace_size", "fovea_workspace_init", "fovea_retrieve_fuse", "fovea_sync_errors",
    "fovea_last_error", "fovea_timing_enable", "fovea_timing_read", "fovea_version",
    "fovea_retrieve_fuse_noalloc", "fovea_noalloc_sync_errors", "fovea_memory_folded_keys",
    "fovea_lm_head_topk", "fovea_debug_wait_limit", "fovea_lm_head_workspace_size",
)
NOALLOC_WORKSPACE_BYTES = 32 << 20


class FoveaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class CParams(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int), ("mlp_hidden", ctypes.c_int),
                ("max_depth", ctypes.c_int), ("dtype", ctypes.c_int),
                ("ln_eps", ctypes.c_float), ("rms_eps", ctypes.c_float)] + \
               [(n, ctypes.c_void_p) for n in PARAM_NAMES]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build(); "
                               "the FOVEA path has no CPU fallback")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32p = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32)
        L.fovea_build_memory.argtypes = [ctypes.POINTER(CParams), vp, vp, ctypes.c_int, ctypes.c_int,
                                         vp, ctypes.POINTER(vp)]
        L.fovea_memory_destroy.argtypes = [vp]
        L.fovea_memory_destroy.restype = None
        L.fovea_memory_info.argtypes = [vp, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int), i32p]
        L.fovea_memory_tensors.argtypes = [vp, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(vp),
                                           ctypes.POINTER(ctypes.c_int64)]
        L.fovea_memory_folded_keys.argtypes = [vp, vp, ctypes.POINTER(vp)]
        L.fovea_lm_head_topk.argtypes = [vp, ctypes.c_int, ctypes.c_int, ctypes.c_int, vp,
                                         ctypes.c_int, ctypes.c_int, vp, vp, vp, vp,
                                         ctypes.c_size_t, vp]
        L.fovea_workspace_size.argtypes = [ctypes.POINTER(CParams), vp, i32p, ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_size_t)]
        L.fovea_workspace_init.argtypes = [vp, ctypes.c_size_t, vp]
        L.fovea_retrieve_fuse.argtypes = [ctypes.POINTER(CParams), vp, vp, vp, i32p, vp,
                                          ctypes.c_float, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                          vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
        L.fovea_retrieve_fuse_noalloc.argtypes = [ctypes.POINTER(CParams), vp, vp, vp, i32p, vp,
                                                  ctypes.c_float, ctypes.c_int, ctypes.c_int,
                                                  ctypes.c_int, vp, vp, vp, vp, vp, vp]
        L.fovea_retrieve_fuse_noalloc.restype = ctypes.c_int
        L.fovea_lm_head_workspace_size.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                    ctypes.c_int, ctypes.POINTER(ctypes.c_size_t)]
        L.fovea_lm_head_workspace_size.restype = ctypes.c_int
        L.fovea_noalloc_sync_errors.argtypes = [vp]
        L.fovea_noalloc_sync_errors.restype = ctypes.c_int
        L.fovea_debug_wait_limit.argtypes = [ctypes.c_ulonglong]
        L.fovea_debug_wait_limit.restype = ctypes.c_int
        L.fovea_sync_errors.argtypes = [vp, vp]
        L.fovea_last_error.restype = ctypes.c_char_p
        L.fovea_last_error.argtypes = []
        L.fovea_timing_enable.argtypes = [ctypes.c_int]
        L.fovea_timing_read.argtypes = [ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_double),
                                        ctypes.POINTER(ctypes.c_int), ctypes.c_int]
        L.fovea_timing_read.restype = ctypes.c_int
        L.fovea_version.restype = ctypes.c_int
        for name in ("fovea_build_memory", "fovea_memory_info", "fovea_memory_tensors",
                     "fovea_memory_folded_keys", "fovea_lm_head_topk",
                     "fovea_workspace_size", "fovea_workspace_init", "fovea_retrieve_fuse",
                     "fovea_sync_errors", "fovea_timing_enable"):
            getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def _check(status: int):
    if status != OK:
        raise FoveaError(status, lib().fovea_last_error().decode())


def last_error() -> str:
    return lib().fovea_last_error().decode()


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to libfovea must be contiguous")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def torch_dtype(dtype: int) -> torch.dtype:
    return torch.bfloat16 if dtype == BF16 else torch.float32


class Params:
    """fovea_params over a dict of device tensors named as in PARAM_NAMES."""

    def __init__(self, weights: Dict[str, torch.Tensor], *, d_model: int, mlp_hidden: int = 512,
                 max_depth: int = 6, dtype: int = BF16, ln_eps: float = 1e-5,
                 rms_eps: float = 1e-6):
        self.weights = weights          # keeps the tensors alive
        c = CParams()
        c.d_model, c.mlp_hidden, c.max_depth, c.dtype = d_model, mlp_hidden, max_depth, dtype
        c.ln_eps, c.rms_eps = ln_eps, rms_eps
        for n in PARAM_NAMES:
            t = weights.get(n)
            setattr(c, n, None if t is None else _ptr(t))
        self.c = c
        self.d_model, self.mlp_hidden, self.max_depth, self.dtype = d_model, mlp_hidden, max_depth, dtype

    @property
    def ref(self):
        return ctypes.byref(self.c)


class _CudaView:
    """__cuda_array_interface__ over library-owned device memory (no copy)."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (ptr, False), "version": 3, "strides": None}


class Memory:
    """A fovea_memory handle (library-owned device buffers)."""

    def __init__(self, handle: ctypes.c_void_p, params: Params):
        self.handle = handle
        self.d = params.d_model
        self.dtype = params.dtype
        B, total = ctypes.c_int(), ctypes.c_int()
        _check(lib().fovea_memory_info(handle, ctypes.byref(B), ctypes.byref(total), None))
        self.B, self.total = B.value, total.value
        counts = (ctypes.c_int32 * self.B)()
        _check(lib().fovea_memory_info(handle, None, None, counts))
        self.valid_counts = list(counts)

    def views(self):
        """(keys [total, d], values [total, d], index [total], offsets list) as
        torch views of the handle's device memory (valid while it lives)."""
        k, u, idx = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
        offs = (ctypes.c_int64 * (self.B + 1))()
        _check(lib().fovea_memory_tensors(self.handle, ctypes.byref(k), ctypes.byref(u),
                                          ctypes.byref(idx), offs))
        if self.total == 0:
            e = torch.empty((0, self.d), dtype=torch_dtype(self.dtype), device="cuda")
            return e, e, torch.empty(0, dtype=torch.int32, device="cuda"), list(offs)
        ts = "<i2" if self.dtype == BF16 else "<f4"

        def view(ptr):
            t = torch.as_tensor(_CudaView(ptr, (self.total, self.d), ts), device="cuda")
            return t.view(torch.bfloat16) if self.dtype == BF16 else t
        index = torch.as_tensor(_CudaView(idx.value, (self.total,), "<i4"), device="cuda")
        return view(k.value), view(u.value), index, list(offs)

    def folded_keys(self, params: Params) -> Optional[torch.Tensor]:
        """The folded keys kappa = W_Q^T k as [total, 2d] bf16 (row i: kappa_hi
        then kappa_lo; a view of the handle's memory) when the memory holds
        them for params' W_Q, else None; a step with these params then scores
        against them."""
        f = ctypes.c_void_p()
        _check(lib().fovea_memory_folded_keys(self.handle, params.c.W_Q, ctypes.byref(f)))
        if not f.value:
            return None
        if self.total == 0:
            return torch.empty((0, 2 * self.d), dtype=torch.bfloat16, device="cuda")
        return torch.as_tensor(_CudaView(f.value, (self.total, 2 * self.d), "<i2"),
                               device="cuda").view(torch.bfloat16)

    def destroy(self):
        if self.handle:
            lib().fovea_memory_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def build_memory(params: Params, v: torch.Tensor, mask: Optional[torch.Tensor] = None,
                 stream=None) -> Memory:
    """fovea_build_memory: v [B, M_max, d] (params dtype), mask [B, M_max] uint8 or None."""
    B, M_max = v.shape[0], v.shape[1]
    out = ctypes.c_void_p()
    _check(lib().fovea_build_memory(params.ref, _ptr(v), _ptr(mask), B, M_max, _stream(stream),
                                    ctypes.byref(out)))
    return Memory(out, params)


def _offsets(row_offsets) -> ctypes.Array:
    vals = [int(x) for x in row_offsets]
    return (ctypes.c_int32 * len(vals))(*vals)


def workspace_size(params: Params, memory: Memory, row_offsets, k_max: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().fovea_workspace_size(params.ref, memory.handle, _offsets(row_offsets), k_max,
                                      ctypes.byref(n)))
    return n.value


def new_workspace(params: Params, memory: Memory, row_offsets, k_max: int, stream=None) -> torch.Tensor:
    """Allocate (torch) and initialise a workspace for these shapes."""
    n = workspace_size(params, memory, row_offsets, k_max)
    ws = torch.empty(max(n, 256), dtype=torch.uint8, device="cuda")
    _check(lib().fovea_workspace_init(_ptr(ws), ws.numel(), _stream(stream)))
    return ws


def _l_max(params: Params, l_max: Optional[int]) -> int:
    return params.max_depth if l_max is None else int(l_max)


def retrieve_fuse(params: Params, memory: Memory, h: torch.Tensor, depth: torch.Tensor,
                  row_offsets, row_scale: Optional[torch.Tensor], rho: float, k_min: int,
                  k_max: int, h_out: torch.Tensor, workspace: torch.Tensor, *,
                  counts: Optional[torch.Tensor] = None, indices: Optional[torch.Tensor] = None,
                  readout: Optional[torch.Tensor] = None, gate: Optional[torch.Tensor] = None,
                  l_max: Optional[int] = None, stream=None, offsets_c=None) -> None:
    """fovea_retrieve_fuse into caller-allocated outputs (asynchronous).
    l_max: depth gate (None: every row is corrected)."""
    offs = offsets_c if offsets_c is not None else _offsets(row_offsets)
    _check(lib().fovea_retrieve_fuse(params.ref, memory.handle, _ptr(h), _ptr(depth), offs,
                                     _ptr(row_scale), float(rho), int(k_min), int(k_max),
                                     _l_max(params, l_max), _ptr(h_out), _ptr(counts),
                                     _ptr(indices), _ptr(readout), _ptr(gate), _ptr(workspace),
                                     workspace.numel(), _stream(stream)))


def step(params: Params, memory: Memory, h: torch.Tensor, depth: torch.Tensor, row_offsets,
         row_scale: Optional[torch.Tensor], rho: float, k_min: int, k_max: int, *,
         workspace: Optional[torch.Tensor] = None, want_readout: bool = True,
         l_max: Optional[int] = None, stream=None) -> Dict[str, torch.Tensor]:
    """Allocate outputs with torch and run one draft step; returns them."""
    N = h.shape[0]
    dev = h.device
    if workspace is None:
        workspace = new_workspace(params, memory, row_offsets, k_max, stream)
    out = dict(
        h_out=torch.empty_like(h),
        counts=torch.empty(N, dtype=torch.int32, device=dev),
        indices=torch.empty((N, k_max), dtype=torch.int32, device=dev),
        readout=torch.empty((N, params.d_model), dtype=torch.float32, device=dev) if want_readout else None,
        gate=torch.empty(N, dtype=torch.float32, device=dev),
    )
    retrieve_fuse(params, memory, h, depth, row_offsets, row_scale, rho, k_min, k_max,
                  out["h_out"], workspace, counts=out["counts"], indices=out["indices"],
                  readout=out["readout"], gate=out["gate"], l_max=l_max, stream=stream)
    out["workspace"] = workspace
    return out


def retrieve_fuse_noalloc(params: Params, memory: Memory, h: torch.Tensor, depth: torch.Tensor,
                          row_offsets, row_scale: Optional[torch.Tensor], rho: float, k_min: int,
                          k_max: int, h_out: torch.Tensor, *,
                          counts: Optional[torch.Tensor] = None,
                          indices: Optional[torch.Tensor] = None,
                          readout: Optional[torch.Tensor] = None,
                          gate: Optional[torch.Tensor] = None, l_max: Optional[int] = None,
                          stream=None) -> None:
    """fovea_retrieve_fuse_noalloc: the draft step with the library's static
    scratch instead of a workspace (for callers that cannot allocate)."""
    _check(lib().fovea_retrieve_fuse_noalloc(params.ref, memory.handle, _ptr(h), _ptr(depth),
                                             _offsets(row_offsets), _ptr(row_scale), float(rho),
                                             int(k_min), int(k_max), _l_max(params, l_max),
                                             _ptr(h_out), _ptr(counts), _ptr(indices),
                                             _ptr(readout), _ptr(gate), _stream(stream)))


def noalloc_sync_errors(stream=None) -> None:
    """fovea_noalloc_sync_errors: read and clear the static array's error word."""
    _check(lib().fovea_noalloc_sync_errors(_stream(stream)))


def sync_errors(workspace: torch.Tensor, stream=None) -> None:
    _check(lib().fovea_sync_errors(_ptr(workspace), _stream(stream)))


def debug_wait_limit(limit_ns: int) -> None:
    """fovea_debug_wait_limit: limit of the bounded device waits of later
    launches (0: the default of about 2 s).  For tests of the timeout path."""
    _check(lib().fovea_debug_wait_limit(int(limit_ns)))


def lm_head_workspace(vocab: int, d_model: int, N: int, k_c: int, stream=None) -> torch.Tensor:
    """An initialised workspace for fovea_lm_head_topk of this shape."""
    n = ctypes.c_size_t()
    _check(lib().fovea_lm_head_workspace_size(vocab, d_model, N, k_c, ctypes.byref(n)))
    ws = torch.empty(n.value, dtype=torch.uint8, device="cuda")
    _check(lib().fovea_workspace_init(_ptr(ws), ws.numel(), _stream(stream)))
    return ws


def lm_head_topk(W_LM: torch.Tensor, h_hat: torch.Tensor, k_c: int, workspace: torch.Tensor,
                 logits: Optional[torch.Tensor] = None, stream=None, write_logits: bool = True):
    """fovea_lm_head_topk: z = h_hat W_LM^T [N, V] (fp32) and the k_c largest
    logits per row (token indices, values), descending, smaller index first
    on ties.  Returns (top_idx [N, k_c] int32, top_val [N, k_c], logits);
    with write_logits=False the logits are not written (NULL) and None is
    returned in their place."""
    V, d = W_LM.shape
    N = h_hat.shape[0]
    dt = BF16 if W_LM.dtype == torch.bfloat16 else FP32
    if not write_logits:
        logits = None
    elif logits is None:
        logits = torch.empty((N, V), dtype=torch.float32, device=h_hat.device)
    idx = torch.empty((N, k_c), dtype=torch.int32, device=h_hat.device)
    val = torch.empty((N, k_c), dtype=torch.float32, device=h_hat.device)
    _check(lib().fovea_lm_head_topk(_ptr(W_LM), V, d, dt, _ptr(h_hat), N, k_c,
                                    _ptr(logits) if logits is not None else None,
                                    _ptr(idx), _ptr(val), _ptr(workspace), workspace.numel(),
                                    _stream(stream)))
    return idx, val, logits


def timing_enable(on: bool = True) -> None:
    _check(lib().fovea_timing_enable(1 if on else 0))


def timing_read() -> Dict[str, tuple]:
    """{kernel name: (total ms, launches)} of launches recorded since enabling."""
    cap = 64
    names = (ctypes.c_char_p * cap)()
    ms = (ctypes.c_double * cap)()
    cnt = (ctypes.c_int * cap)()
    n = lib().fovea_timing_read(names, ms, cnt, cap)
    return {names[i].decode(): (ms[i], cnt[i]) for i in range(min(n, cap))}


def version() -> int:
    return lib().fovea_version()
