"""Python binding of libddattn.so (ctypes): argument marshalling only.

Every step of the attention runs in the library's CUDA kernels; this module
only turns torch tensors (device memory) and streams into the C ABI of
include/ddattn.h. There is no fallback: if the library is missing or the
call fails, it raises.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libddattn.so")

(DD_OK, DD_ERR_INVALID_ARG, DD_ERR_UNSUPPORTED, DD_ERR_WORKSPACE, DD_ERR_CUDA, DD_ERR_DEVICE_TIMEOUT,
 DD_ERR_DEVICE_LAYOUT) = range(7)


class DDAttnError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s: %s (status %d)" % (what, status_string(status) if _lib else "?", status))


class Desc(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("L", ctypes.c_int32), ("H", ctypes.c_int32), ("d", ctypes.c_int32),
                ("scale", ctypes.c_float), ("cu_doc_offsets", ctypes.c_void_p), ("n_offsets", ctypes.c_int32),
                ("rope_base", ctypes.c_float)]


_lib = None

EXPORTS = ("dd_attn_workspace_size", "dd_attn_fwd", "dd_attn_fwd_rope", "dd_attn_bwd", "dd_attn_bwd_phases",
           "dd_attn_bwd_noalloc", "dd_rope_qk", "dd_attn_clear_status", "dd_attn_poll_status", "dd_selftest_wait_timeout",
           "dd_status_string")
NOALLOC_SCRATCH_BYTES = 32 << 20
DD_BWD_PRE, DD_BWD_MAIN, DD_BWD_POST, DD_BWD_ALL = 1, 2, 4, 7


def lib() -> ctypes.CDLL:
    """Load libddattn.so (built by __graft_entry__.build() / paper_2405_13226_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libddattn.so is not built (%s); run python -m paper_2405_13226_gb300.build"
                               % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        vp, sz, i32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
        dp = ctypes.POINTER(Desc)
        L.dd_attn_workspace_size.argtypes = [dp, i32]
        L.dd_attn_workspace_size.restype = sz
        L.dd_attn_fwd.argtypes = [dp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.dd_attn_fwd.restype = i32
        L.dd_attn_fwd_rope.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.dd_attn_fwd_rope.restype = i32
        L.dd_attn_bwd.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.dd_attn_bwd.restype = i32
        L.dd_attn_bwd_phases.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, i32, vp]
        L.dd_attn_bwd_phases.restype = i32
        L.dd_attn_bwd_noalloc.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
        L.dd_attn_bwd_noalloc.restype = i32
        L.dd_rope_qk.argtypes = [dp, vp, vp, vp, vp, vp]
        L.dd_rope_qk.restype = i32
        L.dd_attn_clear_status.argtypes = [vp, vp]
        L.dd_attn_clear_status.restype = i32
        L.dd_attn_poll_status.argtypes = [vp]
        L.dd_attn_poll_status.restype = i32
        L.dd_selftest_wait_timeout.argtypes = [vp, ctypes.c_uint32, vp]
        L.dd_selftest_wait_timeout.restype = i32
        L.dd_status_string.argtypes = [i32]
        L.dd_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


def status_string(s: int) -> str:
    return lib().dd_status_string(int(s)).decode()


def make_desc(B: int, L: int, H: int, d: int, scale: float | None = None, cu_doc_offsets=None,
              rope_base: float = 0.0) -> Desc:
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    off_ptr, n_off = None, 0
    if cu_doc_offsets is not None:
        assert cu_doc_offsets.dtype == torch.int32 and cu_doc_offsets.is_cuda and cu_doc_offsets.is_contiguous()
        off_ptr, n_off = cu_doc_offsets.data_ptr(), cu_doc_offsets.numel()
    return Desc(B, L, H, d, float(scale), off_ptr, n_off, float(rope_base))


def workspace_size(desc: Desc, for_bwd: bool = True) -> int:
    return int(lib().dd_attn_workspace_size(ctypes.byref(desc), 1 if for_bwd else 0))


def new_workspace(desc: Desc, device, for_bwd: bool = True) -> torch.Tensor:
    n = workspace_size(desc, for_bwd)
    if n == 0:
        raise DDAttnError(DD_ERR_INVALID_ARG, "workspace_size")
    ws = torch.empty(n, dtype=torch.uint8, device=device)
    ws[:256].zero_()
    return ws


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check_qkv(*ts):
    for t in ts:
        if not (t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous() and t.dim() == 4):
            raise ValueError("expected contiguous CUDA bf16 tensors of shape [B, L, H, d]")


def rope_qk(q, k, rope_base, q_rot=None, k_rot=None, stream=None):
    """q_rot, k_rot = RoPE(q), RoPE(k) with base frequency rope_base (in place
    if q_rot is q / k_rot is k)."""
    _check_qkv(q, k)
    B, L, H, d = q.shape
    desc = make_desc(B, L, H, d, None, None, rope_base)
    q_rot = torch.empty_like(q) if q_rot is None else q_rot
    k_rot = torch.empty_like(k) if k_rot is None else k_rot
    _check_qkv(q_rot, k_rot)
    st = lib().dd_rope_qk(ctypes.byref(desc), q.data_ptr(), k.data_ptr(), q_rot.data_ptr(), k_rot.data_ptr(),
                          _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_rope_qk")
    return q_rot, k_rot


def fwd(q, k, v, scale=None, cu_doc_offsets=None, out=None, lse=None, workspace=None, stream=None):
    """o, lse = attention forward (causal; document-masked if cu_doc_offsets).
    With RoPE, q and k are the rotated tensors from rope_qk."""
    _check_qkv(q, k, v)
    B, L, H, d = q.shape
    desc = make_desc(B, L, H, d, scale, cu_doc_offsets)
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, H, L), dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = new_workspace(desc, q.device, for_bwd=False)
    st = lib().dd_attn_fwd(ctypes.byref(desc), q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                           lse.data_ptr(), workspace.data_ptr(), workspace.numel(), _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_attn_fwd")
    return out, lse


def fwd_rope(q, k, v, rope_base, scale=None, cu_doc_offsets=None, out=None, lse=None, q_rot=None, k_rot=None,
             workspace=None, stream=None):
    """o, lse, q_rot, k_rot = attention forward with RoPE (base rope_base) applied
    inside the kernel to the un-rotated q, k; q_rot, k_rot are the rotated
    tensors the backward takes (bwd(..., rope_base=rope_base))."""
    _check_qkv(q, k, v)
    B, L, H, d = q.shape
    desc = make_desc(B, L, H, d, scale, cu_doc_offsets, rope_base)
    out = torch.empty_like(q) if out is None else out
    lse = torch.empty((B, H, L), dtype=torch.float32, device=q.device) if lse is None else lse
    q_rot = torch.empty_like(q) if q_rot is None else q_rot
    k_rot = torch.empty_like(k) if k_rot is None else k_rot
    _check_qkv(q_rot, k_rot)
    if workspace is None:
        workspace = new_workspace(desc, q.device, for_bwd=False)
    st = lib().dd_attn_fwd_rope(ctypes.byref(desc), q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                lse.data_ptr(), q_rot.data_ptr(), k_rot.data_ptr(), workspace.data_ptr(),
                                workspace.numel(), _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_attn_fwd_rope")
    return out, lse, q_rot, k_rot


def bwd(q, k, v, o, dO, lse, scale=None, cu_doc_offsets=None, dq=None, dk=None, dv=None, workspace=None,
        stream=None, phases=DD_BWD_ALL, rope_base=0.0):
    """dq, dk, dv = attention backward from the forward's o and lse (`phases`:
    a subset of its three kernels, see dd_attn_bwd_phases). With rope_base > 0,
    q and k are the rotated tensors and dq, dk are returned with respect to the
    un-rotated ones."""
    _check_qkv(q, k, v, o, dO)
    B, L, H, d = q.shape
    desc = make_desc(B, L, H, d, scale, cu_doc_offsets, rope_base)
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    if workspace is None:
        workspace = new_workspace(desc, q.device, for_bwd=True)
    st = lib().dd_attn_bwd_phases(ctypes.byref(desc), q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                  dO.data_ptr(), lse.data_ptr(), dq.data_ptr(), dk.data_ptr(), dv.data_ptr(),
                                  workspace.data_ptr(), workspace.numel(), int(phases), _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_attn_bwd")
    return dq, dk, dv


def clear_status(workspace, stream=None) -> None:
    st = lib().dd_attn_clear_status(workspace.data_ptr(), _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_attn_clear_status")


def selftest_wait_timeout(workspace, limit_us: int = 20000, stream=None) -> None:
    """Launch the bounded-wait self-test kernel (see dd_selftest_wait_timeout)."""
    st = lib().dd_selftest_wait_timeout(workspace.data_ptr(), int(limit_us), _stream(stream))
    if st != DD_OK:
        raise DDAttnError(st, "dd_selftest_wait_timeout")


def poll_status(workspace) -> int:
    """Synchronise and return the device status word of `workspace`."""
    return int(lib().dd_attn_poll_status(workspace.data_ptr()))
