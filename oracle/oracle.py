"""ctypes front end of the fp64 CPU attention oracle (attn_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline / reference legs of bench.py. The CUDA path never imports it, and
it imports nothing from the CUDA path.

Inputs are the bf16 values of q, k, v, dO converted exactly to float64; the
definition it computes is written out in attn_oracle.c (causal attention with
the document mask of Sec. 1 / Sec. 3.5; single-document sequences of Sec. 2.1).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attn_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile attn_oracle.c into liboracle.so next to it (gcc, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int32)
        lib.oracle_doc_ids.argtypes = [ctypes.c_int, ctypes.c_int, ip, ctypes.c_int, ip]
        lib.oracle_attn_fwd.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double, ip,
                                        dp, dp, dp, dp, dp]
        lib.oracle_attn_fwd_rows.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_double, ip, dp, dp, dp,
                                             ctypes.c_int, ip, dp, dp]
        lib.oracle_attn_bwd.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double, ip,
                                        dp, dp, dp, dp, dp, dp, dp]
        lib.oracle_attn_bwd_rows.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_double, ip, dp, dp, dp, dp,
                                             ctypes.c_int, ip, dp, ctypes.c_int, ip, dp, dp]
        lib.oracle_live_pairs.argtypes = [ctypes.c_int, ip]
        lib.oracle_live_pairs.restype = ctypes.c_longlong
        _lib = lib
    return _lib


def _d(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _i(a):
    a = np.ascontiguousarray(a, dtype=np.int32)
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def doc_ids(L: int, b: int, cu_doc_offsets=None) -> np.ndarray:
    """Document id of each token of sequence b (see oracle_doc_ids)."""
    lib = _load()
    out = np.zeros(L, dtype=np.int32)
    if cu_doc_offsets is None:
        lib.oracle_doc_ids(L, b, None, 0, out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
    else:
        off, offp = _i(cu_doc_offsets)
        lib.oracle_doc_ids(L, b, offp, len(off), out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
    return out


def attn_fwd(q, k, v, doc, scale):
    """Slices q,k,v: [n, L, d] float64; doc: [n, L] int32. Returns o [n,L,d], lse [n,L]."""
    lib = _load()
    n, L, d = q.shape
    q, qp = _d(q); k, kp = _d(k); v, vp = _d(v); doc, docp = _i(doc)
    o = np.zeros((n, L, d)); lse = np.zeros((n, L))
    lib.oracle_attn_fwd(n, L, d, float(scale), docp, qp, kp, vp,
                        o.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                        lse.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return o, lse


def attn_fwd_rows(q, k, v, doc, scale, rows):
    """One slice q,k,v: [L, d]; returns o [len(rows), d], lse [len(rows)] for the given query rows."""
    lib = _load()
    L, d = q.shape
    q, qp = _d(q); k, kp = _d(k); v, vp = _d(v); doc, docp = _i(doc); rows, rp = _i(rows)
    o = np.zeros((len(rows), d)); lse = np.zeros(len(rows))
    lib.oracle_attn_fwd_rows(L, d, float(scale), docp, qp, kp, vp, len(rows), rp,
                             o.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                             lse.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return o, lse


def attn_bwd(q, k, v, dO, doc, scale):
    """Slices [n, L, d]; returns dq, dk, dv [n, L, d] from the oracle's own fp64 forward."""
    lib = _load()
    n, L, d = q.shape
    q, qp = _d(q); k, kp = _d(k); v, vp = _d(v); dO, gp = _d(dO); doc, docp = _i(doc)
    dq = np.zeros((n, L, d)); dk = np.zeros((n, L, d)); dv = np.zeros((n, L, d))
    P = ctypes.POINTER(ctypes.c_double)
    lib.oracle_attn_bwd(n, L, d, float(scale), docp, qp, kp, vp, gp,
                        dq.ctypes.data_as(P), dk.ctypes.data_as(P), dv.ctypes.data_as(P))
    return dq, dk, dv


def attn_bwd_rows(q, k, v, dO, doc, scale, qrows, krows):
    """One slice [L, d]; dq for query rows `qrows`, dk/dv for key rows `krows`."""
    lib = _load()
    L, d = q.shape
    q, qp = _d(q); k, kp = _d(k); v, vp = _d(v); dO, gp = _d(dO); doc, docp = _i(doc)
    qrows, qrp = _i(qrows); krows, krp = _i(krows)
    dq = np.zeros((len(qrows), d)); dk = np.zeros((len(krows), d)); dv = np.zeros((len(krows), d))
    P = ctypes.POINTER(ctypes.c_double)
    lib.oracle_attn_bwd_rows(L, d, float(scale), docp, qp, kp, vp, gp, len(qrows), qrp, dq.ctypes.data_as(P),
                             len(krows), krp, dk.ctypes.data_as(P), dv.ctypes.data_as(P))
    return dq, dk, dv


def live_pairs(doc) -> int:
    """Live (query, key) pairs of one sequence by enumerating the mask."""
    lib = _load()
    doc, docp = _i(doc)
    return int(lib.oracle_live_pairs(len(doc), docp))
