"""The C ABI loads, exports what include/ddattn.h declares, and rejects bad
arguments on the host before any launch (CPU only: no kernel runs here)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2405_13226_gb300 import build
    build.build()
    from paper_2405_13226_gb300 import ddattn
    return ddattn


def _declared():
    src = open(os.path.join(ROOT, "include", "ddattn.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dd_[a-z0-9_]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert "dd_attn_fwd" in names and "dd_attn_bwd" in names
    L = lib.lib()
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(lib.EXPORTS)


def test_status_strings(lib):
    for s in range(7):
        assert lib.status_string(s) and lib.status_string(s) != "unknown status"
    assert "timed out" in lib.status_string(lib.DD_ERR_DEVICE_TIMEOUT)


def test_workspace_sizes(lib):
    d = lib.make_desc(4, 256, 2, 64)
    assert lib.workspace_size(d, for_bwd=False) == 256
    n = lib.workspace_size(d, for_bwd=True)
    # status + 2 padded vectors + fp32 accumulator [B, H, L128, d]
    assert n == 256 + 2 * 4 * 2 * 256 * 4 + 4 * 2 * 256 * 64 * 4
    ragged = lib.make_desc(3, 200, 2, 128)
    assert lib.workspace_size(ragged, True) == 256 + 2 * 3 * 2 * 256 * 4 + 3 * 2 * 256 * 128 * 4
    assert lib.workspace_size(lib.make_desc(1, 128, 1, 96), True) == 0       # unsupported head dim
    # d = 80: accumulator in 3 chunks of 32 columns
    assert lib.workspace_size(lib.make_desc(3, 200, 2, 80), True) == 256 + 2 * 3 * 2 * 256 * 4 + 3 * 2 * 256 * 96 * 4
    assert lib.workspace_size(lib.make_desc(0, 128, 1, 64), True) == 0       # empty batch


def _fwd(lib, desc, ptrs, ws=0x100000, ws_bytes=1 << 20):
    q, k, v, o, lse = ptrs
    return lib.lib().dd_attn_fwd(ctypes.byref(desc), q, k, v, o, lse, ws, ws_bytes, None)


def test_host_validation_before_launch(lib):
    good = [0x10000, 0x20000, 0x30000, 0x40000, 0x50000]
    d = lib.make_desc(2, 256, 2, 128)
    assert _fwd(lib, d, [None] + good[1:]) == lib.DD_ERR_INVALID_ARG            # null q
    assert _fwd(lib, d, [0x10008] + good[1:]) == lib.DD_ERR_INVALID_ARG         # misaligned q
    assert _fwd(lib, d, good, ws=None) == lib.DD_ERR_WORKSPACE                  # no workspace
    assert _fwd(lib, d, good, ws=0x100010) == lib.DD_ERR_WORKSPACE              # workspace not 256-aligned
    assert _fwd(lib, d, good, ws_bytes=16) == lib.DD_ERR_WORKSPACE              # workspace too small
    assert _fwd(lib, lib.make_desc(2, 256, 2, 96), good) == lib.DD_ERR_UNSUPPORTED
    assert _fwd(lib, lib.make_desc(2, 0, 2, 128), good) == lib.DD_ERR_INVALID_ARG
    bad_scale = lib.make_desc(2, 256, 2, 128)
    bad_scale.scale = float("nan")
    assert _fwd(lib, bad_scale, good) == lib.DD_ERR_INVALID_ARG
    bad_off = lib.make_desc(2, 256, 2, 128)
    bad_off.cu_doc_offsets, bad_off.n_offsets = 0x60000, 1                      # fewer than 2 offsets
    assert _fwd(lib, bad_off, good) == lib.DD_ERR_INVALID_ARG
    L = lib.lib()
    assert L.dd_attn_bwd(ctypes.byref(d), *good[:3], good[3], None, good[4], *good[:3], 0x100000, 1 << 30,
                         None) == lib.DD_ERR_INVALID_ARG                         # null dO
    assert L.dd_attn_bwd(ctypes.byref(d), *good[:3], good[3], good[3], good[4], *good[:3], 0x100000, 256,
                         None) == lib.DD_ERR_WORKSPACE                           # bwd needs more than the status


def test_rope_descriptor_and_workspace(lib):
    """RoPE adds two copies of the (cos, sin) fp32 table to the backward workspace;
    a negative or non-finite base is rejected."""
    plain = lib.make_desc(3, 200, 2, 128)
    roped = lib.make_desc(3, 200, 2, 128, rope_base=1e4)
    tab = (224 * 64 * 8 + 255) // 256 * 256        # warp-blocked layout, positions rounded up to 32
    tab += (200 * 64 * 8 + 255) // 256 * 256       # row-major copy
    assert lib.workspace_size(roped, True) == lib.workspace_size(plain, True) + tab
    # the fused-RoPE forward keeps the row-major table in its workspace
    assert lib.workspace_size(roped, False) == 256 + (200 * 64 * 8 + 255) // 256 * 256
    assert lib.workspace_size(plain, False) == 256
    for bad in (-1.0, float("nan"), float("inf")):
        assert lib.workspace_size(lib.make_desc(3, 200, 2, 128, rope_base=bad), True) == 0


def test_rope_qk_host_validation(lib):
    L = lib.lib()
    p = [0x10000, 0x20000, 0x30000, 0x40000]
    call = lambda desc, ptrs: L.dd_rope_qk(ctypes.byref(desc), *ptrs, None)
    d = lib.make_desc(2, 256, 2, 128, rope_base=1e4)
    assert call(lib.make_desc(2, 256, 2, 128), p) == lib.DD_ERR_INVALID_ARG        # rope_base = 0
    assert call(d, [None] + p[1:]) == lib.DD_ERR_INVALID_ARG                      # null q
    assert call(d, p[:3] + [0x40004]) == lib.DD_ERR_INVALID_ARG                   # misaligned k_rot
    assert call(lib.make_desc(2, 256, 2, 96, rope_base=1e4), p) == lib.DD_ERR_UNSUPPORTED
    assert L.dd_rope_qk(None, *p, None) == lib.DD_ERR_INVALID_ARG


def test_noalloc_bad_descriptor_codes_match_bwd(lib):
    """dd_attn_bwd_noalloc returns the code dd_attn_bwd returns for the same bad
    descriptor, for every supported head dim (d = 80 included), before it looks
    at the scratch array or any device: nothing is launched."""
    L = lib.lib()
    p = [0x10000 * (i + 1) for i in range(9)]
    for d in (64, 80, 128):
        bad = []
        for B, Lq, scale, rope in ((0, 256, None, 0.0), (2, 0, None, 0.0), (2, 256, float("nan"), 0.0),
                                   (2, 256, None, -1.0)):
            desc = lib.make_desc(B, Lq, 2, d, scale, None, rope)
            bad.append(desc)
        neg_scale = lib.make_desc(2, 256, 2, d)
        neg_scale.scale = -0.5
        bad.append(neg_scale)
        for desc in bad:
            want = L.dd_attn_bwd(ctypes.byref(desc), *p, 0x100000, 1 << 30, None)
            got = L.dd_attn_bwd_noalloc(ctypes.byref(desc), *p, None, None)
            assert want == lib.DD_ERR_INVALID_ARG and got == want, (d, desc.B, desc.L, want, got)
    unsupported = lib.make_desc(2, 256, 2, 96)
    assert L.dd_attn_bwd_noalloc(ctypes.byref(unsupported), *p, None, None) == lib.DD_ERR_UNSUPPORTED
    assert L.dd_attn_bwd_noalloc(None, *p, None, None) == lib.DD_ERR_INVALID_ARG


def test_fwd_rope_host_validation(lib):
    """dd_attn_fwd_rope needs rope_base > 0, both rotated outputs, 16-byte alignment and a
    k_rot that does not overlap k (work items still read k while others write k_rot);
    q_rot may be q."""
    L = lib.lib()
    B, S, H, d = 2, 256, 2, 128
    n = B * S * H * d * 2
    q, k, v, o, lse, qr, kr = 0x1000000, 0x2000000, 0x3000000, 0x4000000, 0x5000000, 0x6000000, 0x7000000
    desc = lib.make_desc(B, S, H, d, rope_base=1e4)
    call = lambda dsc, ptrs, ws=None, wsb=0: L.dd_attn_fwd_rope(ctypes.byref(dsc), *ptrs, ws, wsb, None)
    good = [q, k, v, o, lse, qr, kr]
    assert call(lib.make_desc(B, S, H, d), good) == lib.DD_ERR_INVALID_ARG           # rope_base = 0
    assert call(desc, good[:5] + [None, kr]) == lib.DD_ERR_INVALID_ARG               # no q_rot
    assert call(desc, good[:6] + [None]) == lib.DD_ERR_INVALID_ARG                   # no k_rot
    assert call(desc, good[:6] + [kr + 8]) == lib.DD_ERR_INVALID_ARG                 # misaligned k_rot
    assert call(desc, good[:6] + [k]) == lib.DD_ERR_INVALID_ARG                      # k_rot is k
    assert call(desc, good[:6] + [k + n - 16]) == lib.DD_ERR_INVALID_ARG             # overlaps k's end
    assert call(desc, good[:6] + [k - n + 16]) == lib.DD_ERR_INVALID_ARG             # overlaps k's start
    # k_rot right after k, q_rot in place: the arguments pass, then the workspace is checked
    assert call(desc, good[:5] + [q, k + n]) == lib.DD_ERR_WORKSPACE
    assert call(desc, good, 0x100000, 256) == lib.DD_ERR_WORKSPACE                  # no room for the table
    assert call(lib.make_desc(B, S, H, 96, rope_base=1e4), good) == lib.DD_ERR_UNSUPPORTED
