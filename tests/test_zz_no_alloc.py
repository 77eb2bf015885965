"""dd_attn_bwd_noalloc: the backward for callers that cannot allocate device
memory (a runtime whose own allocator owns all device memory, or a step loop
under a fixed memory budget). It runs the same kernels on a library-owned
scratch array instead of a caller workspace, so its dq, dk, dv must match
dd_attn_bwd's within the parity tolerance, on consecutive calls that reuse
the array. This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest

from paper_2405_13226_gb300 import workloads as wl

from attn_cases import TOL_GRAD_REL, default_scale, oracle_full, rel_l2, to_device, to_f64

pytestmark = pytest.mark.gpu


def _noalloc(dd, desc, q, k, v, o, g, lse, dq, dk, dv, status, stream):
    return dd.lib().dd_attn_bwd_noalloc(ctypes.byref(desc), q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                        g.data_ptr(), lse.data_ptr(), dq.data_ptr(), dk.data_ptr(), dv.data_ptr(),
                                        status.data_ptr(), ctypes.c_void_p(stream.cuda_stream))


# (B, L, H, d, document mask, RoPE base): the d = 64 kernels; the walking d = 128 kernel with
# documents; d = 80 with RoPE (its (cos, sin) tables live inside the scratch array); the
# one-CTA-per-key-tile d = 128 kernel (L > 2048).
CASES = [(4, 256, 2, 64, False, 0.0), (2, 1000, 4, 128, True, 0.0), (2, 640, 2, 80, False, 1e4),
         (1, 4096, 2, 128, False, 0.0)]


@pytest.mark.parametrize("B,L,H,d,doc_mask,rope_base", CASES)
def test_noalloc_matches_workspace_entry_point(B, L, H, d, doc_mask, rope_base):
    """Two calls in a row against dd_attn_bwd (same kernels, caller workspace) and
    against the fp64 oracle, within the parity tolerance."""
    import torch
    from paper_2405_13226_gb300 import ddattn as dd
    scale = default_scale(d)
    qb, kb, vb, gb = wl.attn_inputs(B, L, H, d, seed=11)
    q, k, v, g = (to_device(x) for x in (qb, kb, vb, gb))
    off, off_np = None, None
    if doc_mask:
        off_np = wl.concat_and_chunk_offsets(4, n_chunks=B, chunk=L)
        off = torch.from_numpy(off_np).cuda()
    if rope_base:
        q, k = dd.rope_qk(q, k, rope_base)
    o, lse = dd.fwd(q, k, v, scale, off)
    ref = dd.bwd(q, k, v, o, g, lse, scale, off, rope_base=rope_base)
    _, _, odq, odk, odv = oracle_full(qb, kb, vb, gb, scale, off_np, rope_base)
    desc = dd.make_desc(B, L, H, d, scale, off, rope_base)
    assert dd.workspace_size(desc, True) <= dd.NOALLOC_SCRATCH_BYTES
    stream = torch.cuda.current_stream()
    for call in range(2):   # the second call reuses the scratch array left by the first
        dq, dk, dv = (torch.full_like(q, float("nan")) for _ in range(3))
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        st = _noalloc(dd, desc, q, k, v, o, g, lse, dq, dk, dv, status, stream)
        assert st == dd.DD_OK, dd.status_string(st)
        torch.cuda.synchronize()
        assert int(status.item()) == 0, "device status of call %d" % call
        for name, got, want, orc in (("dq", dq, ref[0], odq), ("dk", dk, ref[1], odk), ("dv", dv, ref[2], odv)):
            assert np.isfinite(to_f64(got)).all(), (call, name)
            err = rel_l2(to_f64(got), to_f64(want))
            assert err <= TOL_GRAD_REL, (call, name, "vs dd_attn_bwd", err)
            err = rel_l2(to_f64(got), orc)
            assert err <= TOL_GRAD_REL, (call, name, "vs oracle", err)


def test_noalloc_rejects_sizes_beyond_scratch():
    """A backward whose workspace would exceed the fixed scratch array is
    refused on the host with DD_ERR_WORKSPACE and nothing is launched."""
    import torch
    from paper_2405_13226_gb300 import ddattn as dd
    desc = dd.make_desc(8, 8192, 16, 128)
    assert dd.workspace_size(desc, True) > dd.NOALLOC_SCRATCH_BYTES
    x = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = _noalloc(dd, desc, x, x, x, x, x, x, x, x, x, status, torch.cuda.current_stream())
    assert st == dd.DD_ERR_WORKSPACE
