"""Device-side failure path, exercised without faulting the GPU: a bounded wait
on an mbarrier that nothing arrives on must expire, record
DD_ERR_DEVICE_TIMEOUT in the workspace status word and leave the context
usable for the next attention call."""
import numpy as np
import pytest

from paper_2405_13226_gb300 import workloads as wl

from attn_cases import check_full, default_scale

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_and_reports_timeout():
    import torch
    from paper_2405_13226_gb300 import ddattn as dd
    desc = dd.make_desc(1, 128, 1, 64)
    ws = dd.new_workspace(desc, torch.device("cuda"), for_bwd=False)
    assert dd.poll_status(ws) == dd.DD_OK
    dd.selftest_wait_timeout(ws, limit_us=20000)
    assert dd.poll_status(ws) == dd.DD_ERR_DEVICE_TIMEOUT
    dd.clear_status(ws)
    assert dd.poll_status(ws) == dd.DD_OK
    # the context still runs attention correctly afterwards
    errs, _ = check_full(*wl.attn_inputs(2, 200, 2, 64, seed=9), default_scale(64))
    assert errs["o_rel"] < 5e-3


def test_selftest_argument_checks():
    import torch
    from paper_2405_13226_gb300 import ddattn as dd
    ws = torch.zeros(512, dtype=torch.uint8, device="cuda")
    L = dd.lib()
    s = torch.cuda.current_stream().cuda_stream
    import ctypes
    assert L.dd_selftest_wait_timeout(None, 100, ctypes.c_void_p(s)) == dd.DD_ERR_WORKSPACE
    assert L.dd_selftest_wait_timeout(ws.data_ptr(), 0, ctypes.c_void_p(s)) == dd.DD_ERR_INVALID_ARG
    assert L.dd_selftest_wait_timeout(ws.data_ptr(), 2000000, ctypes.c_void_p(s)) == dd.DD_ERR_INVALID_ARG
