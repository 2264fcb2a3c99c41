"""memoroid_scan_diag_fwd_static: the forward scan for callers that cannot
provide device scratch memory.  It must give the same result as the regular
entry point (which takes a caller-allocated workspace) call after call, even
though every call reuses the same library-owned scratch array, and it must
refuse shapes that do not fit that array.

This file is named so that pytest collects it last.
"""
import numpy as np
import pytest

import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-4


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


def _rel(a, b):
    a = a.view(torch.float32).double()
    b = b.view(torch.float32).double()
    return float((a - b).abs().max() / b.abs().max().clamp_min(1e-30))


def _run_both(m, B, L, D, seed, per_step):
    t = tapegen.diag_tape(B, L, D, seed=seed, mean=70.0, lambda_per_step=per_step, with_h0=True)
    t["start"][0, 0] = 0  # the first tape continues an episode from h0
    dev = torch.device("cuda")
    lam = torch.from_numpy(t["lam"]).to(dev)
    u = torch.from_numpy(t["u"]).to(dev)
    start = torch.from_numpy(t["start"]).to(dev)
    h0 = torch.from_numpy(t["h0"]).to(dev)

    ws = m.diag_workspace(B, L, D, dev)
    h_ref = torch.empty_like(u)
    last_ref = torch.empty((B, D), dtype=u.dtype, device=dev)
    m.memoroid_scan_diag_fwd(lam, int(per_step), u, start, h0, h_ref, last_ref, B, L, D, ws)

    h = torch.full_like(u, float("nan"))
    last = torch.full((B, D), float("nan"), dtype=u.dtype, device=dev)
    m.memoroid_scan_diag_fwd_static(lam, int(per_step), u, start, h0, h, last, B, L, D)
    torch.cuda.synchronize()
    return h, last, h_ref, last_ref


def test_static_workspace_matches_regular_entry_point_twice():
    m = _m()
    # two calls in a row, different shapes and lambda modes: the second call
    # finds the first call's leftovers in the shared scratch array
    for B, L, D, seed, per_step in ((2, 5000, 192, 71, False), (3, 2500, 70, 72, True)):
        h, last, h_ref, last_ref = _run_both(m, B, L, D, seed, per_step)
        assert _rel(h, h_ref) <= TOL
        assert _rel(last, last_ref) <= TOL


def test_static_workspace_rejects_oversized_shapes():
    m = _m()
    B, L, D = 1, 1 << 20, 256
    capacity = 16 << 20  # MEMOROID_STATIC_WORKSPACE_BYTES in include/memoroid.h
    assert m.memoroid_scan_diag_workspace_bytes(B, L, D) > capacity
    dev = torch.device("cuda")
    small = torch.zeros(16, dtype=torch.complex64, device=dev)
    flags = torch.zeros(16, dtype=torch.uint8, device=dev)
    # rejected on the host from the shape alone, before any pointer is used
    with pytest.raises(m.MemoroidError) as e:
        m.memoroid_scan_diag_fwd_static(small, 0, small, flags, None, small, None, B, L, D)
    assert e.value.status == m.MEMOROID_ERR_WORKSPACE


def test_static_workspace_reports_a_timed_out_wait_then_recovers():
    # a look-back wait that runs out is recorded in the library-owned array's
    # header; memoroid_get_static_device_error reads it (the caller never sees
    # the array), and the next call on the same array is correct again
    m = _m()
    B, L, D = 1, 4096, 64
    t = tapegen.diag_tape(B, L, D, seed=73, start_mode="none")
    dev = torch.device("cuda")
    lam = torch.from_numpy(t["lam"]).to(dev)
    u = torch.from_numpy(t["u"]).to(dev)
    start = torch.from_numpy(t["start"]).to(dev)
    h = torch.empty_like(u)
    try:
        m.memoroid_debug_set_wait_limit_ns(20_000_000)  # 20 ms
        m.memoroid_debug_withhold_tile(3)
        m.memoroid_scan_diag_fwd_static(lam, 0, u, start, None, h, None, B, L, D)
        assert m.memoroid_get_static_device_error() == m.MEMOROID_ERR_TIMEOUT
    finally:
        m.memoroid_debug_withhold_tile(-1)
        m.memoroid_debug_set_wait_limit_ns(0)
    m.memoroid_scan_diag_fwd_static(lam, 0, u, start, None, h, None, B, L, D)
    assert m.memoroid_get_static_device_error() == m.MEMOROID_OK
    ws = m.diag_workspace(B, L, D, dev)
    h_ref = torch.empty_like(u)
    m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h_ref, None, B, L, D, ws)
    torch.cuda.synchronize()
    assert _rel(h, h_ref) <= TOL
