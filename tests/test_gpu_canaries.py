"""Memory canaries for every output the kernels write: each output tensor sits
inside a larger buffer whose margins hold a sentinel, and after a call on a
ragged shape (tape lengths that end inside a tile, partial channel slabs) the
margins must be untouched.  This stands in for a memory checker, which is not
available on this pool.
"""
import numpy as np
import pytest

import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

PAD = 4096  # elements on each side


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


class Guarded:
    """A tensor of `shape` inside a buffer with PAD sentinel elements on each side."""

    def __init__(self, shape, dtype, sentinel):
        n = int(np.prod(shape)) if shape else 1
        self.n = n
        self.sentinel = sentinel
        self.buf = torch.full((n + 2 * PAD,), sentinel, dtype=dtype, device="cuda")
        self.t = self.buf[PAD:PAD + n].view(shape)

    def intact(self):
        s = self.sentinel
        return bool((self.buf[:PAD] == s).all()) and bool((self.buf[PAD + self.n:] == s).all())


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def test_linattn_outputs():
    m = _m()
    B, L, H, d = 2, 1000, 3, 64  # 1000 = 7 x 128 + 104
    t = tapegen.linattn_tape(B, L, H, d, d, tapegen.seed_for(900), mean=90.0, gamma_mode="step", with_S0=True)
    q, k, v = bits(t["q"]), bits(t["k"]), bits(t["v"])
    g, st, S0 = dev(t["gamma"]), dev(t["start"]), dev(t["S0"])
    y = Guarded((B, L, H, d), torch.float32, -77.5)
    Sl = Guarded((B, H, d, d), torch.float32, -77.5)
    dq, dk, dv = (Guarded((B, L, H, d), torch.float32, 55.25) for _ in range(3))
    dg = Guarded((B, L, H), torch.float32, 55.25)
    dS0 = Guarded((B, H, d, d), torch.float32, 55.25)
    ws = m.linattn_workspace(B, L, H, d, "cuda")
    m.memoroid_scan_linattn_fwd(q, k, v, m.MEMOROID_BF16, g, 1, st, S0, y.t, Sl.t, B, L, H, d, d, 64, ws)
    m.memoroid_scan_linattn_bwd(q, k, v, m.MEMOROID_BF16, g, 1, st, S0, dev(t["grad_y"]), dev(t["grad_S_last"]),
                                dq.t, dk.t, dv.t, dg.t, dS0.t, B, L, H, d, d, 64, ws)
    torch.cuda.synchronize()
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    for x in (y, Sl, dq, dk, dv, dg, dS0):
        assert x.intact()


def test_linattn_norm_outputs():
    m = _m()
    B, L, H, d = 1, 777, 2, 24
    t = tapegen.linattn_tape(B, L, H, d, d, tapegen.seed_for(901), mean=60.0, gamma_mode="head", scale=1.0,
                             normalize_k=False)
    q, k, v = bits(t["q"]), bits(t["k"]), bits(t["v"])
    g, st = dev(t["gamma"]), dev(t["start"])
    y = Guarded((B, L, H, d), torch.float32, 3.5)
    den = Guarded((B, L, H), torch.float32, 3.5)
    dq, dk, dv = (Guarded((B, L, H, d), torch.float32, -8.0) for _ in range(3))
    ws = m.workspace(m.memoroid_linattn_norm_workspace_bytes(B, L, H, d), "cuda")
    m.memoroid_linattn_norm_fwd(q, k, v, g, 0, st, None, None, y.t, den.t, None, None, B, L, H, d, ws)
    m.memoroid_linattn_norm_bwd(q, k, v, g, 0, st, None, None, y.t, den.t, dev(t["grad_y"]), None, None, dq.t, dk.t,
                                dv.t, None, None, None, B, L, H, d, ws)
    torch.cuda.synchronize()
    for x in (y, den, dq, dk, dv):
        assert x.intact()


def test_linattn_norm_fused_forward_outputs():
    # 64-channel heads with a 16-byte aligned y take the fused forward (TMA stores of y,
    # the normalizer written per row); the tape ends inside a tile
    m = _m()
    B, L, H, d = 2, 1111, 3, 64
    t = tapegen.linattn_tape(B, L, H, d, d, tapegen.seed_for(903), mean=70.0, gamma_mode="step", scale=1.0,
                             normalize_k=False, with_S0=True)
    q, k, v = bits(t["q"]), bits(t["k"]), bits(t["v"])
    g, st = dev(t["gamma"]), dev(t["start"])
    rng = np.random.default_rng(9)
    S0 = dev(t["S0"])
    z0 = dev(rng.uniform(0.5, 2.0, (B, H, d)).astype(np.float32))
    y = Guarded((B, L, H, d), torch.float32, 6.5)
    den = Guarded((B, L, H), torch.float32, 6.5)
    Sl = Guarded((B, H, d, d), torch.float32, 6.5)
    zl = Guarded((B, H, d), torch.float32, 6.5)
    assert y.t.data_ptr() % 16 == 0
    ws = m.workspace(m.memoroid_linattn_norm_workspace_bytes(B, L, H, d), "cuda")
    m.memoroid_linattn_norm_fwd(q, k, v, g, 1, st, S0, z0, y.t, den.t, Sl.t, zl.t, B, L, H, d, ws)
    torch.cuda.synchronize()
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    for x in (y, den, Sl, zl):
        assert x.intact()
    assert bool(torch.isfinite(y.t).all()) and bool((den.t > 0).all())


def test_returns_outputs():
    m = _m()
    rng = np.random.default_rng(3)
    B, L = 3, 5003  # not a multiple of 8: the scalar path; and a multiple of 8 below
    for LL in (L, 4096):
        r = rng.standard_normal((B, LL)).astype(np.float32)
        v = rng.standard_normal((B, LL)).astype(np.float32)
        start = tapegen.geometric_tape_starts(rng, LL, 40.0)[None].repeat(B, 0)
        G = Guarded((B, LL), torch.float32, 9.75)
        A = Guarded((B, LL), torch.float32, 9.75)
        ws = m.workspace(m.memoroid_returns_workspace_bytes(B, LL), "cuda")
        m.memoroid_discounted_return(dev(r), dev(start), 0.99, None, G.t, B, LL, ws)
        m.memoroid_gae(dev(r), dev(v), dev(start), 0.99, 0.95, None, A.t, B, LL, ws)
        torch.cuda.synchronize()
        assert G.intact() and A.intact()


def test_ffm_outputs():
    m = _m()
    B, L, mm, c = 2, 1111, 12, 4  # D = 48: a partial slab
    t = tapegen.ffm_tape(B, L, mm, c, tapegen.seed_for(902), mean=50.0, with_S0=True)
    al, om, st = dev(t["alpha"]), dev(t["omega"]), dev(t["start"])
    S0 = dev(t["S0"])
    z = Guarded((B, L, 2 * mm * c), torch.float32, 1.25)
    Sl = Guarded((B, mm, c), torch.complex64, complex(1.25, 2.5))
    gx = Guarded((B, L, mm), torch.float32, 1.25)
    ga = Guarded((mm,), torch.float32, 1.25)
    go = Guarded((c,), torch.float32, 1.25)
    gS0 = Guarded((B, mm, c), torch.complex64, complex(1.25, 2.5))
    ws = m.ffm_workspace(B, L, mm, c, "cuda")
    m.memoroid_ffm_fwd(dev(t["x"]), al, om, st, S0, z.t, Sl.t, B, L, mm, c, ws)
    m.memoroid_ffm_bwd(al, om, st, S0, z.t, dev(t["grad_z"]), dev(t["grad_S_last"]), gx.t, ga.t, go.t, gS0.t,
                       B, L, mm, c, ws)
    torch.cuda.synchronize()
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    for x in (z, Sl, gx, ga, go, gS0):
        assert x.intact()


def test_tbb_outputs():
    m = _m()
    rng = np.random.default_rng(4)
    N, B = 3000, 2345
    begin = np.flatnonzero(tapegen.geometric_tape_starts(rng, N, 20.0))
    draws = rng.integers(0, len(begin), size=B)
    start = Guarded((B,), torch.uint8, 7)
    src = Guarded((B,), torch.int64, -5)
    n_used = Guarded((1,), torch.int64, -5)
    ws = m.workspace(m.memoroid_tbb_workspace_bytes(len(draws)), "cuda")
    m.memoroid_tbb_sample(dev(begin), len(begin), N, dev(draws), len(draws), B, start.t, src.t, n_used.t, ws)
    rows = torch.randn((N, 6), device="cuda")  # 24-byte rows: the 4-byte path
    out = Guarded((B, 6), torch.float32, 0.5)
    m.memoroid_gather_rows(rows, N, 24, src.t, B, out.t, ws)
    torch.cuda.synchronize()
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    for x in (start, src, n_used, out):
        assert x.intact()
