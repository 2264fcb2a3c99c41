"""GPU parity of the diagonal resettable scan (forward and backward) against
the fp64 oracle, through the C ABI.

Bar: max |gpu - ref| / max |ref| <= 1e-4 over real components for every
output and gradient (fp32 arithmetic); episode-boundary behaviour bit-exact.
"""
import numpy as np
import pytest

import oracle
import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-4


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


def rel_err(got, ref):
    g = np.asarray(got)
    g = (g.view(np.float32) if g.dtype == np.complex64 else g).astype(np.float64)
    r = np.asarray(ref)
    r = r.view(np.float64) if np.iscomplexobj(r) else r.astype(np.float64)
    return float(np.max(np.abs(g - r))) / max(float(np.max(np.abs(r))), 1e-30)


def dev(a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_gpu(t, h0=None, g_last=None, want_h0=False):
    m = _m()
    lam, u, start = dev(t["lam"]), dev(t["u"]), dev(t["start"])
    B, L, D = t["u"].shape
    ws = m.diag_workspace(B, L, D, "cuda")
    h0d = dev(h0)
    h, h_last = m.diag_fwd(lam, u, start, h0d, ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    out = dict(h=h, h_last=h_last)
    if "grad_h" in t:
        gu, gl, gh0 = m.diag_bwd(lam, start, h, dev(t["grad_h"]), dev(g_last), h0d, want_h0=want_h0, ws=ws)
        assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
        out.update(grad_u=gu, grad_lambda=gl, grad_h0=gh0)
    torch.cuda.synchronize()
    return {k: (None if v is None else v.cpu().numpy()) for k, v in out.items()}


def run_oracle(t, h0=None, g_last=None):
    h, h_last = oracle.diag_fwd(t["lam"], t["u"], t["start"], h0)
    out = dict(h=h, h_last=h_last)
    if "grad_h" in t:
        gu, gl, gh0 = oracle.diag_bwd(t["lam"], t["start"], h, t["grad_h"], g_last, h0)
        out.update(grad_u=gu, grad_lambda=gl, grad_h0=gh0)
    return out


def check(t, h0=None, g_last=None, tol=TOL):
    got = run_gpu(t, h0, g_last, want_h0=True)
    ref = run_oracle(t, h0, g_last)
    errs = {k: rel_err(got[k], ref[k]) for k in ref if got.get(k) is not None}
    for k, e in errs.items():
        assert e <= tol, (k, e, errs)
    return got, ref, errs


# ---------------------------------------------------------------------------
# parity on shapes that span several tiles and a ragged tail
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("B,L,D", [(1, 4096, 64), (3, 1000, 192), (2, 777, 70), (1, 333, 2),
                                   (130, 517, 64)])  # the last: >= 128 chains, the unsegmented tiles
def test_parity_shapes(per_step, B, L, D):
    t = tapegen.diag_tape(B, L, D, seed=100 + L + D, mean=60.0, lambda_per_step=per_step, with_h0=True)
    t["start"][0, 0] = 0  # tape 0 continues an episode from h0
    check(t, h0=t["h0"], g_last=t["grad_h_last"])


def test_config1_full():
    t = tapegen.diag_config(1)
    got = run_gpu(t)
    ref, _ = oracle.diag_fwd(t["lam"], t["u"], t["start"])
    assert rel_err(got["h"], ref) <= TOL


@pytest.mark.parametrize("mode", ["all", "none", "open"])
def test_degenerate_flags(mode):
    # every step a begin flag; one episode; no begin flag at all (continues from h0)
    t = tapegen.diag_tape(2, 3000, 128, seed=7, start_mode=mode, with_h0=True)
    check(t, h0=t["h0"], g_last=t["grad_h_last"])


def test_long_single_episode():
    t = tapegen.diag_tape(1, 40000, 64, seed=8, start_mode="none")
    check(t, g_last=t["grad_h_last"])


def test_resets_on_tile_edges():
    L = 1024
    t = tapegen.diag_tape(1, L, 64, seed=9, start_mode="none")
    # around 16-, 32-, 64- and 128-step edges and the 96-step tiles of the scans
    for s in (1, 11, 12, 13, 15, 16, 17, 23, 24, 25, 63, 64, 65, 95, 96, 97, 127, 128, 129, 191, 192, 193, 255,
              256, 287, 288, 512, 1023):
        t["start"][0, s] = 1
    check(t, g_last=t["grad_h_last"])


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("period", [5, 13, 37, 50])
@pytest.mark.parametrize("L", [997, 1152])
def test_periodic_resets_every_row_offset(per_step, period, L):
    # begin flags every `period` steps, at two phases: across the scan warps' row
    # blocks (24 steps forward, 12 backward) a flag falls on every position of a
    # block, some blocks hold none, and the tape ends inside a block (997) or on a
    # tile edge (1152 = 12 x 96); tape 1 continues an episode from h0
    t = tapegen.diag_tape(2, L, 64, seed=12 + period + L, start_mode="none", lambda_per_step=per_step,
                          with_h0=True)
    t["start"][0, ::period] = 1
    t["start"][1, :] = 0
    t["start"][1, period // 2::period] = 1
    check(t, h0=t["h0"], g_last=t["grad_h_last"])


@pytest.mark.parametrize("L", [1, 2, 31, 33, 95, 96, 97, 191, 193])
def test_tiny_tapes(L):
    t = tapegen.diag_tape(2, L, 4, seed=10 + L, mean=3.0, with_h0=True)
    t["start"][1, 0] = 0
    check(t, h0=t["h0"], g_last=t["grad_h_last"])


def test_empty_tape_h_last_is_h0():
    m = _m()
    h0 = dev(tapegen.complex_normal(np.random.default_rng(0), (3, 8)))
    lam = dev(np.ones(8, np.complex64))
    u = torch.empty((3, 0, 8), dtype=torch.complex64, device="cuda")
    start = torch.empty((3, 0), dtype=torch.uint8, device="cuda")
    _, h_last = m.diag_fwd(lam, u, start, h0)
    torch.cuda.synchronize()
    assert torch.equal(h_last, h0)


# ---------------------------------------------------------------------------
# exact episode-boundary behaviour
# ---------------------------------------------------------------------------

def _tape_for_boundaries():
    t = tapegen.diag_tape(1, 5000, 128, seed=11, mean=150.0)
    return t


def test_start_steps_equal_u_bitwise():
    t = _tape_for_boundaries()
    got = run_gpu(t)
    s = t["start"][0].astype(bool)
    np.testing.assert_array_equal(got["h"][0, s], t["u"][0, s])


def test_perturbation_confined_to_episode():
    t = _tape_for_boundaries()
    base = run_gpu(t)
    eps = tapegen.episode_bounds(t["start"][0])
    s, e = eps[len(eps) // 2]
    t2 = dict(t)
    t2["u"] = t["u"].copy()
    t2["u"][0, s:e] *= np.complex64(1.5 - 0.25j)
    t2["grad_h"] = t["grad_h"].copy()
    t2["grad_h"][0, s:e] += np.complex64(3.0)
    pert = run_gpu(t2)
    outside = np.ones(t["u"].shape[1], bool)
    outside[s:e] = False
    np.testing.assert_array_equal(pert["h"][0, outside], base["h"][0, outside])
    np.testing.assert_array_equal(pert["grad_u"][0, outside], base["grad_u"][0, outside])
    assert not np.array_equal(pert["h"][0, s:e], base["h"][0, s:e])


def test_nan_confined_to_episode():
    t = _tape_for_boundaries()
    eps = tapegen.episode_bounds(t["start"][0])
    s, e = eps[len(eps) // 3]
    t2 = dict(t)
    t2["u"] = t["u"].copy()
    t2["u"][0, s + (e - s) // 2] = np.complex64(np.nan)
    t2["grad_h"] = t["grad_h"].copy()
    t2["grad_h"][0, s + (e - s) // 2] = np.complex64(np.inf)
    got = run_gpu(t2)
    base = run_gpu(t)
    outside = np.ones(t["u"].shape[1], bool)
    outside[s:e] = False
    np.testing.assert_array_equal(got["h"][0, outside], base["h"][0, outside])
    np.testing.assert_array_equal(got["grad_u"][0, outside], base["grad_u"][0, outside])
    assert np.isfinite(got["h"][0, outside]).all()


def test_split_resume():
    t = tapegen.diag_tape(2, 6000, 64, seed=12, mean=400.0)
    full = run_gpu(t)
    t1 = {k: (v[:, :2500] if k in ("u", "start", "grad_h") else v) for k, v in t.items()}
    t2 = {k: (v[:, 2500:] if k in ("u", "start", "grad_h") else v) for k, v in t.items()}
    t2["start"] = t2["start"].copy()
    t2["start"][:, 0] = 0
    t_full = dict(t)
    t_full["start"] = t["start"].copy()
    t_full["start"][:, 2500] = 0
    full = run_gpu(t_full)
    a = run_gpu({k: v for k, v in t1.items() if k != "grad_h"})
    b = run_gpu({k: v for k, v in t2.items() if k != "grad_h"}, h0=a["h_last"])
    joined = np.concatenate([a["h"], b["h"]], axis=1)
    assert rel_err(joined, full["h"].astype(np.complex128)) <= 1e-5


def test_deterministic_grad_lambda():
    t = tapegen.diag_tape(2, 20000, 128, seed=13, mean=300.0)
    a = run_gpu(t)
    b = run_gpu(t)
    np.testing.assert_array_equal(a["grad_lambda"], b["grad_lambda"])
    np.testing.assert_array_equal(a["grad_u"], b["grad_u"])


def test_autograd_wrapper_matches_oracle():
    m = _m()
    t = tapegen.diag_tape(1, 900, 64, seed=14, mean=80.0, with_h0=True)
    t["start"][0, 0] = 0
    lam = dev(t["lam"]).requires_grad_(True)
    u = dev(t["u"]).requires_grad_(True)
    h0 = dev(t["h0"]).requires_grad_(True)
    h = m.DiagScan.apply(lam, u, dev(t["start"]), h0)
    g = dev(t["grad_h"])
    (torch.conj(g) * h).real.sum().backward()
    rh, _ = oracle.diag_fwd(t["lam"], t["u"], t["start"], t["h0"])
    rgu, rgl, rgh0 = oracle.diag_bwd(t["lam"], t["start"], rh, t["grad_h"], None, t["h0"])
    assert rel_err(h.detach().cpu().numpy(), rh) <= TOL
    assert rel_err(u.grad.cpu().numpy(), rgu) <= TOL
    assert rel_err(lam.grad.cpu().numpy(), rgl) <= TOL
    assert rel_err(h0.grad.cpu().numpy(), rgh0) <= TOL


# ---------------------------------------------------------------------------
# full-size workloads (the benchmark's launch configuration)
# ---------------------------------------------------------------------------

def _sample_episodes(start_row, rng, n=64):
    eps = tapegen.episode_bounds(start_row)
    idx = set(rng.choice(len(eps), size=min(n, len(eps)), replace=False).tolist())
    idx |= {0, len(eps) - 1, int(np.argmax([e - s for s, e in eps]))}
    return [eps[i] for i in sorted(idx)]


@pytest.mark.parametrize("cfg", [2, 4])
def test_full_config_sampled(cfg):
    t = tapegen.diag_config(cfg)
    got = run_gpu(t)
    rng = np.random.default_rng(cfg)
    B = t["B"]
    rows = [0, B - 1] if B > 1 else [0]
    for b in rows:
        for s, e in _sample_episodes(t["start"][b], rng, 64 if B == 1 else 16):
            sub = dict(lam=t["lam"], u=t["u"][b:b + 1, s:e], start=t["start"][b:b + 1, s:e],
                       grad_h=t["grad_h"][b:b + 1, s:e])
            rh, _ = oracle.diag_fwd(sub["lam"], sub["u"], sub["start"])
            rgu, _, _ = oracle.diag_bwd(sub["lam"], sub["start"], rh, sub["grad_h"])
            scale_h = np.max(np.abs(rh.view(np.float64)))
            scale_g = np.max(np.abs(rgu.view(np.float64)))
            assert np.max(np.abs(got["h"][b, s:e].astype(np.complex128) - rh).view(np.float64)) <= TOL * scale_h
            assert np.max(np.abs(got["grad_u"][b, s:e].astype(np.complex128) - rgu).view(np.float64)) <= TOL * scale_g
    # grad_lambda sums over the whole tape: full oracle run (fp64)
    rh, _ = oracle.diag_fwd(t["lam"], t["u"], t["start"])
    _, rgl, _ = oracle.diag_bwd(t["lam"], t["start"], rh, t["grad_h"])
    assert rel_err(got["grad_lambda"], rgl) <= TOL


# ---------------------------------------------------------------------------
# bounded waits: a withheld look-back flag yields MEMOROID_ERR_TIMEOUT
# ---------------------------------------------------------------------------

def test_lookback_timeout_reported():
    m = _m()
    t = tapegen.diag_tape(1, 4096, 64, seed=15, start_mode="none")
    lam, u, start = dev(t["lam"]), dev(t["u"]), dev(t["start"])
    ws = m.diag_workspace(1, 4096, 64, "cuda")
    h = torch.empty_like(u)
    try:
        m.memoroid_debug_set_wait_limit_ns(20_000_000)  # 20 ms
        m.memoroid_debug_withhold_tile(3)
        m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, 1, 4096, 64, ws)
        assert m.memoroid_get_device_error(ws) == m.MEMOROID_ERR_TIMEOUT
    finally:
        m.memoroid_debug_withhold_tile(-1)
        m.memoroid_debug_set_wait_limit_ns(0)
    m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, 1, 4096, 64, ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    ref, _ = oracle.diag_fwd(t["lam"], t["u"], t["start"])
    assert rel_err(h.cpu().numpy(), ref) <= TOL


@pytest.mark.parametrize("fill", [0xFF, 0x00, 0xA5])
def test_garbage_workspace(fill):
    # a fresh workspace full of leftover bytes: the look-back summaries' region
    # is zeroed on the workspace's first use, so no old word is taken for a
    # summary of this launch; forward and backward against the oracle, twice
    m = _m()
    B, L, D = 2, 6000, 128
    t = tapegen.diag_tape(B, L, D, seed=tapegen.seed_for(77), mean=150.0)
    lam, u, start, gh = dev(t["lam"]), dev(t["u"]), dev(t["start"]), dev(t["grad_h"])
    ws = torch.full((m.memoroid_scan_diag_workspace_bytes(B, L, D),), fill, dtype=torch.uint8, device="cuda")
    ref_h, _ = oracle.diag_fwd(t["lam"], t["u"], t["start"])
    ref_gu, ref_gl, _ = oracle.diag_bwd(t["lam"], t["start"], ref_h, t["grad_h"])
    for _ in range(2):
        h = torch.empty_like(u)
        m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, B, L, D, ws)
        gu, gl = torch.empty_like(u), torch.empty_like(lam)
        m.memoroid_scan_diag_bwd(lam, 0, start, None, h, gh, None, gu, gl, None, B, L, D, ws)
        assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
        assert rel_err(h.cpu().numpy(), ref_h) <= TOL
        assert rel_err(gu.cpu().numpy(), ref_gu) <= TOL
        assert rel_err(gl.cpu().numpy(), ref_gl) <= TOL


def test_guard_bands_untouched():
    m = _m()
    B, L, D = 2, 1000, 70
    t = tapegen.diag_tape(B, L, D, seed=16, mean=90.0)
    n = B * L * D
    pad = 4096
    sentinel = np.complex64(complex(1234.5, -987.25))
    buf = torch.full((n + 2 * pad,), complex(sentinel), dtype=torch.complex64, device="cuda")
    h = buf[pad:pad + n].view(B, L, D)
    gbuf = torch.full((n + 2 * pad,), complex(sentinel), dtype=torch.complex64, device="cuda")
    gu = gbuf[pad:pad + n].view(B, L, D)
    lam, u, start = dev(t["lam"]), dev(t["u"]), dev(t["start"])
    ws = m.diag_workspace(B, L, D, "cuda")
    m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, B, L, D, ws)
    m.memoroid_scan_diag_bwd(lam, 0, start, None, h, dev(t["grad_h"]), None, gu, None, None, B, L, D, ws)
    torch.cuda.synchronize()
    for b in (buf, gbuf):
        assert bool((b[:pad] == complex(sentinel)).all()) and bool((b[pad + n:] == complex(sentinel)).all())


# ---------------------------------------------------------------------------
# episode index list <-> begin flags
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("L", [1, 9, 4096, 100_003, 1 << 20])
def test_tape_index_round_trip(L):
    m = _m()
    rng = np.random.default_rng(L)
    start = (rng.random(L) < 0.01).astype(np.uint8)
    start[0] = 1
    offs_ref = oracle.offsets_from_starts(start)
    offs, count = m.offsets_from_starts(dev(start))
    torch.cuda.synchronize()
    n = int(count.item())
    np.testing.assert_array_equal(offs[:n].cpu().numpy(), offs_ref)
    back = m.starts_from_offsets(dev(offs_ref), L)
    np.testing.assert_array_equal(back.cpu().numpy(), oracle.starts_from_offsets(offs_ref, L))
