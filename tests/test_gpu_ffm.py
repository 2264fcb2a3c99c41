"""GPU parity of the Fast and Forgetful Memory memoroid (forward and backward)
against the fp64 oracle, through the C ABI.

Bar: max |gpu - ref| / max |ref| <= 1e-4 over real components for every
output and gradient (fp32 arithmetic; lambda_ij is rounded to fp32 once);
episode-boundary behaviour bit-exact.  Cases cover every supported context
size c (1..16), partial 64-channel slabs, segmented tapes (the segment
fix-up pass), rows that continue an episode from S0 and the degenerate reset
patterns.
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


def run_gpu(t, S0=None, gSl=None, want_S0=False):
    m = _m()
    B, L, mm, c = t["B"], t["L"], t["m"], t["c"]
    ws = m.ffm_workspace(B, L, mm, c, "cuda")
    a, o, st, S0d = dev(t["alpha"]), dev(t["omega"]), dev(t["start"]), dev(S0)
    z, S_last = m.ffm_fwd(dev(t["x"]), a, o, st, S0d, ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    gx, ga, go, gS0 = m.ffm_bwd(a, o, st, z, dev(t["grad_z"]), dev(gSl), S0d, want_S0=want_S0, ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    torch.cuda.synchronize()
    out = dict(z=z, S_last=S_last, grad_x=gx, grad_alpha=ga, grad_omega=go, grad_S0=gS0)
    return {k: (None if v is None else v.cpu().numpy()) for k, v in out.items()}


def run_oracle(t, S0=None, gSl=None):
    z, S_last = oracle.ffm_fwd(t["alpha"], t["omega"], t["x"], t["start"], S0)
    gx, ga, go, gS0 = oracle.ffm_bwd(t["alpha"], t["omega"], t["start"], z, t["grad_z"], gSl, S0)
    return dict(z=z, S_last=S_last, grad_x=gx, grad_alpha=ga, grad_omega=go, grad_S0=gS0)


def check(t, with_S0=True, tol=TOL):
    S0 = t.get("S0") if with_S0 else None
    gSl = t["grad_S_last"]
    got = run_gpu(t, S0, gSl, want_S0=True)
    ref = run_oracle(t, S0, gSl)
    errs = {k: rel_err(got[k], ref[k]) for k in ref}
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, (bad, errs)
    return got, ref


SHAPES = [
    # B, L, m, c, mean, S0
    (2, 3000, 8, 4, 200.0, False),    # D = 32: one partial slab
    (1, 5000, 64, 4, 500.0, True),    # D = 256: four slabs
    (3, 2000, 12, 16, 100.0, True),   # D = 192, c = 16
    (2, 1500, 4, 1, 80.0, False),     # c = 1: two rows i per lane; D = 4
    (2, 777, 16, 2, 50.0, True),      # c = 2, ragged last tile
    (1, 40000, 32, 8, 500.0, False),  # long tape: segments and the fix-up pass
    (1, 30000, 8, 8, 3000.0, True),   # long episodes across segment edges
]


@pytest.mark.parametrize("B,L,m,c,mean,with_S0", SHAPES)
def test_ffm_parity_shapes(B, L, m, c, mean, with_S0):
    t = tapegen.ffm_tape(B, L, m, c, tapegen.seed_for(700 + B * L + m * c), mean=mean, with_S0=with_S0)
    if with_S0:
        t["start"][:, 0] = 0  # rows continue an episode from S0
    check(t, with_S0)


@pytest.mark.parametrize("mode", ["all", "none", "open"])
def test_ffm_degenerate_flags(mode):
    t = tapegen.ffm_tape(2, 20000, 16, 4, tapegen.seed_for(710), start_mode=mode, with_S0=True)
    check(t, with_S0=True)


@pytest.mark.parametrize("period", [7, 31, 32, 45])
def test_ffm_periodic_resets_every_row_offset(period):
    # begin flags every `period` steps at two phases: a flag falls on every position
    # of the scan warps' row blocks (31 steps forward, 12 backward), some blocks hold
    # none, and the tape ends inside a block; row 1 continues an episode from S0
    t = tapegen.ffm_tape(2, 1001, 16, 4, tapegen.seed_for(740 + period), start_mode="none", with_S0=True)
    t["start"][0, :] = 0
    t["start"][0, ::period] = 1
    t["start"][1, :] = 0
    t["start"][1, period // 2::period] = 1
    check(t, with_S0=True)


@pytest.mark.parametrize("L", [1, 2, 95, 96, 97, 185, 186, 187, 373])
def test_ffm_tiny_tapes(L):
    # around the forward's 186-step and the backward's 96-step tile edges
    t = tapegen.ffm_tape(2, L, 8, 2, tapegen.seed_for(720 + L), mean=3.0, with_S0=True)
    t["start"][1, 0] = 0
    check(t, with_S0=True)


def test_ffm_episode_isolation_bitwise():
    # changing one episode's input leaves every other episode's state bit-identical;
    # changing one episode's upstream gradient leaves grad_x elsewhere bit-identical
    m = _m()
    t = tapegen.ffm_tape(1, 60000, 32, 4, tapegen.seed_for(730), mean=400.0)
    heads = np.flatnonzero(t["start"][0])
    s, e = int(heads[40]), int(heads[41])
    base = run_gpu(t)
    t2 = dict(t)
    t2["x"] = t["x"].copy()
    t2["x"][0, s:e] += 1.0
    t2["grad_z"] = t["grad_z"].copy()
    t2["grad_z"][0, s:e] -= 0.5
    pert = run_gpu(t2)
    outside = np.ones(t["L"], dtype=bool)
    outside[s:e] = False
    assert np.array_equal(base["z"][0, outside], pert["z"][0, outside])
    assert np.array_equal(base["grad_x"][0, outside], pert["grad_x"][0, outside])
    assert not np.array_equal(base["z"][0, s:e], pert["z"][0, s:e])
    del m


def test_ffm_deterministic():
    t = tapegen.ffm_tape(2, 50000, 64, 4, tapegen.seed_for(731), mean=300.0)
    a = run_gpu(t)
    b = run_gpu(t)
    for k in ("z", "grad_x", "grad_alpha", "grad_omega"):
        assert np.array_equal(a[k], b[k]), k


def test_ffm_large_full_compare():
    # the measured shape (m = 64, c = 4, D = 256) on a 2^18-step tape, every output compared
    t = tapegen.ffm_tape(1, 1 << 18, 64, 4, tapegen.seed_for(732), mean=500.0, hi=10000)
    check(t, with_S0=False)


def test_ffm_bench_size_sampled_episodes():
    # the measured workload (L = 2^20): states and grad_x on three whole-episode
    # windows (each starts at a begin flag and ends right before one, so the
    # oracle on the window alone is exact there)
    t = tapegen.ffm_tape(1, 1 << 20, 64, 4, tapegen.seed_for(733), mean=500.0, hi=10000)
    got = run_gpu(t)
    heads = np.flatnonzero(t["start"][0])
    for pick in (5, len(heads) // 2, len(heads) - 20):
        s, e = int(heads[pick]), int(heads[pick + 10])
        z, _ = oracle.ffm_fwd(t["alpha"], t["omega"], t["x"][:, s:e], t["start"][:, s:e])
        gx, _, _, _ = oracle.ffm_bwd(t["alpha"], t["omega"], t["start"][:, s:e], z, t["grad_z"][:, s:e])
        assert rel_err(got["z"][:, s:e], z) <= TOL
        assert rel_err(got["grad_x"][:, s:e], gx) <= TOL
