"""GPU parity of the decayed linear-attention memoroid (forward and backward)
against the fp64 oracle, through the C ABI.

Bar: max |gpu - ref| / max |ref| <= 2e-2 for every output (bf16 q, k, v;
the oracle takes the same bf16 values upcast, so only the arithmetic counts).
Cases span several 128-step tiles with a ragged tail, every segment layout
(one tile per segment up to one segment per tape), both decay modes, S0, and
the degenerate reset patterns.
"""
import numpy as np
import pytest

import oracle
import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 2e-2


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


def rel_err(got, ref):
    g = np.asarray(got, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(g - r))) / max(float(np.max(np.abs(r))), 1e-30)


def dev(a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()


def bits_dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def run_gpu_fwd(t, chunk=64, S0=None, ws=None):
    m = _m()
    q, k, v = bits_dev(t["q"]), bits_dev(t["k"]), bits_dev(t["v"])
    gamma, start = dev(t["gamma"]), dev(t["start"])
    B, L, H, d = t["q"].shape
    if ws is None:
        ws = m.linattn_workspace(B, L, H, d, "cuda", chunk)
    y, S_last = m.linattn_fwd(q, k, v, gamma, start, dev(S0), chunk=chunk, ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    torch.cuda.synchronize()
    return y.cpu().numpy(), S_last.cpu().numpy()


def run_oracle_fwd(t, S0=None):
    f = oracle.bf16_bits_to_f64
    return oracle.linattn_fwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"], S0)


CASES = [
    # B, L, H, d, gamma_mode, mean, with_S0
    (2, 1000, 3, 64, "head", 60.0, False),
    (2, 1000, 3, 128, "step", 60.0, True),
    (1, 3000, 2, 64, "step", 400.0, True),
    (1, 3000, 1, 128, "head", 2000.0, False),
    (3, 777, 2, 128, "head", 30.0, True),
]


@pytest.mark.parametrize("B,L,H,d,gm,mean,with_S0", CASES)
def test_fwd_matches_oracle(B, L, H, d, gm, mean, with_S0):
    t = tapegen.linattn_tape(B, L, H, d, d, seed=tapegen.seed_for(100 + L + d + H), mean=mean, gamma_mode=gm,
                             gammas=(0.95, 0.99, 1.0), with_grad=False, with_S0=with_S0)
    S0 = t.get("S0")
    if S0 is not None:
        t["start"][:, 0] = 0  # the first episode continues from S0
    y, S_last = run_gpu_fwd(t, S0=S0)
    y_ref, S_ref = run_oracle_fwd(t, S0)
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL


@pytest.mark.parametrize("mode", ["all", "none", "open"])
@pytest.mark.parametrize("d", [64, 128])
def test_fwd_degenerate_resets(mode, d):
    # every step a start / one episode over the whole tape / no start at all
    t = tapegen.linattn_tape(2, 700, 2, d, d, seed=tapegen.seed_for(7 + d), gamma_mode="step",
                             with_grad=False, with_S0=True, start_mode=mode)
    S0 = t["S0"]
    y, S_last = run_gpu_fwd(t, S0=S0)
    y_ref, S_ref = run_oracle_fwd(t, S0)
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL


@pytest.mark.parametrize("L", [1, 5, 127, 128, 129, 256, 300])
def test_fwd_short_tapes(L):
    t = tapegen.linattn_tape(1, L, 2, 64, 64, seed=tapegen.seed_for(900 + L), mean=40.0, gamma_mode="step",
                             with_grad=False, with_S0=True)
    t["start"][:, 0] = 0
    y, S_last = run_gpu_fwd(t, S0=t["S0"])
    y_ref, S_ref = run_oracle_fwd(t, t["S0"])
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL


def test_fwd_chunk_128_same_function():
    t = tapegen.linattn_tape(1, 900, 2, 64, 64, seed=tapegen.seed_for(55), mean=100.0, with_grad=False)
    y64, _ = run_gpu_fwd(t, chunk=64)
    y128, _ = run_gpu_fwd(t, chunk=128)
    assert np.array_equal(y64, y128)


def test_fwd_one_segment_per_tape():
    # B * H >= 152 CTAs: one segment per (tape, head), no carry between segments
    t = tapegen.linattn_tape(4, 600, 40, 64, 64, seed=tapegen.seed_for(56), mean=150.0, gamma_mode="step",
                             with_grad=False)
    y, S_last = run_gpu_fwd(t)
    y_ref, S_ref = run_oracle_fwd(t)
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL


def _long_episode_tape(d, gamma_lo, gamma_hi, seed, starts=()):
    # B = 1, L = 2^16, 2 heads: 512 tiles cut into many segments, begin flags
    # only at the given steps (none: one episode continuing from S0), a
    # per-step gamma drawn from [gamma_lo, gamma_hi]
    L = 1 << 16
    t = tapegen.linattn_tape(1, L, 2, d, d, seed=seed, gamma_mode="step", with_grad=True, with_S0=True,
                             start_mode="open")
    rng = np.random.default_rng(seed + 1)
    t["gamma"] = rng.uniform(gamma_lo, gamma_hi, size=(1, L, 2)).astype(np.float32)
    for s_ in starts:
        t["start"][0, s_] = 1
    return t


@pytest.mark.parametrize("d,gamma_lo,gamma_hi,starts", [
    (64, 0.9995, 1.0, ()),              # one episode: the state crosses every segment boundary
    (128, 0.9999, 1.0, (40000,)),       # two episodes, the second from the middle of a segment
    (64, 0.5, 0.6, ()),                 # strong decay: the segment summaries skip underflowing tiles
    (128, 1.0, 1.0, (777, 30001)),      # gamma = 1, flags in two segments only
])
def test_reset_sparse_long_tape(d, gamma_lo, gamma_hi, starts):
    # the inter-segment carry: a tape with few or no begin flags runs on as
    # many segments (CTAs) as any other, each starting from the state that
    # the carry brings in; forward and backward against the oracle
    t = _long_episode_tape(d, gamma_lo, gamma_hi, tapegen.seed_for(70 + d + len(starts)), starts)
    y, S_last = run_gpu_fwd(t, S0=t["S0"])
    y_ref, S_ref = run_oracle_fwd(t, t["S0"])
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL
    check_bwd(t, t["S0"], t["grad_S_last"])


def test_fwd_episode_isolation_bitwise():
    # changing q/k/v inside one episode leaves every other episode's outputs unchanged, bit for bit
    t = tapegen.linattn_tape(1, 2000, 2, 64, 64, seed=tapegen.seed_for(57), mean=200.0, with_grad=False)
    y0, _ = run_gpu_fwd(t)
    starts = np.flatnonzero(t["start"][0])
    s, e = int(starts[3]), int(starts[4])
    t2 = dict(t)
    for key in ("q", "k", "v"):
        a = t[key].copy()
        a[0, s:e] ^= np.uint16(0x0040)
        t2[key] = a
    y1, _ = run_gpu_fwd(t2)
    outside = np.ones(2000, dtype=bool)
    outside[s:e] = False
    assert np.array_equal(y0[0, outside], y1[0, outside])
    assert not np.array_equal(y0[0, s:e], y1[0, s:e])


@pytest.mark.parametrize("d", [64, 128])
def test_fwd_nonfinite_q_k_confined_to_their_episode(d):
    # a NaN in q (one episode) and in k (another, ending in the middle of a tile) stays
    # in its episode: every other episode's outputs are bit for bit those of the tape
    # without them (the masks, the rows scaled into the state and the inter-tile term
    # are selects, not products).  v is not covered: the tile-wide contractions
    # multiply it by the zero weights of other episodes' rows.
    t = tapegen.linattn_tape(1, 6000, 2, d, d, seed=tapegen.seed_for(59), mean=300.0, with_grad=False)
    y0, s0 = run_gpu_fwd(t)
    starts = np.flatnonzero(t["start"][0])
    spans = [(int(starts[i]), int(starts[i + 1])) for i in (4, 9)]
    t2 = dict(t)
    nan = np.uint16(0x7FC0)
    for key, (s, e) in zip(("q", "k"), spans):
        a = t[key].copy()
        a[0, s:e, 0, 3] = nan
        t2[key] = a
    y1, s1 = run_gpu_fwd(t2)
    outside = np.ones(6000, dtype=bool)
    for s, e in spans:
        outside[s:e] = False
        assert np.isnan(y1[0, s:e, 0]).any()
    assert np.array_equal(y0[0, outside], y1[0, outside])
    assert np.array_equal(y0[0, :, 1], y1[0, :, 1])  # the other head
    assert np.array_equal(s0, s1)


def test_fwd_deterministic():
    t = tapegen.linattn_tape(1, 5000, 2, 128, 128, seed=tapegen.seed_for(58), mean=500.0, gamma_mode="step",
                             with_grad=False)
    a, sa = run_gpu_fwd(t)
    b, sb = run_gpu_fwd(t)
    assert np.array_equal(a, b) and np.array_equal(sa, sb)


def test_fwd_config3_full():
    # the full L = 2^18, 4-head, d = 64 tape with per-head gamma: every output
    # against the oracle run over the whole tape
    t = tapegen.linattn_config(3)
    y, S_last = run_gpu_fwd(t, chunk=t["chunk"])
    y_ref, S_ref = run_oracle_fwd(t)
    assert rel_err(y, y_ref) <= TOL
    assert rel_err(S_last, S_ref) <= TOL


# ---------------------------------------------------------------------------
# backward
# ---------------------------------------------------------------------------

def run_gpu_bwd(t, S0=None, dS_last=None, chunk=64):
    m = _m()
    q, k, v = bits_dev(t["q"]), bits_dev(t["k"]), bits_dev(t["v"])
    gamma, start = dev(t["gamma"]), dev(t["start"])
    B, L, H, d = t["q"].shape
    ws = m.linattn_workspace(B, L, H, d, "cuda", chunk)
    out = m.linattn_bwd(q, k, v, gamma, start, dev(t["grad_y"]), dev(dS_last), dev(S0), want_S0=True, chunk=chunk,
                        ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    torch.cuda.synchronize()
    return [o.cpu().numpy() for o in out]


def run_oracle_bwd(t, S0=None, dS_last=None):
    f = oracle.bf16_bits_to_f64
    return oracle.linattn_bwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"], t["grad_y"], dS_last, S0)


def check_bwd(t, S0=None, dS_last=None):
    got = run_gpu_bwd(t, S0, dS_last)
    ref = run_oracle_bwd(t, S0, dS_last)
    errs = {name: rel_err(g, r) for name, g, r in zip(("dq", "dk", "dv", "dgamma", "dS0"), got, ref)}
    assert all(e <= TOL for e in errs.values()), errs
    return errs


BWD_CASES = [
    # B, L, H, d, gamma_mode, mean, with_S0, with_dS_last
    (2, 1000, 3, 64, "head", 60.0, False, False),
    (2, 1000, 3, 128, "step", 60.0, True, True),
    (1, 3000, 2, 64, "step", 400.0, True, True),
    (1, 3000, 1, 128, "head", 2000.0, False, True),
    (3, 777, 2, 128, "head", 30.0, True, False),
]


@pytest.mark.parametrize("B,L,H,d,gm,mean,with_S0,with_dS", BWD_CASES)
def test_bwd_matches_oracle(B, L, H, d, gm, mean, with_S0, with_dS):
    t = tapegen.linattn_tape(B, L, H, d, d, seed=tapegen.seed_for(300 + L + d + H), mean=mean, gamma_mode=gm,
                             gammas=(0.95, 0.99, 1.0), with_grad=True, with_S0=with_S0)
    S0 = t.get("S0")
    if S0 is not None:
        t["start"][:, 0] = 0
    check_bwd(t, S0, t["grad_S_last"] if with_dS else None)


@pytest.mark.parametrize("mode", ["all", "none", "open"])
@pytest.mark.parametrize("d", [64, 128])
def test_bwd_degenerate_resets(mode, d):
    t = tapegen.linattn_tape(2, 700, 2, d, d, seed=tapegen.seed_for(17 + d), gamma_mode="step", with_grad=True,
                             with_S0=True, start_mode=mode)
    check_bwd(t, t["S0"], t["grad_S_last"])


@pytest.mark.parametrize("L", [1, 5, 127, 128, 129, 300])
def test_bwd_short_tapes(L):
    t = tapegen.linattn_tape(1, L, 2, 64, 64, seed=tapegen.seed_for(950 + L), mean=40.0, gamma_mode="step",
                             with_grad=True, with_S0=True)
    t["start"][:, 0] = 0
    check_bwd(t, t["S0"], t["grad_S_last"])


def test_bwd_deterministic():
    t = tapegen.linattn_tape(1, 5000, 2, 128, 128, seed=tapegen.seed_for(59), mean=500.0, gamma_mode="head",
                             with_grad=True)
    a = run_gpu_bwd(t)
    b = run_gpu_bwd(t)
    assert all(np.array_equal(x, y) for x, y in zip(a, b))


def test_bwd_config3_full():
    # the full L = 2^18, 4-head, d = 64 tape with per-head gamma, every output
    t = tapegen.linattn_config(3)
    t["grad_y"] = np.random.default_rng(tapegen.seed_for(3) + 1).standard_normal(t["q"].shape, dtype=np.float32)
    errs = check_bwd(t)
    assert errs["dgamma"] <= TOL



def test_bwd_episode_isolation_bitwise():
    # changing grad_y inside one episode leaves dq, dk, dv of every other episode unchanged, bit for bit
    t = tapegen.linattn_tape(1, 2000, 2, 64, 64, seed=tapegen.seed_for(60), mean=200.0, gamma_mode="step",
                             with_grad=True)
    a = run_gpu_bwd(t)
    starts = np.flatnonzero(t["start"][0])
    s, e = int(starts[3]), int(starts[4])
    t2 = dict(t)
    t2["grad_y"] = t["grad_y"].copy()
    t2["grad_y"][0, s:e] += 0.75
    b = run_gpu_bwd(t2)
    outside = np.ones(2000, dtype=bool)
    outside[s:e] = False
    for name, x, y in zip(("dq", "dk", "dv"), a[:3], b[:3]):
        assert np.array_equal(x[0, outside], y[0, outside]), name
        assert not np.array_equal(x[0, s:e], y[0, s:e]), name


@pytest.mark.parametrize("cut,tol,tol_b", [(1280, 1e-5, 2.0 ** -8), (1300, TOL, TOL)])
def test_split_resume_fwd_and_bwd(cut, tol, tol_b):
    # a tape scanned in two calls (S_last of the first is S0 of the second) gives the
    # one-call outputs; the second call's dS0 fed as the first call's dS_last gives
    # the one-call gradients.  A cut on a 128-step tile edge leaves every tile's
    # operands as in one call, so the forward agrees to fp32 rounding; the backward
    # recomputes the state at the cut with transposed operands, whose fp32 sum can
    # round to the neighbouring bf16 value (one bf16 ulp, 2^-8 relative, of the
    # carried state).  A ragged cut re-tiles the rest of the tape, so its bf16
    # roundings of the masked scores and states differ and the bar is the kernels' own.
    L = 3000
    t = tapegen.linattn_tape(2, L, 2, 64, 64, seed=tapegen.seed_for(62), mean=400.0, gamma_mode="step",
                             with_grad=True, with_S0=True)
    t["start"][:, 0] = 0
    t["start"][:, cut] = 0  # an episode runs across the cut

    def part(sl):
        return dict(q=t["q"][:, sl], k=t["k"][:, sl], v=t["v"][:, sl], gamma=t["gamma"][:, sl],
                    start=t["start"][:, sl], grad_y=t["grad_y"][:, sl])

    y, S_last = run_gpu_fwd(t, S0=t["S0"])
    p1, p2 = part(slice(0, cut)), part(slice(cut, L))
    y1, S1 = run_gpu_fwd(p1, S0=t["S0"])
    y2, S2 = run_gpu_fwd(p2, S0=S1)
    assert rel_err(np.concatenate([y1, y2], axis=1), y) <= tol
    assert rel_err(S2, S_last) <= tol
    full = run_gpu_bwd(t, t["S0"], t["grad_S_last"])
    g2 = run_gpu_bwd(p2, S1, t["grad_S_last"])
    g1 = run_gpu_bwd(p1, t["S0"], g2[4])
    for i, name in enumerate(("dq", "dk", "dv", "dgamma")):
        assert rel_err(np.concatenate([g1[i], g2[i]], axis=1), full[i]) <= tol_b, name
    assert rel_err(g1[4], full[4]) <= tol_b

def test_config5_sampled_episodes():
    # L = 2^22, 8 heads, d = 128, per-step gamma, drawn on the device.  The
    # first episode continues from S0 and the last one is cut by the tape's
    # end (it gives S_last and takes grad_S_last); every episode depends on
    # nothing outside itself (the reset of Theorem 3.2), so the oracle checks
    # them one at a time: the first, the last, the longest and 64 others
    # drawn at random, every output (y, S_last, dq, dk, dv, dgamma, dS0).
    m = _m()
    c = tapegen.LINATTN_CONFIGS[5]
    B, L, H, d = c["B"], c["L"], c["H"], c["d"]
    t = tapegen.linattn_tape_device(B, L, H, d, tapegen.seed_for(5), c["mean"], c["gamma"], with_grad=True)
    t["start"][:, 0] = 0
    rng = np.random.default_rng(tapegen.seed_for(5) + 1)
    S0 = (rng.standard_normal((B, H, d, d)) * 0.3).astype(np.float32)
    dS_last = rng.standard_normal((B, H, d, d)).astype(np.float32)
    ws = m.linattn_workspace(B, L, H, d, "cuda")
    y, S_last = m.linattn_fwd(t["q"], t["k"], t["v"], t["gamma"], t["start"], dev(S0), want_last=True, ws=ws)
    dq, dk, dv, dg, dS0 = m.linattn_bwd(t["q"], t["k"], t["v"], t["gamma"], t["start"], t["grad_y"], dev(dS_last),
                                        dev(S0), want_S0=True, ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_OK
    torch.cuda.synchronize()
    start = t["start"].cpu().numpy()
    heads = np.flatnonzero(start[0])
    bounds = np.concatenate([[0], heads, [L]])
    episodes = list(zip(bounds[:-1].tolist(), bounds[1:].tolist()))
    first, last = episodes[0], episodes[-1]
    inner = episodes[1:-1]
    longest = max(inner, key=lambda se: se[1] - se[0])
    others = [se for se in inner if se != longest]
    picks = [others[i] for i in sorted(rng.choice(len(others), size=64, replace=False))]
    worst = {}

    def note(name, got, ref):
        worst[name] = max(worst.get(name, 0.0), rel_err(got, ref))

    for s, e in [first, longest, *picks, last]:
        sl = slice(s, e)
        sub = dict(q=t["q"][:, sl].cpu().numpy().view(np.uint16), k=t["k"][:, sl].cpu().numpy().view(np.uint16),
                   v=t["v"][:, sl].cpu().numpy().view(np.uint16), gamma=t["gamma"][:, sl].cpu().numpy(),
                   start=start[:, sl], grad_y=t["grad_y"][:, sl].cpu().numpy())
        s0 = S0 if s == 0 else None
        ds = dS_last if e == L else None
        y_ref, S_ref = run_oracle_fwd(sub, s0)
        rq, rk, rv, rg, rS0 = run_oracle_bwd(sub, s0, ds)
        for name, got, ref in (("y", y[:, sl], y_ref), ("dq", dq[:, sl], rq), ("dk", dk[:, sl], rk),
                               ("dv", dv[:, sl], rv), ("dgamma", dg[:, sl], rg)):
            note(name, got.cpu().numpy(), ref)
        if s == 0:
            note("dS0", dS0.cpu().numpy(), rS0)
        if e == L:
            note("S_last", S_last.cpu().numpy(), S_ref)
    assert set(worst) == {"y", "dq", "dk", "dv", "dgamma", "dS0", "S_last"}
    assert all(v <= TOL for v in worst.values()), worst


@pytest.mark.parametrize("d", [64, 128])
def test_injected_wait_failure_reported_then_recovers(d):
    # CTA 0 treats its first tensor-core wait as timed out: it drains its
    # in-flight work, records the error and stops; no GPU fault, and the next
    # calls on the same context are correct again
    m = _m()
    t = tapegen.linattn_tape(1, 3000, 2, d, d, seed=tapegen.seed_for(61 + d), mean=300.0, with_grad=True)
    q, k, v = bits_dev(t["q"]), bits_dev(t["k"]), bits_dev(t["v"])
    gamma, start = dev(t["gamma"]), dev(t["start"])
    ws = m.linattn_workspace(1, 3000, 2, d, "cuda")
    m.memoroid_debug_withhold_tile(0)
    try:
        m.linattn_fwd(q, k, v, gamma, start, ws=ws)
        fwd_status = m.memoroid_get_device_error(ws)
        m.linattn_bwd(q, k, v, gamma, start, dev(t["grad_y"]), ws=ws)
        bwd_status = m.memoroid_get_device_error(ws)
    finally:
        m.memoroid_debug_withhold_tile(-1)
    assert fwd_status == m.MEMOROID_ERR_TIMEOUT
    assert bwd_status == m.MEMOROID_ERR_TIMEOUT
    y, S_last = run_gpu_fwd(t, ws=ws)
    y_ref, S_ref = run_oracle_fwd(t)
    assert rel_err(y, y_ref) <= TOL and rel_err(S_last, S_ref) <= TOL
    check_bwd(t)
