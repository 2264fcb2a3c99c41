"""Pins of the fp64 oracle against facts that do not come from the oracle.

Each test checks the oracle against something the paper or mathematics fixes:
the case table of Theorem 3.2's proof, hand-worked examples, closed forms,
library routines (scipy.signal.lfilter, numpy.cumsum, numpy matmul), brute
force, torch.autograd in float64 through an independent loop, and central
finite differences.
"""
import os

import numpy as np
import pytest
import scipy.signal

import oracle
import tapegen

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


def _rand_c(rng, *shape):
    return rng.standard_normal(shape) + 1j * rng.standard_normal(shape)


def _rand_lam(rng, *shape):
    return rng.uniform(0.3, 0.99, shape) * np.exp(1j * rng.uniform(0, 2 * np.pi, shape))


def _random_starts(rng, B, L, p=0.15, first=True):
    s = (rng.random((B, L)) < p).astype(np.uint8)
    if first and L:
        s[:, 0] = 1
    return s


# ---------------------------------------------------------------------------
# the resettable combine (Theorem 3.2)
# ---------------------------------------------------------------------------

def _s5(e1, e2):
    # S5/LRU monoid with diagonal X (Appendix "Simplified State Space Models"):
    # (X, x) . (X', x') = (X' X, X' x + x'), applied to one channel.
    return (e2[0] * e1[0], e2[0] * e1[1] + e2[1])


def _read_table():
    rows = []
    with open(os.path.join(GOLDEN, "resettable_cases.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def test_combine_case_table():
    rng = _rng(1)
    table = _read_table()
    assert sum(r[0] == "pair" for r in table) == 4 and sum(r[0] == "triple" for r in table) == 8
    for _ in range(5):
        A, A1, A2 = [(complex(*rng.standard_normal(2)), complex(*rng.standard_normal(2))) for _ in range(3)]
        eI = (1.0 + 0j, 0j)
        expect_elems = {
            "AA'": _s5(A, A1), "eA'": _s5(eI, A1),
            "AA'A''": _s5(_s5(A, A1), A2), "eA'A''": _s5(_s5(eI, A1), A2), "eA''": _s5(eI, A2),
        }
        for row in table:
            if row[0] == "pair":
                b, b1 = int(row[1]), int(row[2])
                got, gb = oracle.diag_combine(A, b, A1, b1)
                res, flag = row[3], int(row[4])
            else:
                b, b1, b2 = int(row[1]), int(row[2]), int(row[3])
                left, lb = oracle.diag_combine(A, b, A1, b1)
                got, gb = oracle.diag_combine(left, lb, A2, b2)
                res, flag = row[4], int(row[5])
            assert gb == flag
            np.testing.assert_allclose(np.array(got), np.array(expect_elems[res]), rtol=1e-13, atol=1e-13)


def test_combine_associative_all_flag_patterns():
    rng = _rng(2)
    for trial in range(200):
        els = [(complex(*rng.standard_normal(2)), complex(*rng.standard_normal(2))) for _ in range(3)]
        for pattern in range(8):
            fl = [(pattern >> i) & 1 for i in range(3)]
            l1, lb1 = oracle.diag_combine(els[0], fl[0], els[1], fl[1])
            left, lb = oracle.diag_combine(l1, lb1, els[2], fl[2])
            r1, rb1 = oracle.diag_combine(els[1], fl[1], els[2], fl[2])
            right, rb = oracle.diag_combine(els[0], fl[0], r1, rb1)
            assert lb == rb
            scale = max(1.0, max(abs(z) for z in left + right))
            assert max(abs(a - b) for a, b in zip(left, right)) <= 1e-12 * scale


def test_combine_identity_exact():
    rng = _rng(3)
    gI = ((1.0 + 0j, 0j), 0)
    for _ in range(50):
        e = (complex(*rng.standard_normal(2)), complex(*rng.standard_normal(2)))
        for b in (0, 1):
            got, gb = oracle.diag_combine(gI[0], gI[1], e, b)
            assert got == e and gb == b
            got, gb = oracle.diag_combine(e, b, gI[0], gI[1])
            assert got == e and gb == b


# ---------------------------------------------------------------------------
# diagonal scan, forward
# ---------------------------------------------------------------------------

def test_diag_worked_example():
    vals = {}
    with open(os.path.join(GOLDEN, "diag_worked_example.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, *v = line.split()
                vals[k] = [float(x) for x in v]
    lam = np.array([vals["lambda"][0]], dtype=np.complex128)
    u = np.array(vals["u"], dtype=np.complex128).reshape(1, -1, 1)
    start = np.array(vals["start"], dtype=np.uint8).reshape(1, -1)
    h, h_last = oracle.diag_fwd(lam, u, start)
    np.testing.assert_array_equal(h.reshape(-1).real, np.array(vals["h"]))
    assert h_last[0, 0] == vals["h"][-1]


def _closed_form(lam, u, start, h0=None):
    # h_t = sum_{r=s}^{t} (prod_{j=r+1}^{t} lambda_j) u_r over t's episode [s, ..],
    # plus (prod_{j=0}^{t} lambda_j) h0 for a row that continues an episode.
    B, L, D = u.shape
    per_step = lam.ndim == 3
    out = np.zeros((B, L, D), dtype=np.complex128)
    for b in range(B):
        for t in range(L):
            s = t
            while s > 0 and not start[b, s]:
                s -= 1
            for d in range(D):
                lams = lam[b, :, d] if per_step else np.full(L, lam[d])
                acc = 0j
                for r in range(s, t + 1):
                    acc += np.prod(lams[r + 1:t + 1]) * u[b, r, d]
                if s == 0 and not start[b, 0] and h0 is not None:
                    acc += np.prod(lams[0:t + 1]) * h0[b, d]
                out[b, t, d] = acc
    return out


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_diag_fwd_closed_form(per_step, first):
    rng = _rng(4)
    B, L, D = 2, 40, 3
    lam = _rand_lam(rng, B, L, D) if per_step else _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    start = _random_starts(rng, B, L, 0.12, first=first)
    h0 = _rand_c(rng, B, D)
    h, h_last = oracle.diag_fwd(lam, u, start, h0)
    ref = _closed_form(lam, u, start, h0)
    np.testing.assert_allclose(h, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(h_last, ref[:, -1], rtol=1e-12, atol=1e-12)


def test_diag_lambda_zero_is_identity_map():
    rng = _rng(5)
    u = _rand_c(rng, 2, 50, 4)
    start = _random_starts(rng, 2, 50)
    h, _ = oracle.diag_fwd(np.zeros(4, np.complex128), u, start)
    np.testing.assert_array_equal(h, u)


def test_diag_lambda_one_is_segmented_cumsum():
    rng = _rng(6)
    B, L, D = 3, 200, 5
    u = _rand_c(rng, B, L, D)
    start = _random_starts(rng, B, L, 0.05)
    h, _ = oracle.diag_fwd(np.ones(D, np.complex128), u, start)
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            np.testing.assert_allclose(h[b, s:e], np.cumsum(u[b, s:e], axis=0), rtol=1e-12, atol=1e-12)


def test_diag_matches_lfilter_per_episode():
    # h_t = lambda h_{t-1} + u_t is the IIR filter b = [1], a = [1, -lambda].
    rng = _rng(7)
    B, L, D = 2, 3000, 6
    lam = _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    start = _random_starts(rng, B, L, 0.01)
    h, _ = oracle.diag_fwd(lam, u, start)
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            for d in range(D):
                ref = scipy.signal.lfilter([1.0], [1.0, -lam[d]], u[b, s:e, d])
                np.testing.assert_allclose(h[b, s:e, d], ref, rtol=1e-11, atol=1e-11)


def test_diag_fold_matches_definition():
    rng = _rng(8)
    for per_step in (False, True):
        B, L, D = 2, 300, 4
        lam = _rand_lam(rng, B, L, D) if per_step else _rand_lam(rng, D)
        u = _rand_c(rng, B, L, D)
        start = _random_starts(rng, B, L, 0.05, first=False)
        h0 = _rand_c(rng, B, D)
        h, _ = oracle.diag_fwd(lam, u, start, h0)
        hf = oracle.diag_fold(lam, u, start, h0)
        np.testing.assert_allclose(hf, h, rtol=1e-12, atol=1e-12)


def test_diag_all_start_and_reset_invariant():
    rng = _rng(9)
    B, L, D = 2, 64, 4
    lam = _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    h, _ = oracle.diag_fwd(lam, u, np.ones((B, L), np.uint8))
    np.testing.assert_array_equal(h, u)
    # tape over many episodes == each episode scanned on its own
    start = _random_starts(rng, B, L, 0.2)
    h, _ = oracle.diag_fwd(lam, u, start)
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            one, _ = oracle.diag_fwd(lam, u[b:b + 1, s:e], np.eye(1, e - s, dtype=np.uint8))
            np.testing.assert_array_equal(one[0], h[b, s:e])


def test_diag_tbb_equals_sbb_for_equal_lengths():
    # With every episode exactly L_ep long, the tape equals a [E, L_ep] batch
    # of independent segments (Section 5, TBB vs SBB).
    rng = _rng(10)
    E, Lep, D = 7, 13, 3
    lam = _rand_lam(rng, D)
    u = _rand_c(rng, 1, E * Lep, D)
    start = np.zeros((1, E * Lep), np.uint8)
    start[0, ::Lep] = 1
    h_tape, _ = oracle.diag_fwd(lam, u, start)
    sb = np.zeros((E, Lep), np.uint8)
    sb[:, 0] = 1
    h_seg, _ = oracle.diag_fwd(lam, u.reshape(E, Lep, D), sb)
    np.testing.assert_array_equal(h_tape.reshape(E, Lep, D), h_seg)


def test_diag_split_resume():
    rng = _rng(11)
    B, L, D = 2, 100, 3
    lam = _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    start = _random_starts(rng, B, L, 0.05)
    start[:, 50] = 0
    h, h_last = oracle.diag_fwd(lam, u, start)
    h1, hl1 = oracle.diag_fwd(lam, u[:, :50], start[:, :50])
    h2, hl2 = oracle.diag_fwd(lam, u[:, 50:], start[:, 50:], h0=hl1)
    np.testing.assert_allclose(np.concatenate([h1, h2], 1), h, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(hl2, h_last, rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------------------
# diagonal scan, backward
# ---------------------------------------------------------------------------

def _torch_diag_loss(torch, lam, u, start, h0, g, g_last, per_step):
    # An independent forward loop in torch (complex128): h_t = lambda h_{t-1} + u_t,
    # h_t = u_t at begin flags; loss = sum Re(conj(g) h) + Re(conj(g_last) h_last),
    # whose torch-convention gradient w.r.t. h is g.
    B, L, D = u.shape
    loss = 0.0
    for b in range(B):
        prev = h0[b] if h0 is not None else torch.zeros(D, dtype=torch.complex128)
        for t in range(L):
            lt = lam[b, t] if per_step else lam
            cur = u[b, t] if start[b, t] else lt * prev + u[b, t]
            loss = loss + (torch.conj(g[b, t]) * cur).real.sum()
            prev = cur
        loss = loss + (torch.conj(g_last[b]) * prev).real.sum()
    return loss


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_diag_bwd_vs_torch_autograd(per_step, first):
    torch = pytest.importorskip("torch")
    rng = _rng(12)
    B, L, D = 2, 24, 3
    lam = _rand_lam(rng, B, L, D) if per_step else _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    start = _random_starts(rng, B, L, 0.2, first=first)
    start[0, 5] = 1
    start[0, 6] = 1
    h0 = _rand_c(rng, B, D)
    g = _rand_c(rng, B, L, D)
    g_last = _rand_c(rng, B, D)
    tl = torch.tensor(lam, requires_grad=True)
    tu = torch.tensor(u, requires_grad=True)
    th0 = torch.tensor(h0, requires_grad=True)
    loss = _torch_diag_loss(torch, tl, tu, start, th0, torch.tensor(g), torch.tensor(g_last), per_step)
    loss.backward()
    h, _ = oracle.diag_fwd(lam, u, start, h0)
    gu, glam, gh0 = oracle.diag_bwd(lam, start, h, g, g_last, h0)
    np.testing.assert_allclose(gu, tu.grad.numpy(), rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(glam, tl.grad.numpy(), rtol=1e-11, atol=1e-11)
    ref_h0 = np.zeros_like(gh0) if th0.grad is None else th0.grad.numpy()
    np.testing.assert_allclose(gh0, ref_h0, rtol=1e-11, atol=1e-11)


def test_diag_bwd_finite_differences():
    rng = _rng(13)
    B, L, D = 1, 12, 2
    lam = _rand_lam(rng, D)
    u = _rand_c(rng, B, L, D)
    start = np.zeros((B, L), np.uint8)
    start[0, [4, 9]] = 1  # row continues an episode from h0, then two resets
    h0 = _rand_c(rng, B, D)
    g = _rand_c(rng, B, L, D)
    g_last = _rand_c(rng, B, D)

    def loss(lam_, u_, h0_):
        h, hl = oracle.diag_fwd(lam_, u_, start, h0_)
        return float(np.sum((np.conj(g) * h).real) + np.sum((np.conj(g_last) * hl).real))

    h, _ = oracle.diag_fwd(lam, u, start, h0)
    gu, glam, gh0 = oracle.diag_bwd(lam, start, h, g, g_last, h0)
    eps = 1e-6

    def fd(arr, idx, f):
        out = 0j
        for part, unit in ((0, 1.0), (1, 1j)):
            a1, a2 = arr.copy(), arr.copy()
            a1[idx] += eps * unit
            a2[idx] -= eps * unit
            d = (f(a1) - f(a2)) / (2 * eps)
            out += d if part == 0 else 1j * d
        return out

    for idx in [(0, 0, 0), (0, 3, 1), (0, 4, 0), (0, 8, 1), (0, 11, 0)]:
        assert abs(fd(u, idx, lambda a: loss(lam, a, h0)) - gu[idx]) < 1e-6
    for d in range(D):
        assert abs(fd(lam, (d,), lambda a: loss(a, u, h0)) - glam[d]) < 1e-6
        assert abs(fd(h0, (0, d), lambda a: loss(lam, u, a)) - gh0[0, d]) < 1e-6


# ---------------------------------------------------------------------------
# linear attention, forward
# ---------------------------------------------------------------------------

def _la_inputs(rng, B, L, H, dk, dv, per_step, p=0.1, first=True):
    q = rng.standard_normal((B, L, H, dk)) * 0.5
    k = rng.standard_normal((B, L, H, dk)) * 0.5
    v = rng.standard_normal((B, L, H, dv)) * 0.5
    gamma = rng.uniform(0.5, 1.0, (B, L, H)) if per_step else rng.uniform(0.5, 1.0, H)
    start = _random_starts(rng, B, L, p, first=first)
    return q, k, v, gamma, start


def _la_brute(q, k, v, gamma, start, S0=None):
    # y_t = sum_{r in ep(t), r <= t} (prod_{j=r+1}^{t} gamma_j) (q_t . k_r) v_r
    #       (+ (prod_{j=0}^{t} gamma_j) S0^T q_t for a row continuing an episode)
    B, L, H, dk = q.shape
    per_step = gamma.ndim == 3
    y = np.zeros(v.shape)
    for b in range(B):
        for h in range(H):
            gam = gamma[b, :, h] if per_step else np.full(L, gamma[h])
            for t in range(L):
                s = t
                while s > 0 and not start[b, s]:
                    s -= 1
                for r in range(s, t + 1):
                    y[b, t, h] += np.prod(gam[r + 1:t + 1]) * (q[b, t, h] @ k[b, r, h]) * v[b, r, h]
                if s == 0 and not start[b, 0] and S0 is not None:
                    y[b, t, h] += np.prod(gam[0:t + 1]) * (S0[b, h].T @ q[b, t, h])
    return y


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_linattn_fwd_brute_force(per_step, first):
    rng = _rng(20)
    B, L, H, dk, dv = 2, 30, 2, 3, 4
    q, k, v, gamma, start = _la_inputs(rng, B, L, H, dk, dv, per_step, first=first)
    S0 = rng.standard_normal((B, H, dk, dv))
    y, S_last = oracle.linattn_fwd(q, k, v, gamma, start, S0)
    np.testing.assert_allclose(y, _la_brute(q, k, v, gamma, start, S0), rtol=1e-11, atol=1e-11)
    # S_last: the decayed sum of outer products of the last episode
    for b in range(B):
        for h in range(H):
            s = L - 1
            while s > 0 and not start[b, s]:
                s -= 1
            gam = gamma[b, :, h] if per_step else np.full(L, gamma[h])
            ref = sum(np.prod(gam[r + 1:L]) * np.outer(k[b, r, h], v[b, r, h]) for r in range(s, L))
            if s == 0 and not start[b, 0]:
                ref = ref + np.prod(gam[0:L]) * S0[b, h]
            np.testing.assert_allclose(S_last[b, h], ref, rtol=1e-11, atol=1e-11)


def test_linattn_gamma_one_is_causal_attention():
    rng = _rng(21)
    B, L, H, d = 1, 300, 2, 8
    q, k, v, _, start = _la_inputs(rng, B, L, H, d, d, False, p=0.02)
    y, _ = oracle.linattn_fwd(q, k, v, np.ones(H), start)
    for s, e in tapegen.episode_bounds(start[0]):
        for h in range(H):
            Q, K, V = q[0, s:e, h], k[0, s:e, h], v[0, s:e, h]
            ref = np.tril(Q @ K.T) @ V
            np.testing.assert_allclose(y[0, s:e, h], ref, rtol=1e-10, atol=1e-10)


def test_linattn_all_start():
    rng = _rng(22)
    q, k, v, gamma, _ = _la_inputs(rng, 2, 20, 2, 4, 3, True)
    y, _ = oracle.linattn_fwd(q, k, v, gamma, np.ones((2, 20), np.uint8))
    ref = np.einsum("blhi,blhi->blh", q, k)[..., None] * v
    np.testing.assert_allclose(y, ref, rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------------------
# linear attention, backward
# ---------------------------------------------------------------------------

def _torch_la_loss(torch, q, k, v, gamma, start, S0, dy, dS_last, per_step):
    B, L, H, dk = q.shape
    dv = v.shape[-1]
    loss = 0.0
    for b in range(B):
        for h in range(H):
            S = S0[b, h] if S0 is not None else torch.zeros(dk, dv, dtype=torch.float64)
            for t in range(L):
                g = gamma[b, t, h] if per_step else gamma[h]
                kv = torch.outer(k[b, t, h], v[b, t, h])
                S = kv if start[b, t] else g * S + kv
                loss = loss + (dy[b, t, h] * (S.T @ q[b, t, h])).sum()
            loss = loss + (dS_last[b, h] * S).sum()
    return loss


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_linattn_bwd_vs_torch_autograd(per_step, first):
    torch = pytest.importorskip("torch")
    rng = _rng(23)
    B, L, H, dk, dv = 2, 16, 2, 3, 2
    q, k, v, gamma, start = _la_inputs(rng, B, L, H, dk, dv, per_step, p=0.2, first=first)
    start[0, 7] = 1
    start[0, 8] = 1
    S0 = rng.standard_normal((B, H, dk, dv))
    dy = rng.standard_normal((B, L, H, dv))
    dS_last = rng.standard_normal((B, H, dk, dv))
    t = {n: torch.tensor(a, requires_grad=True) for n, a in
         dict(q=q, k=k, v=v, gamma=gamma, S0=S0).items()}
    loss = _torch_la_loss(torch, t["q"], t["k"], t["v"], t["gamma"], start, t["S0"],
                          torch.tensor(dy), torch.tensor(dS_last), per_step)
    loss.backward()
    dq, dk_, dv_, dg, dS0 = oracle.linattn_bwd(q, k, v, gamma, start, dy, dS_last, S0)
    for name, got in dict(q=dq, k=dk_, v=dv_, gamma=dg, S0=dS0).items():
        ref = t[name].grad
        ref = np.zeros_like(got) if ref is None else ref.numpy()
        np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-11, err_msg=name)


def test_linattn_bwd_finite_differences():
    rng = _rng(24)
    B, L, H, dk, dv = 1, 10, 1, 2, 3
    q, k, v, gamma, start = _la_inputs(rng, B, L, H, dk, dv, True, first=False)
    start[0, :] = 0
    start[0, 6] = 1
    S0 = rng.standard_normal((B, H, dk, dv))
    dy = rng.standard_normal((B, L, H, dv))
    dS_last = rng.standard_normal((B, H, dk, dv))

    def loss(q_, k_, v_, g_, S0_):
        y, Sl = oracle.linattn_fwd(q_, k_, v_, g_, start, S0_)
        return float(np.sum(dy * y) + np.sum(dS_last * Sl))

    dq, dk_, dv_, dg, dS0 = oracle.linattn_bwd(q, k, v, gamma, start, dy, dS_last, S0)
    eps = 1e-6
    args = [q, k, v, gamma, S0]
    grads = [dq, dk_, dv_, dg, dS0]
    for ai in range(5):
        arr = args[ai]
        for _ in range(6):
            idx = tuple(rng.integers(0, n) for n in arr.shape)
            a1, a2 = arr.copy(), arr.copy()
            a1[idx] += eps
            a2[idx] -= eps
            f1 = loss(*[a1 if j == ai else args[j] for j in range(5)])
            f2 = loss(*[a2 if j == ai else args[j] for j in range(5)])
            assert abs((f1 - f2) / (2 * eps) - grads[ai][idx]) < 1e-6, (ai, idx)


# ---------------------------------------------------------------------------
# episode index list <-> begin flags
# ---------------------------------------------------------------------------

def test_figure2_tape_indices():
    vals = {}
    with open(os.path.join(GOLDEN, "tbb_figure2.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, *v = line.split()
                vals[k] = [int(x) for x in v]
    start = oracle.starts_from_offsets(vals["I"], len(vals["episode"]))
    np.testing.assert_array_equal(start, vals["start"])
    np.testing.assert_array_equal(oracle.offsets_from_starts(start), vals["I"])
    # the episode labels change exactly at the begin indices
    ep = np.array(vals["episode"])
    np.testing.assert_array_equal(np.flatnonzero(np.r_[1, np.diff(ep) != 0]), vals["I"])


def test_offsets_round_trip_random():
    rng = _rng(30)
    for L in (1, 7, 1000):
        start = (rng.random(L) < 0.1).astype(np.uint8)
        offs = oracle.offsets_from_starts(start)
        np.testing.assert_array_equal(offs, np.flatnonzero(start))
        np.testing.assert_array_equal(oracle.starts_from_offsets(offs, L), start)


# ---------------------------------------------------------------------------
# discounted return and GAE memoroids (appendix "The Discounted Return as a
# Memoroid" and "The Generalized Advantage Estimate as a Memoroid")
# ---------------------------------------------------------------------------

def _ret_combine(x, y):
    # (a, r) . (a', r') = (a a', a r' + r), the left operand earlier in time
    return (x[0] * y[0], x[0] * y[1] + x[1])


def test_return_golden_worked_example():
    rows = np.loadtxt(os.path.join(GOLDEN, "return_expansion.txt"))
    r = rows[:, 1][None, :]
    start = rows[:, 2].astype(np.uint8)[None, :]
    G = oracle.discounted_return(r, start, 0.5)
    assert np.array_equal(G[0], rows[:, 3])


def test_return_equals_memoroid_fold_at_episode_heads():
    rng = np.random.default_rng(41)
    gamma = 0.9
    r = rng.standard_normal((3, 200))
    start = np.stack([tapegen.geometric_tape_starts(rng, 200, 15.0) for _ in range(3)])
    G = oracle.discounted_return(r, start, gamma)
    for b in range(3):
        for s, e in tapegen.episode_bounds(start[b]):
            acc = (1.0, 0.0)  # e_I
            for t in range(s, e):
                acc = _ret_combine(acc, (gamma, r[b, t]))
            assert acc[0] == pytest.approx(gamma ** (e - s), rel=1e-12)
            assert G[b, s] == pytest.approx(acc[1], rel=1e-12, abs=1e-12)


def test_return_brute_force_suffix_sums_with_bootstrap():
    rng = np.random.default_rng(42)
    gamma = 0.8
    r = rng.standard_normal((2, 60))
    start = np.stack([tapegen.geometric_tape_starts(rng, 60, 8.0) for _ in range(2)])
    boot = rng.standard_normal(2)
    G = oracle.discounted_return(r, start, gamma, boot)
    for b in range(2):
        bounds = tapegen.episode_bounds(start[b])
        for s, e in bounds:
            for t in range(s, e):
                want = sum(gamma ** (l - t) * r[b, l] for l in range(t, e))
                if e == 60:
                    want += gamma ** (e - t) * boot[b]
                assert G[b, t] == pytest.approx(want, rel=1e-12, abs=1e-12)


def test_return_matches_reverse_diagonal_scan():
    # the return is the diagonal backward recurrence with a real multiplier:
    # delta_t = g_t + [b_{t+1} = 0] gamma delta_{t+1}, g_last = gamma * boot
    rng = np.random.default_rng(43)
    gamma = 0.95
    B, L = 2, 300
    r = rng.standard_normal((B, L))
    start = np.stack([tapegen.geometric_tape_starts(rng, L, 30.0) for _ in range(B)])
    boot = rng.standard_normal(B)
    G = oracle.discounted_return(r, start, gamma, boot)
    lam = np.full(2, gamma, dtype=np.complex128)
    g = np.zeros((B, L, 2), dtype=np.complex128)
    g[:, :, 0] = r
    h = np.zeros_like(g)
    g_last = np.zeros((B, 2), dtype=np.complex128)
    g_last[:, 0] = gamma * boot
    gu, _, _ = oracle.diag_bwd(lam, start, h, g, g_last)
    assert np.allclose(gu[:, :, 0].real, G, rtol=1e-12, atol=1e-12)


def test_gae_special_cases_and_brute_force():
    rng = np.random.default_rng(44)
    gamma, lam = 0.9, 0.7
    B, L = 2, 80
    r = rng.standard_normal((B, L))
    v = rng.standard_normal((B, L))
    start = np.stack([tapegen.geometric_tape_starts(rng, L, 10.0) for _ in range(B)])
    v_boot = rng.standard_normal(B)
    # delta_t = r_t + gamma V_{t+1} - V_t (V after an episode's end: 0; after the tape: v_boot)
    delta = np.zeros((B, L))
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            for t in range(s, e):
                nv = v[b, t + 1] if t + 1 < e else (v_boot[b] if e == L else 0.0)
                delta[b, t] = r[b, t] + gamma * nv - v[b, t]
    # lambda = 0: one-step TD error
    assert np.allclose(oracle.gae(r, v, start, gamma, 0.0, v_boot), delta, rtol=1e-12, atol=1e-12)
    # lambda = 1: the discounted return (bootstrapped by v_boot) minus the value
    G = oracle.discounted_return(r, start, gamma, v_boot)
    assert np.allclose(oracle.gae(r, v, start, gamma, 1.0, v_boot), G - v, rtol=1e-10, atol=1e-10)
    # general lambda: sum_l (gamma lambda)^l delta_{t+l} within the episode
    A = oracle.gae(r, v, start, gamma, lam, v_boot)
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            for t in range(s, e):
                want = sum((gamma * lam) ** (l - t) * delta[b, l] for l in range(t, e))
                assert A[b, t] == pytest.approx(want, rel=1e-12, abs=1e-12)


# ---------------------------------------------------------------------------
# Fast and Forgetful Memory (Appendix "Fast and Forgetful Memory")
# ---------------------------------------------------------------------------

def _ffm_inputs(rng, B, L, m, c, p=0.15, first=True):
    alpha = rng.uniform(-0.3, 0.3, m)  # signed: the memoroid uses |alpha|
    omega = rng.uniform(-np.pi, np.pi, c)
    xt = rng.standard_normal((B, L, m))
    start = _random_starts(rng, B, L, p, first=first)
    S0 = _rand_c(rng, B, m, c)
    return alpha, omega, xt, start, S0


def _planar(X):
    # Re(X) || Im(X), each flattened (i * c + j)
    B, L, m, c = X.shape
    return np.concatenate([X.real.reshape(B, L, m * c), X.imag.reshape(B, L, m * c)], axis=-1)


def _ffm_aggregator(alpha, omega, xt, start, S0):
    # The original FFM aggregator in closed form, episode by episode: for an
    # episode that starts at step k, row i of the aggregator gives
    #   S_{k+i} = Gamma(i + 1) * S_{k-1} + Gamma(i - t) * sum_{j<=i} Gamma(t - j) * (o_{k+j} 1^T)
    # with Gamma(tau)[a, b] = exp(-tau (|alpha_a| + i w_b)) and t the episode's
    # last row.  The aggregator's Gamma carries exp(-i tau w) while the
    # memoroid's multiplier is exp(+i omega): w = -omega.  The positive powers
    # Gamma(i - t) for i < t are what the memoroid form avoids; at these sizes
    # they are exact enough in fp64.
    B, L, m = xt.shape
    c = omega.shape[0]
    w = -omega
    expo = np.abs(alpha)[:, None] + 1j * w[None, :]

    def gamma(tau):
        return np.exp(-tau * expo)

    X = np.zeros((B, L, m, c), dtype=np.complex128)
    for b in range(B):
        for s, e in tapegen.episode_bounds(start[b]):
            prev = S0[b] if (s == 0 and not start[b, 0]) else np.zeros((m, c), np.complex128)
            t = e - 1 - s
            for i in range(e - s):
                acc = np.zeros((m, c), np.complex128)
                for j in range(i + 1):
                    acc += gamma(t - j) * np.repeat(xt[b, s + j][:, None], c, axis=1)
                X[b, s + i] = gamma(i + 1) * prev + gamma(i - t) * acc
    return X


@pytest.mark.parametrize("first", [True, False])
def test_ffm_fwd_matches_aggregator_closed_form(first):
    rng = _rng(60)
    B, L, m, c = 2, 40, 3, 4
    alpha, omega, xt, start, S0 = _ffm_inputs(rng, B, L, m, c, 0.12, first=first)
    z, S_last = oracle.ffm_fwd(alpha, omega, xt, start, S0)
    X = _ffm_aggregator(alpha, omega, xt, start, S0)
    np.testing.assert_allclose(z, _planar(X), rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(S_last, X[:, -1], rtol=1e-10, atol=1e-10)


def test_ffm_is_diag_scan_with_outer_sum_multiplier():
    # lambda_ij = exp(-|alpha_i| + i omega_j) per channel, input x~_i in every column
    rng = _rng(61)
    B, L, m, c = 2, 50, 4, 3
    alpha, omega, xt, start, S0 = _ffm_inputs(rng, B, L, m, c, 0.1, first=False)
    lam = np.exp(-np.abs(alpha)[:, None] + 1j * omega[None, :]).reshape(m * c)
    u = np.repeat(xt[..., None], c, axis=-1).reshape(B, L, m * c).astype(np.complex128)
    h, hl = oracle.diag_fwd(lam, u, start, S0.reshape(B, m * c))
    z, S_last = oracle.ffm_fwd(alpha, omega, xt, start, S0)
    np.testing.assert_allclose(z, np.concatenate([h.real, h.imag], axis=-1), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(S_last.reshape(B, m * c), hl, rtol=1e-12, atol=1e-12)


def test_ffm_all_start_is_broadcast_input():
    rng = _rng(62)
    B, L, m, c = 1, 9, 2, 5
    alpha, omega, xt, _, S0 = _ffm_inputs(rng, B, L, m, c)
    start = np.ones((B, L), np.uint8)
    z, _ = oracle.ffm_fwd(alpha, omega, xt, start, S0)
    D = m * c
    np.testing.assert_array_equal(z[..., :D], np.repeat(xt[..., None], c, axis=-1).reshape(B, L, D))
    np.testing.assert_array_equal(z[..., D:], 0.0)


def _torch_ffm_loss(torch, alpha, omega, xt, start, S0, gz, gSl):
    # independent loop: X_t = lambda * X_{t-1} + x~_t (columns), X_t = x~_t at begin flags;
    # loss = <gz, Re || Im> + Re(conj(gSl) X_last)
    B, L, m = xt.shape
    c = omega.shape[0]
    lam = torch.exp(-torch.abs(alpha)[:, None] + 1j * omega[None, :])
    loss = 0.0
    for b in range(B):
        X = S0[b]
        for t in range(L):
            inp = xt[b, t][:, None].expand(m, c).to(torch.complex128)
            X = inp if start[b, t] else lam * X + inp
            flat = torch.cat([X.real.reshape(-1), X.imag.reshape(-1)])
            loss = loss + (gz[b, t] * flat).sum()
        loss = loss + (torch.conj(gSl[b]) * X).real.sum()
    return loss


@pytest.mark.parametrize("first", [True, False])
def test_ffm_bwd_vs_torch_autograd(first):
    torch = pytest.importorskip("torch")
    rng = _rng(63)
    B, L, m, c = 2, 20, 3, 2
    alpha, omega, xt, start, S0 = _ffm_inputs(rng, B, L, m, c, 0.2, first=first)
    alpha[1] = -alpha[1] if alpha[1] > 0 else alpha[1]  # one negative alpha: sign(alpha) enters
    gz = rng.standard_normal((B, L, 2 * m * c))
    gSl = _rand_c(rng, B, m, c)
    ta, to = torch.tensor(alpha, requires_grad=True), torch.tensor(omega, requires_grad=True)
    tx, ts = torch.tensor(xt, requires_grad=True), torch.tensor(S0, requires_grad=True)
    loss = _torch_ffm_loss(torch, ta, to, tx, start, ts, torch.tensor(gz), torch.tensor(gSl))
    loss.backward()
    z, _ = oracle.ffm_fwd(alpha, omega, xt, start, S0)
    gx, ga, go, gS0 = oracle.ffm_bwd(alpha, omega, start, z, gz, gSl, S0)
    np.testing.assert_allclose(gx, tx.grad.numpy(), rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(ga, ta.grad.numpy(), rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(go, to.grad.numpy(), rtol=1e-10, atol=1e-10)
    ref_S0 = np.zeros_like(gS0) if ts.grad is None else ts.grad.numpy()
    np.testing.assert_allclose(gS0, ref_S0, rtol=1e-10, atol=1e-10)


def test_ffm_bwd_finite_differences():
    rng = _rng(64)
    B, L, m, c = 1, 14, 2, 3
    alpha, omega, xt, start, S0 = _ffm_inputs(rng, B, L, m, c, 0.0, first=False)
    start[0, [5, 10]] = 1
    gz = rng.standard_normal((B, L, 2 * m * c))
    gSl = _rand_c(rng, B, m, c)

    def loss(a, o, x, s0):
        z, Sl = oracle.ffm_fwd(a, o, x, start, s0)
        return float(np.sum(gz * z) + np.sum((np.conj(gSl) * Sl).real))

    z, _ = oracle.ffm_fwd(alpha, omega, xt, start, S0)
    gx, ga, go, gS0 = oracle.ffm_bwd(alpha, omega, start, z, gz, gSl, S0)
    eps = 1e-6

    def fd(arr, idx, f, unit=1.0):
        a1, a2 = arr.copy(), arr.copy()
        a1[idx] += eps * unit
        a2[idx] -= eps * unit
        return (f(a1) - f(a2)) / (2 * eps)

    for i in range(m):
        assert abs(fd(alpha, (i,), lambda a: loss(a, omega, xt, S0)) - ga[i]) < 1e-6
    for j in range(c):
        assert abs(fd(omega, (j,), lambda o: loss(alpha, o, xt, S0)) - go[j]) < 1e-6
    for idx in [(0, 0, 0), (0, 4, 1), (0, 5, 0), (0, 13, 1)]:
        assert abs(fd(xt, idx, lambda x: loss(alpha, omega, x, S0)) - gx[idx]) < 1e-6
    for idx in [(0, 0, 0), (0, 1, 2)]:
        d = fd(S0, idx, lambda s: loss(alpha, omega, xt, s)) + 1j * fd(S0, idx, lambda s: loss(alpha, omega, xt, s), 1j)
        assert abs(d - gS0[idx]) < 1e-6


# ---------------------------------------------------------------------------
# tape-based batching, sampling (Algorithm 2)
# ---------------------------------------------------------------------------

FIG2_I = np.array([0, 4, 6, 7])
FIG2_N = 9


def test_tbb_sample_figure2_worked_by_hand():
    with open(os.path.join(GOLDEN, "tbb_sample_figure2.txt")) as f:
        rows = [l for l in f if l.strip() and not l.startswith("#")]
    assert len(rows) == 2
    for row in rows:
        head, draws, used, src, start = [c.split() for c in row.split("|")]
        B = int(head[1])
        s, x, n = oracle.tbb_sample(FIG2_I, FIG2_N, np.array(draws, dtype=np.int64), B)
        assert n == int(used[0])
        assert np.array_equal(x, np.array(src, dtype=np.int64))
        assert np.array_equal(s, np.array(start, dtype=np.uint8))


def _episode_range(I, N, i):
    return int(I[i]), int(I[i + 1]) if i + 1 < len(I) else N


@pytest.mark.parametrize("seed", range(6))
def test_tbb_sample_defining_properties(seed):
    rng = np.random.default_rng(900 + seed)
    N = int(rng.integers(50, 3000))
    starts = tapegen.geometric_tape_starts(rng, N, float(rng.choice([1.5, 8.0, 60.0])))
    I = np.flatnonzero(starts)
    if seed == 5:
        I = I[1:] if len(I) > 1 else I  # a buffer whose first transitions belong to a popped episode
    B = int(rng.integers(1, 2 * N))
    ep = rng.integers(0, len(I), size=4 * B + 8)
    start, src, n = oracle.tbb_sample(I, N, ep, B)
    heads = np.flatnonzero(start)
    # one piece per draw used, starting at step 0, in draw order
    assert len(heads) == n and heads[0] == 0
    bounds = list(heads) + [B]
    full = 0
    for k in range(n):
        lo, hi = _episode_range(I, N, int(ep[k]))
        piece = src[bounds[k]:bounds[k + 1]]
        # a piece is the drawn episode's transitions, consecutive, from its first one
        assert piece[0] == lo
        assert np.all(np.diff(piece) == 1)
        if k < n - 1:
            assert len(piece) == hi - lo  # whole episodes before the last
            full += hi - lo
        else:
            assert 1 <= len(piece) <= hi - lo  # the last one is cut at B
    # the fewest draws: the pieces before the last do not fill the batch
    assert full < B


def test_tbb_sample_exact_fit_and_errors():
    # the episodes fill B exactly: nothing is cut
    start, src, n = oracle.tbb_sample(FIG2_I, FIG2_N, np.array([1, 3, 2]), 5)
    assert n == 3 and np.array_equal(src, [4, 5, 7, 8, 6]) and np.array_equal(start, [1, 0, 1, 0, 1])
    assert oracle.tbb_sample(FIG2_I, FIG2_N, np.array([], dtype=np.int64), 0)[2] == 0
    with pytest.raises(ValueError):
        oracle.tbb_sample(FIG2_I, FIG2_N, np.array([2, 2]), 5)  # two 1-step episodes cannot fill 5 steps
    with pytest.raises(ValueError):
        oracle.tbb_sample(FIG2_I, FIG2_N, np.array([4]), 2)  # no episode 4


# ---------------------------------------------------------------------------
# the Linear Transformer with phi = 1 + ELU and its normalizer (Appendix "Linear Transformer")
# ---------------------------------------------------------------------------

def _phi_np(z):
    return np.where(z > 0, 1.0 + z, np.exp(np.minimum(z, 0.0)))


def _norm_inputs(rng, B, L, H, d, per_step, p=0.1, first=True):
    q = rng.standard_normal((B, L, H, d))
    k = rng.standard_normal((B, L, H, d))
    v = rng.standard_normal((B, L, H, d))
    gamma = rng.uniform(0.7, 1.0, (B, L, H) if per_step else (H,))
    start = _random_starts(rng, B, L, p, first=first)
    S0 = rng.standard_normal((B, H, d, d))
    z0 = rng.uniform(0.5, 2.0, (B, H, d))  # a normalizer state is a sum of positive features
    return q, k, v, gamma, start, S0, z0


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_linattn_norm_brute_force_weighted_average(per_step, first):
    # y_t = sum_r w_tr v_r / sum_r w_tr with w_tr = (prod of gamma over (r, t]) phi(q_t).phi(k_r)
    # over the steps r <= t of t's episode (plus the incoming state for a continued row)
    rng = _rng(70)
    B, L, H, d = 2, 30, 2, 3
    q, k, v, gamma, start, S0, z0 = _norm_inputs(rng, B, L, H, d, per_step, first=first)
    y, den, S_last, z_last = oracle.linattn_norm_fwd(q, k, v, gamma, start, S0, z0)
    for b in range(B):
        for h in range(H):
            for t in range(L):
                s = t
                while s > 0 and not start[b, s]:
                    s -= 1
                num = np.zeros(d)
                dd = 0.0
                for r in range(s, t + 1):
                    w = 1.0
                    for j in range(r + 1, t + 1):
                        w *= gamma[b, j, h] if per_step else gamma[h]
                    a = w * float(_phi_np(q[b, t, h]) @ _phi_np(k[b, r, h]))
                    num += a * v[b, r, h]
                    dd += a
                if not start[b, s]:  # a continued row carries (S0, z0) decayed over [0, t]
                    w = 1.0
                    for j in range(0, t + 1):
                        w *= gamma[b, j, h] if per_step else gamma[h]
                    num += w * (S0[b, h].T @ _phi_np(q[b, t, h]))
                    dd += w * float(z0[b, h] @ _phi_np(q[b, t, h]))
                np.testing.assert_allclose(y[b, t, h], num / dd, rtol=1e-10, atol=1e-12)
                assert den[b, t, h] == pytest.approx(dd, rel=1e-10)


def test_linattn_norm_all_start_and_shift_equivariance():
    rng = _rng(71)
    B, L, H, d = 1, 40, 2, 4
    q, k, v, gamma, _, _, _ = _norm_inputs(rng, B, L, H, d, False)
    ones = np.ones((B, L), np.uint8)
    y, _, _, _ = oracle.linattn_norm_fwd(q, k, v, gamma, ones)
    np.testing.assert_allclose(y, v, rtol=1e-12, atol=1e-12)  # one term: the weight cancels
    start = _random_starts(rng, B, L, 0.15)
    y1, _, _, _ = oracle.linattn_norm_fwd(q, k, v, gamma, start)
    y2, _, _, _ = oracle.linattn_norm_fwd(q, k, v + 3.5, gamma, start)
    np.testing.assert_allclose(y2, y1 + 3.5, rtol=1e-12, atol=1e-11)  # normalised weights sum to 1
    # each output lies within the range of v over its episode so far
    for t in range(L):
        s = t
        while s > 0 and not start[0, s]:
            s -= 1
        lo = v[0, s:t + 1].min(axis=0)
        hi = v[0, s:t + 1].max(axis=0)
        assert np.all(y1[0, t] >= lo - 1e-12) and np.all(y1[0, t] <= hi + 1e-12)


def _torch_norm_loss(torch, q, k, v, gamma, start, S0, z0, dy, dSl, dzl, per_step):
    def phi(z):
        return torch.where(z > 0, 1.0 + z, torch.exp(torch.clamp(z, max=0.0)))
    B, L, H, d = q.shape
    loss = 0.0
    for b in range(B):
        for h in range(H):
            X, x = S0[b, h], z0[b, h]
            for t in range(L):
                g = gamma[b, t, h] if per_step else gamma[h]
                pk, pq = phi(k[b, t, h]), phi(q[b, t, h])
                if start[b, t]:
                    X, x = torch.outer(pk, v[b, t, h]), pk
                else:
                    X, x = g * X + torch.outer(pk, v[b, t, h]), g * x + pk
                y = (X.T @ pq) / (x @ pq)
                loss = loss + (dy[b, t, h] * y).sum()
            loss = loss + (dSl[b, h] * X).sum() + (dzl[b, h] * x).sum()
    return loss


@pytest.mark.parametrize("per_step", [False, True])
@pytest.mark.parametrize("first", [True, False])
def test_linattn_norm_bwd_vs_torch_autograd(per_step, first):
    torch = pytest.importorskip("torch")
    rng = _rng(72)
    B, L, H, d = 2, 14, 2, 3
    q, k, v, gamma, start, S0, z0 = _norm_inputs(rng, B, L, H, d, per_step, 0.2, first=first)
    dy = rng.standard_normal((B, L, H, d))
    dSl = rng.standard_normal((B, H, d, d))
    dzl = rng.standard_normal((B, H, d))
    T = [torch.tensor(a, requires_grad=True) for a in (q, k, v, gamma, S0, z0)]
    loss = _torch_norm_loss(torch, *T[:4], start, T[4], T[5], torch.tensor(dy), torch.tensor(dSl),
                            torch.tensor(dzl), per_step)
    loss.backward()
    got = oracle.linattn_norm_bwd(q, k, v, gamma, start, dy, dSl, dzl, S0, z0)
    for g, t in zip(got, T):
        ref = np.zeros_like(g) if t.grad is None else t.grad.numpy()
        np.testing.assert_allclose(g, ref, rtol=1e-9, atol=1e-10)


def test_linattn_norm_bwd_finite_differences():
    rng = _rng(73)
    B, L, H, d = 1, 10, 1, 2
    q, k, v, gamma, start, S0, z0 = _norm_inputs(rng, B, L, H, d, False, 0.0, first=False)
    start[0, 6] = 1
    dy = rng.standard_normal((B, L, H, d))

    def loss(q_, k_, v_, g_):
        y, _, _, _ = oracle.linattn_norm_fwd(q_, k_, v_, g_, start, S0, z0)
        return float(np.sum(dy * y))

    dq, dk, dv, dg, _, _ = oracle.linattn_norm_bwd(q, k, v, gamma, start, dy, None, None, S0, z0)
    eps = 1e-6

    def fd(arr, idx, f):
        a1, a2 = arr.copy(), arr.copy()
        a1[idx] += eps
        a2[idx] -= eps
        return (f(a1) - f(a2)) / (2 * eps)

    for idx in [(0, 0, 0, 0), (0, 5, 0, 1), (0, 6, 0, 0), (0, 9, 0, 1)]:
        assert abs(fd(q, idx, lambda a: loss(a, k, v, gamma)) - dq[idx]) < 1e-6
        assert abs(fd(k, idx, lambda a: loss(q, a, v, gamma)) - dk[idx]) < 1e-6
        assert abs(fd(v, idx, lambda a: loss(q, k, a, gamma)) - dv[idx]) < 1e-6
    assert abs(fd(gamma, (0,), lambda a: loss(q, k, v, a)) - dg[0]) < 1e-6
