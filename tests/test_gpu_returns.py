"""GPU parity of the per-step discounted return and GAE with resets (the
return and GAE memoroids of the appendices) against the fp64 oracle, through
the C ABI.

Bar: max |gpu - ref| / max |ref| <= 1e-4 (fp32 arithmetic).  Cases cover many
short tapes, long and single-episode tapes (the carry between warp ranges),
the tape bootstrap, block edges and the degenerate reset patterns.
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
    g = np.asarray(got, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(g - r))) / max(float(np.max(np.abs(r))), 1e-30)


def tape(B, L, mean, seed, mode="geometric"):
    rng = np.random.default_rng(seed)
    r = rng.standard_normal((B, L), dtype=np.float32)
    v = rng.standard_normal((B, L), dtype=np.float32)
    boot = rng.standard_normal(B).astype(np.float32)
    start = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        if mode == "all":
            start[b] = 1
        elif mode == "none":
            start[b, 0] = 1
        elif mode == "open":
            pass
        else:
            start[b] = tapegen.geometric_tape_starts(rng, L, mean)
    return r, v, start, boot


def dev(a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()


CASES = [
    # B, L, mean, gamma, lambda, with_boot
    (4, 5000, 30.0, 0.99, 0.95, True),
    (1, 20000, 500.0, 0.9, 0.9, False),
    (64, 1000, 5.0, 0.5, 0.0, True),
    (3, 2049, 100.0, 0.97, 1.0, True),
    (2, 7, 2.0, 0.9, 0.5, True),
    (1, 1, 1.0, 0.9, 0.5, True),
]


@pytest.mark.parametrize("B,L,mean,gamma,lam,with_boot", CASES)
def test_return_and_gae_match_oracle(B, L, mean, gamma, lam, with_boot):
    m = _m()
    r, v, start, boot = tape(B, L, mean, tapegen.seed_for(500 + B + L))
    boot = boot if with_boot else None
    G = m.discounted_return(dev(r), dev(start), gamma, dev(boot))
    A = m.gae(dev(r), dev(v), dev(start), gamma, lam, dev(boot))
    torch.cuda.synchronize()
    assert rel_err(G.cpu().numpy(), oracle.discounted_return(r, start, gamma, boot)) <= TOL
    assert rel_err(A.cpu().numpy(), oracle.gae(r, v, start, gamma, lam, boot)) <= TOL


@pytest.mark.parametrize("mode", ["all", "none", "open"])
def test_degenerate_resets(mode):
    # every step its own episode / one episode over the tape / a tape that
    # continues an episode (no begin flag): in the last two every warp range
    # takes its value from the ranges after it
    m = _m()
    r, v, start, boot = tape(2, 30000, 0.0, tapegen.seed_for(600), mode)
    G = m.discounted_return(dev(r), dev(start), 0.999, dev(boot))
    A = m.gae(dev(r), dev(v), dev(start), 0.999, 0.97, dev(boot))
    torch.cuda.synchronize()
    assert rel_err(G.cpu().numpy(), oracle.discounted_return(r, start, 0.999, boot)) <= TOL
    assert rel_err(A.cpu().numpy(), oracle.gae(r, v, start, 0.999, 0.97, boot)) <= TOL


@pytest.mark.parametrize("gamma,lam,flags", [(0.9999, 0.99, ()), (1.0, 1.0, (123457, 700001))])
def test_long_tape_few_begin_flags(gamma, lam, flags):
    # 2^20 steps with a begin flag at t = 0 only, or at two more steps: the tape
    # is still cut into thousands of warp ranges, each of which gets the value
    # entering it from the maps of the ranges after it
    m = _m()
    B, L = 1, 1 << 20
    r, v, start, boot = tape(B, L, 0.0, tapegen.seed_for(605 + len(flags)), "none")
    for f in flags:
        start[0, f] = 1
    # the call takes gamma and lambda as fp32: over a horizon of 10^4 steps the
    # oracle must see the same values (0.9999 and its fp32 rounding differ by
    # 1.7e-9, which moves the return by about 1e-4 of its size)
    gamma, lam = float(np.float32(gamma)), float(np.float32(lam))
    G = m.discounted_return(dev(r), dev(start), gamma, dev(boot))
    A = m.gae(dev(r), dev(v), dev(start), gamma, lam, dev(boot))
    torch.cuda.synchronize()
    assert rel_err(G.cpu().numpy(), oracle.discounted_return(r, start, gamma, boot)) <= TOL
    assert rel_err(A.cpu().numpy(), oracle.gae(r, v, start, gamma, lam, boot)) <= TOL


def test_episode_heads_bitwise_independent_of_other_episodes():
    # changing the rewards of one episode leaves every other episode's returns unchanged, bit for bit
    m = _m()
    r, v, start, boot = tape(1, 50000, 300.0, tapegen.seed_for(601))
    G0 = m.discounted_return(dev(r), dev(start), 0.99, dev(boot)).cpu().numpy()
    heads = np.flatnonzero(start[0])
    s, e = int(heads[10]), int(heads[11])
    r2 = r.copy()
    r2[0, s:e] += 1.0
    G1 = m.discounted_return(dev(r2), dev(start), 0.99, dev(boot)).cpu().numpy()
    outside = np.ones(50000, dtype=bool)
    outside[s:e] = False
    assert np.array_equal(G0[0, outside], G1[0, outside])
    assert not np.array_equal(G0[0, s:e], G1[0, s:e])


def test_deterministic():
    m = _m()
    r, v, start, boot = tape(8, 100000, 200.0, tapegen.seed_for(602))
    a = m.gae(dev(r), dev(v), dev(start), 0.99, 0.95, dev(boot)).cpu().numpy()
    b = m.gae(dev(r), dev(v), dev(start), 0.99, 0.95, dev(boot)).cpu().numpy()
    assert np.array_equal(a, b)


def _offset(a, k):
    # the same values at a base address k elements past an allocation's start
    flat = torch.zeros(a.size + k, dtype=getattr(torch, str(a.dtype))).cuda()
    out = flat[k:].view(a.shape)
    out.copy_(torch.from_numpy(np.ascontiguousarray(a)))
    return out


@pytest.mark.parametrize("k", [1, 3])
def test_unaligned_base_pointers(k):
    # tapes whose length is a multiple of 8 but whose buffers start off a 16-byte boundary
    m = _m()
    r, v, start, boot = tape(3, 4096, 40.0, tapegen.seed_for(603 + k))
    G = m.discounted_return(_offset(r, k), _offset(start, k), 0.98, dev(boot))
    A = m.gae(_offset(r, k), _offset(v, k), _offset(start, k), 0.98, 0.9, dev(boot))
    torch.cuda.synchronize()
    assert rel_err(G.cpu().numpy(), oracle.discounted_return(r, start, 0.98, boot)) <= TOL
    assert rel_err(A.cpu().numpy(), oracle.gae(r, v, start, 0.98, 0.9, boot)) <= TOL


def test_full_size_tape_set():
    # the measured workload: 64 tapes of 2^20 steps, episode lengths geometric with
    # mean 200 (Bernoulli(1/200) begin flags); four tapes checked against the oracle
    m = _m()
    B, L, p = 64, 1 << 20, 1.0 / 200.0
    rng = np.random.default_rng(tapegen.seed_for(604))
    r = rng.standard_normal((B, L), dtype=np.float32)
    v = rng.standard_normal((B, L), dtype=np.float32)
    boot = rng.standard_normal(B).astype(np.float32)
    start = (rng.random((B, L)) < p).astype(np.uint8)
    start[:, 0] = 1
    G = m.discounted_return(dev(r), dev(start), 0.99, dev(boot)).cpu().numpy()
    A = m.gae(dev(r), dev(v), dev(start), 0.99, 0.95, dev(boot)).cpu().numpy()
    rows = [0, 17, 40, 63]
    assert rel_err(G[rows], oracle.discounted_return(r[rows], start[rows], 0.99, boot[rows])) <= TOL
    assert rel_err(A[rows], oracle.gae(r[rows], v[rows], start[rows], 0.99, 0.95, boot[rows])) <= TOL
