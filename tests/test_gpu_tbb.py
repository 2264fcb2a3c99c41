"""GPU parity of tape-based batching (Algorithm 2: sampling with the draws
given, and the row gather that builds the batch) against the oracle,
through the C ABI.  Integer work: every output must match bit for bit.
"""
import os

import numpy as np
import pytest

import oracle
import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def sample_gpu(I, N, draws, B):
    m = _m()
    ws = m.workspace(m.memoroid_tbb_workspace_bytes(len(draws)), "cuda")
    start, src, n = m.tbb_sample(dev(np.asarray(I, np.int64)), N, dev(np.asarray(draws, np.int64)), B, ws=ws)
    status = m.memoroid_get_device_error(ws)
    torch.cuda.synchronize()
    return start.cpu().numpy(), src.cpu().numpy(), int(n.item()), status


def random_buffer(rng, N, mean):
    return np.flatnonzero(tapegen.geometric_tape_starts(rng, N, mean))


def test_figure2_golden_cases():
    m = _m()
    I, N = np.array([0, 4, 6, 7]), 9
    with open(os.path.join(GOLDEN, "tbb_sample_figure2.txt")) as f:
        rows = [l for l in f if l.strip() and not l.startswith("#")]
    for row in rows:
        head, draws, used, src, start = [c.split() for c in row.split("|")]
        s, x, n, st = sample_gpu(I, N, np.array(draws, dtype=np.int64), int(head[1]))
        assert st == m.MEMOROID_OK
        assert n == int(used[0])
        assert np.array_equal(x, np.array(src, dtype=np.int64))
        assert np.array_equal(s, np.array(start, dtype=np.uint8))


@pytest.mark.parametrize("N,mean,B", [
    (3000, 8.0, 2500),        # many short episodes: several scan chunks of draws
    (50000, 500.0, 20000),    # long episodes, last one cut
    (10000, 1.0, 9000),       # every episode one step: one draw per step (K > 4096)
    (100000, 40.0, 100000),   # batch as large as the buffer
    (777, 3000.0, 5000),      # one episode covering the buffer, drawn repeatedly
])
def test_sample_matches_oracle(N, mean, B):
    m = _m()
    rng = np.random.default_rng(int(N + B + mean))
    I = random_buffer(rng, N, mean)
    draws = rng.integers(0, len(I), size=B + 16)
    s, x, n, st = sample_gpu(I, N, draws, B)
    rs, rx, rn = oracle.tbb_sample(I, N, draws, B)
    assert st == m.MEMOROID_OK
    assert n == rn
    assert np.array_equal(s, rs)
    assert np.array_equal(x, rx)


def test_popped_buffer_head_and_last_episode_to_end():
    # I[0] > 0 (the buffer's first transitions belong to a popped episode) and
    # draws of the last index, whose episode runs to the end of the buffer
    m = _m()
    I, N = np.array([5, 9, 20]), 31
    draws = np.array([2, 0, 2, 1, 2])
    s, x, n, st = sample_gpu(I, N, draws, 30)
    rs, rx, rn = oracle.tbb_sample(I, N, draws, 30)
    assert st == m.MEMOROID_OK and n == rn
    assert np.array_equal(s, rs) and np.array_equal(x, rx)


def test_too_few_draws_and_bad_index_reported():
    m = _m()
    I, N = np.array([0, 4, 6, 7]), 9
    s, x, n, st = sample_gpu(I, N, np.array([2, 2]), 5)  # two 1-step episodes for 5 steps
    assert st == m.MEMOROID_ERR_BAD_DATA
    assert n == 2 and np.array_equal(x[:2], [6, 6]) and np.all(x[2:] == -1) and np.all(s[2:] == 0)
    s, x, n, st = sample_gpu(I, N, np.array([1, 4, 0]), 5)  # no episode 4
    assert st == m.MEMOROID_ERR_BAD_DATA
    s, x, n, st = sample_gpu(I, N, np.array([0, 1]), 6)  # a good call clears the status
    assert st == m.MEMOROID_OK and n == 2


@pytest.mark.parametrize("shape,dtype", [
    ((512,), np.complex64),   # 4 KB rows: 16-byte copies, warp per row
    ((4,), np.float32),       # 16-byte rows: 16-byte units, thread per row
    ((), np.float32),         # 4-byte rows
    ((10,), np.int32),        # 40-byte rows: 4-byte units, warp per row
    ((3,), np.uint8),         # 3-byte rows: byte copies
    ((), np.uint8),           # 1-byte rows (begin flags, done flags)
])
def test_gather_rows_matches_indexing(shape, dtype):
    m = _m()
    rng = np.random.default_rng(17)
    N, B = 5000, 7000
    rows = (rng.integers(0, 250, size=(N,) + shape)).astype(dtype)
    if np.iscomplexobj(rows):
        rows = rows + 1j * rng.standard_normal((N,) + shape).astype(np.float32)
    src = rng.integers(0, N, size=B)
    got = m.gather_rows(dev(rows), dev(src)).cpu().numpy()
    assert np.array_equal(got, rows[src])  # the definition: out[t] = rows[src[t]]


def test_gather_bad_source_is_zero_row_and_reported():
    m = _m()
    rows = np.arange(40, dtype=np.float32).reshape(10, 4)
    src = np.array([3, -1, 9, 10])
    ws = m.workspace(256, "cuda")
    got = m.gather_rows(dev(rows), dev(src), ws=ws)
    assert m.memoroid_get_device_error(ws) == m.MEMOROID_ERR_BAD_DATA
    got = got.cpu().numpy()
    assert np.array_equal(got[0], rows[3]) and np.array_equal(got[2], rows[9])
    assert np.all(got[1] == 0) and np.all(got[3] == 0)


def test_sampled_tape_feeds_the_scan():
    # buffer -> Algorithm 2 batch -> diagonal scan, against the oracle on the
    # oracle-built batch: the sampler's flags make the scan reset exactly at
    # the appended episodes' first steps
    m = _m()
    rng = np.random.default_rng(23)
    N, D, B = 20000, 64, 12000
    I = random_buffer(rng, N, 150.0)
    u = tapegen.complex_normal(rng, (N, D))
    lam = tapegen.diag_lambda(rng, (D,))
    draws = rng.integers(0, len(I), size=B)
    start, src, n = m.tbb_sample(dev(I), N, dev(draws), B)
    tape_u = m.gather_rows(dev(u), src)
    h, _ = m.diag_fwd(dev(lam), tape_u.view(1, B, D), start.view(1, B))
    torch.cuda.synchronize()
    rs, rx, rn = oracle.tbb_sample(I, N, draws, B)
    rh, _ = oracle.diag_fwd(lam, u[rx][None], rs[None])
    g = h.cpu().numpy().view(np.float32).astype(np.float64)
    r = rh.view(np.float64)
    assert float(np.max(np.abs(g - r))) / float(np.max(np.abs(r))) <= 1e-4


def test_bench_size_sample_and_gather():
    # the measured workload: 2^20-step batch from a 2^21-transition buffer,
    # Geometric(500) episodes, 2 KB rows (256 complex64 channels)
    m = _m()
    rng = np.random.default_rng(29)
    N, B, D = 1 << 21, 1 << 20, 256
    I = random_buffer(rng, N, 500.0)
    draws = rng.integers(0, len(I), size=B // 100)
    s, x, n, st = sample_gpu(I, N, draws, B)
    rs, rx, rn = oracle.tbb_sample(I, N, draws, B)
    assert st == m.MEMOROID_OK and n == rn
    assert np.array_equal(s, rs) and np.array_equal(x, rx)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(29)
    rows = torch.randn((N, 2 * D), generator=gen, device="cuda")
    out = m.gather_rows(rows, dev(x))
    pick = rng.integers(0, B, size=2000)
    assert torch.equal(out[dev(pick)], rows[dev(rx[pick])])
