"""CUDA-graph capture of the library's calls (GB300).

A fwd + bwd captured into a graph records its workspace clears, its look-back
tags and its dependent launches once; replayed on fresh inputs copied into the
captured buffers, it must give the bits the same calls give when made one by
one, and calls made afterwards on the same workspace must still be right.
(Every replay reuses the captured tag, so a captured call clears its tag
region; without that clear a reader that polled a summary before this replay
wrote it would take the previous replay's value.  That race depends on timing
and does not show here; these tests check the replays' results.)
"""
import numpy as np
import pytest
import torch

import tapegen

pytestmark = pytest.mark.gpu


def _m():
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def bits(a):
    return dev(np.ascontiguousarray(a).view(np.int16))


def graph_matches_eager(tapes, load, step, ws):
    """load(t) copies tape t into the static inputs; step() makes the calls and
    returns their output tensors."""
    m = _m()
    eager = []
    for t in tapes:
        load(t)
        outs = step()
        torch.cuda.synchronize()
        eager.append([o.cpu().numpy().copy() for o in outs])
    # warm-up on a side stream, then capture
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        load(tapes[0])
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        outs = step()
    for _ in range(2):
        for t, ref in zip(tapes, eager):
            load(t)
            g.replay()
            torch.cuda.synchronize()
            for o, r in zip(outs, ref):
                assert np.array_equal(o.cpu().numpy(), r)
    for w in ws:
        assert m.memoroid_get_device_error(w) == m.MEMOROID_OK
    # an eager call on the same workspace after the replays is still right
    load(tapes[1])
    again = step()
    torch.cuda.synchronize()
    for o, r in zip(again, eager[1]):
        assert np.array_equal(o.cpu().numpy(), r)


def test_diag_fwd_bwd_graph():
    m = _m()
    B, L, D = 2, 1 << 16, 256  # many tiles per chain, several segments
    tapes = [tapegen.diag_tape(B, L, D, seed=tapegen.seed_for(700 + i), mean=300.0) for i in range(3)]
    t0 = tapes[0]
    lam, u, start = dev(t0["lam"]), dev(t0["u"]), dev(t0["start"])
    gh, ghl = dev(t0["grad_h"]), dev(t0["grad_h_last"])
    ws = m.diag_workspace(B, L, D, "cuda")

    def load(t):
        for x, key in ((lam, "lam"), (u, "u"), (start, "start"), (gh, "grad_h"), (ghl, "grad_h_last")):
            x.copy_(dev(t[key]))

    def step():
        h, h_last = m.diag_fwd(lam, u, start, ws=ws)
        gu, gl, _ = m.diag_bwd(lam, start, h, gh, ghl, ws=ws)
        return [h, h_last, gu, gl]

    graph_matches_eager(tapes, load, step, [ws])


def test_linattn_fwd_bwd_graph():
    m = _m()
    B, L, H, d = 1, 8192, 2, 64
    tapes = [tapegen.linattn_tape(B, L, H, d, d, seed=tapegen.seed_for(710 + i), mean=300.0) for i in range(3)]
    t0 = tapes[0]
    q, k, v = bits(t0["q"]), bits(t0["k"]), bits(t0["v"])
    gamma, start, gy = dev(t0["gamma"]), dev(t0["start"]), dev(t0["grad_y"])
    ws = m.linattn_workspace(B, L, H, d, "cuda")

    def load(t):
        for x, key in ((q, "q"), (k, "k"), (v, "v")):
            x.copy_(bits(t[key]))
        for x, key in ((gamma, "gamma"), (start, "start"), (gy, "grad_y")):
            x.copy_(dev(t[key]))

    def step():
        y, S_last = m.linattn_fwd(q, k, v, gamma, start, ws=ws)
        dq, dk, dv, dgamma, _ = m.linattn_bwd(q, k, v, gamma, start, gy, ws=ws)
        return [y, S_last, dq, dk, dv, dgamma]

    graph_matches_eager(tapes, load, step, [ws])


def test_returns_graph():
    m = _m()
    B, L = 8, 100000
    tapes = []
    for i in range(3):
        rng = np.random.default_rng(tapegen.seed_for(720 + i))
        start = (rng.random((B, L)) < (0.0 if i == 2 else 1.0 / 300.0)).astype(np.uint8)
        start[:, 0] = 1
        tapes.append(dict(r=rng.standard_normal((B, L), dtype=np.float32),
                          v=rng.standard_normal((B, L), dtype=np.float32),
                          boot=rng.standard_normal(B).astype(np.float32), start=start))
    t0 = tapes[0]
    r, v, start, boot = dev(t0["r"]), dev(t0["v"]), dev(t0["start"]), dev(t0["boot"])
    ws = m.workspace(m.memoroid_returns_workspace_bytes(B, L), "cuda")

    def load(t):
        for x, key in ((r, "r"), (v, "v"), (start, "start"), (boot, "boot")):
            x.copy_(dev(t[key]))

    def step():
        G = m.discounted_return(r, start, 0.99, boot, ws=ws)
        A = m.gae(r, v, start, 0.99, 0.95, boot, ws=ws)
        return [G, A]

    graph_matches_eager(tapes, load, step, [ws])
