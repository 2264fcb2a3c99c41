"""The torch.autograd wrappers of the memoroids (linear attention, the
normalised Linear Transformer and Fast and Forgetful Memory): outputs and the
gradients that loss.backward() leaves on the leaves match the fp64 oracle,
and a two-layer graph through the wrappers back-propagates end to end.
"""
import numpy as np
import pytest

import oracle
import tapegen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


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
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def bf16_leaf(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16).requires_grad_(True)


def np32(t):
    return t.detach().float().cpu().numpy()


def test_linattn_autograd_matches_oracle():
    m = _m()
    t = tapegen.linattn_tape(2, 900, 2, 64, 64, seed=tapegen.seed_for(1200), mean=120.0, gamma_mode="step",
                             with_grad=True, with_S0=True)
    t["start"][:, 0] = 0
    q, k, v = bf16_leaf(t["q"]), bf16_leaf(t["k"]), bf16_leaf(t["v"])
    gamma = dev(t["gamma"]).requires_grad_(True)
    S0 = dev(t["S0"]).requires_grad_(True)
    y = m.LinAttnScan.apply(q, k, v, gamma, dev(t["start"]), S0)
    (y * dev(t["grad_y"])).sum().backward()
    f = oracle.bf16_bits_to_f64
    ry, _ = oracle.linattn_fwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"], t["S0"])
    rq, rk, rv, rg, rS0 = oracle.linattn_bwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"], t["grad_y"],
                                             None, t["S0"])
    assert q.grad.dtype == torch.bfloat16 and gamma.grad.dtype == torch.float32
    # dq, dk, dv come back rounded to bf16: 2e-2 covers the kernel's bar plus one rounding
    for name, got, ref in (("y", y, ry), ("dq", q.grad, rq), ("dk", k.grad, rk), ("dv", v.grad, rv),
                           ("dgamma", gamma.grad, rg), ("dS0", S0.grad, rS0)):
        assert rel_err(np32(got), ref) <= 2e-2, name


@pytest.mark.parametrize("d", [32, 64])  # 64: the fused forward
def test_linattn_norm_autograd_matches_oracle(d):
    m = _m()
    t = tapegen.linattn_tape(1, 800, 2, d, d, seed=tapegen.seed_for(1201 + d), mean=90.0, gamma_mode="head",
                             scale=1.0, normalize_k=False, with_grad=True)
    q, k, v = bf16_leaf(t["q"]), bf16_leaf(t["k"]), bf16_leaf(t["v"])
    gamma = dev(t["gamma"]).requires_grad_(True)
    y = m.LinAttnNormScan.apply(q, k, v, gamma, dev(t["start"]))
    (y * dev(t["grad_y"])).sum().backward()
    f = oracle.bf16_bits_to_f64
    ry, _, _, _ = oracle.linattn_norm_fwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"])
    rq, rk, rv, rg, _, _ = oracle.linattn_norm_bwd(f(t["q"]), f(t["k"]), f(t["v"]), t["gamma"], t["start"],
                                                   t["grad_y"])
    for name, got, ref in (("y", y, ry), ("dq", q.grad, rq), ("dk", k.grad, rk), ("dv", v.grad, rv),
                           ("dgamma", gamma.grad, rg)):
        assert rel_err(np32(got), ref) <= 2e-2, name


def test_ffm_autograd_matches_oracle():
    m = _m()
    t = tapegen.ffm_tape(2, 1500, 16, 4, tapegen.seed_for(1202), mean=100.0, with_S0=True)
    t["start"][:, 0] = 0
    x = dev(t["x"]).requires_grad_(True)
    alpha = dev(t["alpha"]).requires_grad_(True)
    omega = dev(t["omega"]).requires_grad_(True)
    S0 = dev(t["S0"]).requires_grad_(True)
    z = m.FFMScan.apply(x, alpha, omega, dev(t["start"]), S0)
    (z * dev(t["grad_z"])).sum().backward()
    rz, _ = oracle.ffm_fwd(t["alpha"], t["omega"], t["x"], t["start"], t["S0"])
    rgx, rga, rgo, rgS0 = oracle.ffm_bwd(t["alpha"], t["omega"], t["start"], rz, t["grad_z"], None, t["S0"])
    for name, got, ref in (("z", z, rz), ("grad_x", x.grad, rgx), ("grad_alpha", alpha.grad, rga),
                           ("grad_omega", omega.grad, rgo)):
        assert rel_err(got.detach().cpu().numpy(), ref) <= 1e-4, name
    assert rel_err(S0.grad.cpu().numpy(), rgS0) <= 1e-4


def test_two_layer_graph_backpropagates():
    # FFM output -> a linear map -> linear attention.  Each link of the chain
    # is checked on its own: the attention's gradients (returned in bf16, the
    # dtype of its inputs) against the oracle on the same bf16 operands at the
    # attention's 2e-2 bar; the gradient reaching z against those returned
    # gradients pushed through W by hand (fp64); and the gradient reaching x
    # against the FFM oracle's backward of that z gradient.
    m = _m()
    B, L, mm, c, H, d = 1, 600, 8, 2, 2, 64  # the tensor-core path takes d = 64 or 128
    tf = tapegen.ffm_tape(B, L, mm, c, tapegen.seed_for(1203), mean=80.0)
    rng = np.random.default_rng(tapegen.seed_for(1204))
    W = (rng.standard_normal((2 * mm * c, 3 * H * d)) / np.sqrt(2 * mm * c)).astype(np.float32)
    gamma = np.full(H, 0.97, dtype=np.float32)
    gy = rng.standard_normal((B, L, H, d)).astype(np.float32)
    x = dev(tf["x"]).requires_grad_(True)
    z = m.FFMScan.apply(x, dev(tf["alpha"]), dev(tf["omega"]), dev(tf["start"]), None)
    z.retain_grad()
    qkv = (z @ dev(W)).to(torch.bfloat16).view(B, L, 3, H, d)
    q, k, v = qkv[:, :, 0].contiguous(), qkv[:, :, 1].contiguous(), qkv[:, :, 2].contiguous()
    for a in (q, k, v):
        a.retain_grad()
    y = m.LinAttnScan.apply(q, k, v, dev(gamma), dev(tf["start"]), None)
    (y * dev(gy)).sum().backward()
    f = oracle.bf16_bits_to_f64

    def bits(t_):
        return t_.detach().cpu().view(torch.int16).numpy().view(np.uint16)

    rq, rk, rv, _, _ = oracle.linattn_bwd(f(bits(q)), f(bits(k)), f(bits(v)), gamma, tf["start"], gy)
    for name, got, ref in (("dq", q.grad, rq), ("dk", k.grad, rk), ("dv", v.grad, rv)):
        assert rel_err(np32(got), ref) <= 2e-2, name
    got_qkv = np.stack([np32(q.grad), np32(k.grad), np32(v.grad)], axis=2).astype(np.float64).reshape(B, L, 3 * H * d)
    assert rel_err(z.grad.cpu().numpy(), got_qkv @ W.astype(np.float64).T) <= 1e-5
    rz, _ = oracle.ffm_fwd(tf["alpha"], tf["omega"], tf["x"], tf["start"])
    rgx, _, _, _ = oracle.ffm_bwd(tf["alpha"], tf["omega"], tf["start"], rz, z.grad.cpu().numpy().astype(np.float64))
    assert rel_err(x.grad.cpu().numpy(), rgx) <= 1e-4
