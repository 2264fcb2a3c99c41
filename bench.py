"""Benchmark: resettable diagonal memoroid scan, forward + backward, on one
synthetic tape of L = 2^20 steps x D = 256 complex64 channels with
Geometric(500) episodes clipped to [1, 10000] (the tape-based batch of
Section 4.1 at GPU scale).

One step = memoroid_scan_diag_fwd + memoroid_scan_diag_bwd (with grad_lambda)
over the whole tape.  Prints one JSON line.  Its "linattn" object times the
decayed linear-attention memoroid on the largest linattn tape (L = 2^22,
8 heads, d = 128, per-step gamma, Geometric(1000) episodes): one step =
memoroid_scan_linattn_fwd + memoroid_scan_linattn_bwd, plus the tensor-core
throughput of the intra-tile contraction alone (memoroid_bench_linattn_intra).
Its "returns" object times the per-step discounted return and GAE with resets
on 64 tapes of 2^20 steps, its "ffm" object the Fast and Forgetful Memory
memoroid (fwd + bwd) on a 2^20-step tape with a 64 x 4 complex state, its
"tbb" object the device-side sampling of a 2^20-step batch (Algorithm 2) and
the gather of its 2 KB rows, and its "linattn_norm" object the paper's Linear
Transformer (phi = 1 + ELU, normalizer) fwd + bwd on the config-3 shape.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

--impl reference times the fp64 CPU oracle (the plain sequential definition)
on the host cores on a bounded sample of the same workload.
Under torchrun each rank scans its own tape (independent tapes are plain data
parallelism: no collective on the data path); rank 0 reports the max time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import tapegen  # noqa: E402

METRIC = "tape transitions/sec (fwd+bwd) and % of HBM / tensor roofline on 1 GB300"
UNIT = "transitions/s"
CFG = 2
WORKLOAD = ("diag scan fwd+bwd (grad_u, grad_lambda): B=1 tape, L=2^20 steps, D=256 complex64 "
            "channels, per-channel lambda, Geometric(500) episodes clipped to [1,10000]")
# algorithmic bytes per (step, channel): fwd reads u, writes h; bwd reads grad_h and h, writes grad_u
FWD_BYTES_PER_STEP_CH = 16
BWD_BYTES_PER_STEP_CH = 24
PROFILE_TRAFFIC = os.path.join(ROOT, "profiles", "diag_scan_traffic_L1M_D256.md")
LA_CFG = 5
LA_WORKLOAD = ("linattn fwd+bwd (dq, dk, dv, per-step dgamma): B=1 tape, L=2^22 steps, H=8 heads, d_k=d_v=128, "
               "bf16 q/k/v, per-step gamma=sigmoid(N(3,1)), Geometric(1000) episodes")
KERNEL_SRC = os.path.join(ROOT, "paper_2402_09900_gb300", "csrc", "diag_scan.cu")
DATASHEET_HBM_GBS = 7900.0  # nominal HBM3e bandwidth, printed beside the fraction of the measured peak
E2E_BLOCKS = 3  # end-to-end timing: blocks of --e2e-steps steps, the median reported


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(value, ws, device):
    """The largest `value` over the ranks of the job (its time is its slowest
    rank's); `value` itself for a single rank."""
    if ws <= 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ws, units_per_rank, ms_per_step):
    """Whole-job throughput: the units every rank processed in one step,
    divided by the step time (weak scaling: each rank has its own tape)."""
    return ws * units_per_rank / (ms_per_step / 1e3)


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _tensor_peaks():
    """(bf16 burst TFLOP/s, sustained TFLOP/s, kind)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 1900.0, 1700.0, "fallback"


RET_WORKLOAD = ("per-step discounted return and GAE with resets: B=64 tapes x L=2^20 steps (64 Mi steps), "
                "fp32 rewards and values, Geometric(200) episodes (and, *_single_episode, one episode per tape), "
                "gamma=0.99, lambda=0.95")


def returns_leg(args, m, dev, stream):
    """Times memoroid_discounted_return and memoroid_gae on 64 tapes of 2^20 steps."""
    import torch

    B, L = 64, 1 << 20
    rng = np.random.default_rng(tapegen.seed_for(6))
    start = np.stack([tapegen.geometric_tape_starts(rng, L, 200.0) for _ in range(B)])
    gen = torch.Generator(device=dev)
    gen.manual_seed(tapegen.seed_for(6))
    r = torch.randn((B, L), generator=gen, device=dev, dtype=torch.float32)
    v = torch.randn((B, L), generator=gen, device=dev, dtype=torch.float32)
    st = torch.from_numpy(start).to(dev)
    boot = torch.randn(B, generator=gen, device=dev, dtype=torch.float32)
    ws = m.workspace(m.memoroid_returns_workspace_bytes(B, L), dev)
    G = torch.empty_like(r)
    A = torch.empty_like(r)
    out = {"workload": RET_WORKLOAD}
    peak, peak_kind = _peaks()
    one = torch.zeros_like(st)  # one episode per tape: the reset-density extreme
    one[:, 0] = 1
    for name, fn, byts in (
            ("return", lambda: m.memoroid_discounted_return(r, st, 0.99, boot, G, B, L, ws, stream), B * L * 9 + B * 4),
            ("gae", lambda: m.memoroid_gae(r, v, st, 0.99, 0.95, boot, A, B, L, ws, stream), B * L * 13 + B * 4),
            ("return_single_episode", lambda: m.memoroid_discounted_return(r, one, 0.99, boot, G, B, L, ws, stream),
             B * L * 9 + B * 4),
            ("gae_single_episode", lambda: m.memoroid_gae(r, v, one, 0.99, 0.95, boot, A, B, L, ws, stream),
             B * L * 13 + B * 4)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.ret_steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / args.ret_steps
        gbs = byts / (ms * 1e-3) / 1e9
        out[name] = {"value": B * L / (ms * 1e-3), "unit": "steps/s", "ms": ms,
                     "roofline": {"bound": "hbm", "algorithmic_bytes_per_call": byts, "achieved": gbs, "unit": "GB/s",
                                  "peak": peak, "frac": gbs / peak, "peak_kind": f"{peak_kind} (copy bandwidth)"}}
    # one map launch and one scan launch per call (64 tapes: several ranges per tape)
    out["gpu_launches"] = 4 * 2 * args.ret_steps
    del r, v, G, A, ws
    torch.cuda.empty_cache()
    return out


FFM_WORKLOAD = ("Fast and Forgetful Memory memoroid fwd+bwd: B=1 tape x L=2^20 steps, m=64 trace x c=4 context "
                "(D=256 complex state), fp32, Geometric(500) episodes clipped to [1, 10000]")


def ffm_leg(args, m, dev, stream):
    """Times memoroid_ffm_fwd + memoroid_ffm_bwd (with the alpha / omega
    gradients) on one 2^20-step tape, m = 64, c = 4."""
    import torch

    B, L, mm, c = 1, (args.ffm_tape_steps or (1 << 20)), 64, 4
    D = mm * c
    small = tapegen.ffm_tape(B, 1, mm, c, tapegen.seed_for(7), with_grad=False)  # alpha, omega
    rng = np.random.default_rng(tapegen.seed_for(7))
    start = torch.from_numpy(np.stack([tapegen.geometric_tape_starts(rng, L, 500.0, 1, 10000)
                                       for _ in range(B)])).to(dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(tapegen.seed_for(7))
    x = torch.randn((B, L, mm), generator=gen, device=dev, dtype=torch.float32)
    gz = torch.randn((B, L, 2 * D), generator=gen, device=dev, dtype=torch.float32)
    alpha = torch.from_numpy(small["alpha"]).to(dev)
    omega = torch.from_numpy(small["omega"]).to(dev)
    ws = m.ffm_workspace(B, L, mm, c, dev)
    z = torch.empty((B, L, 2 * D), dtype=torch.float32, device=dev)
    gx = torch.empty_like(x)
    ga, go = torch.empty_like(alpha), torch.empty_like(omega)

    def fwd():
        m.memoroid_ffm_fwd(x, alpha, omega, start, None, z, None, B, L, mm, c, ws, stream)

    def bwd():
        m.memoroid_ffm_bwd(alpha, omega, start, None, z, gz, None, gx, ga, go, None, B, L, mm, c, ws, stream)

    for _ in range(3):
        fwd()
        bwd()
    torch.cuda.synchronize()
    steps = args.ffm_steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        evs[i][0].record(stream)
        fwd()
        evs[i][1].record(stream)
        bwd()
        evs[i][2].record(stream)
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the FFM timed region")
    f_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    b_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    # algorithmic bytes: fwd reads x~ (4 m) and the flag, writes z (8 D); bwd reads
    # grad_z and z (8 D each) and the flag, writes grad_x~ (4 m)
    fb = B * L * (4 * mm + 1 + 8 * D)
    bb = B * L * (16 * D + 1 + 4 * mm)
    peak, peak_kind = _peaks()
    kpc = (m.memoroid_ffm_kernels_per_call(B, L, mm, c, 0, 0) + m.memoroid_ffm_kernels_per_call(B, L, mm, c, 1, 1))
    out = {
        "workload": FFM_WORKLOAD if not args.ffm_tape_steps else f"{FFM_WORKLOAD} (first {L} steps only)",
        "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT, "steps": steps,
        "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms, "episodes": int(start.sum().item()),
        "roofline": {"bound": "hbm", "peak": peak, "unit": "GB/s", "peak_kind": f"{peak_kind} (copy bandwidth)",
                     "fwd": {"algorithmic_bytes_per_call": fb, "achieved": fb / (f_ms * 1e-3) / 1e9,
                             "frac": fb / (f_ms * 1e-3) / 1e9 / peak},
                     "bwd": {"algorithmic_bytes_per_call": bb, "achieved": bb / (b_ms * 1e-3) / 1e9,
                             "frac": bb / (b_ms * 1e-3) / 1e9 / peak},
                     "step_frac": (fb + bb) / ((f_ms + b_ms) * 1e-3) / 1e9 / peak},
        "gpu_launches": steps * kpc,
    }
    del x, gz, z, gx, ws
    torch.cuda.empty_cache()
    return out


LNORM_WORKLOAD = ("Linear Transformer with phi = 1 + ELU and its normalizer, fwd+bwd: B=1 tape x L=2^18 steps, "
                  "4 heads, d=64, bf16 q/k/v ~ N(0,1), per-head gamma in {0.9, 0.99, 0.999, 1.0}, Geometric(300) episodes")


PS_WORKLOAD = ("diag scan fwd+bwd with a per-step lambda (input-dependent decay): B=1 tape, L=2^20 steps, "
               "D=256 complex64 channels, |lambda_t| ~ U(0.9, 0.999), Geometric(500) episodes clipped to [1,10000]")


def per_step_leg(args, m, dev, stream):
    """Times the diagonal scan with a per-step lambda ([B, L, D], grad_lambda per
    step) on the bench tape's shape."""
    import torch

    B, L, D = 1, 1 << 20, 256
    gen = torch.Generator(device=dev)
    gen.manual_seed(tapegen.seed_for(10))
    mag = 0.9 + 0.099 * torch.rand((B, L, D), generator=gen, device=dev)
    ph = 2 * np.pi * torch.rand((B, L, D), generator=gen, device=dev)
    lam = torch.polar(mag, ph).to(torch.complex64)
    u = torch.randn((B, L, D), generator=gen, device=dev, dtype=torch.complex64)
    g = torch.randn((B, L, D), generator=gen, device=dev, dtype=torch.complex64)
    rng = np.random.default_rng(tapegen.seed_for(10))
    st = torch.from_numpy(tapegen.geometric_tape_starts(rng, L, 500.0, 1, 10000)[None]).to(dev)
    h, gu, gl = torch.empty_like(u), torch.empty_like(u), torch.empty_like(lam)
    ws = m.diag_workspace(B, L, D, dev)

    def fwd():
        m.memoroid_scan_diag_fwd(lam, 1, u, st, None, h, None, B, L, D, ws, stream)

    def bwd():
        m.memoroid_scan_diag_bwd(lam, 1, st, None, h, g, None, gu, gl, None, B, L, D, ws, stream)

    for _ in range(3):
        fwd()
        bwd()
    torch.cuda.synchronize()
    steps = args.ps_steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        evs[i][0].record(stream)
        fwd()
        evs[i][1].record(stream)
        bwd()
        evs[i][2].record(stream)
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the per-step lambda leg")
    f_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    b_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    # fwd reads u and lambda, writes h; bwd reads grad_h, h and lambda, writes grad_u and grad_lambda
    fb = B * L * D * 24 + B * L
    bb = B * L * D * 40 + B * L
    peak, peak_kind = _peaks()
    kpc = (m.memoroid_scan_diag_kernels_per_call(B, L, D, 1, 0, 0) + m.memoroid_scan_diag_kernels_per_call(B, L, D, 1, 1, 1))
    out = {"workload": PS_WORKLOAD, "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT, "steps": steps,
           "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms,
           "roofline": {"bound": "hbm", "peak": peak, "unit": "GB/s", "peak_kind": f"{peak_kind} (copy bandwidth)",
                        "fwd": {"algorithmic_bytes_per_call": fb, "achieved": fb / (f_ms * 1e-3) / 1e9,
                                "frac": fb / (f_ms * 1e-3) / 1e9 / peak},
                        "bwd": {"algorithmic_bytes_per_call": bb, "achieved": bb / (b_ms * 1e-3) / 1e9,
                                "frac": bb / (b_ms * 1e-3) / 1e9 / peak},
                        "step_frac": (fb + bb) / ((f_ms + b_ms) * 1e-3) / 1e9 / peak},
           "gpu_launches": steps * kpc}
    del lam, u, g, h, gu, gl, ws
    torch.cuda.empty_cache()
    return out


CFG3_WORKLOAD = ("linattn fwd+bwd (dq, dk, dv, per-head dgamma): B=1 tape, L=2^18 steps, H=4 heads, d_k=d_v=64, "
                 "bf16 q/k/v (k L2-normalised), gamma per head in {0.9, 0.99, 0.999, 1.0}, Geometric(300) "
                 "episodes, chunk 64")
CFG4_WORKLOAD = ("diag scan fwd+bwd (grad_u, grad_lambda): B=64 tapes x L=16384 steps, D=128 complex64 channels, "
                 "tapes 0-31 Geometric(20) episodes, tapes 32-63 one episode each")


def _timed_pair(fwd, bwd, steps, stream):
    """Mean milliseconds of fwd and bwd over `steps` back-to-back pairs (CUDA
    events on `stream`, after 3 untimed pairs)."""
    import torch

    for _ in range(3):
        fwd()
        bwd()
    torch.cuda.synchronize()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        evs[i][0].record(stream)
        fwd()
        evs[i][1].record(stream)
        bwd()
        evs[i][2].record(stream)
    torch.cuda.synchronize()
    f_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    b_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    return f_ms, b_ms


def _hbm_roofline(fb, bb, f_ms, b_ms):
    peak, peak_kind = _peaks()
    return {"bound": "hbm", "peak": peak, "unit": "GB/s", "peak_kind": f"{peak_kind} (copy bandwidth)",
            "fwd": {"algorithmic_bytes_per_call": fb, "achieved": fb / (f_ms * 1e-3) / 1e9,
                    "frac": fb / (f_ms * 1e-3) / 1e9 / peak},
            "bwd": {"algorithmic_bytes_per_call": bb, "achieved": bb / (b_ms * 1e-3) / 1e9,
                    "frac": bb / (b_ms * 1e-3) / 1e9 / peak},
            "step_frac": (fb + bb) / ((f_ms + b_ms) * 1e-3) / 1e9 / peak}


def linattn_cfg3_leg(args, m, dev, stream):
    """Times the linear-attention memoroid (fwd, bwd with per-head dgamma) on the
    L = 2^18, 4-head, d = 64 tape with per-head decays."""
    import torch

    c = tapegen.LINATTN_CONFIGS[3]
    B, L, H, d = c["B"], c["L"], c["H"], c["d"]
    t = tapegen.linattn_tape_device(B, L, H, d, tapegen.seed_for(3), c["mean"], c["gamma"], device=dev)
    ws = m.linattn_workspace(B, L, H, d, dev)
    y = torch.empty((B, L, H, d), dtype=torch.float32, device=dev)
    dq, dk, dv = torch.empty_like(y), torch.empty_like(y), torch.empty_like(y)
    dg = torch.empty_like(t["gamma"])

    def fwd():
        m.memoroid_scan_linattn_fwd(t["q"], t["k"], t["v"], m.MEMOROID_BF16, t["gamma"], 0, t["start"], None, y,
                                    None, B, L, H, d, d, c["chunk"], ws, stream)

    def bwd():
        m.memoroid_scan_linattn_bwd(t["q"], t["k"], t["v"], m.MEMOROID_BF16, t["gamma"], 0, t["start"], None,
                                    t["grad_y"], None, dq, dk, dv, dg, None, B, L, H, d, d, c["chunk"], ws, stream)

    f_ms, b_ms = _timed_pair(fwd, bwd, args.cfg3_steps, stream)
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the config-3 linattn leg")
    el = B * L * H * d
    fb = el * (3 * 2 + 4) + H * 4 + B * L
    bb = el * (3 * 2 + 4 + 3 * 4) + H * 8 + B * L
    kpc = (m.memoroid_scan_linattn_kernels_per_call(B, L, H, d, d, 0, 0)
           + m.memoroid_scan_linattn_kernels_per_call(B, L, H, d, d, 1, 1))
    out = {"workload": CFG3_WORKLOAD, "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT,
           "steps": args.cfg3_steps, "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms,
           "episodes": int(t["start"].sum().item()), "roofline": _hbm_roofline(fb, bb, f_ms, b_ms),
           "l2": "q, k, v 32 MiB each, y and gradients 64 MiB each: the working set of a call (0.67 / 1.48 GB) "
                 "exceeds the 129 MB L2",
           "gpu_launches": args.cfg3_steps * kpc}
    del t, y, dq, dk, dv, ws
    torch.cuda.empty_cache()
    return out


def diag_cfg4_leg(args, m, dev, stream):
    """Times the diagonal scan (fwd, bwd with grad_lambda) on 64 tapes of 16384
    steps at D = 128: half the tapes with short Geometric(20) episodes, half
    one episode each (the extremes of reset density)."""
    import torch

    B, L, D = 64, 16384, 128
    gen = torch.Generator(device=dev)
    gen.manual_seed(tapegen.seed_for(4))
    mag = 0.9 + 0.099 * torch.rand((D,), generator=gen, device=dev)
    ph = 2 * np.pi * torch.rand((D,), generator=gen, device=dev)
    lam = torch.polar(mag, ph).to(torch.complex64)
    u = torch.randn((B, L, D), generator=gen, device=dev, dtype=torch.complex64)
    g = torch.randn((B, L, D), generator=gen, device=dev, dtype=torch.complex64) * np.sqrt(2.0)
    rng = np.random.default_rng(tapegen.seed_for(4))
    st_np = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        if b < B // 2:
            st_np[b] = tapegen.geometric_tape_starts(rng, L, 20.0)
        else:
            st_np[b, 0] = 1
    st = torch.from_numpy(st_np).to(dev)
    h, gu, gl = torch.empty_like(u), torch.empty_like(u), torch.empty_like(lam)
    ws = m.diag_workspace(B, L, D, dev)

    def fwd():
        m.memoroid_scan_diag_fwd(lam, 0, u, st, None, h, None, B, L, D, ws, stream)

    def bwd():
        m.memoroid_scan_diag_bwd(lam, 0, st, None, h, g, None, gu, gl, None, B, L, D, ws, stream)

    f_ms, b_ms = _timed_pair(fwd, bwd, args.cfg4_steps, stream)
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the config-4 diag leg")
    fb = B * L * D * FWD_BYTES_PER_STEP_CH + B * L
    bb = B * L * D * BWD_BYTES_PER_STEP_CH + B * L
    kpc = (m.memoroid_scan_diag_kernels_per_call(B, L, D, 0, 0, 0)
           + m.memoroid_scan_diag_kernels_per_call(B, L, D, 0, 1, 1))
    out = {"workload": CFG4_WORKLOAD, "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT,
           "steps": args.cfg4_steps, "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms,
           "fwd_value": B * L / (f_ms * 1e-3), "episodes": int(st_np.sum()),
           "roofline": _hbm_roofline(fb, bb, f_ms, b_ms),
           "l2": "inputs 1 GiB per tensor vs 129 MB L2; no flush needed",
           "gpu_launches": args.cfg4_steps * kpc}
    del lam, u, g, h, gu, gl, ws
    torch.cuda.empty_cache()
    return out


def lnorm_leg(args, m, dev, stream):
    """Times memoroid_linattn_norm_fwd + _bwd on the config-3 shape."""
    import torch

    B, L, H, d = 1, 1 << 18, 4, 64
    t = tapegen.linattn_tape(B, L, H, d, d, tapegen.seed_for(9), mean=300.0, gamma_mode="head", scale=1.0,
                             normalize_k=False)

    def bits(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev)

    q, k, v = bits(t["q"]), bits(t["k"]), bits(t["v"])
    gamma, start = torch.from_numpy(t["gamma"]).to(dev), torch.from_numpy(t["start"]).to(dev)
    dy = torch.from_numpy(t["grad_y"]).to(dev)
    ws = m.workspace(m.memoroid_linattn_norm_workspace_bytes(B, L, H, d), dev)
    y = torch.empty((B, L, H, d), dtype=torch.float32, device=dev)
    den = torch.empty((B, L, H), dtype=torch.float32, device=dev)
    dq, dk, dv = torch.empty_like(y), torch.empty_like(y), torch.empty_like(y)
    dg = torch.empty_like(gamma)

    def fwd():
        m.memoroid_linattn_norm_fwd(q, k, v, gamma, 0, start, None, None, y, den, None, None, B, L, H, d, ws, stream)

    def bwd():
        m.memoroid_linattn_norm_bwd(q, k, v, gamma, 0, start, None, None, y, den, dy, None, None, dq, dk, dv, dg,
                                    None, None, B, L, H, d, ws, stream)

    for _ in range(3):
        fwd()
        bwd()
    torch.cuda.synchronize()
    steps = args.lnorm_steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        evs[i][0].record(stream)
        fwd()
        evs[i][1].record(stream)
        bwd()
        evs[i][2].record(stream)
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the normalised linattn leg")
    f_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    b_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    el = B * L * H * d
    # algorithmic bytes: fwd reads q, k, v (bf16) and the flags, writes y and den; bwd reads
    # q, k, v, y, den, dy and the flags, writes dq, dk, dv
    fb = el * (3 * 2 + 4) + B * L * H * 4 + B * L
    bb = el * (3 * 2 + 4 + 4 + 3 * 4) + B * L * H * 4 + B * L
    peak, peak_kind = _peaks()
    kpc = (m.memoroid_linattn_norm_kernels_per_call(B, L, H, d, 0, 0, 0)
           + m.memoroid_linattn_norm_kernels_per_call(B, L, H, d, 1, 0, 0))
    out = {"workload": LNORM_WORKLOAD, "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT, "steps": steps,
           "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms,
           "roofline": {"bound": "hbm", "peak": peak, "unit": "GB/s", "peak_kind": f"{peak_kind} (copy bandwidth)",
                        "fwd": {"algorithmic_bytes_per_call": fb, "achieved": fb / (f_ms * 1e-3) / 1e9,
                                "frac": fb / (f_ms * 1e-3) / 1e9 / peak},
                        "bwd": {"algorithmic_bytes_per_call": bb, "achieved": bb / (b_ms * 1e-3) / 1e9,
                                "frac": bb / (b_ms * 1e-3) / 1e9 / peak}},
           "gpu_launches": steps * kpc}
    del q, k, v, y, dq, dk, dv, ws
    torch.cuda.empty_cache()
    return out


TBB_WORKLOAD = ("tape-based batching (Algorithm 2): a batch of B=2^20 steps sampled from a buffer of N=2^21 "
                "transitions with Geometric(500) episodes, rows of 256 complex64 channels (2 KB) gathered into the tape")


def tbb_leg(args, m, dev, stream):
    """Times memoroid_tbb_sample (flags and source indices of the batch) and
    memoroid_gather_rows (the batch's 2 KB rows) on the bench buffer."""
    import torch

    N, B, D = 1 << 21, 1 << 20, 256
    rng = np.random.default_rng(tapegen.seed_for(8))
    begin = torch.from_numpy(np.flatnonzero(tapegen.geometric_tape_starts(rng, N, 500.0))).to(dev)
    E = begin.numel()
    draws = torch.from_numpy(rng.integers(0, E, size=B // 100)).to(dev)  # ~2100 draws are used
    K = draws.numel()
    gen = torch.Generator(device=dev)
    gen.manual_seed(tapegen.seed_for(8))
    rows = torch.randn((N, 2 * D), generator=gen, device=dev, dtype=torch.float32)
    ws = m.workspace(m.memoroid_tbb_workspace_bytes(K), dev)
    start = torch.empty(B, dtype=torch.uint8, device=dev)
    src = torch.empty(B, dtype=torch.int64, device=dev)
    n_used = torch.empty(1, dtype=torch.int64, device=dev)
    out = torch.empty((B, 2 * D), dtype=torch.float32, device=dev)
    row_bytes = 2 * D * 4

    def sample():
        m.memoroid_tbb_sample(begin, E, N, draws, K, B, start, src, n_used, ws, stream)

    def gather():
        m.memoroid_gather_rows(rows, N, row_bytes, src, B, out, ws, stream)

    res = {"workload": TBB_WORKLOAD}
    peak, peak_kind = _peaks()
    for name, fn, byts in (("sample", sample, B * 9), ("gather", gather, B * (8 + 2 * row_bytes))):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.tbb_steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / args.tbb_steps
        gbs = byts / (ms * 1e-3) / 1e9
        res[name] = {"ms": ms, "value": B / (ms * 1e-3), "unit": "steps/s",
                     "roofline": {"bound": "hbm", "algorithmic_bytes_per_call": byts, "achieved": gbs, "unit": "GB/s",
                                  "peak": peak, "frac": gbs / peak, "peak_kind": f"{peak_kind} (copy bandwidth)"}}
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side data check failed in the TBB leg")
    res["draws_used"] = int(n_used.item())
    res["gpu_launches"] = args.tbb_steps * 3  # offsets + fill, gather
    del rows, out
    torch.cuda.empty_cache()
    return res


def linattn_leg(args, m, dev, stream):
    """Times the linear-attention memoroid (fwd + bwd) on the L = 2^22, 8-head,
    d = 128 tape, and the intra-tile contraction alone."""
    import torch

    c = tapegen.LINATTN_CONFIGS[LA_CFG]
    B, L, H, d = c["B"], c["L"], c["H"], c["d"]
    if args.la_tape_steps:
        L = args.la_tape_steps  # a shorter tape of the same workload (profiler captures)
    t = tapegen.linattn_tape_device(B, L, H, d, tapegen.seed_for(LA_CFG), c["mean"], c["gamma"], device=dev)
    if args.la_single_gamma1:
        # profiling mode: the timed steps run one episode per tape with gamma = 1
        t["start"].zero_()
        t["start"][:, 0] = 1
        t["gamma"].fill_(1.0)
    per = 1 if t["gamma"].dim() == 3 else 0
    ws = m.linattn_workspace(B, L, H, d, dev)
    y = torch.empty((B, L, H, d), dtype=torch.float32, device=dev)
    dq, dk, dv = torch.empty_like(y), torch.empty_like(y), torch.empty_like(y)
    dg = torch.empty_like(t["gamma"])

    def fwd(start=t["start"], gamma=t["gamma"]):
        m.memoroid_scan_linattn_fwd(t["q"], t["k"], t["v"], m.MEMOROID_BF16, gamma, per, start, None, y,
                                    None, B, L, H, d, d, c["chunk"], ws, stream)

    def bwd(start=t["start"], gamma=t["gamma"]):
        m.memoroid_scan_linattn_bwd(t["q"], t["k"], t["v"], m.MEMOROID_BF16, gamma, per, start, None,
                                    t["grad_y"], None, dq, dk, dv, dg, None, B, L, H, d, d, c["chunk"], ws, stream)

    for _ in range(args.la_warmup):
        fwd()
        bwd()
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the linattn warm-up")
    steps = args.la_steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        evs[i][0].record(stream)
        fwd()
        evs[i][1].record(stream)
        bwd()
        evs[i][2].record(stream)
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the linattn timed region")
    f_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / steps
    b_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / steps
    el = B * L * H * d
    # algorithmic bytes: fwd reads q, k, v (bf16), gamma, start and writes y (fp32);
    # bwd reads q, k, v, gamma, start, dy and writes dq, dk, dv, dgamma
    fb = el * (3 * 2 + 4) + t["gamma"].numel() * 4 + B * L
    bb = el * (3 * 2 + 4 + 3 * 4) + t["gamma"].numel() * 8 + B * L
    peak, peak_kind = _peaks()
    kpc = (m.memoroid_scan_linattn_kernels_per_call(B, L, H, d, d, 0, 0)
           + m.memoroid_scan_linattn_kernels_per_call(B, L, H, d, d, 1, 0))

    # the intra-tile contraction alone, operands resident in shared memory
    scratch = m.workspace(m.memoroid_bench_linattn_intra_scratch_bytes(d), dev)
    scratch.random_(0, 256)
    reps, ctas = args.la_intra_reps, 152
    m.memoroid_bench_linattn_intra(d, reps, ctas, scratch, stream)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    m.memoroid_bench_linattn_intra(d, reps, ctas, scratch, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(scratch) != m.MEMOROID_OK:
        raise RuntimeError("device-side error in the intra-tile benchmark")
    i_ms = e0.elapsed_time(e1)
    i_tf = ctas * reps * 4 * 128 * 128 * d / (i_ms * 1e-3) / 1e12
    burst, sustained, tkind = _tensor_peaks()

    # the same tape with a single begin flag (t = 0): one episode, the extreme of
    # reset density; with the workload's decays and with gamma = 1 (no decay, so
    # every state reaches across the whole tape)
    one = torch.zeros_like(t["start"])
    one[:, 0] = 1
    sparse = {}
    for name, gam in (("workload_gamma", t["gamma"]), ("gamma_1", torch.ones_like(t["gamma"]))):
        sf, sb = _timed_pair(lambda: fwd(one, gam), lambda: bwd(one, gam), steps, stream)
        if m.memoroid_get_device_error(ws) != m.MEMOROID_OK:
            raise RuntimeError("device-side error in the single-episode linattn steps")
        sparse[name] = {"fwd_ms": sf, "bwd_ms": sb, "ms_per_step": sf + sb,
                        "vs_workload_step": (sf + sb) / (f_ms + b_ms),
                        "value": B * L / ((sf + sb) * 1e-3)}
    out = {
        "workload": LA_WORKLOAD if not args.la_tape_steps else f"{LA_WORKLOAD} (first {L} steps only)",
        "value": B * L / ((f_ms + b_ms) * 1e-3), "unit": UNIT, "steps": steps,
        "ms_per_step": f_ms + b_ms, "fwd_ms": f_ms, "bwd_ms": b_ms,
        "episodes": int(t["start"].sum().item()),
        "single_episode": sparse,
        "roofline": {"bound": "hbm", "peak": peak, "unit": "GB/s", "peak_kind": f"{peak_kind} (copy bandwidth)",
                     "fwd": {"algorithmic_bytes_per_call": fb, "achieved": fb / (f_ms * 1e-3) / 1e9,
                             "frac": fb / (f_ms * 1e-3) / 1e9 / peak},
                     "bwd": {"algorithmic_bytes_per_call": bb, "achieved": bb / (b_ms * 1e-3) / 1e9,
                             "frac": bb / (b_ms * 1e-3) / 1e9 / peak},
                     "step_frac": (fb + bb) / ((f_ms + b_ms) * 1e-3) / 1e9 / peak},
        "intra_chunk_tensor": {"bound": "tensor", "achieved": i_tf, "unit": "TFLOP/s", "peak": burst,
                               "frac": i_tf / burst, "frac_of_sustained": i_tf / sustained,
                               "peak_kind": f"{tkind} bf16 dense (burst; sustained {sustained})",
                               "ms": i_ms, "ctas": ctas, "reps": reps,
                               "flops": ctas * reps * 4 * 128 * 128 * d,
                               "what": "P = Q K^T (128x128x128) and Y = Pm V (128x128x128) per rep, tcgen05 "
                                       "kind::f16 bf16->fp32, operands resident in shared memory"},
        "gpu_launches": 3 * steps * kpc + 2,  # timed: the workload and the two single-episode cases, the microbenchmark
    }
    del t, y, dq, dk, dv, ws
    torch.cuda.empty_cache()
    return out


def _traffic_record():
    """(bytes per launch at the bench size, note) from the committed ncu
    summary, or (None, why) if the kernel source changed since."""
    try:
        rec = {}
        with open(PROFILE_TRAFFIC) as f:
            for line in f:
                if ":" in line and not line.startswith(("#", "|", " ")):
                    k, v = line.split(":", 1)
                    rec[k.strip()] = v.strip()
        src = hashlib.sha256(open(KERNEL_SRC, "rb").read()).hexdigest()
        if rec.get("source_sha256") != src:
            return None, "kernel changed since the ncu capture"
        return float(rec["traffic_bytes_per_launch_at_bench_size"]), rec.get("note", "")
    except Exception as e:  # no capture yet
        return None, f"no ncu capture ({type(e).__name__})"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu), "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------

def oracle_sample(t, steps):
    """A bounded sample of the workload: the first `steps` steps of the tape."""
    return {"lam": t["lam"], "u": t["u"][:, :steps], "start": t["start"][:, :steps],
            "grad_h": t["grad_h"][:, :steps]}


def time_oracle_step(sample):
    import oracle
    t0 = time.perf_counter()
    h, _ = oracle.diag_fwd(sample["lam"], sample["u"], sample["start"])
    oracle.diag_bwd(sample["lam"], sample["start"], h, sample["grad_h"])
    return time.perf_counter() - t0


def _calibrate(t):
    """Seconds per transition of the oracle (fwd+bwd), from a short warm run."""
    probe = min(t["L"], 32768)
    time_oracle_step(oracle_sample(t, 1024))  # page-in, thread pool start
    return time_oracle_step(oracle_sample(t, probe)) / probe


def cpu_baseline(t, target_s):
    """The oracle timed on about `target_s` seconds of the workload's first steps."""
    import oracle
    oracle.build()
    per = _calibrate(t)
    steps = int(min(t["L"], max(4096, target_s / per)))
    s = oracle_sample(t, steps)
    dt = time_oracle_step(s)
    B = s["u"].shape[0]
    # the same oracle on one thread, on a tenth of the sample
    cores = oracle.max_threads()
    steps1 = max(1024, steps // 10)
    oracle.set_threads(1)
    try:
        dt1 = time_oracle_step(oracle_sample(t, steps1))
    finally:
        oracle.set_threads(cores)
    return {"value": B * steps / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_thread_value": B * steps1 / dt1,
            "sample": f"first {steps} steps of the tape (x {s['u'].shape[2]} channels), fwd+bwd incl. "
                      f"grad_lambda, fp64 C oracle with OpenMP over channels; {dt:.2f} s "
                      f"(one thread: first {steps1} steps, {dt1:.2f} s)"}


def linattn_cpu_baseline(target_steps):
    """The linear-attention oracle (fwd+bwd with per-step dgamma) on the first
    whole episodes of the linattn tape reaching `target_steps` steps, on the host
    cores: transitions (steps) per second."""
    import oracle
    oracle.build()
    c = tapegen.LINATTN_CONFIGS[LA_CFG]
    rng = np.random.default_rng(tapegen.seed_for(LA_CFG))
    starts = tapegen.geometric_tape_starts(rng, 4 * target_steps, c["mean"])
    heads = np.flatnonzero(starts)
    n = int(heads[np.searchsorted(heads, target_steps)]) if heads[-1] >= target_steps else len(starts)
    t = tapegen.linattn_tape(1, n, c["H"], c["d"], c["d"], tapegen.seed_for(LA_CFG), mean=c["mean"],
                             gamma_mode="step")
    f = oracle.bf16_bits_to_f64
    q, k, v = f(t["q"]), f(t["k"]), f(t["v"])
    t0 = time.perf_counter()
    oracle.linattn_fwd(q, k, v, t["gamma"], t["start"])
    oracle.linattn_bwd(q, k, v, t["gamma"], t["start"], t["grad_y"])
    dt = time.perf_counter() - t0
    return {"value": n / dt, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "sample": f"{n} steps of whole episodes (the workload's recipe: {c['H']} heads, d={c['d']}, "
                      f"per-step gamma, Geometric({c['mean']:.0f})), fwd+bwd incl. per-step dgamma, "
                      f"fp64 C oracle with OpenMP over heads; {dt:.2f} s"}


def run_reference(args):
    """The reference arm: the oracle on the host cores, each step a bounded
    sample of the tape sized so that all steps take about --ref-seconds."""
    ws, rank, _ = _dist_env()
    if rank != 0:
        return
    import oracle
    oracle.build()
    t = tapegen.diag_config(CFG)
    per = _calibrate(t)
    # at most 2^18 steps per step: the oracle's rate is flat well below that, and
    # its fp64 copies of a sample stay near 1 GB whatever --steps is
    steps = int(min(t["L"], 1 << 18, max(1024, args.ref_seconds / max(args.steps, 1) / per)))
    s = oracle_sample(t, steps)
    for _ in range(args.warmup):
        time_oracle_step(oracle_sample(t, min(steps, 1024)))
    times = [time_oracle_step(s) for _ in range(args.steps)]
    dt = sum(times) / len(times)
    value = t["B"] * steps / dt
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "B": t["B"], "L": t["L"], "D": t["D"],
                   "sample_steps_per_step": steps},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
                         "sample": f"first {steps} steps x {t['D']} channels per step, fwd+bwd incl. "
                                   f"grad_lambda, fp64 C oracle"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def run_ours(args):
    import torch
    import torch.distributed as dist

    ws, rank, local = _dist_env()
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2402_09900_gb300 import build as native_build
    native_build.build()
    from paper_2402_09900_gb300 import memoroid as m
    m.load()
    if args.only_linattn:
        # profiling mode: the linattn leg alone (no diag step, no JSON contract line)
        print(json.dumps({"linattn": linattn_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_returns:
        # profiling mode: the discounted-return / GAE leg alone
        print(json.dumps({"returns": returns_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_lnorm:
        # profiling mode: the normalised Linear Transformer leg alone
        print(json.dumps({"linattn_norm": lnorm_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_per_step:
        # profiling mode: the per-step lambda diag leg alone
        print(json.dumps({"diag_per_step_lambda": per_step_leg(args, m, dev, torch.cuda.current_stream())}),
              flush=True)
        return
    if args.only_tbb:
        # profiling mode: the tape-based batching leg alone
        print(json.dumps({"tbb": tbb_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_ffm:
        # profiling mode: the Fast and Forgetful Memory leg alone
        print(json.dumps({"ffm": ffm_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_cfg3:
        # profiling mode: the L=2^18, 4-head, d=64 linattn leg alone
        print(json.dumps({"linattn_cfg3": linattn_cfg3_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return
    if args.only_cfg4:
        # profiling mode: the 64-tape, D=128 diag leg alone
        print(json.dumps({"diag_cfg4": diag_cfg4_leg(args, m, dev, torch.cuda.current_stream())}), flush=True)
        return

    t = tapegen.diag_config(CFG)
    if args.tape_steps:
        # a shorter tape of the same workload (used for profiler captures)
        t = {k: (v[:, :args.tape_steps] if k in ("u", "start", "grad_h") else v) for k, v in t.items()}
        t["L"] = args.tape_steps
    B, L, D = t["B"], t["L"], t["D"]
    lam = torch.from_numpy(t["lam"]).to(dev)
    u = torch.from_numpy(t["u"]).to(dev)
    start = torch.from_numpy(t["start"]).to(dev)
    grad_h = torch.from_numpy(t["grad_h"]).to(dev)
    h = torch.empty_like(u)
    grad_u = torch.empty_like(u)
    grad_lam = torch.empty_like(lam)
    wsb = m.memoroid_scan_diag_workspace_bytes(B, L, D)
    work = m.workspace(wsb, dev)
    stream = torch.cuda.current_stream()

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, B, L, D, work, stream)
        if ev is not None:
            ev[1].record(stream)
        m.memoroid_scan_diag_bwd(lam, 0, start, None, h, grad_h, None, grad_u, grad_lam, None, B, L, D,
                                 work, stream)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if m.memoroid_get_device_error(work) != m.MEMOROID_OK:
        raise RuntimeError("device-side error during warm-up")

    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    ids = [x for x in vis.split(",") if x.strip()]
    smi_index = int(ids[local]) if len(ids) > local and ids[local].strip().isdigit() else local
    sampler = ClockSampler(smi_index)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    t_begin = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)  # let the sampler attach
    t_begin.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    if ws > 1:
        dist.barrier()
    if m.memoroid_get_device_error(work) != m.MEMOROID_OK:
        raise RuntimeError("device-side error during the timed region")
    elapsed_ms = max_over_ranks(t_begin.elapsed_time(t_end), ws, dev)
    fwd_ms = [e[0].elapsed_time(e[1]) for e in evs]
    bwd_ms = [e[1].elapsed_time(e[2]) for e in evs]
    ms_per_step = elapsed_ms / args.steps
    value = job_throughput(ws, B * L, ms_per_step)

    # ---- end to end through the C ABI with pinned host buffers ----
    e2e = None
    if args.e2e_steps > 0:
        hu = torch.from_numpy(t["u"]).pin_memory()
        hg = torch.from_numpy(t["grad_h"]).pin_memory()
        hs = torch.from_numpy(t["start"]).pin_memory()
        hl = torch.from_numpy(t["lam"]).pin_memory()
        oh = torch.empty(h.shape, dtype=h.dtype).pin_memory()
        ogu = torch.empty(grad_u.shape, dtype=grad_u.dtype).pin_memory()
        ogl = torch.empty(grad_lam.shape, dtype=grad_lam.dtype).pin_memory()
        h2d = sum(x.numel() * x.element_size() for x in (hu, hg, hs, hl))
        d2h = sum(x.numel() * x.element_size() for x in (oh, ogu, ogl))

        # Copies run on their own streams so that the two directions overlap each
        # other and the kernels: inputs go up on s_in, results come down on s_out,
        # the scans run on `stream`; every buffer is reused only after the last
        # reader or writer of the previous step is done with it (events).
        s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
        ev = {k: torch.cuda.Event() for k in ("u_in", "g_in", "fwd", "bwd", "h_out", "gu_out")}
        for e in ev.values():
            e.record(stream)

        def e2e_step():
            with torch.cuda.stream(s_in):
                s_in.wait_event(ev["fwd"])  # the previous forward has read u
                u.copy_(hu, non_blocking=True)
                s_in.wait_event(ev["bwd"])  # the previous backward has read start, lambda, grad_h
                start.copy_(hs, non_blocking=True)
                lam.copy_(hl, non_blocking=True)
                ev["u_in"].record(s_in)
                grad_h.copy_(hg, non_blocking=True)
                ev["g_in"].record(s_in)
            stream.wait_event(ev["u_in"])
            stream.wait_event(ev["h_out"])  # h of the previous step is on the host
            m.memoroid_scan_diag_fwd(lam, 0, u, start, None, h, None, B, L, D, work, stream)
            ev["fwd"].record(stream)
            stream.wait_event(ev["g_in"])
            stream.wait_event(ev["gu_out"])  # grad_u / grad_lambda of the previous step are on the host
            m.memoroid_scan_diag_bwd(lam, 0, start, None, h, grad_h, None, grad_u, grad_lam, None, B, L, D,
                                     work, stream)
            ev["bwd"].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev["fwd"])
                oh.copy_(h, non_blocking=True)
                ev["h_out"].record(s_out)
                s_out.wait_event(ev["bwd"])
                ogu.copy_(grad_u, non_blocking=True)
                ogl.copy_(grad_lam, non_blocking=True)
                ev["gu_out"].record(s_out)

        # the host link's floor for a step: the same host->device and device->host copies on
        # two streams with no ordering between them and no scans; the link of a shared host
        # varies from second to second, so the floor is taken before and after the timed
        # end-to-end steps and the faster of the two is reported
        def copies_only():
            with torch.cuda.stream(s_in):
                for dst, src in ((u, hu), (start, hs), (lam, hl), (grad_h, hg)):
                    dst.copy_(src, non_blocking=True)
            with torch.cuda.stream(s_out):
                for dst, src in ((oh, h), (ogu, grad_u), (ogl, grad_lam)):
                    dst.copy_(src, non_blocking=True)

        def floor_ms():
            copies_only()
            torch.cuda.synchronize()
            c0 = time.perf_counter()
            for _ in range(args.e2e_steps):
                copies_only()
            torch.cuda.synchronize()
            return max_over_ranks((time.perf_counter() - c0) * 1e3 / args.e2e_steps, ws, dev)

        c_before = floor_ms()
        e2e_step()
        torch.cuda.synchronize()
        # E2E_BLOCKS blocks of e2e_steps steps; the median block is reported (the shared
        # host's link and memory bandwidth vary from second to second) beside all blocks
        blocks = []
        for _ in range(E2E_BLOCKS):
            if ws > 1:
                dist.barrier()
            e0 = time.perf_counter()
            for _ in range(args.e2e_steps):
                e2e_step()
            torch.cuda.synchronize()
            blocks.append(max_over_ranks((time.perf_counter() - e0) * 1e3 / args.e2e_steps, ws, dev))
        e_ms = sorted(blocks)[len(blocks) // 2]
        c_ms = min(c_before, floor_ms())
        e2e = {"value": job_throughput(ws, B * L, e_ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": args.e2e_steps, "ms_per_step": e_ms,
               "blocks_ms_per_step": blocks, "timing": f"median of {E2E_BLOCKS} blocks of {args.e2e_steps} steps",
               "link_floor_ms_per_step": c_ms, "link_floor_GBps": (h2d + d2h) / c_ms / 1e6}

    if rank != 0:
        if ws > 1:
            dist.destroy_process_group()
        return

    peak, peak_kind = _peaks()
    fwd_bytes = B * L * D * FWD_BYTES_PER_STEP_CH + B * L
    bwd_bytes = B * L * D * BWD_BYTES_PER_STEP_CH + B * L
    fwd_avg = sum(fwd_ms) / len(fwd_ms)
    bwd_avg = sum(bwd_ms) / len(bwd_ms)
    traffic, traffic_note = _traffic_record()
    if args.tape_steps:
        traffic, traffic_note = None, "the record is for the full tape; this run used a shorter one"

    bwd_gbs = bwd_bytes / (bwd_avg * 1e-3) / 1e9
    fwd_gbs = fwd_bytes / (fwd_avg * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": bwd_gbs, "peak": peak, "unit": "GB/s",
                "frac": bwd_gbs / peak, "traffic": traffic,
                "kernel": "memoroid_scan_diag_bwd (reverse scan + grad_lambda reduction)",
                "algorithmic_bytes_per_launch": bwd_bytes, "avg_launch_ms": bwd_avg,
                "peak_kind": f"{peak_kind} (copy bandwidth)", "traffic_note": traffic_note,
                "fwd": {"achieved": fwd_gbs, "frac": fwd_gbs / peak, "avg_launch_ms": fwd_avg,
                        "algorithmic_bytes_per_launch": fwd_bytes},
                "step_frac": (fwd_bytes + bwd_bytes) / (ms_per_step * 1e-3) / 1e9 / peak,
                "frac_of_datasheet": bwd_gbs / DATASHEET_HBM_GBS,
                "step_frac_of_datasheet": (fwd_bytes + bwd_bytes) / (ms_per_step * 1e-3) / 1e9 / DATASHEET_HBM_GBS}
    la = None
    if ws == 1 and not args.skip_linattn:
        la = linattn_leg(args, m, dev, stream)
        if not args.skip_cpu_baseline:
            la["cpu_baseline"] = linattn_cpu_baseline(args.la_cpu_steps)
    rt = None
    if ws == 1 and not args.skip_returns:
        rt = returns_leg(args, m, dev, stream)
    ff = None
    if ws == 1 and not args.skip_ffm:
        ff = ffm_leg(args, m, dev, stream)
    ps = None
    if ws == 1 and not args.skip_per_step:
        ps = per_step_leg(args, m, dev, stream)
    ln = None
    if ws == 1 and not args.skip_lnorm:
        ln = lnorm_leg(args, m, dev, stream)
    tb = None
    if ws == 1 and not args.skip_tbb:
        tb = tbb_leg(args, m, dev, stream)
    c3 = None
    if ws == 1 and not args.skip_cfg3:
        c3 = linattn_cfg3_leg(args, m, dev, stream)
    c4 = None
    if ws == 1 and not args.skip_cfg4:
        c4 = diag_cfg4_leg(args, m, dev, stream)
    # the other legs' roofline fractions, also inside the headline roofline object
    legs = {}
    for name, leg in (("linattn_cfg5", la), ("linattn_cfg3", c3), ("diag_cfg4", c4), ("diag_per_step_lambda", ps),
                      ("linattn_norm", ln), ("ffm", ff)):
        if leg is not None:
            r = leg["roofline"]
            legs[name] = {"fwd_frac": r["fwd"]["frac"], "bwd_frac": r["bwd"]["frac"], "step_frac": r.get("step_frac"),
                          "fwd_ms": leg["fwd_ms"], "bwd_ms": leg["bwd_ms"], "value": leg["value"]}
    if rt is not None:
        legs["returns"] = {k: rt[k]["roofline"]["frac"] for k in ("return", "gae") if k in rt}
    roofline["legs"] = legs
    cpu = None
    if ws == 1 and not args.skip_cpu_baseline:
        cpu = cpu_baseline(t, args.cpu_seconds)
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "B": B, "L": L, "D": D, "episodes": int(t["start"].sum()),
                   "l2": "inputs larger than L2 (each tensor 2 GiB vs 129 MB L2); no flush needed",
                   "parallelism": f"independent tape per GPU x{ws}"},
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": args.steps * (m.memoroid_scan_diag_kernels_per_call(B, L, D, 0, 0, 0)
                                      + m.memoroid_scan_diag_kernels_per_call(B, L, D, 0, 1, 1)),
        "clocks": clocks,
        "linattn": la,
        "returns": rt,
        "ffm": ff,
        "tbb": tb,
        "linattn_norm": ln,
        "diag_per_step_lambda": ps,
        "linattn_cfg3": c3,
        "diag_cfg4": c4,
    }
    print(json.dumps(out), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="approximate CPU time of the cpu_baseline oracle sample")
    ap.add_argument("--ref-seconds", type=float, default=90.0,
                    help="approximate total oracle time of the --impl reference steps")
    ap.add_argument("--skip-cpu-baseline", action="store_true")
    ap.add_argument("--skip-linattn", action="store_true", help="omit the linear-attention leg")
    ap.add_argument("--la-steps", type=int, default=10, help="timed linattn fwd+bwd steps")
    ap.add_argument("--la-warmup", type=int, default=3, help="untimed linattn fwd+bwd steps")
    ap.add_argument("--la-single-gamma1", action="store_true",
                    help="profiling: the linattn leg's timed tape has one episode and gamma = 1")
    ap.add_argument("--la-tape-steps", type=int, default=0,
                    help="linattn tape length (profiler captures); 0 = the full L = 2^22 workload")
    ap.add_argument("--only-linattn", action="store_true",
                    help="profiling mode: run and print only the linattn leg")
    ap.add_argument("--skip-returns", action="store_true", help="omit the discounted-return / GAE leg")
    ap.add_argument("--only-returns", action="store_true",
                    help="profiling mode: run and print only the discounted-return / GAE leg")
    ap.add_argument("--ret-steps", type=int, default=20, help="timed calls of each returns kernel")
    ap.add_argument("--skip-ffm", action="store_true", help="omit the Fast and Forgetful Memory leg")
    ap.add_argument("--skip-tbb", action="store_true", help="omit the tape-based batching leg")
    ap.add_argument("--skip-lnorm", action="store_true", help="omit the normalised Linear Transformer leg")
    ap.add_argument("--skip-per-step", action="store_true", help="omit the per-step lambda diag leg")
    ap.add_argument("--only-cfg3", action="store_true", help="profiling: the config-3 linattn leg alone")
    ap.add_argument("--only-cfg4", action="store_true", help="profiling: the config-4 diag leg alone")
    ap.add_argument("--skip-cfg3", action="store_true", help="omit the L=2^18, 4-head, d=64 linattn leg")
    ap.add_argument("--cfg3-steps", type=int, default=20, help="timed config-3 linattn fwd+bwd steps")
    ap.add_argument("--skip-cfg4", action="store_true", help="omit the 64-tape, D=128 diag leg")
    ap.add_argument("--cfg4-steps", type=int, default=20, help="timed config-4 diag fwd+bwd steps")
    ap.add_argument("--ps-steps", type=int, default=20, help="timed per-step lambda fwd+bwd steps")
    ap.add_argument("--only-per-step", action="store_true",
                    help="profiling mode: run and print only the per-step lambda diag leg")
    ap.add_argument("--only-lnorm", action="store_true",
                    help="profiling mode: run and print only the normalised Linear Transformer leg")
    ap.add_argument("--lnorm-steps", type=int, default=10, help="timed normalised Linear Transformer steps")
    ap.add_argument("--only-tbb", action="store_true",
                    help="profiling mode: run and print only the tape-based batching leg")
    ap.add_argument("--tbb-steps", type=int, default=20, help="timed calls of the sampler and of the gather")
    ap.add_argument("--only-ffm", action="store_true",
                    help="profiling mode: run and print only the Fast and Forgetful Memory leg")
    ap.add_argument("--ffm-steps", type=int, default=20, help="timed FFM fwd+bwd steps")
    ap.add_argument("--ffm-tape-steps", type=int, default=0,
                    help="FFM tape length (profiler captures); 0 = the full L = 2^20 workload")
    ap.add_argument("--la-cpu-steps", type=int, default=1 << 16,
                    help="steps (whole episodes) of the linattn oracle baseline")
    ap.add_argument("--la-intra-reps", type=int, default=2000,
                    help="repetitions of the intra-tile contraction per CTA in the tensor benchmark")
    ap.add_argument("--tape-steps", type=int, default=0,
                    help="use only the first N steps of the tape (profiler captures); 0 = full workload")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
