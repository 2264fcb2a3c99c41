"""Seeded synthetic tapes for the memoroid scans.

This module only draws random inputs; it holds none of the scan arithmetic, so
both the CUDA path and the fp64 oracle can take their inputs from it.

A tape is built the way tape-based batching samples one (Section 4.1,
Algorithm 2): whole episodes are drawn and concatenated until the tape holds
at least L steps, then the tape is cut to exactly L steps (the last episode is
truncated).  The begin flag b_t is 1 on the first step of every episode
(Section 2.1), so start[0] = 1 for every generated tape.

The paper's workloads are POPGym and Atari replay tapes (Section 5, Appendix
"Experiment Setup"); those environments are not available, so these
synthetic tapes with the same structure stand in for them.

Distributions:
  * Geometric(mean mu): support {1, 2, ...} with success probability 1/mu.
  * complex normal CN(0, 1): Re and Im i.i.d. N(0, 1/2).
  * diagonal lambda: |lambda| ~ U(0.9, 0.999), arg(lambda) ~ U(0, 2 pi).
  * bf16 values are produced from fp32 by round-to-nearest-even and carried
    as uint16 bit patterns (numpy has no bf16 type).
"""
from __future__ import annotations

import numpy as np

SEED_BASE = 20240209


def seed_for(config_id: int) -> int:
    return SEED_BASE + int(config_id)


# ----------------------------------------------------------------------------
# episode structure
# ----------------------------------------------------------------------------

def episode_lengths_geometric(rng: np.random.Generator, total: int, mean: float,
                              lo: int = 1, hi: int | None = None) -> np.ndarray:
    """Draw Geometric(mean) episode lengths (clipped to [lo, hi]) until their
    sum reaches `total`; the last one is cut so that the sum is exactly
    `total`."""
    if total <= 0:
        return np.zeros(0, dtype=np.int64)
    p = 1.0 / float(mean)
    out = []
    acc = 0
    while acc < total:
        n = max(int(total - acc) // max(int(mean), 1), 16)
        draw = rng.geometric(p, size=n).astype(np.int64)
        if hi is not None:
            draw = np.clip(draw, lo, hi)
        else:
            draw = np.maximum(draw, lo)
        out.append(draw)
        acc += int(draw.sum())
    lens = np.concatenate(out)
    csum = np.cumsum(lens)
    k = int(np.searchsorted(csum, total, side="left"))
    lens = lens[: k + 1].copy()
    lens[-1] -= int(csum[k] - total)
    assert int(lens.sum()) == total and lens.min() >= 1
    return lens


def starts_from_lengths(lens: np.ndarray, total: int) -> np.ndarray:
    start = np.zeros(total, dtype=np.uint8)
    if len(lens):
        offs = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)
        start[offs] = 1
    return start


def geometric_tape_starts(rng: np.random.Generator, L: int, mean: float,
                          lo: int = 1, hi: int | None = None) -> np.ndarray:
    return starts_from_lengths(episode_lengths_geometric(rng, L, mean, lo, hi), L)


def episode_bounds(start_row: np.ndarray) -> list[tuple[int, int]]:
    """[s, e) bounds of the episodes (and of a leading partial episode, when
    start[0] = 0) of one tape row."""
    L = len(start_row)
    heads = np.flatnonzero(start_row).tolist()
    if not heads or heads[0] != 0:
        heads = [0] + heads
    ends = heads[1:] + [L]
    return [(s, e) for s, e in zip(heads, ends) if e > s]


# ----------------------------------------------------------------------------
# value distributions
# ----------------------------------------------------------------------------

def complex_normal(rng: np.random.Generator, shape, scale: float = 1.0) -> np.ndarray:
    """CN(0, scale^2): Re, Im i.i.d. N(0, scale^2 / 2), as complex64."""
    s = np.float32(scale / np.sqrt(2.0))
    re = rng.standard_normal(shape, dtype=np.float32) * s
    im = rng.standard_normal(shape, dtype=np.float32) * s
    out = np.empty(shape, dtype=np.complex64)
    out.real = re
    out.imag = im
    return out


def diag_lambda(rng: np.random.Generator, shape) -> np.ndarray:
    mag = rng.uniform(0.9, 0.999, size=shape)
    ph = rng.uniform(0.0, 2.0 * np.pi, size=shape)
    return (mag * np.exp(1j * ph)).astype(np.complex64)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round to nearest, ties to even) -> uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    nan = (u & 0x7FFFFFFF) > 0x7F800000
    rounding = ((u >> 16) & 1) + np.uint32(0x7FFF)
    r = ((u + rounding) >> 16).astype(np.uint16)
    r[nan] = ((u[nan] >> 16) | 0x40).astype(np.uint16)
    return r


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ----------------------------------------------------------------------------
# workload builders
# ----------------------------------------------------------------------------

DIAG_CONFIGS = {
    # id: (B, L, D, episode mean, clip hi, with backward)
    1: dict(B=1, L=4096, D=64, mean=200.0, hi=None, bwd=False),
    2: dict(B=1, L=1 << 20, D=256, mean=500.0, hi=10000, bwd=True),
    4: dict(B=64, L=16384, D=128, mean=20.0, hi=None, bwd=True),
}

LINATTN_CONFIGS = {
    3: dict(B=1, L=1 << 18, H=4, d=64, chunk=64, mean=300.0, gamma="head"),
    5: dict(B=1, L=1 << 22, H=8, d=128, chunk=64, mean=1000.0, gamma="step"),
}


def diag_tape(B: int, L: int, D: int, seed: int, mean: float = 200.0, hi: int | None = None,
              lambda_per_step: bool = False, single_episode_rows=(), with_grad: bool = True,
              with_h0: bool = False, start_mode: str = "geometric"):
    """A diag-scan workload: lambda, u, start, optional upstream grads and h0.

    start_mode: "geometric" (Algorithm 2 style concatenation), "all" (every
    step starts an episode), "none" (one episode per row, start[0] = 1) or
    "open" (no start flags at all: the row continues an earlier episode).
    """
    rng = np.random.default_rng(seed)
    lam = diag_lambda(rng, (B, L, D) if lambda_per_step else (D,))
    u = complex_normal(rng, (B, L, D))
    start = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        if start_mode == "all":
            start[b, :] = 1
        elif start_mode == "none" or b in single_episode_rows:
            start[b, 0] = 1 if L else 0
        elif start_mode == "open":
            pass
        else:
            start[b] = geometric_tape_starts(rng, L, mean, 1, hi)
    out = dict(B=B, L=L, D=D, lam=lam, lambda_per_step=lambda_per_step, u=u, start=start)
    if with_grad:
        # upstream gradient: Re, Im ~ N(0, 1)
        out["grad_h"] = complex_normal(rng, (B, L, D), scale=np.sqrt(2.0))
        out["grad_h_last"] = complex_normal(rng, (B, D), scale=np.sqrt(2.0))
    if with_h0:
        out["h0"] = complex_normal(rng, (B, D))
    return out


def diag_config(cfg: int):
    c = DIAG_CONFIGS[cfg]
    rows = tuple(range(c["B"] // 2, c["B"])) if cfg == 4 else ()
    t = diag_tape(c["B"], c["L"], c["D"], seed_for(cfg), mean=c["mean"], hi=c["hi"],
                  single_episode_rows=rows, with_grad=c["bwd"])
    t["grad_h_last"] = None
    return t


def ffm_tape(B: int, L: int, m: int, c: int, seed: int, mean: float = 500.0, hi: int | None = None,
             with_grad: bool = True, with_S0: bool = False, start_mode: str = "geometric"):
    """A Fast-and-Forgetful-Memory workload: alpha [m] with |alpha| ~
    U(0.001, 0.105) and a random sign (so exp(-|alpha|) spans the decays of
    the diagonal configs, 0.9 .. 0.999), omega [c] ~ U(-pi, pi), the gated
    input x~ [B, L, m] ~ N(0, 1) (fp32), begin flags as in diag_tape,
    optional S0 [B, m, c] ~ CN(0, 1) (complex64) and upstream gradients
    grad_z [B, L, 2 m c] ~ N(0, 1), grad_S_last [B, m, c] with Re, Im ~ N(0, 1)."""
    rng = np.random.default_rng(seed)
    alpha = (rng.uniform(0.001, 0.105, m) * rng.choice([-1.0, 1.0], m)).astype(np.float32)
    omega = rng.uniform(-np.pi, np.pi, c).astype(np.float32)
    x = rng.standard_normal((B, L, m), dtype=np.float32)
    start = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        if start_mode == "all":
            start[b, :] = 1
        elif start_mode == "none":
            start[b, 0] = 1 if L else 0
        elif start_mode == "open":
            pass
        else:
            start[b] = geometric_tape_starts(rng, L, mean, 1, hi)
    out = dict(B=B, L=L, m=m, c=c, alpha=alpha, omega=omega, x=x, start=start)
    if with_grad:
        out["grad_z"] = rng.standard_normal((B, L, 2 * m * c), dtype=np.float32)
        out["grad_S_last"] = complex_normal(rng, (B, m, c), scale=np.sqrt(2.0))
    if with_S0:
        out["S0"] = complex_normal(rng, (B, m, c))
    return out


def linattn_tape(B: int, L: int, H: int, dk: int, dv: int, seed: int, mean: float = 300.0,
                 gamma_mode: str = "head", gammas=(0.9, 0.99, 0.999, 1.0), scale: float | None = None,
                 with_grad: bool = True, with_S0: bool = False, start_mode: str = "geometric",
                 normalize_k: bool = True):
    """A linear-attention workload: bf16 q, k, v (as uint16 bits), fp32 gamma,
    start flags and optional upstream gradients.

    q, v ~ N(0, 1) * scale; k ~ N(0, 1), L2-normalised over d_k in fp32 before
    the bf16 cast unless normalize_k is False.  gamma_mode "head": one decay per head (cycled from
    `gammas`); "step": gamma[b, t, h] = sigmoid(N(3, 1)).
    """
    rng = np.random.default_rng(seed)
    if scale is None:
        scale = 1.0 / np.sqrt(dk)
    q = rng.standard_normal((B, L, H, dk), dtype=np.float32) * np.float32(scale)
    k = rng.standard_normal((B, L, H, dk), dtype=np.float32)
    if normalize_k:
        k /= np.maximum(np.linalg.norm(k, axis=-1, keepdims=True), np.float32(1e-12))
    v = rng.standard_normal((B, L, H, dv), dtype=np.float32) * np.float32(scale)
    if gamma_mode == "head":
        gamma = np.array([gammas[h % len(gammas)] for h in range(H)], dtype=np.float32)
    else:
        z = rng.standard_normal((B, L, H)).astype(np.float64) + 3.0
        gamma = (1.0 / (1.0 + np.exp(-z))).astype(np.float32)
    start = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        if start_mode == "all":
            start[b, :] = 1
        elif start_mode == "none":
            start[b, 0] = 1 if L else 0
        elif start_mode == "open":
            pass
        else:
            start[b] = geometric_tape_starts(rng, L, mean)
    out = dict(B=B, L=L, H=H, dk=dk, dv=dv, q=f32_to_bf16_bits(q), k=f32_to_bf16_bits(k),
               v=f32_to_bf16_bits(v), gamma=gamma, gamma_per_step=(gamma_mode != "head"),
               start=start)
    if with_grad:
        out["grad_y"] = rng.standard_normal((B, L, H, dv), dtype=np.float32)
        out["grad_S_last"] = rng.standard_normal((B, H, dk, dv), dtype=np.float32)
    if with_S0:
        out["S0"] = rng.standard_normal((B, H, dk, dv), dtype=np.float32) * np.float32(0.1)
    return out


def linattn_config(cfg: int):
    c = LINATTN_CONFIGS[cfg]
    t = linattn_tape(c["B"], c["L"], c["H"], c["d"], c["d"], seed_for(cfg), mean=c["mean"],
                     gamma_mode=c["gamma"])
    t["grad_S_last"] = None
    t["chunk"] = c["chunk"]
    return t


def linattn_tape_device(B: int, L: int, H: int, d: int, seed: int, mean: float, gamma_mode: str = "step",
                        gammas=(0.9, 0.99, 0.999, 1.0), device="cuda", with_grad: bool = True,
                        rows_per_draw: int = 1 << 18):
    """The linattn_tape recipe drawn on the device with torch's seeded CUDA
    generator, for tapes too large to draw and copy from the host (the L = 2^22,
    8-head, d = 128 workload holds 26 GB of q, k, v).  Start flags come from the
    host generator (numpy, same recipe as linattn_tape).  q, k, v are returned
    as int16 tensors holding bf16 bit patterns; gamma, grad_y as fp32.

    Values differ from linattn_tape for the same seed (another generator);
    parity tests compare the GPU path with the oracle on slices copied back.
    """
    import torch

    rng = np.random.default_rng(seed)
    start = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        start[b] = geometric_tape_starts(rng, L, mean)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    scale = 1.0 / float(np.sqrt(d))

    def draw(normalise: bool, s: float):
        out = torch.empty((B, L, H, d), dtype=torch.bfloat16, device=device)
        for b in range(B):
            for r0 in range(0, L, rows_per_draw):
                r1 = min(L, r0 + rows_per_draw)
                x = torch.randn((r1 - r0, H, d), generator=gen, device=device, dtype=torch.float32)
                if normalise:
                    x = x / x.norm(dim=-1, keepdim=True).clamp_min(1e-12)
                else:
                    x = x * s
                out[b, r0:r1] = x.to(torch.bfloat16)
        return out.view(torch.int16)

    q = draw(False, scale)
    k = draw(True, 1.0)
    v = draw(False, scale)
    if gamma_mode == "head":
        gamma = torch.tensor([gammas[h % len(gammas)] for h in range(H)], dtype=torch.float32, device=device)
    else:
        z = torch.randn((B, L, H), generator=gen, device=device, dtype=torch.float32) + 3.0
        gamma = torch.sigmoid(z)
    out = dict(B=B, L=L, H=H, dk=d, dv=d, q=q, k=k, v=v, gamma=gamma, gamma_per_step=(gamma_mode != "head"),
               start=torch.from_numpy(start).to(device))
    if with_grad:
        out["grad_y"] = torch.randn((B, L, H, d), generator=gen, device=device, dtype=torch.float32)
    return out
