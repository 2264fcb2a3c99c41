"""fp64 CPU oracle for the resettable memoroid scans (test infrastructure).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline leg are the only users.  The product path never imports this
package, and this package never imports the product package.

The arithmetic lives in `memoroid_oracle.c` (plain fp64 loops written from
the paper's definitions); this module compiles it with gcc and marshals numpy
arrays through ctypes.  Inputs are upcast exactly (complex64 -> complex128,
bf16 bits -> float64), so input quantisation is not counted as error.

Parity status of each routine (what pins it, in tests/test_oracle_pins.py):
  diag_combine       case table of Theorem 3.2's proof, associativity, identity
  diag_fwd           closed-form sums (brute force), lambda=0, lambda=1
                     (segmented cumsum), scipy.signal.lfilter per episode,
                     fold of diag_combine, all-start tapes
  diag_bwd           torch.autograd (fp64) through an independent loop,
                     central finite differences
  linattn_fwd        brute-force O(L^2) sums, gamma=1 causal attention via
                     matmul, all-start tapes
  linattn_bwd        torch.autograd (fp64), finite differences
  starts/offsets     the tape example of Figure 2, numpy.flatnonzero
  discounted_return  the appendix expansion worked by hand, the fold at each
                     episode head, brute-force suffix sums, diag_bwd with a
                     real multiplier
  gae                brute-force sums of (gamma lambda)^l delta, lambda = 0
                     (TD error) and lambda = 1 (return minus value)
  ffm_fwd            the original FFM aggregator in closed form (Gamma(t)
                     powers), diag_fwd with lambda_ij and broadcast input,
                     all-start tapes
  ffm_bwd            torch.autograd (fp64) through an independent loop,
                     central finite differences in alpha and omega
  linattn_norm_fwd   brute-force normalised weighted sums (gamma = 1: the
                     paper's model), all-start tapes (y = v), shift equivariance
                     in v, outputs inside each episode's range of v
  linattn_norm_bwd   torch.autograd (fp64) through an independent loop,
                     finite differences
  tbb_sample         the Figure 2 tape worked by hand, and on random inputs the
                     properties that define the batch (whole episodes in draw
                     order, cut at B, flags at piece starts, fewest draws)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "memoroid_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_c = ctypes
_p = ctypes.c_void_p
_i64 = ctypes.c_int64


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp contraction off, so that both hosts
    round identically)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", _SRC,
            "-o", _LIB_PATH + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            L.oracle_diag_fwd.argtypes = [_i64, _i64, _i64, _p, _c.c_int, _p, _p, _p, _p, _p]
            L.oracle_diag_fold.argtypes = [_i64, _i64, _i64, _p, _c.c_int, _p, _p, _p, _p]
            L.oracle_diag_bwd.argtypes = [_i64, _i64, _i64, _p, _c.c_int, _p, _p, _p, _p, _p,
                                          _p, _p, _p]
            L.oracle_diag_combine.argtypes = [_p, _c.c_int, _p, _c.c_int, _p, _p]
            L.oracle_linattn_fwd.argtypes = [_i64] * 5 + [_p] * 4 + [_c.c_int] + [_p] * 4
            L.oracle_linattn_bwd.argtypes = [_i64] * 5 + [_p] * 4 + [_c.c_int] + [_p] * 9
            L.oracle_starts_from_offsets.argtypes = [_p, _i64, _i64, _p]
            L.oracle_discounted_return.argtypes = [_i64, _i64, _p, _p, _c.c_double, _p, _p]
            L.oracle_gae.argtypes = [_i64, _i64, _p, _p, _p, _c.c_double, _c.c_double, _p, _p]
            L.oracle_offsets_from_starts.argtypes = [_p, _i64, _p]
            L.oracle_linattn_norm_fwd.argtypes = [_i64] * 5 + [_p] * 4 + [_c.c_int] + [_p] * 7
            L.oracle_linattn_norm_bwd.argtypes = [_i64] * 5 + [_p] * 4 + [_c.c_int] + [_p] * 12
            L.oracle_tbb_sample.argtypes = [_p, _i64, _i64, _p, _i64, _i64, _p, _p]
            L.oracle_tbb_sample.restype = _i64
            L.oracle_ffm_fwd.argtypes = [_i64] * 4 + [_p] * 7
            L.oracle_ffm_bwd.argtypes = [_i64] * 4 + [_p] * 11
            L.oracle_offsets_from_starts.restype = _i64
            L.oracle_set_threads.argtypes = [_c.c_int]
            L.oracle_max_threads.restype = _c.c_int
            _lib = L
    return _lib


def set_threads(n: int) -> None:
    lib().oracle_set_threads(int(n))


def max_threads() -> int:
    return int(lib().oracle_max_threads())


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_p)


def _c128(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.complex128)


def _f64(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float64)


def _u8(a):
    return np.ascontiguousarray(a, dtype=np.uint8)


def _check(rc):
    if rc != 0:
        raise RuntimeError(f"oracle returned {rc}")


# ---------------------------------------------------------------------------
# diagonal scan
# ---------------------------------------------------------------------------

def diag_combine(left, b_left, right, b_right):
    """Resettable S5/LRU combine of two elements; left/right = (a, x) complex."""
    l = np.array([left[0].real, left[0].imag, left[1].real, left[1].imag], dtype=np.float64)
    r = np.array([right[0].real, right[0].imag, right[1].real, right[1].imag], dtype=np.float64)
    out = np.zeros(4, dtype=np.float64)
    bo = ctypes.c_int(0)
    lib().oracle_diag_combine(_ptr(l), int(b_left), _ptr(r), int(b_right), _ptr(out),
                              ctypes.cast(ctypes.pointer(bo), _p))
    return (complex(out[0], out[1]), complex(out[2], out[3])), int(bo.value)


def _diag_shapes(u, start):
    u = np.asarray(u)
    B, L, D = u.shape
    assert np.asarray(start).shape == (B, L)
    return B, L, D


def diag_fwd(lam, u, start, h0=None, lambda_per_step=None):
    B, L, D = _diag_shapes(u, start)
    lam = _c128(lam)
    if lambda_per_step is None:
        lambda_per_step = lam.ndim == 3
    u = _c128(u)
    start = _u8(start)
    h0 = _c128(h0)
    h = np.zeros((B, L, D), dtype=np.complex128)
    h_last = np.zeros((B, D), dtype=np.complex128)
    _check(lib().oracle_diag_fwd(B, L, D, _ptr(lam), int(lambda_per_step), _ptr(u), _ptr(start),
                                 _ptr(h0), _ptr(h), _ptr(h_last)))
    return h, h_last


def diag_fold(lam, u, start, h0=None, lambda_per_step=None):
    B, L, D = _diag_shapes(u, start)
    lam = _c128(lam)
    if lambda_per_step is None:
        lambda_per_step = lam.ndim == 3
    u = _c128(u)
    start = _u8(start)
    h0 = _c128(h0)
    h = np.zeros((B, L, D), dtype=np.complex128)
    _check(lib().oracle_diag_fold(B, L, D, _ptr(lam), int(lambda_per_step), _ptr(u), _ptr(start),
                                  _ptr(h0), _ptr(h)))
    return h


def diag_bwd(lam, start, h, g, g_last=None, h0=None, lambda_per_step=None):
    """Returns (grad_u, grad_lambda, grad_h0)."""
    h = _c128(h)
    B, L, D = h.shape
    lam = _c128(lam)
    if lambda_per_step is None:
        lambda_per_step = lam.ndim == 3
    start = _u8(start)
    g = _c128(g)
    g_last = _c128(g_last)
    h0 = _c128(h0)
    grad_u = np.zeros((B, L, D), dtype=np.complex128)
    grad_lam = np.zeros((B, L, D) if lambda_per_step else (D,), dtype=np.complex128)
    grad_h0 = np.zeros((B, D), dtype=np.complex128)
    _check(lib().oracle_diag_bwd(B, L, D, _ptr(lam), int(lambda_per_step), _ptr(start), _ptr(h0),
                                 _ptr(h), _ptr(g), _ptr(g_last), _ptr(grad_u), _ptr(grad_lam),
                                 _ptr(grad_h0)))
    return grad_u, grad_lam, grad_h0


# ---------------------------------------------------------------------------
# linear attention
# ---------------------------------------------------------------------------

def bf16_bits_to_f64(bits):
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def linattn_fwd(q, k, v, gamma, start, S0=None, gamma_per_step=None):
    """q, k: [B,L,H,dk]; v: [B,L,H,dv] (float arrays; bf16 callers upcast
    first with bf16_bits_to_f64).  Returns (y [B,L,H,dv], S_last [B,H,dk,dv])."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    B, L, H, dk = q.shape
    dv = v.shape[-1]
    gamma = _f64(gamma)
    if gamma_per_step is None:
        gamma_per_step = gamma.ndim == 3
    start = _u8(start)
    S0 = _f64(S0)
    y = np.zeros((B, L, H, dv), dtype=np.float64)
    S_last = np.zeros((B, H, dk, dv), dtype=np.float64)
    _check(lib().oracle_linattn_fwd(B, L, H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gamma),
                                    int(gamma_per_step), _ptr(start), _ptr(S0), _ptr(y),
                                    _ptr(S_last)))
    return y, S_last


def linattn_bwd(q, k, v, gamma, start, dy, dS_last=None, S0=None, gamma_per_step=None):
    """Returns (dq, dk, dv, dgamma, dS0)."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    B, L, H, dk = q.shape
    dv = v.shape[-1]
    gamma = _f64(gamma)
    if gamma_per_step is None:
        gamma_per_step = gamma.ndim == 3
    start = _u8(start)
    S0 = _f64(S0)
    dy = _f64(dy)
    dS_last = _f64(dS_last)
    dq = np.zeros((B, L, H, dk))
    dkk = np.zeros((B, L, H, dk))
    dvv = np.zeros((B, L, H, dv))
    dgamma = np.zeros((B, L, H) if gamma_per_step else (H,))
    dS0 = np.zeros((B, H, dk, dv))
    _check(lib().oracle_linattn_bwd(B, L, H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gamma),
                                    int(gamma_per_step), _ptr(start), _ptr(S0), _ptr(dy),
                                    _ptr(dS_last), _ptr(dq), _ptr(dkk), _ptr(dvv), _ptr(dgamma),
                                    _ptr(dS0)))
    return dq, dkk, dvv, dgamma, dS0


def linattn_norm_fwd(q, k, v, gamma, start, S0=None, z0=None, gamma_per_step=None):
    """The Linear Transformer memoroid with phi = 1 + ELU and its normalizer
    (decayed by gamma; gamma = 1 is the paper's model): returns y [B,L,H,dv],
    den [B,L,H], S_last [B,H,dk,dv], z_last [B,H,dk]."""
    q, k, v, gamma = _f64(q), _f64(k), _f64(v), _f64(gamma)
    B, L, H, dk = q.shape
    dv = v.shape[-1]
    if gamma_per_step is None:
        gamma_per_step = gamma.ndim == 3
    start = _u8(start)
    S0, z0 = _f64(S0), _f64(z0)
    y = np.zeros((B, L, H, dv))
    den = np.zeros((B, L, H))
    S_last = np.zeros((B, H, dk, dv))
    z_last = np.zeros((B, H, dk))
    _check(lib().oracle_linattn_norm_fwd(B, L, H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gamma), int(gamma_per_step),
                                         _ptr(start), _ptr(S0), _ptr(z0), _ptr(y), _ptr(den), _ptr(S_last),
                                         _ptr(z_last)))
    return y, den, S_last, z_last


def linattn_norm_bwd(q, k, v, gamma, start, dy, dS_last=None, dz_last=None, S0=None, z0=None, gamma_per_step=None):
    """Reverse mode of linattn_norm_fwd: dq, dk, dv, dgamma, dS0, dz0."""
    q, k, v, gamma, dy = _f64(q), _f64(k), _f64(v), _f64(gamma), _f64(dy)
    B, L, H, dk = q.shape
    dv = v.shape[-1]
    if gamma_per_step is None:
        gamma_per_step = gamma.ndim == 3
    start = _u8(start)
    S0, z0, dS_last, dz_last = _f64(S0), _f64(z0), _f64(dS_last), _f64(dz_last)
    dq, dkk, dvv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    dgamma = np.zeros_like(gamma)
    dS0 = np.zeros((B, H, dk, dv))
    dz0 = np.zeros((B, H, dk))
    _check(lib().oracle_linattn_norm_bwd(B, L, H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gamma), int(gamma_per_step),
                                         _ptr(start), _ptr(S0), _ptr(z0), _ptr(dy), _ptr(dS_last), _ptr(dz_last),
                                         _ptr(dq), _ptr(dkk), _ptr(dvv), _ptr(dgamma), _ptr(dS0), _ptr(dz0)))
    return dq, dkk, dvv, dgamma, dS0, dz0


# ---------------------------------------------------------------------------
# episode index list <-> begin flags
# ---------------------------------------------------------------------------

def discounted_return(r, start, gamma, boot=None):
    """G [B, L]: per-step discounted return within episodes (boot: [B] value
    after the tape's last step, or None)."""
    r = _f64(r)
    B, L = r.shape
    start = _u8(start)
    boot = _f64(boot)
    G = np.zeros((B, L), dtype=np.float64)
    _check(lib().oracle_discounted_return(B, L, _ptr(r), _ptr(start), float(gamma), _ptr(boot), _ptr(G)))
    return G


def gae(r, v, start, gamma, lam, v_boot=None):
    """A [B, L]: per-step generalised advantage estimate within episodes."""
    r, v = _f64(r), _f64(v)
    B, L = r.shape
    start = _u8(start)
    v_boot = _f64(v_boot)
    A = np.zeros((B, L), dtype=np.float64)
    _check(lib().oracle_gae(B, L, _ptr(r), _ptr(v), _ptr(start), float(gamma), float(lam), _ptr(v_boot), _ptr(A)))
    return A


def ffm_fwd(alpha, omega, xt, start, S0=None):
    """Fast and Forgetful Memory memoroid.  alpha [m], omega [c], xt [B, L, m]
    (the cell's gated input x~), start [B, L], S0 [B, m, c] complex or None.
    Returns z [B, L, 2*m*c] (Re(X_t) || Im(X_t), each flattened i*c + j) and
    S_last [B, m, c] complex."""
    alpha, omega, xt = _f64(alpha), _f64(omega), _f64(xt)
    B, L, m = xt.shape
    c = omega.shape[0]
    start = _u8(start)
    S0 = _c128(S0)
    z = np.zeros((B, L, 2 * m * c), dtype=np.float64)
    S_last = np.zeros((B, m, c), dtype=np.complex128)
    _check(lib().oracle_ffm_fwd(B, L, m, c, _ptr(alpha), _ptr(omega), _ptr(xt), _ptr(start), _ptr(S0),
                                _ptr(z), _ptr(S_last)))
    return z, S_last


def ffm_bwd(alpha, omega, start, z, grad_z, grad_S_last=None, S0=None):
    """Reverse-mode of ffm_fwd: returns grad_xt [B, L, m], grad_alpha [m],
    grad_omega [c], grad_S0 [B, m, c] complex."""
    alpha, omega, z, grad_z = _f64(alpha), _f64(omega), _f64(z), _f64(grad_z)
    m, c = alpha.shape[0], omega.shape[0]
    B, L = z.shape[0], z.shape[1]
    start = _u8(start)
    S0, grad_S_last = _c128(S0), _c128(grad_S_last)
    gx = np.zeros((B, L, m), dtype=np.float64)
    ga = np.zeros(m, dtype=np.float64)
    go = np.zeros(c, dtype=np.float64)
    gS0 = np.zeros((B, m, c), dtype=np.complex128)
    _check(lib().oracle_ffm_bwd(B, L, m, c, _ptr(alpha), _ptr(omega), _ptr(start), _ptr(S0), _ptr(z),
                                _ptr(grad_z), _ptr(grad_S_last), _ptr(gx), _ptr(ga), _ptr(go), _ptr(gS0)))
    return gx, ga, go, gS0


def tbb_sample(I, N, ep, B):
    """Algorithm 2 with the draws given: I [E] episode begin indices into a
    buffer of N transitions, ep [K] the drawn indices, B the batch size.
    Returns (start [B] uint8, src [B] int64, draws used); raises ValueError
    on an out-of-range index or too few draws."""
    I = np.ascontiguousarray(I, dtype=np.int64)
    ep = np.ascontiguousarray(ep, dtype=np.int64)
    start = np.zeros(B, dtype=np.uint8)
    src = np.zeros(B, dtype=np.int64)
    n = lib().oracle_tbb_sample(_ptr(I), len(I), N, _ptr(ep), len(ep), B, _ptr(start), _ptr(src))
    if n == -2:
        raise ValueError("episode index out of range")
    if n == -3:
        raise ValueError("the draws do not fill the batch")
    _check(0 if n >= 0 else n)
    return start, src, int(n)


def starts_from_offsets(offsets, L):
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    start = np.zeros(L, dtype=np.uint8)
    _check(lib().oracle_starts_from_offsets(_ptr(offsets), len(offsets), L, _ptr(start)))
    return start


def offsets_from_starts(start):
    start = _u8(start)
    out = np.zeros(max(len(start), 1), dtype=np.int64)
    n = lib().oracle_offsets_from_starts(_ptr(start), len(start), _ptr(out))
    return out[:n].copy()
