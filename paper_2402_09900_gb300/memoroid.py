"""ctypes binding of the C ABI in include/memoroid.h.

Argument marshalling only: every step of every scan runs in the CUDA kernels
of libmemoroid.so.  PyTorch supplies device memory (outputs and workspace are
torch tensors) and the current CUDA stream.  There is no fallback: if the
library is missing or no GPU is present, the calls raise.

The raw entry points keep the C names (memoroid_scan_diag_fwd, ...) and take
torch tensors (or None) where the C call takes a pointer; the short helpers
(diag_fwd, diag_bwd, ...) allocate outputs and workspace and return tensors.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

MEMOROID_OK = 0
MEMOROID_ERR_INVALID_ARG = 1
MEMOROID_ERR_UNSUPPORTED = 2
MEMOROID_ERR_WORKSPACE = 3
MEMOROID_ERR_CUDA = 4
MEMOROID_ERR_TIMEOUT = 5
MEMOROID_ERR_BAD_DATA = 6
MEMOROID_F32 = 0
MEMOROID_BF16 = 1

_lock = threading.Lock()
_lib = None

_p = ctypes.c_void_p
_i64 = ctypes.c_int64
_int = ctypes.c_int
_sz = ctypes.c_size_t

# name -> (restype, argtypes); mirrors include/memoroid.h
SIGNATURES = {
    "memoroid_status_string": (ctypes.c_char_p, [_int]),
    "memoroid_version": (_int, []),
    "memoroid_scan_diag_workspace_bytes": (_sz, [_i64, _i64, _i64]),
    "memoroid_scan_diag_kernels_per_call": (_int, [_i64, _i64, _i64, _int, _int, _int]),
    "memoroid_scan_diag_fwd": (_int, [_p, _int, _p, _p, _p, _p, _p, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_scan_diag_bwd": (_int, [_p, _int, _p, _p, _p, _p, _p, _p, _p, _p, _i64, _i64, _i64,
                                      _p, _sz, _p]),
    "memoroid_scan_diag_fwd_static": (_int, [_p, _int, _p, _p, _p, _p, _p, _i64, _i64, _i64, _p]),
    "memoroid_scan_linattn_workspace_bytes": (_sz, [_i64, _i64, _i64, _i64, _i64, _i64]),
    "memoroid_scan_linattn_kernels_per_call": (_int, [_i64, _i64, _i64, _i64, _i64, _int, _int]),
    "memoroid_scan_linattn_fwd": (_int, [_p, _p, _p, _int, _p, _int, _p, _p, _p, _p, _i64, _i64, _i64,
                                         _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_scan_linattn_bwd": (_int, [_p, _p, _p, _int, _p, _int, _p, _p, _p, _p, _p, _p, _p, _p, _p, _i64,
                                         _i64, _i64, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_bench_linattn_intra_scratch_bytes": (_sz, [_i64]),
    "memoroid_bench_linattn_intra": (_int, [_i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_returns_workspace_bytes": (_sz, [_i64, _i64]),
    "memoroid_linattn_norm_workspace_bytes": (_sz, [_i64, _i64, _i64, _i64]),
    "memoroid_linattn_norm_kernels_per_call": (_int, [_i64, _i64, _i64, _i64, _int, _int, _int]),
    "memoroid_linattn_norm_fwd": (_int, [_p, _p, _p, _p, _int, _p, _p, _p, _p, _p, _p, _p,
                                         _i64, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_linattn_norm_bwd": (_int, [_p, _p, _p, _p, _int, _p, _p, _p, _p, _p, _p, _p, _p,
                                         _p, _p, _p, _p, _p, _p, _i64, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_tbb_workspace_bytes": (_sz, [_i64]),
    "memoroid_tbb_sample": (_int, [_p, _i64, _i64, _p, _i64, _i64, _p, _p, _p, _p, _sz, _p]),
    "memoroid_gather_rows": (_int, [_p, _i64, _i64, _p, _i64, _p, _p, _sz, _p]),
    "memoroid_ffm_workspace_bytes": (_sz, [_i64, _i64, _i64, _i64]),
    "memoroid_ffm_kernels_per_call": (_int, [_i64, _i64, _i64, _i64, _int, _int]),
    "memoroid_ffm_fwd": (_int, [_p, _p, _p, _p, _p, _p, _p, _i64, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_ffm_bwd": (_int, [_p] * 11 + [_i64, _i64, _i64, _i64, _p, _sz, _p]),
    "memoroid_discounted_return": (_int, [_p, _p, ctypes.c_float, _p, _p, _i64, _i64, _p, _sz, _p]),
    "memoroid_gae": (_int, [_p, _p, _p, ctypes.c_float, ctypes.c_float, _p, _p, _i64, _i64, _p, _sz, _p]),
    "memoroid_starts_from_offsets": (_int, [_p, _i64, _i64, _p, _p]),
    "memoroid_offsets_workspace_bytes": (_sz, [_i64]),
    "memoroid_offsets_from_starts": (_int, [_p, _i64, _p, _p, _p, _sz, _p]),
    "memoroid_get_device_error": (_int, [_p, _p]),
    "memoroid_get_static_device_error": (_int, [_p]),
    "memoroid_debug_set_wait_limit_ns": (None, [ctypes.c_uint64]),
    "memoroid_debug_withhold_tile": (None, [_i64]),
    "memoroid_debug_lnorm_padded": (None, [_int]),
}


class MemoroidError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


def lib_path() -> str:
    return _build.lib_path()


def load():
    """Loads libmemoroid.so (it must have been built: __graft_entry__.build()
    or paper_2402_09900_gb300.build.build())."""
    global _lib
    with _lock:
        if _lib is None:
            path = lib_path()
            if not os.path.exists(path):
                raise RuntimeError(f"{path} is missing: build the CUDA library first")
            L = ctypes.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def status_string(status: int) -> str:
    return load().memoroid_status_string(int(status)).decode()


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(status, where):
    if status != MEMOROID_OK:
        raise MemoroidError(status, where)


def _need_cuda(*ts):
    for t in ts:
        if t is not None:
            if not t.is_cuda:
                raise ValueError("memoroid kernels take CUDA tensors only")
            if not t.is_contiguous():
                raise ValueError("memoroid kernels take contiguous tensors only")


# ---------------------------------------------------------------------------
# raw entry points (same names as the C ABI)
# ---------------------------------------------------------------------------

def memoroid_scan_diag_workspace_bytes(B, L, D) -> int:
    return int(load().memoroid_scan_diag_workspace_bytes(B, L, D))


def memoroid_scan_diag_kernels_per_call(B, L, D, lambda_per_step, backward, with_grad_lambda) -> int:
    return int(load().memoroid_scan_diag_kernels_per_call(B, L, D, int(lambda_per_step), int(backward),
                                                          int(with_grad_lambda)))


def memoroid_scan_diag_fwd(lam, lambda_per_step, u, start, h0, h, h_last, B, L, D, workspace,
                           stream=None):
    _need_cuda(lam, u, start, h0, h, h_last, workspace)
    st = load().memoroid_scan_diag_fwd(_ptr(lam), int(lambda_per_step), _ptr(u), _ptr(start), _ptr(h0),
                                       _ptr(h), _ptr(h_last), B, L, D, _ptr(workspace),
                                       workspace.numel() if workspace is not None else 0, _stream(stream))
    _check(st, "memoroid_scan_diag_fwd")


def memoroid_scan_diag_bwd(lam, lambda_per_step, start, h0, h, grad_h, grad_h_last, grad_u, grad_lambda,
                           grad_h0, B, L, D, workspace, stream=None):
    _need_cuda(lam, start, h0, h, grad_h, grad_h_last, grad_u, grad_lambda, grad_h0, workspace)
    st = load().memoroid_scan_diag_bwd(_ptr(lam), int(lambda_per_step), _ptr(start), _ptr(h0), _ptr(h),
                                       _ptr(grad_h), _ptr(grad_h_last), _ptr(grad_u), _ptr(grad_lambda),
                                       _ptr(grad_h0), B, L, D, _ptr(workspace),
                                       workspace.numel() if workspace is not None else 0, _stream(stream))
    _check(st, "memoroid_scan_diag_bwd")


def memoroid_scan_diag_fwd_static(lam, lambda_per_step, u, start, h0, h, h_last, B, L, D, stream=None):
    """Forward scan that takes no workspace: it uses a fixed-size scratch array
    owned by the library (see include/memoroid.h for the rules of use)."""
    _need_cuda(lam, u, start, h0, h, h_last)
    st = load().memoroid_scan_diag_fwd_static(_ptr(lam), int(lambda_per_step), _ptr(u), _ptr(start), _ptr(h0),
                                              _ptr(h), _ptr(h_last), B, L, D, _stream(stream))
    _check(st, "memoroid_scan_diag_fwd_static")


def memoroid_scan_linattn_workspace_bytes(B, L, H, dk, dv, chunk) -> int:
    return int(load().memoroid_scan_linattn_workspace_bytes(B, L, H, dk, dv, chunk))


def memoroid_scan_linattn_kernels_per_call(B, L, H, dk, dv, backward, with_dgamma_per_head) -> int:
    return int(load().memoroid_scan_linattn_kernels_per_call(B, L, H, dk, dv, int(backward),
                                                             int(with_dgamma_per_head)))


def memoroid_scan_linattn_fwd(q, k, v, in_dtype, gamma, gamma_per_step, start, S0, y, S_last, B, L, H, dk, dv,
                              chunk, workspace, stream=None):
    _need_cuda(q, k, v, gamma, start, S0, y, S_last, workspace)
    st = load().memoroid_scan_linattn_fwd(_ptr(q), _ptr(k), _ptr(v), int(in_dtype), _ptr(gamma),
                                          int(gamma_per_step), _ptr(start), _ptr(S0), _ptr(y), _ptr(S_last),
                                          B, L, H, dk, dv, chunk, _ptr(workspace),
                                          workspace.numel() if workspace is not None else 0, _stream(stream))
    _check(st, "memoroid_scan_linattn_fwd")


def memoroid_scan_linattn_bwd(q, k, v, in_dtype, gamma, gamma_per_step, start, S0, grad_y, grad_S_last, dq, dk_out,
                              dv_out, dgamma, dS0, B, L, H, dk, dv, chunk, workspace, stream=None):
    _need_cuda(q, k, v, gamma, start, S0, grad_y, grad_S_last, dq, dk_out, dv_out, dgamma, dS0, workspace)
    st = load().memoroid_scan_linattn_bwd(_ptr(q), _ptr(k), _ptr(v), int(in_dtype), _ptr(gamma), int(gamma_per_step),
                                          _ptr(start), _ptr(S0), _ptr(grad_y), _ptr(grad_S_last), _ptr(dq),
                                          _ptr(dk_out), _ptr(dv_out), _ptr(dgamma), _ptr(dS0), B, L, H, dk, dv, chunk,
                                          _ptr(workspace), workspace.numel() if workspace is not None else 0,
                                          _stream(stream))
    _check(st, "memoroid_scan_linattn_bwd")


def memoroid_bench_linattn_intra_scratch_bytes(d) -> int:
    return int(load().memoroid_bench_linattn_intra_scratch_bytes(d))


def memoroid_bench_linattn_intra(d, reps, ctas, scratch, stream=None):
    _need_cuda(scratch)
    _check(load().memoroid_bench_linattn_intra(d, reps, ctas, _ptr(scratch), scratch.numel(), _stream(stream)),
           "memoroid_bench_linattn_intra")


def memoroid_returns_workspace_bytes(B, L) -> int:
    return int(load().memoroid_returns_workspace_bytes(B, L))


def memoroid_discounted_return(r, start, gamma, boot, G, B, L, workspace, stream=None):
    _need_cuda(r, start, boot, G, workspace)
    _check(load().memoroid_discounted_return(_ptr(r), _ptr(start), float(gamma), _ptr(boot), _ptr(G), B, L,
                                             _ptr(workspace), workspace.numel() if workspace is not None else 0,
                                             _stream(stream)), "memoroid_discounted_return")


def memoroid_gae(r, v, start, gamma, lam, v_boot, A, B, L, workspace, stream=None):
    _need_cuda(r, v, start, v_boot, A, workspace)
    _check(load().memoroid_gae(_ptr(r), _ptr(v), _ptr(start), float(gamma), float(lam), _ptr(v_boot), _ptr(A), B, L,
                               _ptr(workspace), workspace.numel() if workspace is not None else 0, _stream(stream)),
           "memoroid_gae")


def memoroid_linattn_norm_workspace_bytes(B, L, H, d) -> int:
    return int(load().memoroid_linattn_norm_workspace_bytes(B, L, H, d))


def memoroid_linattn_norm_kernels_per_call(B, L, H, d, backward, with_dgamma_per_head, with_states) -> int:
    return int(load().memoroid_linattn_norm_kernels_per_call(B, L, H, d, int(backward), int(with_dgamma_per_head),
                                                             int(with_states)))


def memoroid_linattn_norm_fwd(q, k, v, gamma, gamma_per_step, start, S0, z0, y, den, S_last, z_last, B, L, H, d,
                              workspace, stream=None):
    _need_cuda(q, k, v, gamma, start, S0, z0, y, den, S_last, z_last, workspace)
    _check(load().memoroid_linattn_norm_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(gamma), int(gamma_per_step), _ptr(start),
                                            _ptr(S0), _ptr(z0), _ptr(y), _ptr(den), _ptr(S_last), _ptr(z_last),
                                            B, L, H, d, _ptr(workspace),
                                            workspace.numel() if workspace is not None else 0, _stream(stream)),
           "memoroid_linattn_norm_fwd")


def memoroid_linattn_norm_bwd(q, k, v, gamma, gamma_per_step, start, S0, z0, y, den, grad_y, grad_S_last, grad_z_last,
                              dq, dk, dv, dgamma, dS0, dz0, B, L, H, d, workspace, stream=None):
    _need_cuda(q, k, v, gamma, start, S0, z0, y, den, grad_y, grad_S_last, grad_z_last, dq, dk, dv, dgamma, dS0, dz0,
               workspace)
    _check(load().memoroid_linattn_norm_bwd(_ptr(q), _ptr(k), _ptr(v), _ptr(gamma), int(gamma_per_step), _ptr(start),
                                            _ptr(S0), _ptr(z0), _ptr(y), _ptr(den), _ptr(grad_y), _ptr(grad_S_last),
                                            _ptr(grad_z_last), _ptr(dq), _ptr(dk), _ptr(dv), _ptr(dgamma), _ptr(dS0),
                                            _ptr(dz0), B, L, H, d, _ptr(workspace),
                                            workspace.numel() if workspace is not None else 0, _stream(stream)),
           "memoroid_linattn_norm_bwd")


def memoroid_tbb_workspace_bytes(K) -> int:
    return int(load().memoroid_tbb_workspace_bytes(K))


def memoroid_tbb_sample(begin, E, N, draws, K, B, start, src, n_used, workspace, stream=None):
    _need_cuda(begin, draws, start, src, n_used, workspace)
    _check(load().memoroid_tbb_sample(_ptr(begin), E, N, _ptr(draws), K, B, _ptr(start), _ptr(src), _ptr(n_used),
                                      _ptr(workspace), workspace.numel() if workspace is not None else 0,
                                      _stream(stream)), "memoroid_tbb_sample")


def memoroid_gather_rows(rows, N, row_bytes, src, B, out, workspace, stream=None):
    _need_cuda(rows, src, out, workspace)
    _check(load().memoroid_gather_rows(_ptr(rows), N, row_bytes, _ptr(src), B, _ptr(out), _ptr(workspace),
                                       workspace.numel() if workspace is not None else 0, _stream(stream)),
           "memoroid_gather_rows")


def memoroid_ffm_workspace_bytes(B, L, m, c) -> int:
    return int(load().memoroid_ffm_workspace_bytes(B, L, m, c))


def memoroid_ffm_kernels_per_call(B, L, m, c, backward, with_param_grads) -> int:
    return int(load().memoroid_ffm_kernels_per_call(B, L, m, c, int(backward), int(with_param_grads)))


def memoroid_ffm_fwd(x, alpha, omega, start, S0, z, S_last, B, L, m, c, workspace, stream=None):
    _need_cuda(x, alpha, omega, start, S0, z, S_last, workspace)
    _check(load().memoroid_ffm_fwd(_ptr(x), _ptr(alpha), _ptr(omega), _ptr(start), _ptr(S0), _ptr(z), _ptr(S_last),
                                   B, L, m, c, _ptr(workspace), workspace.numel() if workspace is not None else 0,
                                   _stream(stream)), "memoroid_ffm_fwd")


def memoroid_ffm_bwd(alpha, omega, start, S0, z, grad_z, grad_S_last, grad_x, grad_alpha, grad_omega, grad_S0,
                     B, L, m, c, workspace, stream=None):
    _need_cuda(alpha, omega, start, S0, z, grad_z, grad_S_last, grad_x, grad_alpha, grad_omega, grad_S0, workspace)
    _check(load().memoroid_ffm_bwd(_ptr(alpha), _ptr(omega), _ptr(start), _ptr(S0), _ptr(z), _ptr(grad_z),
                                   _ptr(grad_S_last), _ptr(grad_x), _ptr(grad_alpha), _ptr(grad_omega),
                                   _ptr(grad_S0), B, L, m, c, _ptr(workspace),
                                   workspace.numel() if workspace is not None else 0, _stream(stream)),
           "memoroid_ffm_bwd")


def memoroid_starts_from_offsets(offsets, E, L, start, stream=None):
    _need_cuda(offsets, start)
    _check(load().memoroid_starts_from_offsets(_ptr(offsets), E, L, _ptr(start), _stream(stream)),
           "memoroid_starts_from_offsets")


def memoroid_offsets_workspace_bytes(L) -> int:
    return int(load().memoroid_offsets_workspace_bytes(L))


def memoroid_offsets_from_starts(start, L, offsets, count, workspace, stream=None):
    _need_cuda(start, offsets, count, workspace)
    _check(load().memoroid_offsets_from_starts(_ptr(start), L, _ptr(offsets), _ptr(count), _ptr(workspace),
                                               workspace.numel() if workspace is not None else 0,
                                               _stream(stream)),
           "memoroid_offsets_from_starts")


def memoroid_get_device_error(workspace, stream=None) -> int:
    return int(load().memoroid_get_device_error(_ptr(workspace), _stream(stream)))


def memoroid_get_static_device_error(stream=None) -> int:
    return int(load().memoroid_get_static_device_error(_stream(stream)))


def memoroid_debug_set_wait_limit_ns(ns: int) -> None:
    load().memoroid_debug_set_wait_limit_ns(int(ns))


def memoroid_debug_withhold_tile(ticket: int) -> None:
    load().memoroid_debug_withhold_tile(int(ticket))


def memoroid_debug_lnorm_padded(on: bool) -> None:
    load().memoroid_debug_lnorm_padded(1 if on else 0)


# ---------------------------------------------------------------------------
# allocating helpers
# ---------------------------------------------------------------------------

def workspace(nbytes: int, device) -> torch.Tensor:
    # torch's caching allocator returns 512-byte aligned blocks
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def diag_workspace(B, L, D, device) -> torch.Tensor:
    return workspace(memoroid_scan_diag_workspace_bytes(B, L, D), device)


def diag_fwd(lam, u, start, h0=None, want_last=True, ws=None, out=None, stream=None):
    """h, h_last = scan of u ([B,L,D] complex64) with lambda ([D] or [B,L,D])."""
    B, L, D = u.shape
    per_step = lam.dim() == 3
    if ws is None:
        ws = diag_workspace(B, L, D, u.device)
    h = torch.empty_like(u) if out is None else out
    h_last = torch.empty((B, D), dtype=u.dtype, device=u.device) if want_last else None
    memoroid_scan_diag_fwd(lam, per_step, u, start, h0, h, h_last, B, L, D, ws, stream)
    return h, h_last


def diag_bwd(lam, start, h, grad_h, grad_h_last=None, h0=None, want_lambda=True, want_h0=False,
             ws=None, out=None, stream=None):
    """grad_u, grad_lambda, grad_h0 of the diagonal scan."""
    B, L, D = grad_h.shape
    per_step = lam.dim() == 3
    if ws is None:
        ws = diag_workspace(B, L, D, grad_h.device)
    grad_u = torch.empty_like(grad_h) if out is None else out
    grad_lambda = torch.empty_like(lam) if want_lambda else None
    grad_h0 = torch.empty((B, D), dtype=grad_h.dtype, device=grad_h.device) if want_h0 else None
    memoroid_scan_diag_bwd(lam, per_step, start, h0, h, grad_h, grad_h_last, grad_u, grad_lambda, grad_h0,
                           B, L, D, ws, stream)
    return grad_u, grad_lambda, grad_h0


def linattn_workspace(B, L, H, d, device, chunk=64) -> torch.Tensor:
    return workspace(memoroid_scan_linattn_workspace_bytes(B, L, H, d, d, chunk), device)


def linattn_fwd(q, k, v, gamma, start, S0=None, want_last=True, chunk=64, ws=None, out=None, stream=None):
    """y, S_last of the decayed linear-attention memoroid.  q, k, v: bf16
    [B,L,H,d] (torch.bfloat16, or their bits as int16/uint16); gamma: fp32 [H]
    or [B,L,H]; start: uint8 [B,L]; S0: fp32 [B,H,d,d] or None."""
    B, L, H, d = q.shape
    per_step = gamma.dim() == 3
    if ws is None:
        ws = linattn_workspace(B, L, H, d, q.device, chunk)
    y = torch.empty((B, L, H, d), dtype=torch.float32, device=q.device) if out is None else out
    S_last = torch.empty((B, H, d, d), dtype=torch.float32, device=q.device) if want_last else None
    memoroid_scan_linattn_fwd(q, k, v, MEMOROID_BF16, gamma, per_step, start, S0, y, S_last, B, L, H, d, d, chunk,
                              ws, stream)
    return y, S_last


def linattn_bwd(q, k, v, gamma, start, grad_y, grad_S_last=None, S0=None, want_gamma=True, want_S0=False, chunk=64,
                ws=None, stream=None):
    """dq, dk, dv, dgamma, dS0 of the decayed linear-attention memoroid."""
    B, L, H, d = q.shape
    per_step = gamma.dim() == 3
    if ws is None:
        ws = linattn_workspace(B, L, H, d, q.device, chunk)
    dq = torch.empty((B, L, H, d), dtype=torch.float32, device=q.device)
    dk = torch.empty_like(dq)
    dv = torch.empty_like(dq)
    dgamma = torch.empty_like(gamma) if want_gamma else None
    dS0 = torch.empty((B, H, d, d), dtype=torch.float32, device=q.device) if want_S0 else None
    memoroid_scan_linattn_bwd(q, k, v, MEMOROID_BF16, gamma, per_step, start, S0, grad_y, grad_S_last, dq, dk, dv,
                              dgamma, dS0, B, L, H, d, d, chunk, ws, stream)
    return dq, dk, dv, dgamma, dS0


def discounted_return(r, start, gamma, boot=None, ws=None, stream=None):
    """G [B, L]: per-step discounted return within episodes."""
    B, L = r.shape
    if ws is None:
        ws = workspace(memoroid_returns_workspace_bytes(B, L), r.device)
    G = torch.empty_like(r)
    memoroid_discounted_return(r, start, gamma, boot, G, B, L, ws, stream)
    return G


def gae(r, v, start, gamma, lam, v_boot=None, ws=None, stream=None):
    """A [B, L]: per-step generalised advantage estimate within episodes."""
    B, L = r.shape
    if ws is None:
        ws = workspace(memoroid_returns_workspace_bytes(B, L), r.device)
    A = torch.empty_like(r)
    memoroid_gae(r, v, start, gamma, lam, v_boot, A, B, L, ws, stream)
    return A


def linattn_norm_fwd(q, k, v, gamma, start, S0=None, z0=None, want_last=True, ws=None, stream=None):
    """Linear Transformer with phi = 1 + ELU and its normalizer: q, k, v as
    int16 views of bf16 [B, L, H, d]; returns y, den, S_last, z_last."""
    B, L, H, d = q.shape
    per = 1 if gamma.dim() == 3 else 0
    if ws is None:
        ws = workspace(memoroid_linattn_norm_workspace_bytes(B, L, H, d), q.device)
    y = torch.empty((B, L, H, d), dtype=torch.float32, device=q.device)
    den = torch.empty((B, L, H), dtype=torch.float32, device=q.device)
    S_last = torch.empty((B, H, d, d), dtype=torch.float32, device=q.device) if want_last else None
    z_last = torch.empty((B, H, d), dtype=torch.float32, device=q.device) if want_last else None
    memoroid_linattn_norm_fwd(q, k, v, gamma, per, start, S0, z0, y, den, S_last, z_last, B, L, H, d, ws, stream)
    return y, den, S_last, z_last


def linattn_norm_bwd(q, k, v, gamma, start, y, den, grad_y, grad_S_last=None, grad_z_last=None, S0=None, z0=None,
                     want_gamma=True, want_S0=False, ws=None, stream=None):
    """Backward of linattn_norm_fwd: dq, dk, dv, dgamma, dS0, dz0."""
    B, L, H, d = q.shape
    per = 1 if gamma.dim() == 3 else 0
    if ws is None:
        ws = workspace(memoroid_linattn_norm_workspace_bytes(B, L, H, d), q.device)
    dq = torch.empty((B, L, H, d), dtype=torch.float32, device=q.device)
    dk, dv = torch.empty_like(dq), torch.empty_like(dq)
    dgamma = torch.empty_like(gamma) if want_gamma else None
    dS0 = torch.empty((B, H, d, d), dtype=torch.float32, device=q.device) if want_S0 else None
    dz0 = torch.empty((B, H, d), dtype=torch.float32, device=q.device) if want_S0 else None
    memoroid_linattn_norm_bwd(q, k, v, gamma, per, start, S0, z0, y, den, grad_y, grad_S_last, grad_z_last, dq, dk,
                              dv, dgamma, dS0, dz0, B, L, H, d, ws, stream)
    return dq, dk, dv, dgamma, dS0, dz0


def tbb_sample(begin, N, draws, B, ws=None, stream=None):
    """Algorithm 2 with the draws given: returns start [B] uint8, src [B]
    int64 and n_used [1] int64 (device tensors).  begin: int64 [E] episode
    begin indices into a buffer of N transitions; draws: int64 [K]."""
    E, K = begin.numel(), draws.numel()
    if ws is None:
        ws = workspace(memoroid_tbb_workspace_bytes(K), begin.device)
    start = torch.empty(B, dtype=torch.uint8, device=begin.device)
    src = torch.empty(B, dtype=torch.int64, device=begin.device)
    n_used = torch.empty(1, dtype=torch.int64, device=begin.device)
    memoroid_tbb_sample(begin, E, N, draws, K, B, start, src, n_used, ws, stream)
    return start, src, n_used


def gather_rows(rows, src, ws=None, stream=None):
    """out[t] = rows[src[t]] for a [N, ...] tensor of rows (any dtype)."""
    N = rows.shape[0]
    B = src.numel()
    row_bytes = rows[0].numel() * rows.element_size() if N > 0 else rows.element_size()
    if ws is None:
        ws = workspace(256, rows.device)
    out = torch.empty((B,) + tuple(rows.shape[1:]), dtype=rows.dtype, device=rows.device)
    memoroid_gather_rows(rows, N, row_bytes, src, B, out, ws, stream)
    return out


def ffm_workspace(B, L, m, c, device) -> torch.Tensor:
    return workspace(memoroid_ffm_workspace_bytes(B, L, m, c), device)


def ffm_fwd(x, alpha, omega, start, S0=None, want_last=True, ws=None, stream=None):
    """Fast and Forgetful Memory: x [B, L, m] fp32, alpha [m], omega [c];
    returns z [B, L, 2*m*c] (Re || Im of the state) and S_last [B, m, c]
    complex64 (or None)."""
    B, L, m = x.shape
    c = omega.shape[0]
    if ws is None:
        ws = ffm_workspace(B, L, m, c, x.device)
    z = torch.empty((B, L, 2 * m * c), dtype=torch.float32, device=x.device)
    S_last = torch.empty((B, m, c), dtype=torch.complex64, device=x.device) if want_last else None
    memoroid_ffm_fwd(x, alpha, omega, start, S0, z, S_last, B, L, m, c, ws, stream)
    return z, S_last


def ffm_bwd(alpha, omega, start, z, grad_z, grad_S_last=None, S0=None, want_params=True, want_S0=False, ws=None,
            stream=None):
    """Backward of ffm_fwd: grad_x [B, L, m], grad_alpha [m], grad_omega [c]
    (None unless want_params), grad_S0 [B, m, c] (None unless want_S0)."""
    B, L = z.shape[0], z.shape[1]
    m, c = alpha.shape[0], omega.shape[0]
    if ws is None:
        ws = ffm_workspace(B, L, m, c, z.device)
    gx = torch.empty((B, L, m), dtype=torch.float32, device=z.device)
    ga = torch.empty(m, dtype=torch.float32, device=z.device) if want_params else None
    go = torch.empty(c, dtype=torch.float32, device=z.device) if want_params else None
    gS0 = torch.empty((B, m, c), dtype=torch.complex64, device=z.device) if want_S0 else None
    memoroid_ffm_bwd(alpha, omega, start, S0, z, grad_z, grad_S_last, gx, ga, go, gS0, B, L, m, c, ws, stream)
    return gx, ga, go, gS0


def starts_from_offsets(offsets, L, stream=None):
    start = torch.empty(L, dtype=torch.uint8, device=offsets.device)
    memoroid_starts_from_offsets(offsets, offsets.numel(), L, start, stream)
    return start


def offsets_from_starts(start, stream=None):
    L = start.numel()
    offsets = torch.empty(max(L, 1), dtype=torch.int64, device=start.device)
    count = torch.empty(1, dtype=torch.int64, device=start.device)
    ws = workspace(memoroid_offsets_workspace_bytes(L), start.device)
    memoroid_offsets_from_starts(start, L, offsets, count, ws, stream)
    return offsets, count


class DiagScan(torch.autograd.Function):
    """Autograd wrapper: h = DiagScan.apply(lam, u, start, h0)."""

    @staticmethod
    def forward(ctx, lam, u, start, h0):
        h, _ = diag_fwd(lam, u, start, h0, want_last=False)
        ctx.save_for_backward(lam, start, h0 if h0 is not None else torch.empty(0), h)
        ctx.has_h0 = h0 is not None
        return h

    @staticmethod
    def backward(ctx, grad_h):
        lam, start, h0, h = ctx.saved_tensors
        h0 = h0 if ctx.has_h0 else None
        gu, gl, gh0 = diag_bwd(lam, start, h, grad_h.contiguous(), None, h0,
                               want_lambda=ctx.needs_input_grad[0], want_h0=ctx.has_h0)
        return gl, gu, None, gh0


def _bf16_bits(t):
    """The int16 view the C ABI takes for a bf16 tensor (bf16 tensors in, int16 views pass through)."""
    if t.dtype == torch.bfloat16:
        return t.contiguous().view(torch.int16)
    if t.dtype == torch.int16:
        return t.contiguous()
    raise ValueError("q, k, v must be bfloat16 tensors (or their int16 bit views)")


class LinAttnScan(torch.autograd.Function):
    """Autograd wrapper of the decayed linear-attention memoroid:
    y = LinAttnScan.apply(q, k, v, gamma, start, S0) with q, k, v bfloat16
    [B, L, H, d], gamma fp32 [H] or [B, L, H], S0 fp32 [B, H, d, d] or None.
    Gradients come back in the inputs' dtypes (dq, dk, dv rounded to bf16)."""

    @staticmethod
    def forward(ctx, q, k, v, gamma, start, S0=None):
        qb, kb, vb = _bf16_bits(q), _bf16_bits(k), _bf16_bits(v)
        y, _ = linattn_fwd(qb, kb, vb, gamma.contiguous(), start, S0, want_last=False)
        ctx.save_for_backward(qb, kb, vb, gamma, start, S0 if S0 is not None else torch.empty(0))
        ctx.has_S0 = S0 is not None
        ctx.dtypes = (q.dtype, k.dtype, v.dtype)
        return y

    @staticmethod
    def backward(ctx, grad_y):
        qb, kb, vb, gamma, start, S0 = ctx.saved_tensors
        S0 = S0 if ctx.has_S0 else None
        dq, dk, dv, dg, dS0 = linattn_bwd(qb, kb, vb, gamma.contiguous(), start, grad_y.contiguous(), None, S0,
                                          want_gamma=ctx.needs_input_grad[3], want_S0=ctx.has_S0)

        def cast(g, dt):
            return g.to(torch.bfloat16) if dt == torch.bfloat16 else None  # int16 views take no gradient

        return cast(dq, ctx.dtypes[0]), cast(dk, ctx.dtypes[1]), cast(dv, ctx.dtypes[2]), dg, None, dS0


class FFMScan(torch.autograd.Function):
    """Autograd wrapper of the Fast and Forgetful Memory memoroid:
    z = FFMScan.apply(x, alpha, omega, start, S0) with x fp32 [B, L, m],
    alpha [m], omega [c], S0 complex64 [B, m, c] or None; z = Re(X) || Im(X)."""

    @staticmethod
    def forward(ctx, x, alpha, omega, start, S0=None):
        z, _ = ffm_fwd(x.contiguous(), alpha.contiguous(), omega.contiguous(), start, S0, want_last=False)
        ctx.save_for_backward(alpha, omega, start, S0 if S0 is not None else torch.empty(0), z)
        ctx.has_S0 = S0 is not None
        return z

    @staticmethod
    def backward(ctx, grad_z):
        alpha, omega, start, S0, z = ctx.saved_tensors
        S0 = S0 if ctx.has_S0 else None
        gx, ga, go, gS0 = ffm_bwd(alpha.contiguous(), omega.contiguous(), start, z, grad_z.contiguous(), None, S0,
                                  want_params=ctx.needs_input_grad[1] or ctx.needs_input_grad[2],
                                  want_S0=ctx.has_S0)
        return gx, ga, go, None, gS0


class LinAttnNormScan(torch.autograd.Function):
    """Autograd wrapper of the Linear Transformer with phi = 1 + ELU and its
    normalizer: y = LinAttnNormScan.apply(q, k, v, gamma, start) with q, k, v
    bfloat16 [B, L, H, d] (d a multiple of 8, at most 120)."""

    @staticmethod
    def forward(ctx, q, k, v, gamma, start):
        qb, kb, vb = _bf16_bits(q), _bf16_bits(k), _bf16_bits(v)
        y, den, _, _ = linattn_norm_fwd(qb, kb, vb, gamma.contiguous(), start, want_last=False)
        ctx.save_for_backward(qb, kb, vb, gamma, start, y, den)
        ctx.dtypes = (q.dtype, k.dtype, v.dtype)
        return y

    @staticmethod
    def backward(ctx, grad_y):
        qb, kb, vb, gamma, start, y, den = ctx.saved_tensors
        dq, dk, dv, dg, _, _ = linattn_norm_bwd(qb, kb, vb, gamma.contiguous(), start, y, den, grad_y.contiguous(),
                                                want_gamma=ctx.needs_input_grad[3])

        def cast(g, dt):
            return g.to(torch.bfloat16) if dt == torch.bfloat16 else None

        return cast(dq, ctx.dtypes[0]), cast(dk, ctx.dtypes[1]), cast(dv, ctx.dtypes[2]), dg, None
