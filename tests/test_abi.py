"""The C-ABI library builds, loads on a CPU-only host, and exports every
symbol that include/memoroid.h declares; argument validation runs on the host.

The validation cases below all fail before any CUDA call is made, so they use
dummy pointer values and never touch a device.
"""
import ctypes
import os
import re

import pytest

from paper_2402_09900_gb300 import build as native_build
from paper_2402_09900_gb300 import memoroid as m

HEADER_DIR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")


def _declared():
    names = set()
    for fn in os.listdir(HEADER_DIR):
        if fn.endswith(".h"):
            text = open(os.path.join(HEADER_DIR, fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(memoroid_\w+)\s*\(", text))
    return names


@pytest.fixture(scope="module")
def lib():
    native_build.build()
    return m.load()


def test_exports_every_declared_symbol(lib):
    declared = _declared()
    assert declared, "no declarations found"
    raw = ctypes.CDLL(m.lib_path())
    missing = [n for n in sorted(declared) if not hasattr(raw, n)]
    assert not missing, missing
    # the binding covers the same set of names
    assert declared == set(m.SIGNATURES), declared ^ set(m.SIGNATURES)


def test_status_strings(lib):
    for code in range(7):
        assert m.status_string(code)
    assert lib.memoroid_version() >= 100


def test_workspace_queries(lib):
    assert lib.memoroid_scan_diag_workspace_bytes(1, 1 << 20, 256) > 0
    assert lib.memoroid_scan_diag_workspace_bytes(1, 10, 3) == 0  # odd D
    assert lib.memoroid_scan_diag_workspace_bytes(-1, 10, 4) == 0
    assert lib.memoroid_offsets_workspace_bytes(1000) >= 256


def test_diag_kernel_counts(lib):
    # one tape of 256 channels is 4 chains, cut into segments: the scan, the segment
    # carries and the fix-up; the backward adds the two grad_lambda reduction stages
    assert lib.memoroid_scan_diag_kernels_per_call(1, 1 << 20, 256, 0, 0, 0) == 3
    assert lib.memoroid_scan_diag_kernels_per_call(1, 1 << 20, 256, 0, 1, 1) == 5
    assert lib.memoroid_scan_diag_kernels_per_call(1, 1 << 20, 256, 0, 1, 0) == 3
    # 64 tapes of 128 channels are 128 chains, one segment each: the scan alone
    assert lib.memoroid_scan_diag_kernels_per_call(64, 16384, 128, 0, 0, 0) == 1
    assert lib.memoroid_scan_diag_kernels_per_call(64, 16384, 128, 0, 1, 1) == 3
    # a per-step lambda has no grad_lambda reduction (its gradient is per step)
    assert lib.memoroid_scan_diag_kernels_per_call(1, 1 << 20, 256, 1, 1, 1) == 3


FAKE = 0x10000000  # 256-byte aligned dummy address, never dereferenced


def _fwd(lib, lam=FAKE, ps=0, u=FAKE, start=FAKE, h0=None, h=FAKE, hl=None, B=1, L=8, D=4,
         ws=FAKE, wsb=1 << 30):
    return lib.memoroid_scan_diag_fwd(lam, ps, u, start, h0, h, hl, B, L, D, ws, wsb, None)


def test_fwd_validation(lib):
    assert _fwd(lib, D=3) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, B=-1) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, ps=2) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, u=None) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, lam=None) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, start=None) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, u=FAKE + 8) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, h0=FAKE + 4) == m.MEMOROID_ERR_INVALID_ARG
    assert _fwd(lib, ws=None) == m.MEMOROID_ERR_WORKSPACE
    assert _fwd(lib, ws=FAKE + 16) == m.MEMOROID_ERR_WORKSPACE
    assert _fwd(lib, wsb=16) == m.MEMOROID_ERR_WORKSPACE


def test_bwd_validation(lib):
    def bwd(grad_u=FAKE, h=FAKE + 0x1000, D=4, ws=FAKE, wsb=1 << 30, grad_h=FAKE):
        return lib.memoroid_scan_diag_bwd(FAKE, 0, FAKE, None, h, grad_h, None, grad_u, None, None,
                                          1, 8, D, ws, wsb, None)
    assert bwd(D=5) == m.MEMOROID_ERR_INVALID_ARG
    assert bwd(grad_u=None) == m.MEMOROID_ERR_INVALID_ARG
    assert bwd(grad_u=FAKE + 0x1000) == m.MEMOROID_ERR_INVALID_ARG  # aliases h
    assert bwd(grad_h=FAKE + 8) == m.MEMOROID_ERR_INVALID_ARG
    assert bwd(wsb=0) == m.MEMOROID_ERR_WORKSPACE


def test_tape_index_validation(lib):
    assert lib.memoroid_starts_from_offsets(FAKE, -1, 8, FAKE, None) == m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_starts_from_offsets(None, 3, 8, FAKE, None) == m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_offsets_from_starts(FAKE, 8, FAKE, None, FAKE, 4096, None) == m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_offsets_from_starts(FAKE, 8, FAKE, FAKE, None, 4096, None) == m.MEMOROID_ERR_WORKSPACE
    assert lib.memoroid_offsets_from_starts(FAKE, 8, FAKE, FAKE, FAKE, 8, None) == m.MEMOROID_ERR_WORKSPACE


def test_ffm_validation(lib):
    assert lib.memoroid_ffm_workspace_bytes(1, 1 << 20, 64, 4) > lib.memoroid_scan_diag_workspace_bytes(1, 1 << 20, 256)
    for m_, c_ in ((6, 4), (8, 3), (8, 32), (0, 4)):
        assert lib.memoroid_ffm_workspace_bytes(1, 100, m_, c_) == 0
        assert lib.memoroid_ffm_kernels_per_call(1, 100, m_, c_, 0, 0) == -1

    def fwd(x=FAKE, z=FAKE + 0x1000, m_=8, c_=4, ws=FAKE, wsb=1 << 30, S0=None):
        return lib.memoroid_ffm_fwd(x, FAKE, FAKE, FAKE, S0, z, None, 1, 8, m_, c_, ws, wsb, None)

    assert fwd(m_=6) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(c_=3) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(x=None) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(x=FAKE + 8) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(S0=FAKE + 4) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(ws=None) == m.MEMOROID_ERR_WORKSPACE
    assert fwd(wsb=64) == m.MEMOROID_ERR_WORKSPACE

    def bwd(gx=FAKE + 0x2000, z=FAKE, gz=FAKE + 0x1000, c_=4, wsb=1 << 30):
        return lib.memoroid_ffm_bwd(FAKE, FAKE, FAKE, None, z, gz, None, gx, None, None, None, 1, 8, 8, c_,
                                    FAKE, wsb, None)

    assert bwd(c_=5) == m.MEMOROID_ERR_INVALID_ARG
    assert bwd(gx=None) == m.MEMOROID_ERR_INVALID_ARG
    assert bwd(gx=FAKE) == m.MEMOROID_ERR_INVALID_ARG  # aliases z
    assert bwd(gx=FAKE + 0x1000) == m.MEMOROID_ERR_INVALID_ARG  # aliases grad_z
    assert bwd(wsb=0) == m.MEMOROID_ERR_WORKSPACE


def test_returns_validation(lib):
    assert lib.memoroid_discounted_return(FAKE, FAKE, 0.9, None, FAKE, -1, 8, FAKE, 4096, None) == \
        m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_discounted_return(None, FAKE, 0.9, None, FAKE, 1, 8, FAKE, 4096, None) == \
        m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_discounted_return(FAKE, FAKE, 0.9, None, FAKE, 1, 8, None, 4096, None) == \
        m.MEMOROID_ERR_WORKSPACE
    assert lib.memoroid_gae(FAKE, None, FAKE, 0.9, 0.9, None, FAKE, 1, 8, FAKE, 4096, None) == \
        m.MEMOROID_ERR_INVALID_ARG


def test_linattn_norm_validation(lib):
    assert lib.memoroid_linattn_norm_workspace_bytes(1, 4096, 4, 64) > 0
    for d in (0, 4, 12, 128):
        assert lib.memoroid_linattn_norm_workspace_bytes(1, 100, 2, d) == 0
        assert lib.memoroid_linattn_norm_kernels_per_call(1, 100, 2, d, 0, 0, 0) == -1
    # the forward of 64-channel heads is one fused linear-attention call: no operand
    # padding and no division kernel; other widths keep them
    fwd64 = lib.memoroid_linattn_norm_kernels_per_call(1, 4096, 4, 64, 0, 0, 0)
    fwd32 = lib.memoroid_linattn_norm_kernels_per_call(1, 4096, 4, 32, 0, 0, 0)
    assert fwd32 - fwd64 == 2
    # the backward of 64-channel heads builds its operands and applies the chain rule
    # through phi inside the kernels (no padding kernel, no chain-rule kernel)
    assert lib.memoroid_linattn_norm_kernels_per_call(1, 4096, 4, 32, 1, 0, 0) - \
        lib.memoroid_linattn_norm_kernels_per_call(1, 4096, 4, 64, 1, 0, 0) == 2

    def fwd(q=FAKE, d=64, ws=FAKE, wsb=1 << 40, gps=0):
        return lib.memoroid_linattn_norm_fwd(q, FAKE, FAKE, FAKE, gps, FAKE, None, None, FAKE + 0x1000, None, None,
                                             None, 1, 256, 2, d, ws, wsb, None)

    assert fwd(d=12) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(gps=3) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(q=None) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(q=FAKE + 8) == m.MEMOROID_ERR_INVALID_ARG
    assert fwd(ws=None) == m.MEMOROID_ERR_WORKSPACE
    assert fwd(wsb=1024) == m.MEMOROID_ERR_WORKSPACE
    # the backward needs den, grad_y and the three gradients
    assert lib.memoroid_linattn_norm_bwd(FAKE, FAKE, FAKE, FAKE, 0, FAKE, None, None, FAKE, None, FAKE, None, None,
                                         FAKE, FAKE, FAKE, None, None, None, 1, 256, 2, 64, FAKE, 1 << 40,
                                         None) == m.MEMOROID_ERR_INVALID_ARG


def test_tbb_validation(lib):
    assert lib.memoroid_tbb_workspace_bytes(1000) >= 256 + 8 * 1002
    assert lib.memoroid_tbb_workspace_bytes(-1) == 0
    assert lib.memoroid_tbb_sample(FAKE, 4, 9, FAKE, 3, -1, FAKE, FAKE, None, FAKE, 1 << 20, None) == \
        m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_tbb_sample(FAKE, 4, 9, FAKE, 3, 5, None, FAKE, None, FAKE, 1 << 20, None) == \
        m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_tbb_sample(FAKE, 4, 9, FAKE, 3, 5, FAKE, FAKE + 4, None, FAKE, 1 << 20, None) == \
        m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_tbb_sample(FAKE, 4, 9, FAKE, 3, 5, FAKE, FAKE, None, FAKE, 16, None) == \
        m.MEMOROID_ERR_WORKSPACE
    assert lib.memoroid_gather_rows(FAKE, 10, 0, FAKE, 4, FAKE, FAKE, 256, None) == m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_gather_rows(FAKE, 10, 16, None, 4, FAKE, FAKE, 256, None) == m.MEMOROID_ERR_INVALID_ARG
    assert lib.memoroid_gather_rows(FAKE, 10, 16, FAKE, 4, FAKE, None, 256, None) == m.MEMOROID_ERR_WORKSPACE
