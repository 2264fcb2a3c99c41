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
    for code in range(6):
        assert m.status_string(code)
    assert lib.memoroid_version() >= 100


def test_workspace_queries(lib):
    assert lib.memoroid_scan_diag_workspace_bytes(1, 1 << 20, 256) > 0
    assert lib.memoroid_scan_diag_workspace_bytes(1, 10, 3) == 0  # odd D
    assert lib.memoroid_scan_diag_workspace_bytes(-1, 10, 4) == 0
    assert lib.memoroid_offsets_workspace_bytes(1000) >= 256


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
