"""The C-ABI library builds for sm_103a and exports every entry point that
include/pe.h declares (no device calls: this runs without a GPU)."""
import os
import re

import pytest

from paper_2608_11226_gb300 import build, pe

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared():
    src = open(os.path.join(ROOT, "include", "pe.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pe_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared()
    for must in ("pe_env_create", "pe_rollout", "pe_gae", "pe_ppo_update", "pe_fleet_windows",
                 "pe_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol():
    path = build.build()
    assert os.path.exists(path)
    L = pe.lib()
    for name in declared():
        assert hasattr(L, name), name
    assert set(pe.EXPORTS) <= set(declared())


def test_error_path_without_device():
    """Argument errors are caught on the host before any CUDA call."""
    L = pe.lib()
    import ctypes as C
    assert L.pe_fleet_workspace_bytes(0, 10, 10) == -1
    net = pe.Net(16, 128, 5, 0)
    assert L.pe_param_count(C.byref(net)) == 38150
    rc = L.pe_gae(None, None, None, None, 4, 4, 0.99, 0.95, None, None, None)
    assert rc == pe.PE_EINVAL
    assert b"null" in L.pe_last_error()
