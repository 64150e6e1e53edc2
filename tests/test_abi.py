"""The C-ABI library loads and exports every function include/msi.h declares;
host-only entry points answer without a GPU."""
import ctypes
import os
import re

import pytest

from paper_2608_23805_gb300 import build as B
from paper_2608_23805_gb300 import native as N

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "msi.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return ctypes.CDLL(B.LIB)


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*[A-Za-z_][\w\s\*]*?\b(msi_\w+)\s*\(", src, flags=re.M)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert "msi_moe_forward" in names and "msi_plan_create" in names and len(names) >= 18
    for n in names:
        assert hasattr(lib, n), n
        assert n in N._SIGS, "binding misses " + n


def test_host_only_entry_points(lib):
    l = N.lib()
    assert l.msi_extent_bytes(2048, 512, N.MSI_W_BF16) == 6291456
    assert l.msi_extent_bytes(256, 128, N.MSI_W_BF16) == 196608
    assert l.msi_extent_bytes(2048, 512, N.MSI_W_Q4G32) == 1769472
    assert l.msi_extent_bytes(0, 512, N.MSI_W_BF16) == 0
    assert l.msi_status_string(N.MSI_ERR_STALE_GENERATION) == b"stale generation"
    assert l.msi_plan_create(None, None) == N.MSI_ERR_INVALID_ARG
    assert l.msi_plan_destroy(None) == N.MSI_ERR_INVALID_ARG
    assert l.msi_kernel_launches(None) == 0


def test_struct_layouts_match_header():
    assert ctypes.sizeof(N.msi_trace_rec) == 40
    assert ctypes.sizeof(N.msi_route_event) == 32
    assert ctypes.sizeof(N.msi_counters) == 56
