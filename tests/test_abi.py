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


STRUCTS = ["msi_plan_desc", "msi_route_event", "msi_trace_rec", "msi_counters", "msi_source_desc",
           "msi_source_stats"]


def test_struct_layouts_match_header(tmp_path):
    """Sizes and field offsets of the binding's structures equal those the C
    compiler gives the header's."""
    src = tmp_path / "layout.c"
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "msi.h"', "int main(void) {"]
    for name in STRUCTS:
        lines.append('printf("%s %%zu\\n", sizeof(%s));' % (name, name))
        for f, _ in getattr(N, name)._fields_:
            lines.append('printf("%s.%s %%zu\\n", offsetof(%s, %s));' % (name, f, name, f))
    lines.append("return 0; }")
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    import subprocess
    subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)],
                   check=True)
    got = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                 check=True).stdout.splitlines())
    for name in STRUCTS:
        st = getattr(N, name)
        assert ctypes.sizeof(st) == int(got[name]), name
        for f, _ in st._fields_:
            assert getattr(st, f).offset == int(got[name + "." + f]), (name, f)
