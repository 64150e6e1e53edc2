"""Bounded source service on the host (no GPU): extents read from a file into
fixed aligned windows (paper, Sec. "Bounded Source Service").  Checked: the
bytes delivered equal the file's extent bytes; covering reads under O_DIRECT
add exactly the padding that rounds each extent out to the alignment, and
padding is counted apart from logical bytes; extent overflow, short reads and
an exhausted window set are rejected; reads in flight never exceed the
window count; a source with a window still held refuses to close."""
import ctypes
import os

import numpy as np
import pytest

import synth
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

HEADER = 100  # extents start off the 4096-byte grid


def _file(tmp_path, cfg):
    E, eb = cfg.n_experts, cfg.extent_bytes
    win = np.empty(E * eb, dtype=np.uint8)
    synth.fill_extents(cfg, 0, win)
    path = str(tmp_path / "experts.bin")
    with open(path, "wb") as f:
        f.write(bytes(range(HEADER)))
        f.write(win.tobytes())
    return path, win, [HEADER + e * eb for e in range(E)]


def _open(path, eb, direct, n=4):
    try:
        return api.Source(path, eb + 2 * 4096, n_windows=n, direct=direct)
    except N.MsiError as e:
        if direct and e.status == N.MSI_ERR_UNSUPPORTED:
            pytest.skip("file system refuses O_DIRECT")
        raise


@pytest.mark.parametrize("direct", [False, True])
def test_reads_deliver_the_extents_with_covering_padding(tmp_path, direct):
    cfg = synth.config("tiny")
    eb = cfg.extent_bytes
    path, win, off = _file(tmp_path, cfg)
    src = _open(path, eb, direct)
    phys = 0
    for e in range(cfg.n_experts):
        w, got = src.read(off[e], eb)
        assert np.array_equal(got, win[e * eb:(e + 1) * eb])
        src.release(w)
        lead = off[e] % 4096 if direct else 0
        phys += ((lead + eb + 4095) // 4096) * 4096 if direct else eb
    st = src.stats()
    assert st["reads"] == cfg.n_experts and st["rejected"] == 0
    assert st["logical_bytes"] == cfg.n_experts * eb
    assert st["physical_bytes"] == phys
    assert st["padding_bytes"] == phys - cfg.n_experts * eb
    assert 1 <= st["max_in_flight"] <= src.n_windows
    src.close()


def test_extent_overflow_and_short_read_are_rejected(tmp_path):
    cfg = synth.config("tiny")
    eb = cfg.extent_bytes
    path, win, off = _file(tmp_path, cfg)
    src = _open(path, eb, False)
    size = os.path.getsize(path)
    with pytest.raises(N.MsiError) as ei:
        src.read(size - 10, 100)  # past the end of the file
    assert ei.value.status == N.MSI_ERR_SOURCE
    os.truncate(path, off[-1] + eb // 2)  # the last extent loses its second half
    with pytest.raises(N.MsiError) as ei:
        src.read(off[-1], eb)
    assert ei.value.status == N.MSI_ERR_SOURCE
    w, got = src.read(off[0], eb)  # a whole extent still reads
    assert np.array_equal(got, win[:eb])
    src.release(w)
    assert src.stats()["rejected"] == 2
    src.close()


def test_held_windows_bound_the_reads(tmp_path):
    cfg = synth.config("tiny")
    eb = cfg.extent_bytes
    path, win, off = _file(tmp_path, cfg)
    src = _open(path, eb, False, n=3)
    held = [src.read(off[e], eb)[0] for e in range(3)]
    assert sorted(held) == [0, 1, 2]
    with pytest.raises(N.MsiError) as ei:
        src.read(off[3], eb)  # every window is HostReady and held
    assert ei.value.status == N.MSI_ERR_SLOT_BUSY
    src.release(held[1])
    w, got = src.read(off[3], eb)
    assert w == held[1] and np.array_equal(got, win[3 * eb:4 * eb])
    for x in (held[0], held[2], w):
        src.release(x)
    src.close()


def test_open_rejects_bad_descriptors(tmp_path):
    cfg = synth.config("tiny")
    path, _, _ = _file(tmp_path, cfg)
    buf = np.zeros(8192 * 3, dtype=np.uint8)
    base = buf.ctypes.data + (-buf.ctypes.data) % 4096
    h = ctypes.c_void_p()
    bad = [
        N.msi_source_desc(path.encode(), 0, 4096, 0, base, 8192),          # no window
        N.msi_source_desc(path.encode(), 0, 3000, 2, base, 8192),          # alignment not 2^n
        N.msi_source_desc(path.encode(), 1, 4096, 2, base + 16, 8192),     # direct, misaligned
        N.msi_source_desc(path.encode(), 0, 4096, N.MSI_MAX_WINDOWS + 1, base, 8192),
    ]
    for d in bad:
        assert N.lib().msi_source_open(ctypes.byref(d), ctypes.byref(h)) == N.MSI_ERR_INVALID_ARG
    d = N.msi_source_desc(str(tmp_path / "missing").encode(), 0, 4096, 2, base, 8192)
    assert N.lib().msi_source_open(ctypes.byref(d), ctypes.byref(h)) == N.MSI_ERR_SOURCE


def test_close_refuses_while_a_window_is_held(tmp_path):
    """Shutdown with a live consumer (paper, Table 6): a caller still holds a
    HostReady window, so close refuses and changes nothing; once the window is
    released every window is Free and close succeeds."""
    cfg = synth.config("tiny")
    eb = cfg.extent_bytes
    path, win, off = _file(tmp_path, cfg)
    src = _open(path, eb, False, n=2)
    w, got = src.read(off[1], eb)
    with pytest.raises(N.MsiError) as ei:
        src.close()
    assert ei.value.status == N.MSI_ERR_SLOT_BUSY
    assert src.stats()["windows_busy"] == 1
    assert np.array_equal(got, win[eb:2 * eb])  # the held bytes are untouched
    src.release(w)
    assert src.stats()["windows_busy"] == 0
    src.close()
