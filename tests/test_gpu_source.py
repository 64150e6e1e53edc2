"""Staging through the bounded source service (paper, Sec. "Bounded Source
Service"): extents read from a file into fixed aligned windows, checked, then
copied into slots.  The same calls staged from the file and from host windows
give bit-identical outputs and identical slot traces; a read rejected in the
middle of a streamed call (I/O error, short read) leaves its bundle
unpublished with its slots Vacant, plans no later bundle, writes no output
row, and the next call runs normally."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu

HEADER = 1000  # extents start off the 4096-byte grid: covering reads pad


def _source(case, tmp_path, direct, n_windows=8):
    cfg = case.cfg
    L, E, eb = case.L, cfg.n_experts, cfg.extent_bytes
    path = str(tmp_path / "experts.bin")
    with open(path, "wb") as f:
        f.write(b"\0" * HEADER)
        f.write(case.windows.numpy().tobytes())
    off = np.array([HEADER + i * eb for i in range(L * E)], dtype=np.uint64)
    try:
        src = api.Source(path, eb + 2 * 4096, n_windows=n_windows, direct=direct)
    except N.MsiError as e:
        if direct and e.status == N.MSI_ERR_UNSUPPORTED:
            pytest.skip("file system refuses O_DIRECT")
        raise
    return src, off


@pytest.mark.parametrize("direct,wdtype", [(False, N.MSI_W_BF16), (True, N.MSI_W_BF16),
                                          (True, N.MSI_W_Q4G32)])
def test_streamed_from_file_equals_host_windows(tmp_path, direct, wdtype):
    cfg = synth.config("tiny", wdtype=wdtype)
    a, b = Case(cfg), Case(cfg)
    src, off = _source(b, tmp_path, direct, n_windows=4)
    b.plan.set_source(src, off)
    for call in range(3):
        x = bf16_tensor(synth.hidden(cfg, 0, 50 + call))
        oa, _ = a.plan.forward_streamed(0, x, a.router[0])
        ob, _ = b.plan.forward_streamed(0, x, b.router[0])
        torch.cuda.synchronize()
        assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
        assert torch.equal(oa.view(torch.int16), ob.view(torch.int16))
    assert a.plan.trace() == b.plan.trace()
    st, c = src.stats(), b.plan.counters()
    assert st["reads"] == c["stages"] and st["rejected"] == 0
    assert st["logical_bytes"] == c["stages"] * cfg.extent_bytes
    assert 1 <= st["max_in_flight"] <= 4
    assert st["windows_busy"] == 0  # balanced terminal state: every window Free
    if direct:
        assert st["padding_bytes"] > 0 and st["physical_bytes"] % 4096 == 0
    b.plan.set_source(None)
    src.close()
    a.close()
    b.close()


def test_slot_stage_from_file_matches_oracle(tmp_path):
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    src, off = _source(case, tmp_path, False)
    case.plan.set_source(src, off)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 60)
    out, _ = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out), case.oracle_layer(x_bits)["out"])
    assert src.stats()["reads"] == cfg.n_experts
    case.plan.set_source(None)
    src.close()
    case.close()


@pytest.mark.parametrize("kind", [N.MSI_FAULT_IO_ERROR, N.MSI_FAULT_SHORT_READ,
                                  N.MSI_FAULT_STALE_EPOCH])
def test_rejected_read_mid_call_unwinds_the_remaining_bundles(tmp_path, kind):
    """Qwen-shaped layer with 64 experts, 16 slots (waves of 8): the read of
    an expert in the third wave fails (I/O error, short read, or a completion
    carrying the previous request epoch).  The call returns MSI_ERR_SOURCE; the
    third bundle is not published, its slots are Vacant, no later wave is
    planned; the output buffer keeps its contents; the next call matches the
    oracle."""
    cfg = synth.config("qwen3next_4k", n_experts=64, n_slots=16, tokens=256, lru=True)
    case = Case(cfg)
    src, off = _source(case, tmp_path, False)
    case.plan.set_source(src, off)
    x_bits = synth.hidden(cfg, 0, 61)
    ids = oracle.router(x_bits, case.router_np[0], cfg.top_k)["ids"]
    needed = sorted(set(ids.reshape(-1).tolist()))
    victim = needed[2 * 8 + 3]  # a miss of the third wave (all misses on a cold pool)
    case.plan.inject(kind, 0, victim)
    out = torch.full((cfg.tokens, cfg.hidden), 7.0, dtype=torch.bfloat16, device="cuda")
    rc, out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0], out=out,
                                             check=False)
    torch.cuda.synchronize()
    assert rc == N.MSI_ERR_SOURCE
    assert torch.all(out == 7.0)
    tr = case.plan.trace()
    assert max(r[6] for r in tr) == 2  # no wave after the failing one was planned
    staged3 = [(r[2], r[3]) for r in tr if r[5] == "stage" and r[6] == 2]
    evicted3 = {(r[2], r[3]) for r in tr if r[5] == "evict" and r[6] == 2}
    assert staged3 and all(x in evicted3 for x in staged3)  # the third bundle is unwound
    table = case.plan.slot_table(0)[0]
    assert all(table[e] >= 0 for e in needed[8:16])  # the second wave stays resident
    assert all(table[e] == -1 for e in needed[:8] + needed[16:])  # first evicted by the third
    busy = sum(1 for s in range(cfg.n_slots) if case.plan.slot_state(s) != N.MSI_SLOT_VACANT)
    assert busy == 8
    assert src.stats()["rejected"] == 1
    assert src.stats()["windows_busy"] == 0  # the executor drained: every window Free
    out2, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out2), case.oracle_layer(x_bits)["out"])
    assert src.stats()["windows_busy"] == 0
    case.plan.set_source(None)
    src.close()
    case.close()


def test_reset_and_shutdown_with_source_work(tmp_path):
    """Reset with source work, shutdown with a live consumer (paper, Table 6).
    A streamed call stages through the source, then the plan is reset: the
    reset drains every window copy (all windows Free), advances the epoch and
    evicts every slot; the next call restages everything from the file and
    matches the oracle.  Closing the source while the plan has it attached is
    refused and changes nothing; destroying the plan detaches it, after which
    the source closes."""
    cfg = synth.config("tiny", n_slots=8, lru=True)
    case = Case(cfg)
    src, off = _source(case, tmp_path, False, n_windows=3)
    case.plan.set_source(src, off)
    x_bits = synth.hidden(cfg, 0, 62)
    expect = case.oracle_layer(x_bits)["out"]
    out, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
    reads = src.stats()["reads"]
    epoch = case.plan.reset()
    assert src.stats()["windows_busy"] == 0
    assert all(case.plan.slot_state(s) == N.MSI_SLOT_VACANT for s in range(cfg.n_slots))
    compare_out(bf16_bits(out), expect)
    out2, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out2), expect)
    assert src.stats()["reads"] == 2 * reads and src.stats()["rejected"] == 0
    assert case.plan.reset() == epoch + 1
    with pytest.raises(N.MsiError) as ei:
        src.close()  # still attached
    assert ei.value.status == N.MSI_ERR_SLOT_BUSY
    case.close()  # destroy drains and detaches
    assert src.stats()["windows_busy"] == 0
    src.close()
