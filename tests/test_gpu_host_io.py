"""End-to-end calls from and to host memory (msi_moe_forward_host,
msi_moe_forward_streamed_host): the rows are copied in on the plan's copy
stream, the ids come back beside the GEMMs and the outputs come back in
combine chunks.  They must give exactly what the device-buffer calls give:
outputs, route events and ids bit for bit, the same slot traces, and nothing
past the compute stream's point after the call."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _host(bits, pinned=True):
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.pin_memory() if pinned else t.clone()


@pytest.mark.parametrize("T", [1003, 64, 1])
def test_resident_host_call_equals_device_call(T):
    """Qwen-shape layer (H 2048, I 512, k 10, shared expert) with 64 experts
    resident; T = 1003 makes four uneven combine chunks."""
    cfg = synth.config("qwen3next_4k", n_experts=64, n_slots=64, tokens=T)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 120)
    out_d, ev_d = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    ids_host = torch.empty((T, cfg.top_k), dtype=torch.int32).pin_memory()
    out_h, ev_h = case.plan.forward_host(0, _host(x_bits), case.router[0], table, gens,
                                         ids_host=ids_host)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    assert torch.equal(out_h.view(torch.int16), out_d.cpu().view(torch.int16))
    assert torch.equal(ids_host, ev_d.ids.cpu())
    for f in ("ids", "weights", "counts", "gap"):
        assert torch.equal(getattr(ev_h, f), getattr(ev_d, f))
    if T == 1003:
        compare_out(bf16_bits(out_h), case.oracle_layer(x_bits)["out"])
    case.close()


@pytest.mark.parametrize("pinned", [True, False])
def test_streamed_host_call_equals_device_call(pinned):
    """Tiny layer, 8-slot LRU: the host call stages the same waves (equal
    traces) and returns the same outputs; pageable buffers work too."""
    cfg = synth.config("tiny")
    a, b = Case(cfg), Case(cfg)
    for call in range(3):
        x_bits = synth.hidden(cfg, 0, 130 + call)
        oa, eva = a.plan.forward_streamed(0, bf16_tensor(x_bits), a.router[0], residual=True)
        ids_host = torch.empty((cfg.tokens, cfg.top_k), dtype=torch.int32)
        ob, evb = b.plan.forward_host(0, _host(x_bits, pinned), b.router[0], ids_host=ids_host,
                                      residual=True)
        torch.cuda.synchronize()
        assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
        assert torch.equal(ob.view(torch.int16), oa.cpu().view(torch.int16))
        assert torch.equal(ids_host, eva.ids.cpu())
    assert a.plan.trace() == b.plan.trace()
    compare_out(bf16_bits(ob), a.oracle_layer(x_bits, residual=True)["out"])
    a.close()
    b.close()


def test_host_call_empty_batch_and_workspace():
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    table, gens = case.stage_all()
    empty = torch.empty((0, cfg.hidden), dtype=torch.bfloat16)
    out, ev = case.plan.forward_host(0, empty, case.router[0], table, gens)
    torch.cuda.synchronize()
    assert out.shape == (0, cfg.hidden) and int(ev.counts.sum()) == 0
    # a workspace without room for the row buffers is refused, nothing enqueued
    x = _host(synth.hidden(cfg, 0, 140))
    small = case.plan.workspace(cfg.tokens)
    out_h = torch.empty_like(x)
    ev = case.plan.forward(0, bf16_tensor(synth.hidden(cfg, 0, 140)), case.router[0], table, gens)[1]
    st = np.ascontiguousarray(table, dtype=np.int32)
    ex = np.ascontiguousarray(gens, dtype=np.uint64)
    rc = N.lib().msi_moe_forward_host(case.plan.h, 0, x.data_ptr(), cfg.tokens,
                                      case.router[0].data_ptr(), st.ctypes.data, ex.ctypes.data,
                                      out_h.data_ptr(), None, ctypes.byref(ev.c), small.data_ptr(),
                                      small.numel(), 0, torch.cuda.current_stream().cuda_stream)
    assert rc == N.MSI_ERR_WORKSPACE
    case.close()


def test_streamed_host_call_with_early_staging_equals_device_call():
    """The bench's end-to-end configuration: a host-buffer streamed call on
    a plan with an early-staging buffer (copied after the call's rows have
    crossed) and T k >= 8 E, at the Qwen3-Next layer shape with 64 experts
    and 16 slots (waves of 8, the shared expert after the first miss wave;
    8,200 rows, so eight uneven combine chunks): outputs, ids and slot
    traces equal those of the device-buffer call."""
    cfg = synth.config("prefill32k_lru64", tokens=8200, n_experts=64, n_slots=16)
    a, b = Case(cfg, early_staging=True), Case(cfg, early_staging=True)
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, 150 + call)
        oa, eva = a.plan.forward_streamed(0, bf16_tensor(x_bits), a.router[0])
        ids_host = torch.empty((cfg.tokens, cfg.top_k), dtype=torch.int32).pin_memory()
        ob, evb = b.plan.forward_host(0, _host(x_bits), b.router[0], ids_host=ids_host)
        torch.cuda.synchronize()
        assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
        assert torch.equal(ob.view(torch.int16), oa.cpu().view(torch.int16))
        assert torch.equal(ids_host, eva.ids.cpu())
    assert a.plan.trace() == b.plan.trace()
    toks = np.arange(0, cfg.tokens, 241)
    compare_out(bf16_bits(ob)[toks], a.oracle_layer(x_bits, tokens=toks)["out"])
    a.close()
    b.close()
