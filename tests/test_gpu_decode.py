"""Decode workload: a stack of 48 MoE layers of the tiny shape (hidden 256, 16
experts, top-2, intermediate 128, router + experts only), batch 1 and 64, 64
decode steps, one 64-slot LRU pool shared across the layers' 768 objects.

Step inputs are fresh N(0,1) rows per step; each layer computes
x_{l+1} = bf16(x_l + moe_l(x_l)).  The oracle is teacher-forced per layer with
the GPU's bf16 layer input so that one near-tie cannot cascade; every route
event is compared, and the slot trace is compared with the oracle's slot
simulator fed the same needed sets (the GPU's, which equal the oracle's unless
a near-tie changes a set; such calls are counted)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("batch,steps", [(1, 64), (64, 64)])
def test_decode48_stack(batch, steps):
    cfg = synth.config("decode48", tokens=batch)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    stage = torch.cuda.Stream()
    eb = cfg.extent_bytes
    decoded = {}
    set_diverged = 0
    near_total = 0
    for step in range(steps):
        x_bits = synth.hidden(cfg, 0, 1000 + step, tokens=batch)
        for l in range(cfg.n_layers):
            x = bf16_tensor(x_bits)
            out, ev = case.plan.forward_streamed(l, x, case.router[l], residual=True, stage_stream=stage)
            torch.cuda.synchronize()
            assert case.plan.status() == N.MSI_OK
            ref = oracle.moe_layer(x_bits, case.router_np[l], cfg.top_k,
                                   lambda e: case.extent(l, e), cfg.hidden, cfg.inter,
                                   residual=True)
            ids = ev.ids.cpu().numpy()
            near, _ = compare_routes(ids, ev.weights.cpu().numpy(), ref)
            near_total += near
            gpu_needed = sorted(set(ids.reshape(-1).tolist()))
            ora_needed = sorted(set(ref["ids"].reshape(-1).tolist()))
            if gpu_needed != ora_needed:
                set_diverged += 1
                assert near > 0, "needed sets differ without a near-tie"
            sim.call(l, gpu_needed)
            mask = ~oracle.near_tie_tokens(ref["gap_k"])
            compare_out(bf16_bits(out), ref["out"], mask)
            x_bits = bf16_bits(out)          # the GPU's layer output feeds the next layer
    assert case.plan.trace() == sim.trace
    c = case.plan.counters()
    assert c["streamed_forwards"] == steps * cfg.n_layers
    assert c["hits"] == sum(1 for r in sim.trace if r[5] == "hit")
    print("decode48 batch %d: %d route events, %d near-tie tokens, %d needed-set divergences, "
          "%d stages, %d hits" % (batch, steps * cfg.n_layers, near_total, set_diverged,
                                  c["stages"], c["hits"]))
    case.close()


def test_decode_stack_call_equals_layer_calls():
    """msi_moe_forward_streamed_stack over the 48-layer decode stack (batch 64,
    with the early-staging buffer the bench uses) equals 48 separate
    streamed calls on a twin plan: every layer's route ids, the stack's
    output bit for bit, and the slot traces, over three steps."""
    cfg = synth.config("decode48", tokens=64)
    a = Case(cfg, early_staging=True)
    b = Case(cfg, early_staging=True)
    E, L = cfg.n_experts, cfg.n_layers
    from paper_2608_23805_gb300 import api
    evs = [api.RouteEvent(64, cfg.top_k, E) for _ in range(L)]
    bufs = [torch.empty((64, cfg.hidden), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    stage_a, stage_b = torch.cuda.Stream(), torch.cuda.Stream()
    for step in range(3):
        x = bf16_tensor(synth.hidden(cfg, 0, 3000 + step, tokens=64))
        last = a.plan.forward_streamed_stack(0, x, a.router, bufs[0], bufs[1], evs, residual=True,
                                             stage_stream=stage_a)
        xb = x
        ids_b = []
        for l in range(L):
            xb, evb = b.plan.forward_streamed(l, xb, b.router[l], residual=True, stage_stream=stage_b)
            ids_b.append(evb.ids)
        torch.cuda.synchronize()
        assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
        for l in range(L):
            assert torch.equal(evs[l].ids, ids_b[l]), l
        assert torch.equal(last.view(torch.int16), xb.view(torch.int16))
    assert a.plan.trace() == b.plan.trace()
    # argument checks: a stack past the last layer is refused, nothing enqueued
    rc, done, _ = a.plan.forward_streamed_stack(L - 1, x, a.router[:2], bufs[0], bufs[1], evs[:2],
                                                residual=True, check=False)
    assert rc == N.MSI_ERR_INVALID_ARG and done == 0
    a.close()
    b.close()
