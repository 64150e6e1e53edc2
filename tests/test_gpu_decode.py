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
