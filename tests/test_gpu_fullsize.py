"""The 32K-token single-layer prefills at their full size, in the launch
configuration the bench times (msi_moe_forward_streamed, default flags, a
side stage stream, an early-staging buffer of one wave): 32,768 tokens, 512 experts, top-10, a 64-slot pool in
LRU waves of 32, bf16 and 4-bit experts.  Every route event is compared with
the oracle router, the slot trace with the oracle's simulator (bit-exact),
and the outputs on sampled tokens (the first, the last and random ones)
with the oracle layer.  Two calls: the first stages into an empty pool, the
second starts with the 64 experts left resident as hits and stages the rest."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _needed(ids):
    return sorted(set(np.asarray(ids).reshape(-1).tolist()))


@pytest.mark.parametrize("name,samples", [("prefill32k_lru64", (48, 24)),
                                          ("prefill32k_q4_lru64", (24, 12))])
def test_prefill32k_full_size(name, samples):
    cfg = synth.config(name)
    assert cfg.tokens == 32768 and cfg.n_experts == 512 and cfg.n_slots == 64
    case = Case(cfg, early_staging=True)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    stage = torch.cuda.Stream()
    rng = np.random.default_rng(7)
    for call, ns in enumerate(samples):
        x_bits = synth.hidden(cfg, 0, call)   # call 0 is the bench's input
        out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                             stage_stream=stage)
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        ids = ev.ids.cpu().numpy()
        r = oracle.router(x_bits, case.router_np[0], cfg.top_k, case.gate_np[0])
        compare_routes(ids, ev.weights.cpu().numpy(), r)
        assert np.array_equal(ev.counts.cpu().numpy(), np.bincount(ids.reshape(-1), minlength=512))
        sim.call(0, _needed(ids))
        toks = np.sort(np.concatenate([[0, cfg.tokens - 1],
                                       rng.choice(np.arange(1, cfg.tokens - 1), ns, replace=False)]))
        ref = case.oracle_layer(x_bits, tokens=toks)
        compare_out(bf16_bits(out)[toks], ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    assert case.plan.trace() == sim.trace
    c = case.plan.counters()
    assert c["stages"] == sum(1 for t in sim.trace if t[5] == oracle.TRACE_STAGE)
    assert c["hits"] == sum(1 for t in sim.trace if t[5] == oracle.TRACE_HIT)
    case.close()
