"""Failure detection on the GPU without a GPU fault: a bounded device wait
that runs out.  MSI_FAULT_DEVICE_WAIT makes the next forward's tensor-core
kernels (the router, the routed expert GEMMs and the shared expert's CTA-pair
GEMMs) wait once on a barrier that nothing arrives at; with a short plan wait
limit that wait expires, every such kernel drains the copies and MMAs it
issued, frees its TMEM and returns, and the forward reports MSI_ERR_TIMEOUT
with no `out` row written.  The context stays usable: the next call at the
default limit matches the oracle."""
import numpy as np
import pytest
import torch

import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu

SHORT_WAIT = 2_000_000   # clock64 cycles, ~1 ms at GB300 clocks


@pytest.mark.parametrize("streamed", [False, True])
def test_expired_device_wait_fails_closed_then_recovers(streamed):
    # 1,024 tokens at the Qwen shape: the tensor-core router, single-CTA routed
    # GEMMs and CTA-pair shared-expert GEMMs all run
    T = 1024
    cfg = synth.config("qwen3next_4k", tokens=T, n_slots=512 if not streamed else 64,
                       lru=streamed)
    case = Case(cfg)
    table = gens = None
    if not streamed:
        table, gens = case.stage_all()
    x_bits = synth.hidden(cfg)
    x = bf16_tensor(x_bits)
    sentinel = torch.full_like(x, 7.0)

    def run():
        out = sentinel.clone()
        if streamed:
            case.plan.forward_streamed(0, x, case.router[0], out=out)
        else:
            case.plan.forward(0, x, case.router[0], table, gens, out=out)
        torch.cuda.synchronize()
        return out

    case.plan.set_wait_cycles(SHORT_WAIT)
    case.plan.inject(N.MSI_FAULT_DEVICE_WAIT, 0, 0)
    out = run()
    assert case.plan.status() == N.MSI_ERR_TIMEOUT
    assert torch.equal(out.view(torch.int16), sentinel.view(torch.int16))   # no row written

    # the limit back at its default; the hook was one-shot
    case.plan.set_wait_cycles(0)
    out = run()
    assert case.plan.status() == N.MSI_OK
    toks = np.arange(0, T, 37)
    ref = case.oracle_layer(x_bits, tokens=toks)
    compare_out(bf16_bits(out)[toks], ref["out"])
    case.close()
