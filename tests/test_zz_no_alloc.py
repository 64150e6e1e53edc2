"""msi_moe_forward_static: the resident forward for callers that cannot
allocate device memory (its scratch is a fixed 32 MiB array inside the
library).  Its outputs must match msi_moe_forward's on the same inputs, on
two calls in a row (the shared scratch keeps the previous call's contents).
This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu

STATIC_SCRATCH_BYTES = 32 << 20


def _static_forward(plan, layer, x, router_w, table, gens):
    T = x.shape[0]
    out = torch.empty_like(x)
    ev = api.RouteEvent(T, plan.k, plan.E)
    st = np.ascontiguousarray(table, dtype=np.int32)
    ex = np.ascontiguousarray(gens, dtype=np.uint64)
    rc = N.lib().msi_moe_forward_static(plan.h, layer, x.data_ptr(), T, router_w.data_ptr(),
                                        st.ctypes.data, ex.ctypes.data, out.data_ptr(),
                                        ctypes.byref(ev.c), 0,
                                        torch.cuda.current_stream().cuda_stream)
    return rc, out, ev


@pytest.mark.parametrize("name,T", [("tiny", 200), ("qwen3next_4k", 256)])
def test_static_scratch_forward_matches_workspace_forward(name, T):
    cfg = synth.config(name, n_slots=synth.config(name).n_experts, tokens=T)
    case = Case(cfg)
    table, gens = case.stage_all()
    for call in range(2):                       # two calls in a row share the scratch
        x = bf16_tensor(synth.hidden(cfg, 0, 10 + call))
        out_ref, ev_ref = case.plan.forward(0, x, case.router[0], table, gens)
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        rc, out, ev = _static_forward(case.plan, 0, x, case.router[0], table, gens)
        assert rc == N.MSI_OK
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        assert torch.equal(ev.ids, ev_ref.ids)
        assert torch.equal(ev.counts, ev_ref.counts)
        compare_out(bf16_bits(out), oracle.bf16_to_f64(bf16_bits(out_ref)))
    case.close()


def test_static_scratch_rejects_oversize_batch():
    cfg = synth.config("qwen3next_4k", n_slots=512, tokens=4096)
    case = Case(cfg)
    table, gens = case.stage_all()
    n = ctypes.c_size_t()
    N.check(N.lib().msi_workspace_size(case.plan.h, 4096, ctypes.byref(n)), "ws")
    assert n.value > STATIC_SCRATCH_BYTES
    n0 = case.plan.launches()
    rc, _, _ = _static_forward(case.plan, 0, bf16_tensor(synth.hidden(cfg)), case.router[0], table, gens)
    assert rc == N.MSI_ERR_WORKSPACE
    assert case.plan.launches() == n0            # nothing enqueued
    case.close()
