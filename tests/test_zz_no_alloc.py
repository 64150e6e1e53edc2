"""msi_moe_forward_static: the resident forward for callers that cannot
allocate device memory (code inside another runtime's memory budget, plugins
whose host framework owns every allocation, loops that forbid allocation after
start-up).  Its scratch is a fixed 32 MiB array inside the library, shared by
every call and keeping the previous call's contents.

It runs the same kernels on the same inputs as msi_moe_forward with a caller
workspace, so its route event and outputs must equal that forward's bit for
bit: on two calls in a row, after a larger call has left more router blocks
and permuted rows in the array, and at the largest batch the array holds.
This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from gpu_case import Case, bf16_tensor
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu

STATIC_SCRATCH_BYTES = 32 << 20
# largest batch whose workspace fits the array at the Qwen3-Next layer shape
QWEN_STATIC_MAX_T = 478


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


def _ws_bytes(plan, T):
    n = ctypes.c_size_t()
    N.check(N.lib().msi_workspace_size(plan.h, T, ctypes.byref(n)), "msi_workspace_size")
    return n.value


def _check_equal(case, table, gens, T, call):
    """One static call against the workspace forward on the same rows: every
    field of the route event and every output bit equal."""
    cfg = case.cfg
    x = bf16_tensor(synth.hidden(cfg, 0, 10 + call, tokens=T))
    out_ref, ev_ref = case.plan.forward(0, x, case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    rc, out, ev = _static_forward(case.plan, 0, x, case.router[0], table, gens)
    assert rc == N.MSI_OK
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    assert torch.equal(ev.ids, ev_ref.ids)
    assert torch.equal(ev.counts, ev_ref.counts)
    assert torch.equal(ev.weights, ev_ref.weights)
    assert torch.equal(ev.gap, ev_ref.gap)
    assert torch.equal(out.view(torch.int16), out_ref.view(torch.int16))


@pytest.mark.parametrize("name,T", [("tiny", 200), ("qwen3next_4k", 256)])
def test_static_scratch_forward_matches_workspace_forward(name, T):
    """Two calls in a row, then a larger call followed by a small ragged one
    (37 tokens: fewer router blocks and permuted rows than the array holds
    from the call before)."""
    big = 4000 if name == "tiny" else QWEN_STATIC_MAX_T
    cfg = synth.config(name, n_slots=synth.config(name).n_experts, tokens=big)
    case = Case(cfg)
    table, gens = case.stage_all()
    for call, t in enumerate([T, T, big, 37]):
        _check_equal(case, table, gens, t, call)
    case.close()


def test_static_scratch_limit_at_qwen_shape():
    """The array holds 478 tokens at the Qwen3-Next layer shape (E 512, top-10,
    H 2048, I 512, shared expert): a call at the limit equals the workspace
    forward, one token more is rejected with nothing enqueued."""
    cfg = synth.config("qwen3next_4k", n_slots=512, tokens=QWEN_STATIC_MAX_T + 1)
    case = Case(cfg)
    table, gens = case.stage_all()
    assert _ws_bytes(case.plan, QWEN_STATIC_MAX_T) <= STATIC_SCRATCH_BYTES
    assert _ws_bytes(case.plan, QWEN_STATIC_MAX_T + 1) > STATIC_SCRATCH_BYTES
    _check_equal(case, table, gens, QWEN_STATIC_MAX_T, 0)
    n0 = case.plan.launches()
    x = bf16_tensor(synth.hidden(cfg, 0, 20, tokens=QWEN_STATIC_MAX_T + 1))
    rc, _, _ = _static_forward(case.plan, 0, x, case.router[0], table, gens)
    assert rc == N.MSI_ERR_WORKSPACE
    assert case.plan.launches() == n0            # nothing enqueued
    # a call after the rejection is still exact
    _check_equal(case, table, gens, 100, 1)
    case.close()
