"""Early staging (msi_plan_set_bounce): a long streamed call copies the
extents of its first misses into a device buffer while it routes, and its
waves copy them device to device into their slots.  Residency, victims,
generations, the slot trace and every output must be those of a twin plan
without the buffer, bit for bit, also when some copied extents turn out
not to be needed."""
import numpy as np
import pytest
import torch

import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


class _Twin:
    """The plan of a Case with an early-staging buffer of one wave of extents."""

    def __init__(self, case):
        cfg = case.cfg
        self.router = case.router
        shared_w = gate_w = None
        if cfg.has_shared:
            shared_w = torch.from_numpy(np.concatenate(case.shared_np)).cuda()
            gate_w = torch.from_numpy(np.stack(case.gate_np)).cuda()
        self.plan = api.Plan(n_layers=case.L, n_experts=cfg.n_experts, top_k=cfg.top_k,
                             hidden=cfg.hidden, inter=cfg.inter, n_slots=cfg.n_slots,
                             host_windows=case.windows, has_shared=cfg.has_shared,
                             shared_w=shared_w, shared_gate_w=gate_w, wdtype=cfg.wdtype,
                             early_staging=True)
        assert self.plan.bounce is not None

    def close(self):
        self.plan.close()


def _call(case, x, router):
    case.plan.trace(clear=True)
    out, ev = case.plan.forward_streamed(0, x, router)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    return bf16_bits(out), ev.ids.cpu().numpy(), case.plan.trace(), case.plan.counters()


@pytest.mark.parametrize("name,tokens", [("prefill32k_lru64", 4096), ("prefill32k_q4_lru64", 4096)])
def test_early_staging_equals_plain_staging(name, tokens):
    """Qwen3-Next shape, 64 slots (waves of 32), T k / E = 80: two calls in a
    row (the second starts from the first one's residency)."""
    cfg = synth.config(name, tokens=tokens)
    b = Case(cfg)
    a = _Twin(b)
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, 30 + call)
        x = bf16_tensor(x_bits)
        oa, ia, ta, ca = _call(a, x, a.router[0])
        ob, ib, tb, cb = _call(b, x, b.router[0])
        assert np.array_equal(ia, ib)
        assert ta == tb
        assert ca == cb
        assert np.array_equal(oa, ob)
    toks = np.arange(0, tokens, 97)
    ref = b.oracle_layer(x_bits, tokens=toks)
    compare_out(oa[toks], ref["out"])
    a.close()
    b.close()


def test_early_staging_with_unneeded_experts():
    """Experts 0-5 never win the routing (hidden column 0 is 4.0 in every
    token and their router weight there is -10), so the first extents copied
    early are not needed: the waves must take only the needed ones from the
    buffer."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=4, tokens=1024, n_slots=16)
    b = Case(cfg)
    a = _Twin(b)
    wr = b.router_np[0].copy()
    wr[:6, 0] = -10.0
    router = torch.from_numpy(wr).cuda()
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, 40 + call).copy()
        x_bits[:, 0] = 0x4080                              # bf16 4.0
        x = bf16_tensor(x_bits)
        oa, ia, ta, ca = _call(a, x, router)
        ob, ib, tb, cb = _call(b, x, router)
        assert not np.isin(ia, np.arange(6)).any()
        assert np.array_equal(ia, ib)
        assert ta == tb
        assert np.array_equal(oa, ob)
    a.close()
    b.close()


def test_early_staging_decode_stack_equals_plain_staging():
    """The decode stack at batch 64 (48 layers of the tiny shape, one 64-slot
    pool; T k = 8 E, so every layer call copies its first misses early and
    stages a wave drawn wholly from the early-staging buffer in one launch:
    invalidation, device copies, publication): route ids, outputs and slot
    traces equal those of a plan without the buffer, over four steps."""
    cfg = synth.config("decode48", tokens=64)
    b = Case(cfg)
    a = _Twin(b)
    stage_a, stage_b = torch.cuda.Stream(), torch.cuda.Stream()
    for step in range(4):
        xa = xb = bf16_tensor(synth.hidden(cfg, 0, 2000 + step, tokens=64))
        for l in range(cfg.n_layers):
            oa, eva = a.plan.forward_streamed(l, xa, a.router[l], residual=True, stage_stream=stage_a)
            ob, evb = b.plan.forward_streamed(l, xb, b.router[l], residual=True, stage_stream=stage_b)
            torch.cuda.synchronize()
            assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
            assert torch.equal(eva.ids, evb.ids)
            assert torch.equal(oa.view(torch.int16), ob.view(torch.int16))
            xa, xb = oa, ob
    assert a.plan.trace() == b.plan.trace()
    assert a.plan.counters()["stages"] == b.plan.counters()["stages"]
    a.close()
    b.close()
