"""Lifecycle and fault cells, transposed from the paper's fault-mode table
(Sec. "Integrated Deterministic Faults"): publish only after complete valid
movement, a published version denotes the requested object and version, legal
completion order is not over-constrained, reset drains or invalidates.  Every
fault is made on the host (no GPU fault, trap or hang is ever provoked)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _resident(E=16):
    cfg = synth.config("tiny", n_slots=E)
    return cfg, Case(cfg)


def test_reset_drains_and_invalidates():
    cfg, case = _resident()
    x = bf16_tensor(synth.hidden(cfg, 0, 1))
    for e in range(cfg.n_experts):               # copies still in flight at the reset
        case.plan.stage(e, 0, e)
    table, gens = case.plan.slot_table(0)
    epoch = case.plan.reset()
    assert epoch == 1
    assert all(case.plan.slot_state(s) == N.MSI_SLOT_VACANT for s in range(cfg.n_slots))
    t2, g2 = case.plan.slot_table(0)
    assert np.all(t2 == -1)
    rc, _, _ = case.plan.forward(0, x, case.router[0], table, gens, check=False)
    assert rc == N.MSI_ERR_WRONG_OBJECT           # nothing from before the reset passes
    # generations keep increasing across the reset
    assert case.plan.stage(0, 0, 0) == gens[0] + 1
    case.close()


def test_out_of_order_completion_is_exact():
    """The same bundle staged in order on one stream, and staged on two streams
    whose copies complete in the opposite order, give bit-identical outputs."""
    cfg, a = _resident()
    _, b = _resident()
    x_bits = synth.hidden(cfg, 0, 4)
    ta, ga = a.stage_all()
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    big = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    with torch.cuda.stream(s1):
        big.zero_()                                # delays everything queued on s1 after it
    for e in range(cfg.n_experts // 2):
        b.plan.stage(e, 0, e, s1)
    for e in range(cfg.n_experts // 2, cfg.n_experts):
        b.plan.stage(e, 0, e, s2)
    tb, gb = b.plan.slot_table(0)
    oa, ea = a.plan.forward(0, bf16_tensor(x_bits), a.router[0], ta, ga)
    ob, eb = b.plan.forward(0, bf16_tensor(x_bits), b.router[0], tb, gb)
    torch.cuda.synchronize()
    assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
    assert torch.equal(ea.ids, eb.ids)
    assert torch.equal(oa.view(torch.int16), ob.view(torch.int16))
    a.close()
    b.close()


def test_short_read_publishes_nothing():
    cfg, case = _resident()
    case.plan.inject(N.MSI_FAULT_SHORT_READ, 0, 3)
    with pytest.raises(N.MsiError) as ei:
        case.plan.stage(3, 0, 3)
    assert ei.value.status == N.MSI_ERR_SOURCE
    assert case.plan.slot_state(3) == N.MSI_SLOT_VACANT
    assert case.plan.counters()["stages"] == 0
    assert case.plan.stage(3, 0, 3) == 1          # the hook is one-shot
    case.close()


def test_failed_extent_inside_a_bundle_publishes_no_bundle():
    """Streamed forward: one needed miss has a failed source extent, so no
    bundle of the call is planned, staged or published and no output row is
    written; the route event is still recorded (routing precedes the Plan)."""
    cfg = synth.config("tiny")
    case = Case(cfg)
    x_bits = synth.hidden(cfg, 0, 5)
    ids_ref = oracle.router(x_bits, case.router_np[0], cfg.top_k)["ids"]
    victim = int(ids_ref[7, 1])
    case.plan.inject(N.MSI_FAULT_SHORT_READ, 0, victim)
    out = torch.full((cfg.tokens, cfg.hidden), 3.0, dtype=torch.bfloat16, device="cuda")
    rc, out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0], out=out,
                                             check=False)
    torch.cuda.synchronize()
    assert rc == N.MSI_ERR_SOURCE
    assert case.plan.trace() == []                # nothing staged, evicted or published
    assert all(case.plan.slot_state(s) == N.MSI_SLOT_VACANT for s in range(cfg.n_slots))
    assert torch.all(out == 3.0)
    compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), oracle.router(
        x_bits, case.router_np[0], cfg.top_k))
    # the next call (no fault) runs normally
    out2, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out2), case.oracle_layer(x_bits)["out"])
    case.close()


@pytest.mark.parametrize("kind,status", [(N.MSI_FAULT_STALE_COMPLETION, N.MSI_ERR_STALE_GENERATION),
                                         (N.MSI_FAULT_WRONG_OBJECT, N.MSI_ERR_WRONG_OBJECT)])
def test_stale_or_wrong_publication_fails_closed_on_device(kind, status):
    """The host ledger is right but the slot's published word is not (a late
    stale completion / another object): the GPU re-check rejects the bundle
    before any expert output is computed and no output row becomes visible."""
    cfg, case = _resident()
    x_bits = synth.hidden(cfg, 0, 6)
    ids_ref = oracle.router(x_bits, case.router_np[0], cfg.top_k)["ids"]
    target = int(ids_ref[0, 0])
    for e in range(cfg.n_experts):
        if e == target:
            case.plan.inject(kind, 0, e)
        case.plan.stage(e, 0, e)
    table, gens = case.plan.slot_table(0)
    out = torch.full((cfg.tokens, cfg.hidden), 5.0, dtype=torch.bfloat16, device="cuda")
    case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens, out=out)
    torch.cuda.synchronize()
    assert case.plan.status() == status
    assert torch.all(out == 5.0)
    # restaging publishes a correct version again
    gens[target] = case.plan.stage(target, 0, target)
    out, _ = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out), case.oracle_layer(x_bits)["out"])
    case.close()


def test_balanced_counters_after_streamed_calls():
    cfg = synth.config("tiny")
    case = Case(cfg)
    for call in range(4):
        case.plan.forward_streamed(0, bf16_tensor(synth.hidden(cfg, 0, 30 + call)), case.router[0])
    torch.cuda.synchronize()
    c = case.plan.counters()
    tr = case.plan.trace()
    assert c["stages"] == sum(1 for r in tr if r[5] == "stage")
    assert c["hits"] == sum(1 for r in tr if r[5] == "hit")
    assert c["evicts"] == sum(1 for r in tr if r[5] == "evict")
    assert c["h2d_bytes"] == c["stages"] * cfg.extent_bytes
    occupied = sum(1 for s in range(cfg.n_slots) if case.plan.slot_state(s) != N.MSI_SLOT_VACANT)
    assert occupied == c["stages"] - c["evicts"]
    case.close()


def test_back_to_back_forwards_with_shared_expert_match_sequential():
    """The shared expert of a resident forward runs on the plan's side stream
    (forked after the forward's first kernel, joined before the combine).
    Three forwards enqueued back to back with different inputs, no host sync
    between them, equal the same forwards run one at a time, bit for bit."""
    cfg = synth.config("qwen3next_4k", n_experts=64, tokens=2048, n_slots=64)
    case = Case(cfg)
    table, gens = case.stage_all()
    xs = [bf16_tensor(synth.hidden(cfg, 0, 40 + i)) for i in range(3)]
    seq = []
    for x in xs:
        out, _ = case.plan.forward(0, x, case.router[0], table, gens)
        torch.cuda.synchronize()
        seq.append(out.clone())
    outs = [case.plan.forward(0, x, case.router[0], table, gens)[0] for x in xs]
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    for a, b in zip(seq, outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    toks = np.arange(0, 2048, 64)
    compare_out(bf16_bits(outs[2])[toks], case.oracle_layer(synth.hidden(cfg, 0, 42), tokens=toks)["out"])
    case.close()
