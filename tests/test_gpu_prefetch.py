"""Next-layer prediction, two-bank prefetch and caller pins (the paper's
protected LRU with a two-bank next-layer prefetch, Sec. "Evaluation", "Cache
and storage state"; prediction and pinning over one slot lifecycle, Sec. "A
Shared Cross-Adapter Plan Core").

A predicting call also routes its rows through layer + 1's router and, after
its last wave, stages layer + 1's predicted objects.  Checked: the predicted
route events equal the oracle router's (near-ties excepted); the slot trace,
prefetch records included, equals the oracle simulator's fed the same needed
and predicted sets; prediction changes residency only, so the outputs are
bit-identical to a plan that does not predict; fewer demand stages remain; a
rejected prefetch read unwinds only its bundle; pinned objects are never
evicted."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _predicted_counts(ev_next, E):
    ids = ev_next.ids.cpu().numpy()
    counts = ev_next.counts.cpu().numpy().astype(np.int64)
    assert np.array_equal(counts, np.bincount(ids.reshape(-1), minlength=E))
    return ids, counts


def _check_counters(case, sim):
    tr = case.plan.trace()
    c = case.plan.counters()
    assert c["prefetches"] == sum(1 for r in tr if r[5] == "prefetch") == sim.prefetches
    assert c["prefetch_hits"] == sim.prefetch_hits
    assert c["stages"] == sum(1 for r in tr if r[5] in ("stage", "prefetch"))
    assert c["hits"] == sum(1 for r in tr if r[5] == "hit")
    return c


@pytest.mark.parametrize("batch,steps", [(1, 6), (64, 6)])
def test_decode_stack_with_next_layer_prefetch(batch, steps):
    """The 48-layer decode stack (tiny layer shape, one 64-slot pool): every
    call but the last layer's predicts the next layer.  A twin plan runs the
    same inputs without prediction."""
    cfg = synth.config("decode48", tokens=batch)
    a, b = Case(cfg), Case(cfg)          # a predicts, b does not
    sim_a, sim_b = oracle.LRUWaveSim(cfg.n_slots), oracle.LRUWaveSim(cfg.n_slots)
    stage = torch.cuda.Stream()
    E, L = cfg.n_experts, cfg.n_layers
    near_total = 0
    for step in range(steps):
        x_bits = synth.hidden(cfg, 0, 2000 + step, tokens=batch)
        for l in range(L):
            x = bf16_tensor(x_bits)
            nxt = a.router[l + 1] if l + 1 < L else None
            oa, eva = a.plan.forward_streamed(l, x, a.router[l], residual=True, stage_stream=stage,
                                              next_router_w=nxt)
            ob, evb = b.plan.forward_streamed(l, x, b.router[l], residual=True, stage_stream=stage)
            torch.cuda.synchronize()
            assert a.plan.status() == N.MSI_OK and b.plan.status() == N.MSI_OK
            assert torch.equal(oa.view(torch.int16), ob.view(torch.int16))
            assert torch.equal(eva.ids, evb.ids)
            needed = sorted(set(eva.ids.cpu().numpy().reshape(-1).tolist()))
            predict = None
            if nxt is not None:
                ids, counts = _predicted_counts(eva.next, E)
                ref = oracle.router(x_bits, a.router_np[l + 1], cfg.top_k)
                near, _ = compare_routes(ids, eva.next.weights.cpu().numpy(), ref)
                near_total += near
                predict = (l + 1, counts)
            sim_a.call(l, needed, predict)
            sim_b.call(l, needed)
            x_bits = bf16_bits(oa)
    assert a.plan.trace() == sim_a.trace
    assert b.plan.trace() == sim_b.trace
    ca = _check_counters(a, sim_a)
    cb = b.plan.counters()
    demand_a = ca["stages"] - ca["prefetches"]
    print("decode48 batch %d, %d steps: demand stages %d -> %d with prediction; %d prefetched, "
          "%d prefetch hits; %d near-tie tokens" % (batch, steps, cb["stages"], demand_a,
                                                    ca["prefetches"], ca["prefetch_hits"],
                                                    near_total))
    assert ca["prefetch_hits"] > 0 and demand_a < cb["stages"]
    a.close()
    b.close()


def test_qwen_shape_bundle_is_capped_and_ranked():
    """Two Qwen-shape layers (H 2048, I 512, k 10) with 64 experts and 16
    slots (waves of 8): nearly every expert is predicted, so the bundle takes
    the 8 most-predicted non-resident ones.  Outputs against the oracle; the
    trace against the simulator."""
    cfg = synth.config("qwen3next_4k", n_experts=64, n_slots=16, tokens=256, lru=True, n_layers=2)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    stage = torch.cuda.Stream()
    for call in range(3):
        x_bits = synth.hidden(cfg, 0, 70 + call)
        out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                             stage_stream=stage, next_router_w=case.router[1])
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        compare_out(bf16_bits(out), case.oracle_layer(x_bits, 0)["out"])
        ids, counts = _predicted_counts(ev.next, cfg.n_experts)
        compare_routes(ids, ev.next.weights.cpu().numpy(),
                       oracle.router(x_bits, case.router_np[1], cfg.top_k))
        sim.call(0, sorted(set(ev.ids.cpu().numpy().reshape(-1).tolist())), (1, counts))
        pref = [r for r in sim.trace if r[0] == call and r[5] == "prefetch"]
        assert len(pref) <= 8
        out1, ev1 = case.plan.forward_streamed(1, bf16_tensor(x_bits), case.router[1],
                                               stage_stream=stage)
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        compare_out(bf16_bits(out1), case.oracle_layer(x_bits, 1)["out"])
        sim.call(1, sorted(set(ev1.ids.cpu().numpy().reshape(-1).tolist())))
    assert case.plan.trace() == sim.trace
    c = _check_counters(case, sim)
    # layer 1 runs on the same rows, so the prediction is exact: every
    # prefetched object is consumed by the next call
    assert c["prefetch_hits"] == c["prefetches"] > 0
    case.close()


def test_pins_are_never_evicted():
    """Tiny layer, 8 slots in waves of 2 (room for 4 pins): pinned objects stay
    resident through calls that would evict them; the trace equals the
    simulator's with the same pins; a fifth pin is refused; unpinning makes an
    object an ordinary victim again."""
    cfg = synth.config("tiny")
    case = Case(cfg, wave_capacity=2)
    sim = oracle.LRUWaveSim(cfg.n_slots, 2)
    x0 = synth.hidden(cfg, 0, 80)
    first = sorted(set(oracle.router(x0, case.router_np[0], cfg.top_k)["ids"].reshape(-1).tolist()))
    pins = first[:4]
    for e in pins:
        case.plan.pin(0, e)
        sim.pin(0, e)
    with pytest.raises(N.MsiError) as ei:
        case.plan.pin(0, first[4])
    assert ei.value.status == N.MSI_ERR_SLOT_BUSY
    for call in range(6):
        x_bits = synth.hidden(cfg, 0, 80 + call)
        out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        compare_out(bf16_bits(out), case.oracle_layer(x_bits)["out"])
        sim.call(0, sorted(set(ev.ids.cpu().numpy().reshape(-1).tolist())))
        if call == 3:
            case.plan.pin(0, pins[0], False)
            sim.unpin(0, pins[0])
    tr = case.plan.trace()
    assert tr == sim.trace
    evicted = {(r[1], r[2]) for r in tr if r[5] == "evict"}
    assert not evicted & {(0, e) for e in pins[1:]}
    table = case.plan.slot_table(0)[0]
    assert all(table[e] >= 0 for e in pins[1:])
    case.close()


def test_prediction_arguments_and_empty_batch():
    cfg = synth.config("decode48", tokens=4, n_layers=2)
    case = Case(cfg)
    x = bf16_tensor(synth.hidden(cfg, 0, 90))
    rc, _, _ = case.plan.forward_streamed(1, x, case.router[1], next_router_w=case.router[0],
                                          check=False)
    assert rc == N.MSI_ERR_INVALID_ARG  # no layer after the last
    empty = torch.empty((0, cfg.hidden), dtype=torch.bfloat16, device="cuda")
    nev = api.RouteEvent(0, cfg.top_k, cfg.n_experts)
    nev.counts.fill_(7)
    out, ev = case.plan.forward_streamed(0, empty, case.router[0], next_router_w=case.router[1],
                                         next_ev=nev)
    torch.cuda.synchronize()
    assert torch.all(nev.counts == 0)
    assert case.plan.counters()["prefetches"] == 0 and case.plan.trace() == []
    case.close()


def test_rejected_prefetch_read_unwinds_only_its_bundle(tmp_path):
    """With a source attached, the read of one predicted object fails (EIO):
    the call still succeeds with exact outputs; the bundle's slots are
    evicted (Vacant); the next layer's call stages the object on demand and
    matches the oracle."""
    cfg = synth.config("decode48", tokens=16, n_layers=2)
    case = Case(cfg)
    L, E, eb = case.L, cfg.n_experts, cfg.extent_bytes
    path = str(tmp_path / "experts.bin")
    case.windows.numpy().tofile(path)
    src = api.Source(path, eb + 4096, n_windows=4)
    case.plan.set_source(src, np.arange(L * E, dtype=np.uint64) * eb)
    x_bits = synth.hidden(cfg, 0, 95)
    pred = oracle.router(x_bits, case.router_np[1], cfg.top_k)["ids"]
    victim = sorted(set(pred.reshape(-1).tolist()))[0]
    case.plan.inject(N.MSI_FAULT_IO_ERROR, 1, victim)
    out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                         next_router_w=case.router[1])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out), case.oracle_layer(x_bits, 0)["out"])
    tr = case.plan.trace()
    pref = [(r[2], r[3]) for r in tr if r[5] == "prefetch"]
    unwound = {(r[2], r[3]) for r in tr if r[5] == "evict" and r[1] == 1}
    assert pref and all(x in unwound for x in pref)
    table = case.plan.slot_table(1)[0]
    assert all(table[e] == -1 for e, _ in pref)       # the bundle is unwound
    assert case.plan.counters()["rejections"] == 1 and src.stats()["rejected"] == 1
    out1, ev1 = case.plan.forward_streamed(1, bf16_tensor(x_bits), case.router[1])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out1), case.oracle_layer(x_bits, 1)["out"])
    assert case.plan.slot_table(1)[0][victim] >= 0
    case.plan.set_source(None)
    src.close()
    case.close()


def test_failed_predicting_call_leaves_the_plan_usable():
    """A predicting call that fails after its prediction was launched (a
    caller-held slot times out before the waves are planned) still joins the
    prediction before returning; once the slot is released, the next calls
    (with and without prediction) match the oracle."""
    cfg = synth.config("decode48", tokens=16, n_layers=2)
    case = Case(cfg, wait_timeout_s=0.2)
    x_bits = synth.hidden(cfg, 0, 97)
    out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                         next_router_w=case.router[1])
    torch.cuda.synchronize()
    held = int(case.plan.slot_table(0)[0].max())
    case.plan.hold(held)
    rc, _, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                          next_router_w=case.router[1], check=False)
    assert rc == N.MSI_ERR_TIMEOUT
    case.plan.release(held)
    out1, _ = case.plan.forward_streamed(1, bf16_tensor(x_bits), case.router[1])
    out0, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0],
                                         next_router_w=case.router[1])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out1), case.oracle_layer(x_bits, 1)["out"])
    compare_out(bf16_bits(out0), case.oracle_layer(x_bits, 0)["out"])
    case.close()


def test_pins_with_prediction_match_the_simulator():
    """Pins and the prefetch bundle together (2 layers of the tiny shape, 16
    slots in waves of 4, so four objects may be pinned): over alternating
    layer calls with prediction, the trace equals the simulator's with the same
    pins and predictions, and no pinned object is ever evicted."""
    cfg = synth.config("decode48", tokens=24, n_layers=2, n_slots=16)
    case = Case(cfg, wave_capacity=4)
    sim = oracle.LRUWaveSim(cfg.n_slots, 4)
    pins = [(0, 1), (0, 5), (1, 2), (1, 9)]
    for l, e in pins:
        case.plan.pin(l, e)
        sim.pin(l, e)
    stage = torch.cuda.Stream()
    for step in range(5):
        x_bits = synth.hidden(cfg, 0, 300 + step)
        for l in range(2):
            nxt = case.router[1] if l == 0 else None
            out, ev = case.plan.forward_streamed(l, bf16_tensor(x_bits), case.router[l],
                                                 residual=True, stage_stream=stage,
                                                 next_router_w=nxt)
            torch.cuda.synchronize()
            assert case.plan.status() == N.MSI_OK
            compare_out(bf16_bits(out), case.oracle_layer(x_bits, l, residual=True)["out"])
            predict = None
            if nxt is not None:
                _, counts = _predicted_counts(ev.next, cfg.n_experts)
                predict = (1, counts)
            sim.call(l, sorted(set(ev.ids.cpu().numpy().reshape(-1).tolist())), predict)
            x_bits = bf16_bits(out)
    tr = case.plan.trace()
    assert tr == sim.trace
    assert not {(r[1], r[2]) for r in tr if r[5] == "evict"} & set(pins)
    _check_counters(case, sim)
    case.close()
