"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs.  Route events bit-exact except counted near-ties, slot
traces bit-exact, outputs within norm-relative 5e-3 and max-abs 2e-2."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _needed(ids, E):
    return sorted(set(np.asarray(ids).reshape(-1).tolist()))


def _run_streamed(case, x_bits, layer=0, residual=False):
    x = bf16_tensor(x_bits)
    stage = torch.cuda.Stream()
    out, ev = case.plan.forward_streamed(layer, x, case.router[layer], residual=residual,
                                         stage_stream=stage)
    torch.cuda.synchronize()
    return out, ev


def test_tiny_streamed_lru_full_oracle():
    cfg = synth.config("tiny")
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    for call in range(3):
        x_bits = synth.hidden(cfg, 0, call)
        out, ev = _run_streamed(case, x_bits)
        assert case.plan.status() == N.MSI_OK
        ref = case.oracle_layer(x_bits)
        ids = ev.ids.cpu().numpy()
        compare_routes(ids, ev.weights.cpu().numpy(), ref)
        assert np.array_equal(ev.counts.cpu().numpy(), np.bincount(ids.reshape(-1), minlength=cfg.n_experts))
        sim.call(0, _needed(ids, cfg.n_experts))
        compare_out(bf16_bits(out), ref["out"])
    assert case.plan.trace() == sim.trace
    c = case.plan.counters()
    assert c["stages"] == sum(1 for r in sim.trace if r[5] == "stage")
    case.close()


@pytest.mark.parametrize("T", [1, 33, 97, 200])
def test_tiny_resident_ragged(T):
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 7, tokens=T)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), ref)
    compare_out(bf16_bits(out), ref["out"])
    case.close()


def test_empty_batch():
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    table, gens = case.stage_all()
    x = torch.empty((0, cfg.hidden), dtype=torch.bfloat16, device="cuda")
    out, ev = case.plan.forward(0, x, case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    assert ev.counts.cpu().numpy().sum() == 0
    out, ev = case.plan.forward_streamed(0, x, case.router[0])
    torch.cuda.synchronize()
    assert ev.counts.cpu().numpy().sum() == 0
    case.close()


def test_resident_and_streamed_bitwise_equal():
    """Same inputs through caller-managed residency and through LRU waves give
    bit-identical outputs and route events (per-element accumulation order does
    not depend on the grouping)."""
    cfg = synth.config("tiny", n_slots=16)
    a = Case(cfg)
    table, gens = a.stage_all()
    b = Case(synth.config("tiny"))
    x_bits = synth.hidden(cfg, 0, 3)
    o1, e1 = a.plan.forward(0, bf16_tensor(x_bits), a.router[0], table, gens)
    o2, e2 = _run_streamed(b, x_bits)
    torch.cuda.synchronize()
    assert torch.equal(e1.ids, e2.ids) and torch.equal(e1.weights, e2.weights)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    a.close()
    b.close()


def test_qwen_shape_resident_several_tiles():
    """Qwen3-Next layer shape (H 2048, E 512, k 10, I 512, shared expert) at
    1,000 tokens: ragged 128-row tiles, 4 gate-up and 8 down N tiles, 32 K blocks."""
    cfg = synth.config("qwen3next_4k", tokens=1000)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 0)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    near, near_adj = compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), ref)
    mask = ~oracle.near_tie_tokens(ref["gap_k"])
    compare_out(bf16_bits(out), ref["out"], mask)
    case.close()


def test_qwen_4k_resident_full_routes_sampled_outputs():
    cfg = synth.config("qwen3next_4k")
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 0)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    r = oracle.router(x_bits, case.router_np[0], cfg.top_k)
    compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), r)
    rng = np.random.default_rng(0)
    toks = np.sort(np.concatenate([[0, cfg.tokens - 1], rng.choice(cfg.tokens, 62, replace=False)]))
    ref = case.oracle_layer(x_bits, tokens=toks)
    mask = ~oracle.near_tie_tokens(ref["gap_k"])
    compare_out(bf16_bits(out)[toks], ref["out"], mask)
    case.close()


# ---------------------------------------------------------------------------
# Fail-closed behaviour (host precheck, device re-check, held consumer)
# ---------------------------------------------------------------------------

def test_host_precheck_rejects_stale_and_wrong_object():
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    table, gens = case.stage_all()
    x = bf16_tensor(synth.hidden(cfg, 0, 1))
    n0 = case.plan.launches()
    g2 = gens.copy(); g2[5] += 1
    rc, _, _ = case.plan.forward(0, x, case.router[0], table, g2, check=False)
    assert rc == N.MSI_ERR_STALE_GENERATION
    t2 = table.copy(); t2[3], t2[4] = table[4], table[3]
    rc, _, _ = case.plan.forward(0, x, case.router[0], t2, gens, check=False)
    assert rc == N.MSI_ERR_WRONG_OBJECT
    assert case.plan.launches() == n0          # nothing enqueued
    # restage bumps the generation: the old expectation is now stale
    g_new = case.plan.stage(5, 0, 5)
    assert g_new == gens[5] + 1
    rc, _, _ = case.plan.forward(0, x, case.router[0], table, gens, check=False)
    assert rc == N.MSI_ERR_STALE_GENERATION
    case.close()


def test_device_recheck_not_resident_writes_nothing():
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 2)
    ids_ref = oracle.router(x_bits, case.router_np[0], cfg.top_k)["ids"]
    missing = int(ids_ref[0, 0])
    t2 = table.copy(); t2[missing] = -1
    out = torch.full((cfg.tokens, cfg.hidden), 7.0, dtype=torch.bfloat16, device="cuda")
    case.plan.forward(0, bf16_tensor(x_bits), case.router[0], t2, gens, out=out)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_ERR_NOT_RESIDENT
    assert torch.all(out == 7.0)               # no row became visible
    case.close()


def test_held_consumer_delays_restage():
    cfg = synth.config("tiny", n_slots=16)
    case = Case(cfg, wait_timeout_s=0.2)
    case.stage_all()
    case.plan.hold(3)
    assert case.plan.slot_state(3) == N.MSI_SLOT_IN_USE
    with pytest.raises(N.MsiError) as ei:
        case.plan.stage(3, 0, 3)
    assert ei.value.status == N.MSI_ERR_TIMEOUT
    with pytest.raises(N.MsiError) as ei:
        case.plan.close()                      # destroy with a live consumer
    assert ei.value.status == N.MSI_ERR_SLOT_BUSY
    case.plan.release(3)
    assert case.plan.stage(3, 0, 3) == 2
    torch.cuda.synchronize()
    assert case.plan.slot_state(3) in (N.MSI_SLOT_DEVICE_READY, N.MSI_SLOT_RECYCLABLE)
    case.close()


def test_balanced_teardown_states():
    cfg = synth.config("tiny")
    case = Case(cfg)
    for call in range(2):
        _run_streamed(case, synth.hidden(cfg, 0, call))
    torch.cuda.synchronize()
    states = {case.plan.slot_state(s) for s in range(cfg.n_slots)}
    assert states <= {N.MSI_SLOT_VACANT, N.MSI_SLOT_RECYCLABLE, N.MSI_SLOT_DEVICE_READY}
    case.close()


# ---------------------------------------------------------------------------
# 4-bit block-quantised experts (group 32, fp16 scale), dequantised in the GEMM
# ---------------------------------------------------------------------------

def test_q4_tiny_streamed_lru():
    cfg = synth.config("tiny", wdtype=synth.W_Q4G32)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, 20 + call)
        out, ev = _run_streamed(case, x_bits)
        assert case.plan.status() == N.MSI_OK
        ref = case.oracle_layer(x_bits)
        ids = ev.ids.cpu().numpy()
        compare_routes(ids, ev.weights.cpu().numpy(), ref)
        sim.call(0, _needed(ids, cfg.n_experts))
        compare_out(bf16_bits(out), ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    assert case.plan.trace() == sim.trace
    case.close()


def test_q4_qwen_shape_lru_waves():
    """Qwen3-Next layer shape with 4-bit experts, 64-slot pool, 2,000 tokens
    (all 512 experts needed: 8 waves of 32, 448 stages after the first call)."""
    cfg = synth.config("prefill32k_q4_lru64", tokens=2000)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    rng = np.random.default_rng(1)
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, call)
        out, ev = _run_streamed(case, x_bits)
        assert case.plan.status() == N.MSI_OK
        ids = ev.ids.cpu().numpy()
        r = oracle.router(x_bits, case.router_np[0], cfg.top_k, case.gate_np[0])
        compare_routes(ids, ev.weights.cpu().numpy(), r)
        sim.call(0, _needed(ids, cfg.n_experts))
        toks = np.sort(rng.choice(cfg.tokens, 48, replace=False))
        ref = case.oracle_layer(x_bits, tokens=toks)
        compare_out(bf16_bits(out)[toks], ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    assert case.plan.trace() == sim.trace
    case.close()


def test_simt_router_path_odd_expert_count():
    """E = 20 (not a multiple of 16) routes through the fp32 FFMA router."""
    cfg = synth.config("tiny", n_experts=20, n_slots=8)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    x_bits = synth.hidden(cfg, 0, 5)
    out, ev = _run_streamed(case, x_bits)
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    ids = ev.ids.cpu().numpy()
    compare_routes(ids, ev.weights.cpu().numpy(), ref)
    sim.call(0, _needed(ids, cfg.n_experts))
    compare_out(bf16_bits(out), ref["out"])
    assert case.plan.trace() == sim.trace
    case.close()


@pytest.mark.parametrize("E,k,H", [(64, 31, 1024), (64, 32, 1024), (256, 8, 256), (64, 31, 256)])
def test_router_limits_and_chunks(E, k, H):
    """k = 31 is the largest top-k of the tensor-core router (k + 1 candidates
    per chunk), k = 32 routes through the fp32 FFMA router, E = 256 merges two
    128-expert chunks; small layers (E <= 64, E * H <= 32,768: the last case)
    take the FFMA router sized for 64 experts."""
    cfg = synth.config("tiny", n_experts=E, top_k=k, n_slots=E, tokens=96, hidden=H)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 9)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), ref)
    g = ev.gap.cpu().numpy()
    ok = ~oracle.near_tie_tokens(ref["gap_adj"])
    np.testing.assert_allclose(g[ok], ref["gap_k"][ok], rtol=0, atol=2e-5)
    compare_out(bf16_bits(out), ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    case.close()


@pytest.mark.parametrize("E,H", [(64, 1024), (256, 256), (64, 256)])
def test_exact_logit_ties_rank_lower_id_first(E, H):
    """Duplicated (and amplified) router rows give exactly equal logits; the
    route event must rank the lower expert id first (the oracle's order), the
    pair adjacent with equal weights: tensor router within one 128-expert
    chunk (E = 64, H = 1024) and across chunks through the candidate merge
    (E = 256); FFMA router sized for 64 experts (E = 64, H = 256)."""
    cfg = synth.config("tiny", n_experts=E, n_slots=E, top_k=6, tokens=512, lru=False, hidden=H)
    case = Case(cfg)
    table, gens = case.stage_all()
    w = case.router_np[0].copy()
    pairs = [(3, 40), (10, 11), (0, 63)] if E == 64 else [(5, 133), (120, 200), (7, 8)]
    for lo, hi in pairs:
        w[lo] *= 4.0
        w[hi] = w[lo]
    case.router[0] = torch.from_numpy(w).cuda()
    case.router_np[0] = w
    x_bits = synth.hidden(cfg, 0, 21)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ids = ev.ids.cpu().numpy()
    wts = ev.weights.cpu().numpy()
    seen = 0
    for t in range(cfg.tokens):
        row = ids[t].tolist()
        for lo, hi in pairs:
            if hi in row:
                seen += 1
                j = row.index(hi)
                assert j > 0 and row[j - 1] == lo, f"token {t}: {row}"
                assert wts[t, j] == wts[t, j - 1]
    assert seen > 50  # the amplified pairs are routed often
    compare_routes(ids, wts, oracle.router(x_bits, w, cfg.top_k))
    case.close()


def test_ungated_shared_expert_flag():
    """MSI_FWD_SHARED_UNGATED: the shared expert's output enters with gate 1
    (the other reading of its gate) and matches the oracle taking that
    reading; without the flag the gated output is unchanged."""
    cfg = synth.config("qwen3next_4k", n_experts=64, n_slots=64, tokens=300)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 150)
    out_u, _ = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens,
                                 shared_gate=False)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref_u = oracle.moe_layer(x_bits, case.router_np[0], cfg.top_k, lambda e: case.extent(0, e),
                             cfg.hidden, cfg.inter, shared_extent=case.shared_np[0],
                             w_sg=case.gate_np[0], shared_gated=False)
    compare_out(bf16_bits(out_u), ref_u["out"])
    out_g, _ = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    compare_out(bf16_bits(out_g), case.oracle_layer(x_bits)["out"])
    assert not torch.equal(out_u, out_g)
    case.close()


@pytest.mark.parametrize("E,k,H,I,T", [(512, 32, 256, 128, 200), (16, 16, 256, 128, 64),
                                       (16, 1, 256, 128, 64), (512, 1, 2048, 512, 33)])
def test_extreme_expert_counts_and_top_k(E, k, H, I, T):
    """The library's limits and degenerate routings: E = 512 with k = 32 (the
    largest of both), k = E (every token takes every expert: dense softmax
    mixing, gap +inf), k = 1 at the tiny and the Qwen shape (ragged T)."""
    cfg = synth.config("tiny", n_experts=E, top_k=k, hidden=H, inter=I, tokens=T, n_slots=E,
                       lru=False)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 160)
    out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    ids = ev.ids.cpu().numpy()
    compare_routes(ids, ev.weights.cpu().numpy(), ref)
    assert np.array_equal(ev.counts.cpu().numpy(), np.bincount(ids.reshape(-1), minlength=E))
    if k == E:
        assert np.all(np.sort(ids, axis=1) == np.arange(E)) and np.all(np.isinf(ev.gap.cpu().numpy()))
    compare_out(bf16_bits(out), ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    case.close()
