"""CTA-pair expert GEMMs (256-row tiles, tcgen05 cta_group::2): the forwards
pick them when a launch's groups average at least 1,024 rows.  Each case runs
the same inputs through the pair kernels (default) and through the single-CTA
kernels (MSI_FWD_SINGLE_CTA); both must match the fp64 oracle within the
output tolerance, with route events exact, and agree with each other.  With
4-bit experts the pair kernels take over from 512 rows per group, and each
CTA dequantises only its own half of the B tile."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _both(case, x_bits, table, gens, **kw):
    outs = []
    for single in (False, True):
        out, ev = case.plan.forward(0, bf16_tensor(x_bits), case.router[0], table, gens,
                                    single_cta=single, **kw)
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        outs.append((bf16_bits(out), ev.ids.cpu().numpy(), ev.weights.cpu().numpy()))
    return outs


def _agree(a, b):
    fa, fb = oracle.bf16_to_f64(a), oracle.bf16_to_f64(b)
    assert np.abs(fa - fb).max() <= 2e-2
    assert np.linalg.norm(fa - fb) <= 5e-3 * max(np.linalg.norm(fa), 1e-30)


@pytest.mark.parametrize("tokens", [4100, 6000])
def test_pair_resident_small_shape_full_oracle(tokens):
    """H 512, I 256, 16 experts, top-4, shared expert: ~1,025-1,500 rows per
    expert (ragged pair tiles, several 256-row tiles per expert, partial halves)."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=16, top_k=4, tokens=tokens,
                       n_slots=16, has_shared=True, lru=False)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 11)
    (op, ip, wp), (os_, is_, ws_) = _both(case, x_bits, table, gens)
    ref = case.oracle_layer(x_bits)
    compare_routes(ip, wp, oracle.router(x_bits, case.router_np[0], cfg.top_k))
    assert np.array_equal(ip, is_)
    compare_out(op, ref["out"])
    compare_out(os_, ref["out"])
    _agree(op, os_)
    case.close()


def test_pair_qwen_shape_sampled_tokens():
    """H 2048, I 512, 64 experts, top-10, 8,192 tokens: ~1,280 rows per
    expert, five 256-row tiles each; outputs checked on sampled tokens."""
    cfg = synth.config("qwen3next_4k", n_experts=64, tokens=8192, n_slots=64)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 12)
    (op, ip, wp), (os_, is_, ws_) = _both(case, x_bits, table, gens)
    rng = np.random.default_rng(5)
    toks = np.sort(rng.choice(cfg.tokens, 48, replace=False))
    ref = case.oracle_layer(x_bits, tokens=toks)
    compare_out(op[toks], ref["out"])
    compare_out(os_[toks], ref["out"])
    assert np.array_equal(ip, is_)
    _agree(op, os_)
    case.close()


@pytest.mark.parametrize("tokens,top_k", [(8192, 8), (4096, 5)])
def test_pair_streamed_waves_full_oracle(tokens, top_k):
    """Streamed LRU waves (32 experts, 16 slots, waves of 8): ~2,048 rows per
    expert (pair tiles for both projections) and ~640 rows per expert (pair
    tiles for the down projection only); matches the oracle, with the default
    tiles and with single-CTA tiles."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=top_k, tokens=tokens,
                       n_slots=16, has_shared=False)
    case = Case(cfg)
    x_bits = synth.hidden(cfg, 0, 13)
    out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    ref = case.oracle_layer(x_bits)
    compare_routes(ev.ids.cpu().numpy(), ev.weights.cpu().numpy(),
                   oracle.router(x_bits, case.router_np[0], cfg.top_k))
    compare_out(bf16_bits(out), ref["out"])
    out1, _ = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0], single_cta=True)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    compare_out(bf16_bits(out1), ref["out"])
    case.close()


@pytest.mark.parametrize("tokens", [4100, 2100])
def test_pair_q4_resident_full_oracle(tokens):
    """4-bit experts (group 32, fp16 scales): H 512, I 256, 16 experts, top-4,
    shared expert; ~1,025 and ~525 rows per expert (pair tiles for both
    projections, ragged last tiles)."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=16, top_k=4, tokens=tokens,
                       n_slots=16, has_shared=True, lru=False, wdtype=synth.W_Q4G32)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 14)
    (op, ip, wp), (os_, is_, ws_) = _both(case, x_bits, table, gens)
    ref = case.oracle_layer(x_bits)
    compare_routes(ip, wp, oracle.router(x_bits, case.router_np[0], cfg.top_k))
    assert np.array_equal(ip, is_)
    ok = ~oracle.near_tie_tokens(ref["gap_k"])
    compare_out(op, ref["out"], ok)
    compare_out(os_, ref["out"], ok)
    _agree(op, os_)
    case.close()


def test_pair_q4_qwen_shape_sampled_tokens():
    """Qwen3-Next layer shape (H 2048, I 512, top-10) with 4-bit experts, 64
    experts resident, 8,192 tokens: ~1,280 rows per expert."""
    cfg = synth.config("prefill32k_q4_lru64", n_experts=64, tokens=8192, n_slots=64, lru=False)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 15)
    (op, ip, wp), (os_, is_, ws_) = _both(case, x_bits, table, gens)
    rng = np.random.default_rng(6)
    toks = np.sort(rng.choice(cfg.tokens, 40, replace=False))
    ref = case.oracle_layer(x_bits, tokens=toks)
    compare_out(op[toks], ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    compare_out(os_[toks], ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    assert np.array_equal(ip, is_)
    _agree(op, os_)
    case.close()


def test_pair_q4_streamed_waves_trace_and_oracle():
    """4-bit experts in streamed LRU waves (32 experts, 16 slots, waves of 8),
    8,192 tokens, top-4, shared expert: ~1,024 rows per expert, so both
    projections run on pair tiles while slots are re-staged between waves.
    Two calls: outputs match the oracle, the slot trace the oracle's simulator."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=4, tokens=8192,
                       n_slots=16, has_shared=True, wdtype=synth.W_Q4G32)
    case = Case(cfg)
    sim = oracle.LRUWaveSim(cfg.n_slots)
    for call in range(2):
        x_bits = synth.hidden(cfg, 0, 16 + call)
        out, ev = case.plan.forward_streamed(0, bf16_tensor(x_bits), case.router[0])
        torch.cuda.synchronize()
        assert case.plan.status() == N.MSI_OK
        ids = ev.ids.cpu().numpy()
        ref = case.oracle_layer(x_bits)
        compare_routes(ids, ev.weights.cpu().numpy(), ref)
        sim.call(0, sorted(set(ids.reshape(-1).tolist())))
        compare_out(bf16_bits(out), ref["out"], ~oracle.near_tie_tokens(ref["gap_k"]))
    assert case.plan.trace() == sim.trace
    case.close()


@pytest.mark.parametrize("wdtype", [synth.W_BF16, synth.W_Q4G32])
def test_pair_skewed_routing(wdtype):
    """A heavily skewed routing in one launch: every hidden row carries the
    constant 4.0 in feature 0 and the router's column 0 turns it into a
    per-expert bias 4 * (0.25 - 0.04 e).  The first experts then take most
    tokens (thousands of rows, many pair tiles), the last ones a row or two or
    none.  Pair and single-CTA tiles both match the oracle."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=16, top_k=4, tokens=6000,
                       n_slots=16, has_shared=True, lru=False, wdtype=wdtype)
    case = Case(cfg)
    w = case.router_np[0].copy()
    w[:, 0] = (0.25 - 0.04 * np.arange(cfg.n_experts)).astype(np.float32)
    case.router_np[0] = w
    case.router[0] = torch.from_numpy(w).cuda()
    x_bits = synth.hidden(cfg, 0, 17).copy()
    x_bits[:, 0] = 0x4080  # bf16 4.0
    table, gens = case.stage_all()
    (op, ip, wp), (os_, is_, ws_) = _both(case, x_bits, table, gens)
    counts = np.bincount(ip.reshape(-1), minlength=cfg.n_experts)
    assert counts.max() >= 3 * counts.mean() and (counts <= 2).any()
    ref = case.oracle_layer(x_bits)
    compare_routes(ip, wp, ref)
    assert np.array_equal(ip, is_)
    ok = ~oracle.near_tie_tokens(ref["gap_k"])
    compare_out(op, ref["out"], ok)
    compare_out(os_, ref["out"], ok)
    _agree(op, os_)
    case.close()
