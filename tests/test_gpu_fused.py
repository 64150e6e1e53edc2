"""Fused wave GEMMs: a streamed call runs each bf16 wave's gate-up and down
projections in one launch, the down tiles after the gate-up tiles whose h rows
they read (per-m-tile counters), on single-CTA tiles or, for waves averaging
>= 1,024 rows per expert, on CTA-pair tiles.  The same tiles with the same K
order run as two launches under MSI_FWD_SPLIT_WAVES, so the two must agree
bit for bit; both match the fp64 oracle, with route events exact and the
slot traces of the two runs equal."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_case import Case, bf16_bits, bf16_tensor, compare_out, compare_routes
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _run(case, x, split, single=False):
    case.plan.trace(clear=True)
    out, ev = case.plan.forward_streamed(0, x, case.router[0], split_waves=split, single_cta=single)
    torch.cuda.synchronize()
    assert case.plan.status() == N.MSI_OK
    return bf16_bits(out), ev.ids.cpu().numpy(), ev.weights.cpu().numpy(), case.plan.trace()


def _agree(a, b):
    fa, fb = oracle.bf16_to_f64(a), oracle.bf16_to_f64(b)
    assert np.abs(fa - fb).max() <= 2e-2
    assert np.linalg.norm(fa - fb) <= 5e-3 * max(np.linalg.norm(fa), 1e-30)


@pytest.mark.parametrize("tokens,top_k,tiles", [(2048, 4, "single"), (333, 3, "single"),
                                                (5120, 4, "single"), (12000, 4, "pair")])
def test_fused_waves_small_shape_full_oracle(tokens, top_k, tiles):
    """H 512, I 256, 32 experts, 16 slots (waves of 8): ~256, ~31, ~640 and
    ~1,500 rows per expert (several m-tiles per expert, ragged and
    single-tile groups; the last on 256-row pair tiles).  Single-CTA fused
    waves equal the split single-CTA launches bit for bit; pair-tile fused
    waves equal the split launches, which take pair tiles for both
    projections at ~1,500 rows, bit for bit."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=top_k, tokens=tokens,
                       n_slots=16)
    case = Case(cfg)
    x_bits = synth.hidden(cfg, 0, 21)
    x = bf16_tensor(x_bits)
    of, idf, wf, trf = _run(case, x, split=False)
    case2 = Case(cfg)
    os_, ids_, ws_, trs = _run(case2, x, split=True, single=(tiles == "single"))
    assert np.array_equal(idf, ids_) and np.array_equal(wf, ws_)
    assert trf == trs
    if tiles == "single" or tokens * top_k // 32 >= 1024:
        assert np.array_equal(of, os_)                # bit-identical to the split launches
    else:
        _agree(of, os_)
    ref = case.oracle_layer(x_bits)
    compare_routes(idf, wf, ref)
    compare_out(of, ref["out"])
    case.close()
    case2.close()


def test_fused_waves_qwen_shape_sampled():
    """Qwen3-Next shape, 8,192 tokens, 64 slots (waves of 32): ~160 rows per
    expert, two m-tiles each (a full and a ragged one)."""
    cfg = synth.config("prefill32k_lru64", tokens=8192)
    case = Case(cfg)
    x_bits = synth.hidden(cfg, 0, 22)
    x = bf16_tensor(x_bits)
    of, idf, wf, _ = _run(case, x, split=False)
    os_, ids_, _, _ = _run(case, x, split=True, single=True)   # same plan: the second call's waves differ,
    assert np.array_equal(idf, ids_)                  # the expert work does not
    assert np.array_equal(of, os_)
    rng = np.random.default_rng(9)
    toks = np.sort(rng.choice(cfg.tokens, 40, replace=False))
    ref = case.oracle_layer(x_bits, tokens=toks)
    compare_out(of[toks], ref["out"])
    assert case.plan.launches() > 0
    case.close()


def test_fused_waves_launch_count():
    """One expert-FFN launch per wave instead of two."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=4, tokens=1024, n_slots=16)
    case = Case(cfg)
    x = bf16_tensor(synth.hidden(cfg, 0, 23))
    case.plan.timing(True)
    case.plan.timing_read(reset=True)
    case.plan.forward_streamed(0, x, case.router[0])
    torch.cuda.synchronize()
    kt = case.plan.timing_read(reset=True)
    case.plan.timing(False)
    n_waves = len({r[6] for r in case.plan.trace() if r[5] in ("hit", "stage")})
    assert kt["ffn"][1] == n_waves
    assert kt["gateup"][1] == 0 and kt["down"][1] == 0
    case.close()


@pytest.mark.parametrize("tokens", [1024, 4096])
def test_fused_resident_equals_split_launches(tokens):
    """A resident forward whose groups average < 512 rows (here ~20 and ~80
    rows over 512 experts) runs its two projections in one launch; it equals
    the split launches bit for bit and the oracle on sampled tokens."""
    cfg = synth.config("qwen3next_4k", tokens=tokens)
    case = Case(cfg)
    table, gens = case.stage_all()
    x_bits = synth.hidden(cfg, 0, 24)
    x = bf16_tensor(x_bits)
    outs = []
    for split in (False, True):
        case.plan.timing(True)
        case.plan.timing_read(reset=True)
        out, ev = case.plan.forward(0, x, case.router[0], table, gens, split_waves=split)
        torch.cuda.synchronize()
        kt = case.plan.timing_read(reset=True)
        case.plan.timing(False)
        assert case.plan.status() == N.MSI_OK
        assert (kt["ffn"][1] == 1) == (not split)
        outs.append((bf16_bits(out), ev.ids.cpu().numpy()))
    assert np.array_equal(outs[0][1], outs[1][1])
    assert np.array_equal(outs[0][0], outs[1][0])
    toks = np.arange(0, tokens, max(1, tokens // 48))
    ref = case.oracle_layer(x_bits, tokens=toks)
    compare_out(outs[0][0][toks], ref["out"])
    case.close()


@pytest.mark.parametrize("tokens", [5120, 2600])
def test_fused_q4_waves_equal_split_launches(tokens):
    """4-bit experts: waves whose groups average >= 512 rows (~640 and ~325
    rows per expert here; the smaller one keeps the split single-CTA
    launches) run both projections in one CTA-pair launch with the codes
    dequantised in the kernel; bit-identical to the split pair launches and
    within the output tolerance of the oracle."""
    cfg = synth.config("tiny", hidden=512, inter=256, n_experts=32, top_k=4, tokens=tokens,
                       n_slots=16, wdtype=synth.W_Q4G32)
    case = Case(cfg)
    x_bits = synth.hidden(cfg, 0, 25)
    x = bf16_tensor(x_bits)
    case.plan.timing(True)
    case.plan.timing_read(reset=True)
    of, idf, wf, trf = _run(case, x, split=False)
    kt = case.plan.timing_read(reset=True)
    case.plan.timing(False)
    assert (kt["ffn"][1] > 0) == (tokens * 4 // 32 >= 512)
    case2 = Case(cfg)
    os_, ids_, _, trs = _run(case2, x, split=True)
    assert np.array_equal(idf, ids_)
    assert trf == trs
    assert np.array_equal(of, os_)
    ref = case.oracle_layer(x_bits)
    compare_routes(idf, wf, ref)
    compare_out(of, ref["out"])
    case.close()
    case2.close()
