"""Pins of the oracle's expert FFN, permutation, combine and 4-bit decoding:
closed forms, a library SwiGLU MLP (torch CPU float64), dense masked
evaluation, brute-force stable ordering, exact small-integer dequantisation."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth



def _bits(vals):
    f = np.asarray(vals, dtype=np.float32)
    assert np.all((f.view(np.uint32) & 0xFFFF) == 0)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def _extent_from(w13, w2):
    return np.concatenate([_bits(w13).reshape(-1), _bits(w2).reshape(-1)]).view(np.uint8)


def test_intermediate_one_closed_form():
    """I = 1, unit gate/up/down vectors: y[2] = silu(x0) * x1 and nothing else.
    silu(1) = e / (1 + e) and silu(-2) = -2 / (1 + e^2) in closed form; the
    case is asymmetric, so swapped gate/up rows or a transposed W2 fail."""
    H, I = 4, 1
    w13 = np.zeros((2, H), np.float32); w13[0, 0] = 1.0; w13[1, 1] = 1.0
    w2 = np.zeros((H, I), np.float32); w2[2, 0] = 1.0
    ext = _extent_from(w13, w2)
    Wg, Wu, W2 = oracle.decode_extent(ext, H, I)
    for x0, x1, silu in [(1.0, 2.0, math.e / (1 + math.e)), (-2.0, 3.0, -2.0 / (1 + math.e ** 2)),
                         (0.0, 5.0, 0.0)]:
        y = oracle.swiglu_expert(oracle.bf16_to_f64(_bits([[x0, x1, 0.5, -1.0]])), Wg, Wu, W2)
        want = np.array([0.0, 0.0, silu * x1, 0.0])
        np.testing.assert_allclose(y[0], want, rtol=1e-15, atol=0)


def _tiny(E=4, H=32, I=16, T=24, k=2, seed=3):
    cfg = synth.MoEConfig("t", H, E, k, I, T, 4, False, seed=seed)
    x = synth.hidden(cfg)
    Wr = synth.router_weight(cfg)
    ext = {e: synth.expert_extent(cfg, 0, e) for e in range(E)}
    return cfg, x, Wr, ext


def test_single_expert_is_textbook_swiglu_mlp():
    """E = 1, k = 1 reduces the layer to one SwiGLU MLP: compare with torch's
    F.silu / F.linear in float64 on the same decoded weights."""
    cfg, x, Wr, ext = _tiny(E=1, k=1)
    r = oracle.moe_layer(x, Wr, 1, ext.__getitem__, cfg.hidden, cfg.inter)
    Wg, Wu, W2 = (torch.from_numpy(a) for a in oracle.decode_extent(ext[0], cfg.hidden, cfg.inter))
    xt = torch.from_numpy(oracle.bf16_to_f64(x))
    ref = torch.nn.functional.linear(torch.nn.functional.silu(torch.nn.functional.linear(xt, Wg))
                                     * torch.nn.functional.linear(xt, Wu), W2)
    np.testing.assert_allclose(r["out"], ref.numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(r["weights"], 1.0)


@pytest.mark.parametrize("k", [1, 2, 4])
def test_sparse_equals_dense_masked(k):
    cfg, x, Wr, ext = _tiny(E=6, k=k, T=40)
    r = oracle.moe_layer(x, Wr, k, ext.__getitem__, cfg.hidden, cfg.inter)
    d = oracle.dense_masked_moe(x, Wr, k, ext.__getitem__, cfg.hidden, cfg.inter)
    err = np.linalg.norm(r["out"] - d) / np.linalg.norm(d)
    assert err <= 1e-12


def test_shared_expert_and_residual_terms():
    cfg, x, Wr, ext = _tiny(E=4, k=2)
    cfg2 = synth.MoEConfig("t", cfg.hidden, 4, 2, cfg.inter, cfg.tokens, 4, True, seed=3)
    sh = synth.shared_extent(cfg2)
    wsg = synth.shared_gate_weight(cfg2)
    base = oracle.moe_layer(x, Wr, 2, ext.__getitem__, cfg.hidden, cfg.inter)
    full = oracle.moe_layer(x, Wr, 2, ext.__getitem__, cfg.hidden, cfg.inter,
                            shared_extent=sh, w_sg=wsg, residual=True)
    xf = oracle.bf16_to_f64(x)
    Sg, Su, S2 = (torch.from_numpy(a) for a in oracle.decode_extent(sh, cfg.hidden, cfg.inter))
    xt = torch.from_numpy(xf)
    ys = torch.nn.functional.linear(torch.nn.functional.silu(xt @ Sg.T) * (xt @ Su.T), S2).numpy()
    gate = torch.sigmoid(xt @ torch.from_numpy(wsg.astype(np.float64))).numpy()
    np.testing.assert_allclose(full["out"], base["out"] + gate[:, None] * ys + xf, rtol=1e-12,
                               atol=1e-14)
    # the ungated reading adds the library MLP's output with weight 1
    ungated = oracle.moe_layer(x, Wr, 2, ext.__getitem__, cfg.hidden, cfg.inter,
                               shared_extent=sh, w_sg=wsg, shared_gated=False)
    np.testing.assert_allclose(ungated["out"], base["out"] + ys, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("seed", range(4))
def test_permutation_bijection_and_stable_order(seed):
    rng = np.random.default_rng(seed)
    T, k, E = 37, 3, 8
    ids = np.stack([rng.choice(E, size=k, replace=False) for _ in range(T)])
    counts, offsets, perm, inv = oracle.permutation(ids, E)
    flat = ids.reshape(-1)
    assert counts.sum() == T * k and offsets[-1] == T * k
    # brute force: sort the flat indices by (expert, flat index) in pure Python
    assert list(perm) == sorted(range(T * k), key=lambda i: (flat[i], i))
    assert sorted(perm) == list(range(T * k))             # bijection
    assert np.all(inv[perm] == np.arange(T * k))          # every row unpermuted exactly once
    for e in range(E):
        seg = perm[offsets[e]:offsets[e + 1]]
        assert np.all(flat[seg] == e) and len(seg) == counts[e]


def test_q4_dequant_exact_small_integers():
    rows, cols = 2, 64
    q = np.arange(rows * cols).reshape(rows, cols) % 16
    packed = (q[:, 0::2] | (q[:, 1::2] << 4)).astype(np.uint8)
    scales = np.array([[1.0, 0.5], [-2.0, 0.0]], dtype=np.float16).view(np.uint16)
    w = oracle.dequant_q4g32(packed, scales, rows, cols)
    want = (q - 8).astype(np.float64) * np.repeat(np.array([[1.0, 0.5], [-2.0, 0.0]]), 32, axis=1)
    np.testing.assert_array_equal(w, want)
    assert w[0, 0] == -8.0 and w[0, 1] == -7.0 and w[0, 15] == 7.0   # low nibble = even column


def test_q4_roundtrip_within_half_scale():
    cfg = synth.config("tiny", wdtype=synth.W_Q4G32, hidden=64, inter=32)
    cfgb = synth.config("tiny", hidden=64, inter=32)
    Wg, Wu, W2 = oracle.decode_extent(synth.expert_extent(cfg, 0, 3), 64, 32, 1)
    Bg, Bu, B2 = oracle.decode_extent(synth.expert_extent(cfgb, 0, 3), 64, 32, 0)
    for q, b in [(Wg, Bg), (Wu, Bu), (W2, B2)]:
        amax = np.abs(b.reshape(b.shape[0], -1, 32)).max(axis=2)
        bound = np.repeat(amax / 7.0 * (0.5 + 2 ** -10) + 1e-12, 32, axis=1)
        assert np.all(np.abs(q - b) <= bound)


def test_combine_weighted_sum_order_free():
    """combine against an explicit per-token loop."""
    rng = np.random.default_rng(5)
    T, k, H = 9, 3, 4
    w = rng.random((T, k))
    inv = rng.permutation(T * k)
    Y = rng.normal(size=(T * k, H))
    out = oracle.combine(w, inv, Y)
    for t in range(T):
        want = sum(w[t, j] * Y[inv[t * k + j]] for j in range(k))
        np.testing.assert_allclose(out[t], want, rtol=1e-14)
