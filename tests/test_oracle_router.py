"""Pins of the oracle's router, top-k and route weights against facts other
than the oracle itself: exact-arithmetic brute force, constructed ties, the
dense softmax special case (scipy), renormalisation identities."""
import itertools

import numpy as np
import pytest
import scipy.special

import oracle



def _bf16_bits(vals):
    f = np.asarray(vals, dtype=np.float32)
    assert np.all((f.view(np.uint32) & 0xFFFF) == 0), "value not exactly bf16"
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def _exact_case(T, E, H, seed):
    """Small-integer x and dyadic W: every logit is exact in float64."""
    rng = np.random.default_rng(seed)
    x = rng.integers(-4, 5, size=(T, H)).astype(np.float32)
    W = (rng.integers(-8, 9, size=(E, H)) / 16.0).astype(np.float32)
    return _bf16_bits(x), W, x.astype(np.float64) @ W.astype(np.float64).T


def _rank_by_count(l):
    """Rank of each expert by the counting definition: number of experts that beat it."""
    E = len(l)
    return [sum(1 for f in range(E) if l[f] > l[e] or (l[f] == l[e] and f < e)) for e in range(E)]


@pytest.mark.parametrize("seed", range(5))
@pytest.mark.parametrize("k", [1, 2, 3, 9])
def test_topk_matches_counting_definition(seed, k):
    T, E, H = 40, 9, 6        # small integers make many exact ties
    xb, W, L = _exact_case(T, E, H, seed)
    r = oracle.router(xb, W, k)
    for t in range(T):
        rank = _rank_by_count(list(L[t]))
        want = sorted(range(E), key=lambda e: rank[e])[:k]
        assert list(r["ids"][t]) == want


def test_constructed_exact_ties_prefer_lower_id():
    H, E = 4, 6
    W = np.zeros((E, H), dtype=np.float32)
    W[1] = W[4] = W[5] = [1, 0, 0, 0]       # experts 1, 4, 5 tie for the top
    W[2] = [0.5, 0, 0, 0]
    x = _bf16_bits([[2, 0, 0, 0]])
    r = oracle.router(x, W, 4)
    assert list(r["ids"][0]) == [1, 4, 5, 2]
    assert r["gap_adj"][0] == 0.0
    assert r["gap_k"][0] == pytest.approx(1.0)   # l(2) - l(0) = 1.0 - 0.0
    np.testing.assert_allclose(r["weights"][0, :3], r["weights"][0, 0])


@pytest.mark.parametrize("seed", range(3))
def test_k_equals_E_is_dense_softmax(seed):
    T, E, H = 16, 7, 5
    xb, W, L = _exact_case(T, E, H, seed)
    r = oracle.router(xb, W, E)
    sm = scipy.special.softmax(L, axis=1)
    got = np.zeros_like(sm)
    np.put_along_axis(got, r["ids"], r["weights"], axis=1)
    np.testing.assert_allclose(got, sm, rtol=1e-13, atol=0)
    assert np.all(np.isinf(r["gap_k"]))


@pytest.mark.parametrize("k", [1, 2, 4])
def test_weights_are_renormalised_full_softmax(k):
    T, E, H = 32, 11, 8
    xb, W, L = _exact_case(T, E, H, 7)
    r = oracle.router(xb, W, k)
    sm = scipy.special.softmax(L, axis=1)
    sel = np.take_along_axis(sm, r["ids"], axis=1)
    np.testing.assert_allclose(r["weights"], sel / sel.sum(axis=1, keepdims=True), rtol=1e-13)
    np.testing.assert_allclose(r["weights"].sum(axis=1), 1.0, rtol=1e-14)
    # weights follow the descending logit order
    assert np.all(np.diff(r["weights"], axis=1) <= 1e-15)


def test_gaps_against_masked_definition():
    T, E, H, k = 64, 12, 8, 3
    xb, W, L = _exact_case(T, E, H, 3)
    r = oracle.router(xb, W, k)
    for t in range(T):
        sel = set(r["ids"][t])
        kth = min(L[t, e] for e in sel)
        best_out = max(L[t, e] for e in range(E) if e not in sel)
        assert r["gap_k"][t] == kth - best_out
        vals = sorted(L[t], reverse=True)[:k + 1]
        assert r["gap_adj"][t] == min(a - b for a, b in zip(vals, vals[1:]))


def test_distinct_ids_and_shared_gate_sigmoid():
    rng = np.random.default_rng(0)
    T, E, H, k = 50, 16, 32, 4
    x = _bf16_bits(np.round(rng.normal(size=(T, H)) * 8) / 8)
    W = rng.normal(0, 0.02, size=(E, H)).astype(np.float32)
    wsg = rng.normal(0, 0.02, size=H).astype(np.float32)
    r = oracle.router(x, W, k, wsg)
    for t in range(T):
        assert len(set(r["ids"][t])) == k
    xf = oracle.bf16_to_f64(x)
    np.testing.assert_allclose(r["sg"], scipy.special.expit(xf @ wsg.astype(np.float64)), rtol=1e-14)


def test_bf16_and_f16_decoding_exact():
    import torch
    vals = torch.tensor([0.0, -0.0, 1.0, -2.5, 3.140625, 1e-3, 65504.0, 2.0 ** -14], dtype=torch.float32)
    b = vals.to(torch.bfloat16)
    got = oracle.bf16_to_f64(b.view(torch.int16).numpy().view(np.uint16))
    np.testing.assert_array_equal(got, b.to(torch.float64).numpy())
    h = vals.to(torch.float16)
    got = oracle.f16_to_f64(h.view(torch.int16).numpy().view(np.uint16))
    np.testing.assert_array_equal(got, h.to(torch.float64).numpy())


def test_near_tie_flags():
    g = np.array([0.0, 5e-5, 1e-4, 2e-4, np.inf])
    assert list(oracle.near_tie_tokens(g)) == [True, True, False, False, False]


def test_every_k_subset_brute_force_tiny():
    """Tiny exhaustive check: the selected set maximises the sum of logits over
    all k-subsets when logits are distinct."""
    rng = np.random.default_rng(11)
    T, E, H, k = 12, 6, 4, 3
    x = _bf16_bits(rng.integers(-3, 4, size=(T, H)).astype(np.float32))
    W = (rng.permutation(E * H).reshape(E, H) / 64.0).astype(np.float32)
    r = oracle.router(x, W, k)
    L = r["logits"]
    for t in range(T):
        if len(set(L[t])) < E:
            continue
        best = max(itertools.combinations(range(E), k), key=lambda c: sum(L[t, e] for e in c))
        assert set(best) == set(r["ids"][t])
