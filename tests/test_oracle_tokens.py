"""Pin of oracle.moe_tokens, the sampled-token oracle behind every full-size
output comparison: the outputs, route ids and weights it gives for a token
subset must be the rows of the whole-batch moe_layer at those tokens.

Routing is per token and each routed row's expert output depends only on that
row (paper, Sec. "Output-Exact Execution Beyond the Full-Residency Envelope":
each selected expert runs its complete projections on the token's row), so
the two must agree.  The whole-batch side groups rows by expert before the
matrix products, the subset side groups a different set of rows; a BLAS may
block a product by its row count, so floating-point results are compared to
1e-12 relative, far below any plausible slip (a wrong token index, a dropped
shared or residual term, a mixed-up weight column) which moves them by O(1)."""
import numpy as np
import pytest

import oracle
import synth


def _case(H, E, k, I, T, shared, wdtype=synth.W_BF16, seed=5):
    cfg = synth.MoEConfig("pin", H, E, k, I, T, E, shared, seed=seed, wdtype=wdtype)
    x = synth.hidden(cfg)
    wr = synth.router_weight(cfg)
    ext = {e: synth.expert_extent(cfg, 0, e) for e in range(E)}
    kw = {}
    if shared:
        kw = dict(shared_extent=synth.shared_extent(cfg), w_sg=synth.shared_gate_weight(cfg))
    return cfg, x, wr, ext, kw


def _check(cfg, x, wr, ext, kw, toks, residual):
    full = oracle.moe_layer(x, wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter,
                            cfg.wdtype, residual=residual, **kw)
    sub = oracle.moe_tokens(x, wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter, toks,
                            cfg.wdtype, residual=residual, **kw)
    np.testing.assert_array_equal(sub["ids"], full["ids"][toks])
    np.testing.assert_allclose(sub["weights"], full["weights"][toks], rtol=1e-12, atol=0)
    np.testing.assert_allclose(sub["gap_k"], full["gap_k"][toks], rtol=1e-12, atol=1e-15)
    scale = np.abs(full["out"]).max()
    np.testing.assert_allclose(sub["out"], full["out"][toks], rtol=1e-12, atol=1e-13 * scale)
    if kw:
        np.testing.assert_allclose(sub["sg"], full["sg"][toks], rtol=1e-12, atol=0)
    return full, sub


@pytest.mark.parametrize("residual", [False, True])
@pytest.mark.parametrize("shared", [False, True])
def test_tokens_equal_rows_of_whole_batch_tiny(shared, residual):
    cfg, x, wr, ext, kw = _case(H=64, E=8, k=2, I=32, T=48, shared=shared)
    toks = np.array([41, 3, 17, 3, 0, 47, 22])       # unsorted, non-contiguous, one repeat
    full, sub = _check(cfg, x, wr, ext, kw, toks, residual)
    # the repeated token gives the same row twice
    np.testing.assert_array_equal(sub["out"][1], sub["out"][3])


@pytest.mark.parametrize("wdtype", [synth.W_BF16, synth.W_Q4G32])
def test_tokens_equal_rows_of_whole_batch_mid(wdtype):
    """A mid-size shape with a shared expert and the residual, 4-bit weights too."""
    cfg, x, wr, ext, kw = _case(H=256, E=32, k=4, I=64, T=160, shared=True, wdtype=wdtype)
    rng = np.random.default_rng(11)
    toks = rng.choice(cfg.tokens, size=37, replace=False)   # unsorted random subset
    _check(cfg, x, wr, ext, kw, toks, residual=True)


def test_single_token_subsets_cover_the_batch():
    """Every token alone (a subset of one row: the matrix products degenerate
    to vector products) equals its row of the whole batch."""
    cfg, x, wr, ext, kw = _case(H=64, E=8, k=3, I=32, T=12, shared=True)
    full = oracle.moe_layer(x, wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter, **kw)
    scale = np.abs(full["out"]).max()
    for t in range(cfg.tokens):
        sub = oracle.moe_tokens(x, wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter, [t], **kw)
        np.testing.assert_array_equal(sub["ids"][0], full["ids"][t])
        np.testing.assert_allclose(sub["out"][0], full["out"][t], rtol=1e-12, atol=1e-13 * scale)


def test_planted_token_slip_is_caught():
    """A subset evaluated on the wrong rows (off by one) must fail the pin:
    the comparison is sensitive to the slip it guards against."""
    cfg, x, wr, ext, kw = _case(H=64, E=8, k=2, I=32, T=24, shared=True)
    toks = np.array([5, 9, 2])
    full = oracle.moe_layer(x, wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter, **kw)
    wrong = oracle.moe_layer(x[toks + 1], wr, cfg.top_k, ext.__getitem__, cfg.hidden, cfg.inter, **kw)
    assert not np.allclose(wrong["out"], full["out"][toks], rtol=1e-6)
