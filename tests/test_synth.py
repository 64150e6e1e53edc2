"""The seeded input generator: determinism, stream independence, moments, and
its bf16 rounding against torch's float32 -> bfloat16 conversion."""
import numpy as np
import torch

import synth


def test_deterministic_and_streams_differ():
    a = synth.normal_bf16(0, synth.KIND_W13, 0, 5, 1001, 0.02)
    b = synth.normal_bf16(0, synth.KIND_W13, 0, 5, 1001, 0.02)
    c = synth.normal_bf16(0, synth.KIND_W13, 0, 6, 1001, 0.02)
    d = synth.normal_bf16(1, synth.KIND_W13, 0, 5, 1001, 0.02)
    assert np.array_equal(a, b)
    assert not np.array_equal(a, c) and not np.array_equal(a, d)
    # a prefix of a longer draw is the shorter draw (counter-based)
    assert np.array_equal(synth.normal_bf16(0, 1, 2, 3, 10, 1.0), synth.normal_bf16(0, 1, 2, 3, 99, 1.0)[:10])


def test_moments():
    v = synth.normal_f32(0, synth.KIND_X, 0, 0, 1 << 20, 1.0).astype(np.float64)
    assert abs(v.mean()) < 5e-3 and abs(v.std() - 1.0) < 5e-3
    assert abs((v ** 4).mean() - 3.0) < 0.05          # Gaussian kurtosis
    w = synth.normal_f32(0, synth.KIND_WR, 0, 0, 1 << 18, 0.02).astype(np.float64)
    assert abs(w.std() - 0.02) < 5e-4


def test_bf16_rounding_matches_torch():
    # the generator's bf16 equals torch's RNE conversion of the same float32 draw
    key_args = (7, synth.KIND_X, 3, 1)
    f = synth.normal_f32(*key_args, 4097, 1.0)
    b = synth.normal_bf16(*key_args, 4097, 1.0)
    t = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(b, t)


def test_extent_sizes():
    for name, want in [("tiny", 196608), ("qwen3next_4k", 6291456), ("prefill32k_q4_lru64", 1769472)]:
        cfg = synth.config(name)
        assert cfg.extent_bytes == want
    cfg = synth.config("tiny")
    assert synth.expert_extent(cfg, 0, 0).nbytes == cfg.extent_bytes
    cq = synth.config("tiny", wdtype=synth.W_Q4G32)
    assert synth.expert_extent(cq, 0, 0).nbytes == cq.extent_bytes
