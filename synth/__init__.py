"""Seeded synthetic inputs for the slot-addressed MoE layer forward.

Shared by the fp64 oracle (``oracle/``) and the CUDA path (tests, bench).  This
module draws random inputs and lays them out as bytes; it holds none of the
method's arithmetic (no routing, no FFN, no combine, no dequantisation).

Workload shapes follow the paper's Qwen3-Next identity (48 layers x 512
experts, Sec. 1 and Sec. 6.1; hidden 2048 and expert intermediate 512 are
consistent with its 1,904,640-byte-per-expert semantic demand) and the five
stated workloads (tiny, 4K resident, 32K LRU64 prefill, 48-layer decode,
32K 4-bit prefill).  Distributions: hidden rows N(0,1) bf16, router weights
N(0,0.02) fp32, expert and shared-expert weights N(0,0.02) bf16, shared gate
vector N(0,0.02) fp32; every tensor has its own counter-based stream keyed by
(seed, kind, layer, index), so any one expert's extent can be regenerated
alone.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, replace

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "_synth.so")
_lock = threading.Lock()
_lib = None

# Stream kinds (top byte of the 64-bit stream tag).
KIND_X = 1          # hidden rows of one call:  (layer, call index)
KIND_WR = 2         # router weight of a layer: (layer, 0)
KIND_W13 = 3        # expert gate+up weight:    (layer, expert)
KIND_W2 = 4         # expert down weight:       (layer, expert)
KIND_SH_W13 = 5     # shared-expert gate+up:    (layer, 0)
KIND_SH_W2 = 6      # shared-expert down:       (layer, 0)
KIND_WSG = 7        # shared-expert gate vector (layer, 0)

W_BF16 = 0
W_Q4G32 = 1


def build(force: bool = False) -> str:
    """Compile gen.c into synth/_synth.so with gcc (OpenMP when available)."""
    src = os.path.join(_HERE, "gen.c")
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(src):
        return _SO
    tmp = _SO + ".%d.tmp" % os.getpid()
    base = ["gcc", "-O2", "-shared", "-fPIC", src, "-o", tmp]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:] + ["-lm"], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base + ["-lm"], check=True, capture_output=True)
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.synth_stream_key.restype = ctypes.c_uint64
            lib.synth_stream_key.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
            lib.synth_normal_bf16.restype = None
            lib.synth_normal_bf16.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_double,
                                              ctypes.c_void_p]
            lib.synth_normal_f32.restype = None
            lib.synth_normal_f32.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_double,
                                             ctypes.c_void_p]
            lib.synth_quantize_q4g32.restype = None
            lib.synth_quantize_q4g32.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64,
                                                 ctypes.c_void_p, ctypes.c_void_p]
            lib.synth_raw_u64.restype = None
            lib.synth_raw_u64.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_void_p]
            _lib = lib
    return _lib


def stream_tag(kind: int, layer: int, index: int) -> int:
    return ((kind & 0xFF) << 56) | ((layer & 0xFFFFFF) << 32) | (index & 0xFFFFFFFF)


def stream_key(seed: int, kind: int, layer: int, index: int) -> int:
    return _load().synth_stream_key(seed, stream_tag(kind, layer, index))


def raw_u64(seed: int, kind: int, layer: int, index: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    _load().synth_raw_u64(stream_key(seed, kind, layer, index), n, out.ctypes.data)
    return out


def normal_bf16(seed, kind, layer, index, n, std, out=None) -> np.ndarray:
    """n N(0, std^2) values rounded to bf16, returned as their uint16 bit patterns."""
    if out is None:
        out = np.empty(n, dtype=np.uint16)
    assert out.dtype == np.uint16 and out.size == n and out.flags.c_contiguous
    _load().synth_normal_bf16(stream_key(seed, kind, layer, index), n, float(std), out.ctypes.data)
    return out


def normal_f32(seed, kind, layer, index, n, std, out=None) -> np.ndarray:
    if out is None:
        out = np.empty(n, dtype=np.float32)
    assert out.dtype == np.float32 and out.size == n and out.flags.c_contiguous
    _load().synth_normal_f32(stream_key(seed, kind, layer, index), n, float(std), out.ctypes.data)
    return out


# ---------------------------------------------------------------------------
# Workload configurations
# ---------------------------------------------------------------------------

@dataclass(frozen=True)
class MoEConfig:
    name: str
    hidden: int          # H
    n_experts: int       # E
    top_k: int           # k
    inter: int           # I (routed and shared expert intermediate size)
    tokens: int          # T per layer call
    n_slots: int         # S
    has_shared: bool
    wdtype: int = W_BF16
    n_layers: int = 1
    lru: bool = True     # False: every expert resident, caller-managed tables
    steps: int = 1       # decode steps (decode workload)
    seed: int = 0

    @property
    def extent_bytes(self) -> int:
        return extent_bytes(self.hidden, self.inter, self.wdtype)


def extent_bytes(H: int, I: int, wdtype: int) -> int:
    if wdtype == W_BF16:
        return 3 * H * I * 2
    # packed nibbles (1.5 H I bytes) + fp16 scales, one per 32 weights (3 H I / 32 * 2 bytes)
    return 3 * H * I // 2 + 3 * H * I // 32 * 2


CONFIGS = {
    "tiny": MoEConfig("tiny", 256, 16, 2, 128, 64, 8, False),
    "qwen3next_4k": MoEConfig("qwen3next_4k", 2048, 512, 10, 512, 4096, 512, True, lru=False),
    "prefill32k_lru64": MoEConfig("prefill32k_lru64", 2048, 512, 10, 512, 32768, 64, True),
    "qwen3next_32k": MoEConfig("qwen3next_32k", 2048, 512, 10, 512, 32768, 512, True, lru=False),
    "decode48": MoEConfig("decode48", 256, 16, 2, 128, 64, 64, False, n_layers=48, steps=64),
    "prefill32k_q4_lru64": MoEConfig("prefill32k_q4_lru64", 2048, 512, 10, 512, 32768, 64, True,
                                     wdtype=W_Q4G32),
}


def config(name: str, **over) -> MoEConfig:
    c = CONFIGS[name]
    return replace(c, **over) if over else c


# ---------------------------------------------------------------------------
# Tensors
# ---------------------------------------------------------------------------

def hidden(cfg: MoEConfig, layer: int = 0, call: int = 0, tokens: int | None = None) -> np.ndarray:
    """Hidden rows x, bf16 bits [T, H], N(0,1)."""
    T = cfg.tokens if tokens is None else tokens
    return normal_bf16(cfg.seed, KIND_X, layer, call, T * cfg.hidden, 1.0).reshape(T, cfg.hidden)


def router_weight(cfg: MoEConfig, layer: int = 0) -> np.ndarray:
    """Router weight Wr, fp32 [E, H], N(0, 0.02)."""
    return normal_f32(cfg.seed, KIND_WR, layer, 0, cfg.n_experts * cfg.hidden, 0.02).reshape(
        cfg.n_experts, cfg.hidden)


def shared_gate_weight(cfg: MoEConfig, layer: int = 0) -> np.ndarray:
    """Shared-expert scalar gate vector w_sg, fp32 [H], N(0, 0.02)."""
    return normal_f32(cfg.seed, KIND_WSG, layer, 0, cfg.hidden, 0.02)


def _bf16_weights(seed, kind13, kind2, layer, index, H, I):
    w13 = normal_bf16(seed, kind13, layer, index, 2 * I * H, 0.02).reshape(2 * I, H)
    w2 = normal_bf16(seed, kind2, layer, index, H * I, 0.02).reshape(H, I)
    return w13, w2


def _bf16_bits_to_f32(u16: np.ndarray) -> np.ndarray:
    return (u16.astype(np.uint32) << 16).view(np.float32)


def quantize_q4g32(w_bf16: np.ndarray):
    """Input preparation for the 4-bit workload: per 32-weight group of one row,
    scale = fp16(absmax / 7), q = clip(rint(w / scale) + 8, 0, 15).
    Returns (packed uint8 [rows, cols/2] with the even column in the low
    nibble, scales as fp16 bits uint16 [rows, cols/32])."""
    w = np.ascontiguousarray(w_bf16, dtype=np.uint16)
    rows, cols = w.shape
    assert cols % 32 == 0
    packed = np.empty((rows, cols // 2), dtype=np.uint8)
    scales = np.empty((rows, cols // 32), dtype=np.uint16)
    _load().synth_quantize_q4g32(w.ctypes.data, rows, cols, packed.ctypes.data, scales.ctypes.data)
    return packed, scales


def expert_extent(cfg: MoEConfig, layer: int, expert: int) -> np.ndarray:
    """Canonical byte extent of routed expert (layer, expert), uint8 [extent_bytes].

    bf16 layout: W13 [2I, H] (rows 0..I-1 gate, I..2I-1 up; each row K-major)
    followed by W2 [H, I] (K-major).
    q4 layout: W13 packed [2I, H/2] | W2 packed [H, I/2] | W13 scales fp16 [2I, H/32] |
    W2 scales fp16 [H, I/32]."""
    return _extent(cfg, KIND_W13, KIND_W2, layer, expert)


def shared_extent(cfg: MoEConfig, layer: int = 0) -> np.ndarray:
    """Shared-expert weights in the bf16 extent layout (always bf16, always resident)."""
    w13, w2 = _bf16_weights(cfg.seed, KIND_SH_W13, KIND_SH_W2, layer, 0, cfg.hidden, cfg.inter)
    return np.concatenate([w13.reshape(-1), w2.reshape(-1)]).view(np.uint8)


def _extent(cfg, k13, k2, layer, index):
    H, I = cfg.hidden, cfg.inter
    w13, w2 = _bf16_weights(cfg.seed, k13, k2, layer, index, H, I)
    if cfg.wdtype == W_BF16:
        return np.concatenate([w13.reshape(-1), w2.reshape(-1)]).view(np.uint8)
    p13, s13 = quantize_q4g32(w13)
    p2, s2 = quantize_q4g32(w2)
    return np.concatenate([p13.reshape(-1), p2.reshape(-1),
                           s13.reshape(-1).view(np.uint8), s2.reshape(-1).view(np.uint8)])


def fill_extents(cfg: MoEConfig, layer: int, out: np.ndarray, experts=None, threads: int = 0):
    """Write the extents of `experts` (default: all) of `layer` into
    out[e * extent_bytes : (e + 1) * extent_bytes] (uint8, e.g. a pinned host buffer)."""
    eb = cfg.extent_bytes
    experts = range(cfg.n_experts) if experts is None else experts
    assert out.dtype == np.uint8 and out.size >= cfg.n_experts * eb

    def one(e):
        out[e * eb:(e + 1) * eb] = expert_extent(cfg, layer, e)

    for e in experts:              # the C generator and quantiser are OpenMP-parallel
        one(e)
    return out
