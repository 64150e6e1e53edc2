"""Shared setup of the GPU tests: seeded inputs from ``synth`` placed in pinned
host windows and device buffers, a Plan over them, and comparison helpers
against the fp64 oracle."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import synth
from paper_2608_23805_gb300 import api
from paper_2608_23805_gb300 import native as N

# Tolerances for bf16 weights (outputs); route events are compared exactly.
NORM_REL_TOL = 5e-3
MAX_ABS_TOL = 2e-2
GAP_THRESHOLD = 1e-4


def bf16_tensor(bits: np.ndarray, device="cuda") -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device) if device else t


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().view(torch.int16).numpy().view(np.uint16)


class Case:
    """Inputs of one workload (all layers), host windows filled, plan created."""

    def __init__(self, cfg: synth.MoEConfig, n_slots=None, wave_capacity=0, layers=None,
                 wait_timeout_s=0.0, early_staging=False):
        self.cfg = cfg
        L = cfg.n_layers if layers is None else layers
        self.L = L
        E, H, I = cfg.n_experts, cfg.hidden, cfg.inter
        eb = cfg.extent_bytes
        self.windows = torch.empty(L * E * eb, dtype=torch.uint8, pin_memory=True)
        wnp = self.windows.numpy()
        for l in range(L):
            synth.fill_extents(cfg, l, wnp[l * E * eb:(l + 1) * E * eb])
        self.router_np = [synth.router_weight(cfg, l) for l in range(L)]
        self.router = [torch.from_numpy(w).cuda() for w in self.router_np]
        self.shared_np = None
        shared_w = gate_w = None
        if cfg.has_shared:
            self.shared_np = [synth.shared_extent(cfg, l) for l in range(L)]
            self.gate_np = [synth.shared_gate_weight(cfg, l) for l in range(L)]
            shared_w = torch.from_numpy(np.concatenate(self.shared_np)).cuda()
            gate_w = torch.from_numpy(np.stack(self.gate_np)).cuda()
        self.plan = api.Plan(n_layers=L, n_experts=E, top_k=cfg.top_k, hidden=H, inter=I,
                             n_slots=cfg.n_slots if n_slots is None else n_slots,
                             host_windows=self.windows, has_shared=cfg.has_shared,
                             shared_w=shared_w, shared_gate_w=gate_w, wdtype=cfg.wdtype,
                             wave_capacity=wave_capacity, wait_timeout_s=wait_timeout_s,
                             early_staging=early_staging)

    def extent(self, layer, e):
        eb = self.cfg.extent_bytes
        o = (layer * self.cfg.n_experts + e) * eb
        return self.windows.numpy()[o:o + eb]

    def stage_all(self, layer=0, stream=None):
        """Resident mode: expert e of `layer` into slot e."""
        for e in range(self.cfg.n_experts):
            self.plan.stage(e, layer, e, stream)
        torch.cuda.synchronize()
        return self.plan.slot_table(layer)

    def oracle_layer(self, x_bits, layer=0, tokens=None, residual=False):
        cfg = self.cfg
        kw = {}
        if cfg.has_shared:
            kw = dict(shared_extent=self.shared_np[layer], w_sg=self.gate_np[layer])
        f = (lambda e: self.extent(layer, e))
        if tokens is None:
            return oracle.moe_layer(x_bits, self.router_np[layer], cfg.top_k, f, cfg.hidden,
                                    cfg.inter, cfg.wdtype, residual=residual, **kw)
        return oracle.moe_tokens(x_bits, self.router_np[layer], cfg.top_k, f, cfg.hidden, cfg.inter,
                                 tokens, cfg.wdtype, residual=residual, **kw)

    def close(self):
        self.plan.close()


def compare_routes(ids_gpu: np.ndarray, w_gpu: np.ndarray, ref: dict):
    """Route events: ids compared as sets per token except near-ties (k-th vs
    (k+1)-th gap < 1e-4), ordered ids except tokens with any adjacent gap among
    the top k+1 below 1e-4; weights within 1e-5.  Returns (n_near_tie, n_near_tie_adj)."""
    ids_ref = ref["ids"]
    T = ids_ref.shape[0]
    near = oracle.near_tie_tokens(ref["gap_k"], GAP_THRESHOLD)
    near_adj = oracle.near_tie_tokens(ref["gap_adj"], GAP_THRESHOLD)
    for t in range(T):
        if not near[t]:
            assert set(ids_gpu[t].tolist()) == set(ids_ref[t].tolist()), f"token {t} ids differ"
        if not near_adj[t]:
            assert ids_gpu[t].tolist() == ids_ref[t].tolist(), f"token {t} id order differs"
            np.testing.assert_allclose(w_gpu[t], ref["weights"][t], rtol=0, atol=1e-5)
    assert np.allclose(w_gpu.sum(axis=1), 1.0, atol=1e-5)
    for t in range(T):
        assert len(set(ids_gpu[t].tolist())) == ids_gpu.shape[1]
    return int(near.sum()), int(near_adj.sum())


def compare_out(out_gpu_bits: np.ndarray, out_ref: np.ndarray, mask=None):
    got = oracle.bf16_to_f64(out_gpu_bits)
    if mask is not None:
        got, out_ref = got[mask], out_ref[mask]
    err = got - out_ref
    rel = np.linalg.norm(err) / max(np.linalg.norm(out_ref), 1e-30)
    mx = np.abs(err).max() if err.size else 0.0
    assert rel <= NORM_REL_TOL, f"norm-relative error {rel:.3e}"
    assert mx <= MAX_ABS_TOL, f"max-abs error {mx:.3e}"
    return rel, mx
