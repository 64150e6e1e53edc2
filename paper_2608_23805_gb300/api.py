"""Convenience wrapper over the C ABI for PyTorch callers.

PyTorch supplies device memory, pinned host memory and streams; every step of
the MoE layer forward runs in libmsi.so's CUDA kernels.  This module only
marshals tensors into pointers and checks status codes.
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import native as N


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _flags(residual: bool, single_cta: bool, shared_gate: bool = True, split_waves: bool = False) -> int:
    return ((N.MSI_FWD_RESIDUAL if residual else 0) | (N.MSI_FWD_SINGLE_CTA if single_cta else 0)
            | (0 if shared_gate else N.MSI_FWD_SHARED_UNGATED)
            | (N.MSI_FWD_SPLIT_WAVES if split_waves else 0))


def _stream(s) -> int | None:
    s = torch.cuda.current_stream() if s is None else s
    return s.cuda_stream


class RouteEvent:
    """Device buffers of one layer call's route event."""

    def __init__(self, T: int, k: int, E: int, device="cuda"):
        self.ids = torch.empty((T, k), dtype=torch.int32, device=device)
        self.weights = torch.empty((T, k), dtype=torch.float32, device=device)
        self.counts = torch.empty((E,), dtype=torch.int32, device=device)
        self.gap = torch.empty((T,), dtype=torch.float32, device=device)
        self.c = N.msi_route_event(_ptr(self.ids) if T else None, _ptr(self.weights) if T else None,
                                   _ptr(self.counts), _ptr(self.gap) if T else None)


class Plan:
    """A Plan over one slot pool (see include/msi.h, msi_plan_desc)."""

    def __init__(self, *, n_layers, n_experts, top_k, hidden, inter, n_slots, host_windows,
                 has_shared=False, shared_w=None, shared_gate_w=None, wdtype=N.MSI_W_BF16,
                 slot_pool=None, extent_off=None, wave_capacity=0, wait_timeout_s=0.0,
                 early_staging=False):
        """early_staging: give streamed calls an early-staging buffer of one
        wave of extents (msi_plan_set_bounce)."""
        lib = N.lib()
        self.E, self.k, self.H, self.I = n_experts, top_k, hidden, inter
        self.n_layers, self.S = n_layers, n_slots
        self.extent_bytes = int(lib.msi_extent_bytes(hidden, inter, wdtype))
        if self.extent_bytes == 0:
            raise ValueError("bad shape")
        if slot_pool is None:
            slot_pool = torch.empty(n_slots * self.extent_bytes, dtype=torch.uint8, device="cuda")
        self._keep = [host_windows, slot_pool, shared_w, shared_gate_w]
        self.slot_pool = slot_pool
        self._off = None
        if extent_off is not None:
            self._off = np.ascontiguousarray(extent_off, dtype=np.uint64)
        d = N.msi_plan_desc()
        d.n_layers, d.n_experts, d.top_k = n_layers, n_experts, top_k
        d.hidden, d.inter, d.has_shared, d.wdtype, d.n_slots = hidden, inter, int(has_shared), wdtype, n_slots
        d.slot_pool = slot_pool.data_ptr()
        d.extent_bytes = self.extent_bytes
        d.host_windows = host_windows.data_ptr()
        d.extent_off = self._off.ctypes.data if self._off is not None else None
        d.shared_w = _ptr(shared_w)
        d.shared_gate_w = _ptr(shared_gate_w)
        d.wave_capacity = wave_capacity
        d.wait_timeout_s = wait_timeout_s
        h = ctypes.c_void_p()
        N.check(lib.msi_plan_create(ctypes.byref(d), ctypes.byref(h)), "msi_plan_create")
        self.h = h
        self._ws = {}
        self._ws_bytes = {}
        self.bounce = None
        if early_staging:
            C = wave_capacity if wave_capacity > 0 else n_slots // 2
            self.bounce = torch.empty(C * self.extent_bytes, dtype=torch.uint8, device="cuda")
            N.check(lib.msi_plan_set_bounce(self.h, self.bounce.data_ptr(), self.bounce.numel()),
                    "msi_plan_set_bounce")

    # -- residency ---------------------------------------------------------
    def stage(self, slot: int, layer: int, expert: int, stream=None) -> int:
        g = ctypes.c_uint64()
        N.check(N.lib().msi_slot_stage(self.h, slot, layer, expert, _stream(stream), ctypes.byref(g)),
                "msi_slot_stage")
        return g.value

    def slot_table(self, layer: int):
        st = np.empty(self.E, dtype=np.int32)
        gt = np.empty(self.E, dtype=np.uint64)
        N.check(N.lib().msi_slot_table(self.h, layer, st.ctypes.data, gt.ctypes.data), "msi_slot_table")
        return st, gt

    def slot_state(self, slot: int) -> int:
        s = ctypes.c_int()
        N.check(N.lib().msi_slot_state(self.h, slot, ctypes.byref(s)), "msi_slot_state")
        return s.value

    def reset(self) -> int:
        e = ctypes.c_uint64()
        N.check(N.lib().msi_plan_reset(self.h, ctypes.byref(e)), "msi_plan_reset")
        return e.value

    def inject(self, kind: int, layer: int, expert: int):
        N.check(N.lib().msi_fault_inject(self.h, kind, layer, expert), "msi_fault_inject")

    def set_wait_cycles(self, cycles: int):
        """Limit of every bounded device wait (clock64 cycles); <= 0: default."""
        N.check(N.lib().msi_plan_set_wait_cycles(self.h, int(cycles)), "msi_plan_set_wait_cycles")

    def set_source(self, src: "Source | None", file_off=None):
        """Stage missing extents from `src` (file offsets [L*E]); None detaches."""
        if src is None:
            N.check(N.lib().msi_plan_set_source(self.h, None, None), "msi_plan_set_source")
            self._src = None
            return
        off = np.ascontiguousarray(file_off, dtype=np.uint64)
        N.check(N.lib().msi_plan_set_source(self.h, src.h, off.ctypes.data), "msi_plan_set_source")
        self._src = src  # keep the source alive while attached

    def hold(self, slot: int):
        N.check(N.lib().msi_consumer_hold(self.h, slot), "msi_consumer_hold")

    def release(self, slot: int):
        N.check(N.lib().msi_consumer_release(self.h, slot), "msi_consumer_release")

    # -- forward -------------------------------------------------------------
    def workspace(self, T: int) -> torch.Tensor:
        need = self._ws_bytes.get(T)
        if need is None:  # a pure function of the plan's shape and T
            n = ctypes.c_size_t()
            N.check(N.lib().msi_workspace_size(self.h, T, ctypes.byref(n)), "msi_workspace_size")
            need = self._ws_bytes[T] = n.value
        ws = self._ws.get("buf")
        if ws is None or ws.numel() < need:
            ws = torch.empty(max(need, 256), dtype=torch.uint8, device="cuda")
            self._ws["buf"] = ws
        return ws

    def forward(self, layer, x, router_w, slot_table, expected, out=None, ev=None, residual=False,
                stream=None, check=True, single_cta=False, shared_gate=True, split_waves=False):
        T = x.shape[0]
        out = torch.empty_like(x) if out is None else out
        ev = RouteEvent(T, self.k, self.E) if ev is None else ev
        ws = self.workspace(T)
        st = np.ascontiguousarray(slot_table, dtype=np.int32)
        ex = np.ascontiguousarray(expected, dtype=np.uint64)
        rc = N.lib().msi_moe_forward(self.h, layer, _ptr(x), T, _ptr(router_w), st.ctypes.data,
                                     ex.ctypes.data, _ptr(out), ctypes.byref(ev.c), _ptr(ws),
                                     ws.numel(), _flags(residual, single_cta, shared_gate, split_waves),
                                     _stream(stream))
        if check:
            N.check(rc, "msi_moe_forward")
            return out, ev
        return rc, out, ev

    def forward_streamed(self, layer, x, router_w, out=None, ev=None, residual=False, stream=None,
                         stage_stream=None, check=True, single_cta=False, next_router_w=None,
                         next_ev=None, split_waves=False):
        """Streamed layer forward.  With next_router_w (layer + 1's router), the
        rows are also routed through it and layer + 1's predicted objects are
        prefetched after the last wave; the predicted route event is written to
        next_ev (allocated when None) and returned as ev.next."""
        T = x.shape[0]
        out = torch.empty_like(x) if out is None else out
        ev = RouteEvent(T, self.k, self.E) if ev is None else ev
        ws = self.workspace(T)
        if next_router_w is None:
            rc = N.lib().msi_moe_forward_streamed(self.h, layer, _ptr(x), T, _ptr(router_w), _ptr(out),
                                                  ctypes.byref(ev.c), _ptr(ws), ws.numel(),
                                                  _flags(residual, single_cta, True, split_waves),
                                                  _stream(stream), _stream(stage_stream))
            where = "msi_moe_forward_streamed"
        else:
            next_ev = RouteEvent(T, self.k, self.E) if next_ev is None else next_ev
            ev.next = next_ev
            rc = N.lib().msi_moe_forward_streamed_next(
                self.h, layer, _ptr(x), T, _ptr(router_w), _ptr(out), ctypes.byref(ev.c),
                _ptr(next_router_w), ctypes.byref(next_ev.c), _ptr(ws), ws.numel(),
                _flags(residual, single_cta, True, split_waves), _stream(stream), _stream(stage_stream))
            where = "msi_moe_forward_streamed_next"
        if check:
            N.check(rc, where)
            return out, ev
        return rc, out, ev

    def forward_streamed_stack(self, layer0, x, routers, out_a, out_b, evs, residual=False,
                               stream=None, stage_stream=None, check=True):
        """Streamed forwards of layers layer0 .. layer0 + len(routers) - 1 in
        one call (msi_moe_forward_streamed_stack): layer i reads the previous
        output (x for i = 0) and writes out_a for even i, out_b for odd i.
        evs: one RouteEvent per layer.  Returns the tensor holding the last
        layer's output."""
        n = len(routers)
        assert len(evs) == n
        T = x.shape[0]
        ws = self.workspace(T)
        rw = (ctypes.c_void_p * max(n, 1))(*[r.data_ptr() for r in routers])
        ea = (N.msi_route_event * max(n, 1))(*[e.c for e in evs])
        done = ctypes.c_int()
        rc = N.lib().msi_moe_forward_streamed_stack(
            self.h, layer0, n, _ptr(x), T, ctypes.cast(rw, ctypes.c_void_p), _ptr(out_a), _ptr(out_b),
            ctypes.cast(ea, ctypes.c_void_p), _ptr(ws), ws.numel(), _flags(residual, False),
            _stream(stream), _stream(stage_stream), ctypes.byref(done))
        last = out_a if n % 2 == 1 else out_b
        if check:
            N.check(rc, "msi_moe_forward_streamed_stack")
            return last
        return rc, done.value, last

    def workspace_host(self, T: int) -> torch.Tensor:
        n = ctypes.c_size_t()
        N.check(N.lib().msi_workspace_size_host(self.h, T, ctypes.byref(n)), "msi_workspace_size_host")
        ws = self._ws.get("host")
        if ws is None or ws.numel() < n.value:
            ws = torch.empty(max(n.value, 256), dtype=torch.uint8, device="cuda")
            self._ws["host"] = ws
        return ws

    def forward_host(self, layer, x_host, router_w, slot_table=None, expected=None, out_host=None,
                     ids_host=None, ev=None, residual=False, stream=None, stage_stream=None,
                     check=True, single_cta=False):
        """End-to-end call from and to host memory: x_host and out_host are CPU
        bf16 tensors [T, H] (pinned for the full link rate), ids_host an
        optional CPU int32 [T, k].  With a slot table the resident forward runs,
        without one the streamed forward.  The results are in out_host once the
        compute stream has passed this call."""
        T = x_host.shape[0]
        assert x_host.device.type == "cpu" and x_host.is_contiguous()
        out_host = torch.empty_like(x_host) if out_host is None else out_host
        ev = RouteEvent(T, self.k, self.E) if ev is None else ev
        ws = self.workspace_host(T)
        fl = _flags(residual, single_cta)
        if slot_table is not None:
            st = np.ascontiguousarray(slot_table, dtype=np.int32)
            ex = np.ascontiguousarray(expected, dtype=np.uint64)
            rc = N.lib().msi_moe_forward_host(self.h, layer, x_host.data_ptr(), T, _ptr(router_w),
                                              st.ctypes.data, ex.ctypes.data, out_host.data_ptr(),
                                              _ptr(ids_host), ctypes.byref(ev.c), _ptr(ws), ws.numel(),
                                              fl, _stream(stream))
            where = "msi_moe_forward_host"
        else:
            rc = N.lib().msi_moe_forward_streamed_host(self.h, layer, x_host.data_ptr(), T,
                                                       _ptr(router_w), out_host.data_ptr(),
                                                       _ptr(ids_host), ctypes.byref(ev.c), _ptr(ws),
                                                       ws.numel(), fl, _stream(stream),
                                                       _stream(stage_stream))
            where = "msi_moe_forward_streamed_host"
        if check:
            N.check(rc, where)
            return out_host, ev
        return rc, out_host, ev

    def pin(self, layer: int, expert: int, pinned: bool = True):
        N.check(N.lib().msi_plan_pin(self.h, layer, expert, int(pinned)), "msi_plan_pin")

    def status(self) -> int:
        s = ctypes.c_int()
        N.check(N.lib().msi_forward_status(self.h, ctypes.byref(s)), "msi_forward_status")
        return s.value

    # -- telemetry -------------------------------------------------------------
    def trace(self, clear: bool = False):
        """Slot trace as (call, layer, expert, slot, generation, kind, wave) tuples."""
        cap = 1 << 20
        buf = (N.msi_trace_rec * cap)()
        n = ctypes.c_size_t()
        N.check(N.lib().msi_trace_read(self.h, buf, cap, ctypes.byref(n)), "msi_trace_read")
        kinds = {N.MSI_TRACE_HIT: "hit", N.MSI_TRACE_STAGE: "stage", N.MSI_TRACE_EVICT: "evict",
                 N.MSI_TRACE_PREFETCH: "prefetch"}
        out = [(r.call, r.layer, r.expert, r.slot, int(r.generation), kinds[r.kind], r.wave)
               for r in buf[:n.value]]
        if clear:
            N.check(N.lib().msi_trace_clear(self.h), "msi_trace_clear")
        return out

    def counters(self) -> dict:
        c = N.msi_counters()
        N.check(N.lib().msi_get_counters(self.h, ctypes.byref(c)), "msi_get_counters")
        return {f: getattr(c, f) for f, _ in c._fields_}

    def timing(self, on: bool = True):
        N.check(N.lib().msi_timing_enable(self.h, int(on)), "msi_timing_enable")

    def timing_read(self, reset: bool = True) -> dict:
        """{kind: (milliseconds summed, launches)} of the timed launches."""
        ms = np.zeros(len(N.KERNEL_KINDS), dtype=np.float64)
        n = np.zeros(len(N.KERNEL_KINDS), dtype=np.uint64)
        N.check(N.lib().msi_timing_read(self.h, ms.ctypes.data, n.ctypes.data, int(reset)),
                "msi_timing_read")
        return {k: (float(ms[i]), int(n[i])) for i, k in enumerate(N.KERNEL_KINDS)}

    def launches(self) -> int:
        return int(N.lib().msi_kernel_launches(self.h))

    def close(self):
        if getattr(self, "h", None) is not None and self.h.value:
            N.check(N.lib().msi_plan_destroy(self.h), "msi_plan_destroy")
            self.h = None

    def __del__(self):
        try:
            if getattr(self, "h", None) is not None and self.h.value:
                N.lib().msi_plan_destroy(self.h)
        except Exception:
            pass


class Source:
    """Bounded source service: extents read from `path` into `n_windows`
    fixed, aligned host windows (O_DIRECT covering reads when direct=True).
    The windows are pinned (page-locked) host memory when CUDA is available,
    so that the H2D copies out of them are asynchronous; otherwise aligned
    ordinary host memory (synchronous reads only)."""

    def __init__(self, path: str, window_bytes: int, n_windows: int = 8, direct: bool = True,
                 align: int = 4096):
        wb = (int(window_bytes) + align - 1) // align * align
        nbytes = wb * n_windows + align
        if torch.cuda.is_available():
            self._buf = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
            base = self._buf.data_ptr()
        else:
            self._buf = np.empty(nbytes, dtype=np.uint8)
            base = self._buf.ctypes.data
        self._off = (-base) % align
        self.window_bytes = wb
        self.n_windows = n_windows
        self.direct = direct
        self._path = path.encode()
        d = N.msi_source_desc(self._path, 1 if direct else 0, align, n_windows,
                              base + self._off, wb)
        self.h = ctypes.c_void_p()
        N.check(N.lib().msi_source_open(ctypes.byref(d), ctypes.byref(self.h)), "msi_source_open")

    def read(self, file_off: int, nbytes: int):
        """Synchronous read: (window, bytes of the extent as a numpy copy)."""
        data = ctypes.c_void_p()
        w = ctypes.c_int()
        N.check(N.lib().msi_source_read(self.h, file_off, nbytes, ctypes.byref(data), ctypes.byref(w)),
                "msi_source_read")
        out = np.ctypeslib.as_array((ctypes.c_uint8 * nbytes).from_address(data.value)).copy()
        return w.value, out

    def release(self, window: int):
        N.check(N.lib().msi_source_release(self.h, window), "msi_source_release")

    def stats(self) -> dict:
        st = N.msi_source_stats()
        N.check(N.lib().msi_source_stats_read(self.h, ctypes.byref(st)), "msi_source_stats_read")
        return {n: getattr(st, n) for n, _ in N.msi_source_stats._fields_}

    def close(self):
        if getattr(self, "h", None) is not None and self.h.value:
            N.check(N.lib().msi_source_close(self.h), "msi_source_close")
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
