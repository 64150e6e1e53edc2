"""Thin ctypes binding of the C ABI in include/msi.h (argument marshalling only).

Every function keeps the C name.  Loading fails loudly when libmsi.so is
missing: there is no fallback implementation of any step.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmsi.so")

MSI_OK = 0
MSI_ERR_INVALID_ARG = 1
MSI_ERR_STALE_GENERATION = 2
MSI_ERR_WRONG_OBJECT = 3
MSI_ERR_SLOT_BUSY = 4
MSI_ERR_NOT_RESIDENT = 5
MSI_ERR_TIMEOUT = 6
MSI_ERR_CUDA = 7
MSI_ERR_SHUT_DOWN = 8
MSI_ERR_UNSUPPORTED = 9
MSI_ERR_WORKSPACE = 10
MSI_ERR_SOURCE = 11
(MSI_FAULT_SHORT_READ, MSI_FAULT_STALE_COMPLETION, MSI_FAULT_WRONG_OBJECT, MSI_FAULT_IO_ERROR,
 MSI_FAULT_STALE_EPOCH, MSI_FAULT_DEVICE_WAIT) = 1, 2, 3, 4, 5, 6
MSI_MAX_WINDOWS = 64

MSI_W_BF16 = 0
MSI_W_Q4G32 = 1
MSI_TRACE_HIT, MSI_TRACE_STAGE, MSI_TRACE_EVICT, MSI_TRACE_PREFETCH = 0, 1, 2, 3
MSI_SLOT_VACANT, MSI_SLOT_LOADING, MSI_SLOT_DEVICE_READY, MSI_SLOT_IN_USE, MSI_SLOT_RECYCLABLE = range(5)
MSI_FWD_RESIDUAL = 1
MSI_FWD_SINGLE_CTA = 2
MSI_FWD_SHARED_UNGATED = 4
MSI_FWD_SPLIT_WAVES = 8
KERNEL_KINDS = ["upload", "router", "scan", "scatter", "setup", "gateup", "down", "shared_gateup",
                "shared_down", "combine", "publish", "ffn"]


class msi_plan_desc(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int), ("n_experts", ctypes.c_int), ("top_k", ctypes.c_int),
        ("hidden", ctypes.c_int), ("inter", ctypes.c_int), ("has_shared", ctypes.c_int),
        ("wdtype", ctypes.c_int), ("n_slots", ctypes.c_int),
        ("slot_pool", ctypes.c_void_p), ("extent_bytes", ctypes.c_uint64),
        ("host_windows", ctypes.c_void_p), ("extent_off", ctypes.c_void_p),
        ("shared_w", ctypes.c_void_p), ("shared_gate_w", ctypes.c_void_p),
        ("wave_capacity", ctypes.c_int), ("wait_timeout_s", ctypes.c_double),
    ]


class msi_route_event(ctypes.Structure):
    _fields_ = [("ids", ctypes.c_void_p), ("weights", ctypes.c_void_p),
                ("counts", ctypes.c_void_p), ("gap", ctypes.c_void_p)]


class msi_trace_rec(ctypes.Structure):
    _fields_ = [("seq", ctypes.c_uint64), ("call", ctypes.c_int32), ("layer", ctypes.c_int32),
                ("expert", ctypes.c_int32), ("slot", ctypes.c_int32),
                ("generation", ctypes.c_uint64), ("kind", ctypes.c_int32), ("wave", ctypes.c_int32)]


class msi_counters(ctypes.Structure):
    _fields_ = [(n, ctypes.c_uint64) for n in
                ("forwards", "streamed_forwards", "stages", "hits", "evicts", "h2d_bytes",
                 "rejections", "prefetches", "prefetch_hits")]


class msi_source_desc(ctypes.Structure):
    _fields_ = [("path", ctypes.c_char_p), ("direct", ctypes.c_int), ("align", ctypes.c_uint32),
                ("n_windows", ctypes.c_int), ("windows", ctypes.c_void_p),
                ("window_bytes", ctypes.c_uint64)]


class msi_source_stats(ctypes.Structure):
    _fields_ = [("reads", ctypes.c_uint64), ("rejected", ctypes.c_uint64),
                ("logical_bytes", ctypes.c_uint64), ("physical_bytes", ctypes.c_uint64),
                ("padding_bytes", ctypes.c_uint64), ("read_seconds", ctypes.c_double),
                ("max_in_flight", ctypes.c_int), ("windows_busy", ctypes.c_int)]


_P = ctypes.c_void_p
_SIGS = {
    "msi_extent_bytes": (ctypes.c_uint64, [ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "msi_plan_create": (ctypes.c_int, [ctypes.POINTER(msi_plan_desc), ctypes.POINTER(_P)]),
    "msi_plan_destroy": (ctypes.c_int, [_P]),
    "msi_workspace_size": (ctypes.c_int, [_P, ctypes.c_int, ctypes.POINTER(ctypes.c_size_t)]),
    "msi_slot_stage": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P,
                                      ctypes.POINTER(ctypes.c_uint64)]),
    "msi_slot_table": (ctypes.c_int, [_P, ctypes.c_int, _P, _P]),
    "msi_slot_state": (ctypes.c_int, [_P, ctypes.c_int, ctypes.POINTER(ctypes.c_int)]),
    "msi_moe_forward": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P, _P, _P,
                                       ctypes.POINTER(msi_route_event), _P, ctypes.c_size_t,
                                       ctypes.c_uint, _P]),
    "msi_moe_forward_streamed": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P,
                                                ctypes.POINTER(msi_route_event), _P, ctypes.c_size_t,
                                                ctypes.c_uint, _P, _P]),
    "msi_moe_forward_streamed_next": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P,
                                                     ctypes.POINTER(msi_route_event), _P,
                                                     ctypes.POINTER(msi_route_event), _P,
                                                     ctypes.c_size_t, ctypes.c_uint, _P, _P]),
    "msi_plan_pin": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "msi_workspace_size_host": (ctypes.c_int, [_P, ctypes.c_int, ctypes.POINTER(ctypes.c_size_t)]),
    "msi_moe_forward_host": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P, _P, _P, _P,
                                            ctypes.POINTER(msi_route_event), _P, ctypes.c_size_t,
                                            ctypes.c_uint, _P]),
    "msi_moe_forward_streamed_host": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P, _P,
                                                     ctypes.POINTER(msi_route_event), _P,
                                                     ctypes.c_size_t, ctypes.c_uint, _P, _P]),
    "msi_moe_forward_static": (ctypes.c_int, [_P, ctypes.c_int, _P, ctypes.c_int, _P, _P, _P, _P,
                                              ctypes.POINTER(msi_route_event), ctypes.c_uint, _P]),
    "msi_forward_status": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_int)]),
    "msi_plan_reset": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_uint64)]),
    "msi_fault_inject": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "msi_plan_set_wait_cycles": (ctypes.c_int, [_P, ctypes.c_int64]),
    "msi_plan_set_bounce": (ctypes.c_int, [_P, _P, ctypes.c_size_t]),
    "msi_moe_forward_streamed_stack": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int,
                                                      _P, _P, _P, _P, _P, ctypes.c_size_t, ctypes.c_uint,
                                                      _P, _P, ctypes.POINTER(ctypes.c_int)]),
    "msi_source_open": (ctypes.c_int, [ctypes.POINTER(msi_source_desc), ctypes.POINTER(_P)]),
    "msi_source_close": (ctypes.c_int, [_P]),
    "msi_source_stats_read": (ctypes.c_int, [_P, ctypes.POINTER(msi_source_stats)]),
    "msi_source_read": (ctypes.c_int, [_P, ctypes.c_uint64, ctypes.c_uint64, ctypes.POINTER(_P),
                                       ctypes.POINTER(ctypes.c_int)]),
    "msi_source_release": (ctypes.c_int, [_P, ctypes.c_int]),
    "msi_plan_set_source": (ctypes.c_int, [_P, _P, _P]),
    "msi_consumer_hold": (ctypes.c_int, [_P, ctypes.c_int]),
    "msi_consumer_release": (ctypes.c_int, [_P, ctypes.c_int]),
    "msi_trace_read": (ctypes.c_int, [_P, ctypes.POINTER(msi_trace_rec), ctypes.c_size_t,
                                      ctypes.POINTER(ctypes.c_size_t)]),
    "msi_trace_clear": (ctypes.c_int, [_P]),
    "msi_get_counters": (ctypes.c_int, [_P, ctypes.POINTER(msi_counters)]),
    "msi_kernel_launches": (ctypes.c_uint64, [_P]),
    "msi_timing_enable": (ctypes.c_int, [_P, ctypes.c_int]),
    "msi_timing_read": (ctypes.c_int, [_P, _P, _P, ctypes.c_int]),
    "msi_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "msi_last_cuda_error": (ctypes.c_char_p, []),
}

_lib = None


def lib():
    """Load libmsi.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError("libmsi.so not built: run python -c 'import __graft_entry__ as g; g.build()'")
        l = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


def __getattr__(name):
    if name in _SIGS:
        return getattr(lib(), name)
    raise AttributeError(name)


class MsiError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = lib().msi_status_string(status).decode()
        if status == MSI_ERR_CUDA:
            msg += " (" + lib().msi_last_cuda_error().decode() + ")"
        super().__init__("%s: %s [%d]" % (where, msg, status))
        self.status = status


def check(status: int, where: str) -> None:
    if status != MSI_OK:
        raise MsiError(status, where)
