"""Slot-addressed MoE layer forward for GB300 (sm_103a).

The compute path is the CUDA library libmsi.so (C ABI in include/msi.h);
``native`` binds it with ctypes under the C names and ``api.Plan`` wraps it
for PyTorch callers.  Importing this package loads nothing; the first use of
the binding loads libmsi.so and raises if it has not been built.
"""
__all__ = ["native", "api", "build"]
