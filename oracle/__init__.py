"""fp64 CPU oracle of the slot-addressed MoE layer forward.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference legs may import or run anything in
this package.  The library's compute path never calls it, and this package
shares no code with the CUDA path (no kernels, headers, helpers or tables);
both sides consume the same seeded inputs from ``synth``.

Everything is plain numpy in float64.  Each function cites the passage of the
paper ("Memory-Sovereign Inference: Output-Exact Execution Beyond Full
Residency") it follows; where the paper is silent, the reading taken is named
in the function's docstring.

Parity pins (see ``tests/test_oracle_*.py``): brute force over all experts,
constructed ties, k = E dense softmax, closed-form SwiGLU cases, a library
SwiGLU MLP (torch CPU float64), dense masked evaluation, permutation
bijection, a textbook OrderedDict LRU, hand-worked 3-slot LRU traces in
``tests/golden/``, and exact small-integer dequantisation cases.
"""
from .moe import (  # noqa: F401
    STATUS_OK, STATUS_STALE_GENERATION, STATUS_WRONG_OBJECT, STATUS_NOT_RESIDENT,
    TRACE_HIT, TRACE_STAGE, TRACE_EVICT, TRACE_PREFETCH,
    bf16_to_f64, f16_to_f64, decode_extent, dequant_q4g32,
    router, permutation, swiglu_expert, moe_layer, moe_tokens, dense_masked_moe,
    combine, generation_check, LRUWaveSim, near_tie_tokens,
)
