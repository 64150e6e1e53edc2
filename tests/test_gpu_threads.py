"""Two plans driven from two host threads at once, each on its own streams
(the library's process-wide state -- launch attributes set once per kernel,
cached occupancy, the tensor-map encoder -- is shared between them).  Every
output must equal, bit for bit, what the same calls give when run one plan
after the other."""
import threading

import numpy as np
import pytest
import torch

import synth
from gpu_case import Case, bf16_bits, bf16_tensor
from paper_2608_23805_gb300 import native as N

pytestmark = pytest.mark.gpu


def _runner(case, calls, streamed, out):
    cs, ss = torch.cuda.Stream(), torch.cuda.Stream()
    table = gens = None
    if not streamed:
        table, gens = case.plan.slot_table(0)
    res = []
    with torch.cuda.stream(cs):
        for x_bits in calls:
            x = bf16_tensor(x_bits)
            if streamed:
                o, _ = case.plan.forward_streamed(0, x, case.router[0], stream=cs, stage_stream=ss)
            else:
                o, _ = case.plan.forward(0, x, case.router[0], table, gens, stream=cs)
            res.append(o)
        cs.synchronize()
    out.extend(bf16_bits(o) for o in res)


def test_two_plans_from_two_threads():
    ca = synth.config("tiny")
    cb = synth.config("qwen3next_4k", n_experts=64, n_slots=64, tokens=512)
    calls_a = [synth.hidden(ca, 0, 200 + i) for i in range(6)]
    calls_b = [synth.hidden(cb, 0, 210 + i) for i in range(4)]
    # sequential reference
    a1, b1 = Case(ca), Case(cb)
    b1.stage_all()
    ref_a, ref_b = [], []
    _runner(a1, calls_a, True, ref_a)
    _runner(b1, calls_b, False, ref_b)
    # concurrent
    a2, b2 = Case(ca), Case(cb)
    b2.stage_all()
    got_a, got_b = [], []
    ta = threading.Thread(target=_runner, args=(a2, calls_a, True, got_a))
    tb = threading.Thread(target=_runner, args=(b2, calls_b, False, got_b))
    ta.start()
    tb.start()
    ta.join()
    tb.join()
    assert a2.plan.status() == N.MSI_OK and b2.plan.status() == N.MSI_OK
    assert len(got_a) == len(calls_a) and len(got_b) == len(calls_b)
    for r, g in zip(ref_a + ref_b, got_a + got_b):
        assert np.array_equal(r, g)
    assert a1.plan.trace() == a2.plan.trace()
    for c in (a1, b1, a2, b2):
        c.close()
