"""Pins of the oracle's slot simulator and generation check: hand-worked
traces (tests/golden), a textbook OrderedDict LRU in the special case that
reduces to it, and the reuse / generation invariants."""
import os
from collections import OrderedDict

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "lru_hand_traces.txt")


def _cases():
    cases, cur = [], None
    for line in open(GOLDEN):
        line = line.split("#")[0].strip()
        if not line:
            continue
        tok = line.split()
        if tok[0] == "case":
            cur = {"name": tok[1], "slots": int(tok[2].split("=")[1]), "calls": [], "trace": []}
        elif tok[0] == "call":
            layer = int(tok[1].split("=")[1])
            needed = [int(v) for v in tok[2].split("=")[1].split(",")]
            cur["calls"].append((layer, needed))
        elif tok[0] == "trace":
            pass
        elif tok[0] == "end":
            cases.append(cur)
        else:
            c, l, e, s, g, kind, w = tok
            cur["trace"].append((int(c), int(l), int(e), int(s), int(g), kind, int(w)))
    return cases


@pytest.mark.parametrize("case", _cases(), ids=lambda c: c["name"])
def test_hand_worked_traces(case):
    sim = oracle.LRUWaveSim(case["slots"])
    for layer, needed in case["calls"]:
        sim.call(layer, needed)
    assert sim.trace == case["trace"]


def _textbook_lru(cap, seq):
    """OrderedDict LRU over an access sequence; returns (key, hit, evicted key)."""
    cache, free, where, out = OrderedDict(), list(range(cap)), {}, []
    for key in seq:
        if key in cache:
            cache.move_to_end(key)
            out.append((key, True, None))
            continue
        ev = None
        if free:
            s = free.pop(0)
        else:
            ev, s = cache.popitem(last=False)
        cache[key] = s
        out.append((key, False, ev))
    return out


@pytest.mark.parametrize("seed", range(6))
def test_wave_of_one_without_pinning_is_textbook_lru(seed):
    """Waves of one expert with no pinned previous wave: every access is a
    textbook LRU access, in the per-call order hits-then-misses."""
    rng = np.random.default_rng(seed)
    S, E, L = 5, 12, 3
    sim = oracle.LRUWaveSim(S, wave_capacity=1, pin_previous=False)
    seq = []
    for call in range(40):
        layer = int(rng.integers(L))
        needed = sorted(set(rng.choice(E, size=int(rng.integers(1, 6)), replace=True).tolist()))
        resident = {k for k, _ in sim.where.items()}
        hits = [e for e in needed if (layer, e) in resident]
        misses = [e for e in needed if (layer, e) not in resident]
        seq += [(layer, e) for e in hits + misses]
        sim.call(layer, needed)
    want = _textbook_lru(S, seq)
    got, pending = [], None
    for c, l, e, s, g, kind, w in sim.trace:
        if kind == "evict":
            pending = (l, e)
        elif kind == "hit":
            got.append(((l, e), True, None))
        else:
            got.append(((l, e), False, pending))
            pending = None
    assert got == want


@pytest.mark.parametrize("S", [2, 4, 8, 64])
def test_no_reuse_before_last_consumer_and_generations(S):
    rng = np.random.default_rng(S)
    E = 3 * S + 5
    sim = oracle.LRUWaveSim(S)
    gens = [0] * S
    for call in range(30):
        needed = rng.choice(E, size=int(rng.integers(1, 2 * S + 3)), replace=False)
        waves = sim.call(call % 2, needed)
        recs = [r for r in sim.trace if r[0] == call]
        for w, wave in enumerate(waves):
            assert len(wave) <= sim.C
            busy = {s for _, s in waves[w - 1]} if w > 0 else set()
            for r in recs:
                if r[5] == "stage" and r[6] == w:
                    assert r[3] not in busy                 # previous wave still consuming
            slots = [s for _, s in wave]
            assert len(set(slots)) == len(slots)
        for r in recs:
            if r[5] == "stage":
                gens[r[3]] += 1
                assert r[4] == gens[r[3]]                   # +1 per stage, per slot
        # every needed expert is consumed exactly once per call
        assert sorted(e for wave in waves for e, _ in wave) == sorted(set(int(v) for v in needed))


def test_generation_check_fail_closed():
    obj = [(0, 5), (0, 2), None, (1, 2)]
    gen = [3, 1, 0, 7]
    table = np.full(8, -1)
    table[5], table[2] = 0, 1
    exp = np.zeros(8, dtype=np.int64)
    exp[5], exp[2] = 3, 1
    assert oracle.generation_check(0, [2, 5], table, exp, obj, gen) == ("ok", -1)
    exp2 = exp.copy(); exp2[5] = 2
    assert oracle.generation_check(0, [2, 5], table, exp2, obj, gen) == ("stale_generation", 5)
    t2 = table.copy(); t2[2] = 3                        # slot 3 holds (1, 2), not (0, 2)
    assert oracle.generation_check(0, [2, 5], t2, exp, obj, gen) == ("wrong_object", 2)
    assert oracle.generation_check(0, [2, 5, 6], table, exp, obj, gen) == ("not_resident", 6)
    # the lowest failing expert decides
    assert oracle.generation_check(0, [2, 5, 6], t2, exp2, obj, gen) == ("wrong_object", 2)
