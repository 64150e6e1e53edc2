"""Pins of the oracle's slot simulator and generation check: hand-worked
traces (tests/golden, including prediction, two-bank prefetch and pins), a
textbook OrderedDict LRU in the special case that reduces to it, and the
reuse / generation / prefetch / pin invariants."""
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
            kv = dict(t.split("=") for t in tok[2:])
            cur = {"name": tok[1], "slots": int(kv["slots"]),
                   "wave": int(kv["wave"]) if "wave" in kv else None,
                   "pins": [], "calls": [], "trace": []}
        elif tok[0] == "pin":
            kv = dict(t.split("=") for t in tok[1:])
            cur["pins"].append((int(kv["layer"]), int(kv["expert"])))
        elif tok[0] == "call":
            kv = dict(t.split("=") for t in tok[1:])
            needed = [int(v) for v in kv["needed"].split(",")]
            predict = None
            if "predict" in kv:
                nl, items = kv["predict"].split(":")
                counts = np.zeros(16, dtype=np.int64)
                for it in items.split(","):
                    e, n = it.split("*")
                    counts[int(e)] = int(n)
                predict = (int(nl), counts)
            cur["calls"].append((int(kv["layer"]), needed, predict))
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
    sim = oracle.LRUWaveSim(case["slots"], case["wave"])
    for layer, e in case["pins"]:
        sim.pin(layer, e)
    for layer, needed, predict in case["calls"]:
        sim.call(layer, needed, predict)
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


def _decode_like(rng, sim, L, E, steps, k_max, exact):
    """Calls over layers 0..L-1 per step; each call may predict the next
    layer (the exact next needed set, or a random one)."""
    seq = [(l, sorted(set(rng.integers(0, E, size=rng.integers(1, k_max + 1)).tolist())))
           for _ in range(steps) for l in range(L)]
    misses_after_exact = 0
    for i, (layer, needed) in enumerate(seq):
        predict = None
        if i + 1 < len(seq) and seq[i + 1][0] == layer + 1:
            nl, nxt = seq[i + 1]
            counts = np.zeros(E, dtype=np.int64)
            pool = nxt if exact else rng.integers(0, E, size=len(nxt)).tolist()
            for e in pool:
                counts[e] += 1
            predict = (nl, counts)
        n0 = len(sim.trace)
        sim.call(layer, needed, predict)
        if i > 0 and seq[i - 1][0] == layer - 1 and exact:
            misses_after_exact += sum(1 for r in sim.trace[n0:]
                                      if r[1] == layer and r[5] == oracle.TRACE_STAGE)
    return seq, misses_after_exact


@pytest.mark.parametrize("seed", range(4))
def test_exact_prediction_leaves_no_miss(seed):
    """With the next call's needed set predicted exactly and at most one wave
    of it, every need of that call is a hit: the bundle always finds victims
    (S >= 2C) and never evicts a predicted object already resident."""
    rng = np.random.default_rng(seed)
    sim = oracle.LRUWaveSim(8)
    seq, misses = _decode_like(rng, sim, L=6, E=12, steps=5, k_max=4, exact=True)
    assert misses == 0
    n_pref_hits = sum(1 for r in sim.trace if r[5] == oracle.TRACE_PREFETCH)
    assert sim.prefetches == n_pref_hits == sim.prefetch_hits > 0


@pytest.mark.parametrize("seed", range(4))
def test_prefetch_and_pin_invariants(seed):
    """Random predictions and pins: no pinned object is ever evicted; no
    prefetch evicts a slot of the call's last wave; prefetching never advances
    the tick (tick = number of consumptions); a prediction of zero counts
    leaves the trace of a call without prediction."""
    rng = np.random.default_rng(100 + seed)
    S, E, L = 8, 10, 4
    sim = oracle.LRUWaveSim(S, 2)
    pins = {(int(rng.integers(0, L)), int(rng.integers(0, E))) for _ in range(3)}
    for p in pins:
        sim.pin(*p)
    with pytest.raises(ValueError):
        for e in range(E):
            sim.pin(L, e)  # beyond S - 2C
    for e in range(E):
        sim.unpin(L, e)
    consumed = 0
    for step in range(6):
        for layer in range(L):
            needed = sorted(set(rng.integers(0, E, size=rng.integers(1, 7)).tolist()))
            counts = np.zeros(E, dtype=np.int64)
            for e in rng.integers(0, E, size=rng.integers(0, 6)):
                counts[e] += 1
            n0 = len(sim.trace)
            waves = sim.call(layer, needed, ((layer + 1) % L, counts))
            consumed += len(needed)
            assert sim.tick == consumed
            last = {s for _, s in waves[-1]}
            recs = sim.trace[n0:]
            for r in recs:
                if r[5] == oracle.TRACE_EVICT:
                    assert (r[1], r[2]) not in pins
                if r[6] == len(waves):
                    assert r[3] not in last
    a, b = oracle.LRUWaveSim(S), oracle.LRUWaveSim(S)
    for layer, needed in [(0, [1, 2, 3]), (1, [2, 5]), (0, [1, 7, 8, 9]), (1, [0])]:
        a.call(layer, needed)
        b.call(layer, needed, (layer + 1, np.zeros(E, dtype=np.int64)))
    assert a.trace == b.trace
