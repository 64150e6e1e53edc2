"""fp64 CPU oracle: the slot-addressed MoE layer forward, step by step.

TEST INFRASTRUCTURE ONLY (see the package docstring).  Plain numpy, float64,
no blocking, fusion or reordering beyond what each step's definition states.

Steps, in the order the forward takes them:
  1. decode the stored inputs exactly (bf16 / fp16 / 4-bit codes -> float64);
  2. router logits l[t, e] = sum_h x[t, h] Wr[e, h];
  3. top-k: experts ordered by (logit descending, expert id ascending);
  4. route weights: softmax over the selected k logits (equal to the full
     softmax renormalised over the top-k);
  5. near-tie flags: gap between the k-th and (k+1)-th ordered logits;
  6. histogram, exclusive scan and stable permutation ordered by (e, t, j);
  7. per expert e ascending, per routed row: g = Wg x, u = Wu x,
     h = silu(g) * u, y = W2 h  (the complete gate, up and down projections);
  8. combine: out[t] = sum_j w[t, j] y_(t, j) + sigma(x_t . w_sg) * FFN_shared(x_t);
  9. slot residency: the LRU-wave slot simulator and the generation check;
 10. emit the route event, the slot trace and the outputs.

Readings taken where the paper is silent (it describes no kernels; the MoE
computation runs inside its pinned native runtime):
  R1  renormalise over the selected k (route weights sum to 1);
  R2  equal logits: the lower expert id ranks first;
  R4  shared expert gated by the scalar sigmoid(x . w_sg), always resident;
  R7  LRU-wave slot policy made exact (see LRUWaveSim);
  R9  4-bit weights: symmetric offset 8, low nibble = even column, one fp16
      scale per 32 consecutive weights of a row;
  R10 decode stack: x_{l+1} = x_l + moe_l(x_l) (residual passed to combine);
  R13 next-layer prediction, two-bank prefetch and pins made exact (see
      LRUWaveSim).
"""
from __future__ import annotations

import numpy as np

STATUS_OK = "ok"
STATUS_STALE_GENERATION = "stale_generation"
STATUS_WRONG_OBJECT = "wrong_object"
STATUS_NOT_RESIDENT = "not_resident"

TRACE_HIT = "hit"
TRACE_STAGE = "stage"
TRACE_EVICT = "evict"
TRACE_PREFETCH = "prefetch"

_W_BF16 = 0
_W_Q4G32 = 1


# ---------------------------------------------------------------------------
# Step 1: exact decoding of stored values
# ---------------------------------------------------------------------------

def bf16_to_f64(u16) -> np.ndarray:
    """bf16 bit patterns -> float64 (exact: a bf16 is the top half of a float32)."""
    u16 = np.asarray(u16, dtype=np.uint16)
    return (u16.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f16_to_f64(u16) -> np.ndarray:
    """IEEE half bit patterns -> float64 (exact)."""
    return np.asarray(u16, dtype=np.uint16).view(np.float16).astype(np.float64)


def dequant_q4g32(packed: np.ndarray, scales_u16: np.ndarray, rows: int, cols: int) -> np.ndarray:
    """4-bit block-quantised weights -> float64 (reading R9).

    The paper keeps native quantised bytes and never converts the model
    (Sec. "Exactness Is Scoped by Identity and Horizon", last paragraph), but
    prints no format; the one used here: w[n, c] = s[n, c // 32] * (q[n, c] - 8),
    q the 4-bit code of column c, the even column in the low nibble."""
    packed = np.asarray(packed, dtype=np.uint8).reshape(rows, cols // 2)
    q = np.empty((rows, cols), dtype=np.int64)
    q[:, 0::2] = packed & 0x0F
    q[:, 1::2] = packed >> 4
    s = f16_to_f64(scales_u16).reshape(rows, cols // 32)
    return np.repeat(s, 32, axis=1) * (q - 8)


def decode_extent(extent: np.ndarray, H: int, I: int, wdtype: int = _W_BF16):
    """One expert's canonical extent -> (Wg [I, H], Wu [I, H], W2 [H, I]) in float64.

    The Plan maps a logical (layer, expert) object onto one byte extent
    (Sec. "A Shared Cross-Adapter Plan Core"); its three components are the
    gate, up and down projection weights (Sec. "Output-Exact Execution Beyond
    the Full-Residency Envelope")."""
    extent = np.asarray(extent, dtype=np.uint8)
    if wdtype == _W_BF16:
        v = extent.view(np.uint16)
        w13 = bf16_to_f64(v[: 2 * I * H]).reshape(2 * I, H)
        w2 = bf16_to_f64(v[2 * I * H: 3 * I * H]).reshape(H, I)
    else:
        o = 0
        p13 = extent[o: o + I * H]; o += I * H
        p2 = extent[o: o + H * I // 2]; o += H * I // 2
        s13 = extent[o: o + 2 * I * (H // 32) * 2].view(np.uint16); o += 2 * I * (H // 32) * 2
        s2 = extent[o: o + H * (I // 32) * 2].view(np.uint16)
        w13 = dequant_q4g32(p13, s13, 2 * I, H)
        w2 = dequant_q4g32(p2, s2, H, I)
    return w13[:I], w13[I:], w2


# ---------------------------------------------------------------------------
# Steps 2-5: router, top-k, route weights, near-tie flags
# ---------------------------------------------------------------------------

def router(x_bf16, router_w, k: int, w_sg=None):
    """Route event of one layer call: the router's top-k expert ids and weights.

    The paper records the router's top-k output (``ffn_moe_topk``) once per
    layer and graph evaluation, before any Plan action (Sec. "Output-Exact
    Execution Beyond the Full-Residency Envelope"; Sec. "Exactness Is Scoped
    by Identity and Horizon").  Readings R1 and R2 fix the weights and ties.

    Returns a dict: logits [T, E], ids [T, k] (int64, descending logit),
    weights [T, k], gap_k [T] (l of rank k-1 minus l of rank k; +inf when
    k == E), gap_adj [T] (smallest adjacent gap among ranks 0..k), sg [T]
    (sigmoid(x . w_sg), or None)."""
    x = bf16_to_f64(x_bf16)
    W = np.asarray(router_w, dtype=np.float64)
    T, E = x.shape[0], W.shape[0]
    assert 1 <= k <= E
    logits = x @ W.T                                     # step 2
    order = np.argsort(-logits, axis=1, kind="stable")   # step 3: ties keep ascending id
    ids = order[:, :k]
    kk = min(k + 1, E)
    top = np.take_along_axis(logits, order[:, :kk], axis=1)
    ex = np.exp(top[:, :k] - top[:, :1])                 # step 4
    weights = ex / ex.sum(axis=1, keepdims=True)
    if k < E:                                            # step 5
        gap_k = top[:, k - 1] - top[:, k]
    else:
        gap_k = np.full(T, np.inf)
    gap_adj = np.diff(-top, axis=1).min(axis=1) if kk > 1 else np.full(T, np.inf)
    sg = None
    if w_sg is not None:
        sg = 1.0 / (1.0 + np.exp(-(x @ np.asarray(w_sg, dtype=np.float64))))
    return {"logits": logits, "ids": ids, "weights": weights, "gap_k": gap_k,
            "gap_adj": gap_adj, "sg": sg}


def near_tie_tokens(gap, threshold: float = 1e-4) -> np.ndarray:
    """Tokens whose compared router gap is below the threshold (excluded from
    the bit-exact route comparison and counted)."""
    return np.asarray(gap) < threshold


# ---------------------------------------------------------------------------
# Step 6: histogram, scan, stable permutation
# ---------------------------------------------------------------------------

def permutation(ids, E: int):
    """Group the T*k routed rows by expert.

    counts[e] = #{(t, j): ids[t, j] == e}; offsets = exclusive scan of counts;
    row r in [offsets[e], offsets[e+1]) holds the pairs of expert e in (t, j)
    order; perm[r] = t*k + j and inv[t*k + j] = r."""
    ids = np.asarray(ids)
    flat = ids.reshape(-1)
    counts = np.bincount(flat, minlength=E).astype(np.int64)
    offsets = np.zeros(E + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(counts)
    perm = np.argsort(flat, kind="stable").astype(np.int64)
    inv = np.empty_like(perm)
    inv[perm] = np.arange(flat.size, dtype=np.int64)
    return counts, offsets, perm, inv


# ---------------------------------------------------------------------------
# Step 7: expert SwiGLU FFN
# ---------------------------------------------------------------------------

def swiglu_expert(x_rows: np.ndarray, Wg: np.ndarray, Wu: np.ndarray, W2: np.ndarray) -> np.ndarray:
    """y = W2 (silu(Wg x) * (Wu x)) for each row x (float64).

    Each selected expert runs its complete gate, up and down projections
    (Sec. "Output-Exact Execution Beyond the Full-Residency Envelope")."""
    g = x_rows @ Wg.T
    u = x_rows @ Wu.T
    with np.errstate(over="ignore"):
        h = g / (1.0 + np.exp(-g)) * u
    return h @ W2.T


# ---------------------------------------------------------------------------
# Step 8: combine
# ---------------------------------------------------------------------------

def combine(weights, inv, Y, sg=None, ys=None, residual=None):
    """out[t] = sum_j w[t, j] * Y[inv[t*k + j]] (+ sg[t] * ys[t]) (+ residual[t])."""
    T, k = weights.shape
    out = np.zeros((T, Y.shape[1]), dtype=np.float64)
    for j in range(k):
        out += weights[:, j:j + 1] * Y[inv.reshape(T, k)[:, j]]
    if sg is not None:
        out += sg[:, None] * ys
    if residual is not None:
        out += residual
    return out


# ---------------------------------------------------------------------------
# Composition of steps 1-8 (small and medium cases)
# ---------------------------------------------------------------------------

def moe_layer(x_bf16, router_w, k, extent_of, H, I, wdtype=_W_BF16,
              shared_extent=None, w_sg=None, residual=False, shared_gated=True):
    """The MoE layer forward of one call.

    extent_of(e) returns expert e's canonical extent (uint8).  Returns the
    router dict plus counts, offsets, perm, inv, Y (expert outputs in permuted
    row order) and out [T, H] (float64).  shared_gated=False takes the other
    reading of the shared expert (R4): its output is added with gate 1."""
    r = router(x_bf16, router_w, k,
               w_sg if shared_extent is not None and shared_gated else None)
    E = np.asarray(router_w).shape[0]
    counts, offsets, perm, inv = permutation(r["ids"], E)
    x = bf16_to_f64(x_bf16)
    T = x.shape[0]
    Y = np.zeros((T * k, H), dtype=np.float64)
    for e in range(E):                                   # step 7, experts ascending
        lo, hi = offsets[e], offsets[e + 1]
        if hi == lo:
            continue
        Wg, Wu, W2 = decode_extent(extent_of(e), H, I, wdtype)
        rows = x[perm[lo:hi] // k]
        Y[lo:hi] = swiglu_expert(rows, Wg, Wu, W2)
    ys = None
    if shared_extent is not None:
        Sg, Su, S2 = decode_extent(shared_extent, H, I, _W_BF16)
        ys = swiglu_expert(x, Sg, Su, S2)
    sg = r["sg"] if shared_gated or ys is None else np.ones(T, dtype=np.float64)
    out = combine(r["weights"], inv, Y, sg, ys, x if residual else None)
    r.update(counts=counts, offsets=offsets, perm=perm, inv=inv, Y=Y, ys=ys, out=out)
    return r


def moe_tokens(x_bf16, router_w, k, extent_of, H, I, tokens, wdtype=_W_BF16,
               shared_extent=None, w_sg=None, residual=False):
    """Outputs of a subset of tokens, each computed on its own (routing is per
    token, and each routed row's expert output depends only on that row).
    Used for sampled checks at full workload sizes."""
    tokens = np.asarray(tokens)
    xs = np.asarray(x_bf16)[tokens]
    return moe_layer(xs, router_w, k, extent_of, H, I, wdtype, shared_extent, w_sg, residual)


def dense_masked_moe(x_bf16, router_w, k, extent_of, H, I, wdtype=_W_BF16):
    """Brute-force evaluation: every expert on every token, masked by the top-k
    weights.  Independent of the permutation and combine steps (a pin)."""
    r = router(x_bf16, router_w, k)
    x = bf16_to_f64(x_bf16)
    T, E = x.shape[0], np.asarray(router_w).shape[0]
    mask_w = np.zeros((T, E))
    for j in range(k):
        mask_w[np.arange(T), r["ids"][:, j]] = r["weights"][:, j]
    out = np.zeros((T, H))
    for e in range(E):
        Wg, Wu, W2 = decode_extent(extent_of(e), H, I, wdtype)
        out += mask_w[:, e:e + 1] * swiglu_expert(x, Wg, Wu, W2)
    return out


# ---------------------------------------------------------------------------
# Step 9: slot residency (LRU waves) and the generation check
# ---------------------------------------------------------------------------

def generation_check(layer, needed, slot_table, expected, ledger_obj, ledger_gen):
    """Fail-closed check of a layer's bundle before any consumer reads it.

    A published version must denote the requested object and version, and a
    mismatch is rejected before the data becomes visible (Sec. "Lifetime Is
    Part of Correctness"; Sec. "Stable Slots and Bundle Publication": all
    components are checked before one publication).  For each needed expert,
    ascending: no slot -> not_resident; slot holding another object ->
    wrong_object; generation differing from the expected one ->
    stale_generation.  The lowest failing expert decides.

    Returns (status, expert) with expert = -1 when the bundle passes."""
    for e in sorted(int(v) for v in needed):
        s = int(slot_table[e])
        if s < 0:
            return STATUS_NOT_RESIDENT, e
        if ledger_obj[s] != (layer, e):
            return STATUS_WRONG_OBJECT, e
        if int(ledger_gen[s]) != int(expected[e]):
            return STATUS_STALE_GENERATION, e
    return STATUS_OK, -1


class LRUWaveSim:
    """Explicit slot-pool simulator (reading R7 of the replacement policy).

    The paper fixes only a per-layer LRU with 64 slots (Sec. "Evaluation",
    "Cache and storage state"), that replacement policy is separate from the
    lifecycle (Sec. "A Shared Cross-Adapter Plan Core"), that a slot is not
    reused before its last consumer finishes and that every stage produces a
    new generation (Sec. "Separate Window and GPU-Slot Lifecycles").  Made
    exact here:

      * one global tick, +1 per expert consumption;
      * a call's needed experts (ascending) are split into hits (resident)
        and misses, processed as hits then misses;
      * they are consumed in waves of `wave_capacity` experts (S/2: one half
        of the pool is computed on while the other is staged);
      * the slots of the wave being staged and of the previous wave (being
        computed) are pinned;
      * victim: the lowest-index vacant unpinned slot, else the unpinned slot
        with the smallest last-use tick (ties -> lowest index);
      * each stage bumps the slot's generation by one (a vacant slot has
        generation 0);
      * trace records (call, layer, expert, slot, generation, kind, wave) for
        each hit, each eviction (with the evicted object and its generation)
        and each stage (with the new generation).

    Prediction, two-bank prefetch and pinning (reading R13).  The paper runs a
    protected LRU64 together with a two-bank next-layer prefetch (Sec.
    "Evaluation", "Cache and storage state"; Sec. "Qwen-Specific Natural
    Utility") and states that demand loading, LRU, prediction and pinning pick
    different future objects through one lifecycle (Sec. "A Shared
    Cross-Adapter Plan Core").  It specifies neither the predictor nor the
    banks; made exact here:

      * a call may carry a prediction for another layer: the number of token
        choices predicted per expert of that layer (the forward predicts layer
        l + 1 by routing the call's input through layer l + 1's router);
      * after the call's last wave, one prefetch bundle: the predicted experts
        that are not resident, ranked by predicted count descending (ties ->
        lower id), the first `wave_capacity` of them, assigned in ascending
        expert order;
      * two banks: the slots of the call's last wave (computed on), of the
        prefetch bundle being assigned, and of every predicted object already
        resident are pinned; victims by the same rule; the bundle ends early
        when no unpinned slot is left;
      * a prefetched object's last-use tick is the current tick (prefetching
        is not consumption: the tick does not advance);
      * trace: eviction records and "prefetch" records, wave index = the
        number of waves of the call;
      * caller pins: a pinned object is never a victim; at most
        S - 2 * wave_capacity objects may be pinned (S - wave_capacity
        without previous-wave pinning), so every wave and bundle finds
        victims;
      * counters: objects prefetched, and hits on a prefetched object before
        its first consumption.
    """

    def __init__(self, n_slots: int, wave_capacity: int | None = None, pin_previous: bool = True):
        assert n_slots >= 1
        self.S = n_slots
        self.C = wave_capacity if wave_capacity is not None else max(1, n_slots // 2)
        self.pin_previous = pin_previous
        assert 1 <= self.C and (self.C * (2 if pin_previous else 1) <= n_slots)
        self.obj = [None] * n_slots
        self.gen = [0] * n_slots
        self.last_use = [-1] * n_slots
        self.tick = 0
        self.calls = 0
        self.trace = []
        self.where = {}
        self.pins = set()
        self.prefetched = set()   # slots holding a prefetched, unconsumed object
        self.prefetches = 0
        self.prefetch_hits = 0

    def pin(self, layer: int, e: int):
        """Pin object (layer, e): once resident it is never a victim."""
        limit = self.S - self.C * (2 if self.pin_previous else 1)
        if (layer, e) not in self.pins and len(self.pins) + 1 > limit:
            raise ValueError("too many pinned objects")
        self.pins.add((layer, e))

    def unpin(self, layer: int, e: int):
        self.pins.discard((layer, e))

    def _victim(self, pinned):
        cands = [s for s in range(self.S) if s not in pinned and self.obj[s] not in self.pins]
        if not cands:
            return None
        vacant = [s for s in cands if self.obj[s] is None]
        if vacant:
            return vacant[0]
        return min(cands, key=lambda s: (self.last_use[s], s))

    def _load(self, call, layer, e, s, kind, w):
        if self.obj[s] is not None:
            ol, oe = self.obj[s]
            self.trace.append((call, ol, oe, s, self.gen[s], TRACE_EVICT, w))
            del self.where[self.obj[s]]
        self.prefetched.discard(s)
        self.gen[s] += 1
        self.obj[s] = (layer, e)
        self.where[(layer, e)] = s
        self.trace.append((call, layer, e, s, self.gen[s], kind, w))

    def call(self, layer: int, needed, predict=None) -> list:
        """Process one layer call; returns the waves as lists of (expert, slot).

        predict: None, or (next_layer, counts) with counts[e] the predicted
        number of token choices of expert e in next_layer."""
        call = self.calls
        self.calls += 1
        needed = sorted(set(int(e) for e in needed))
        hits = [e for e in needed if (layer, e) in self.where]
        misses = [e for e in needed if (layer, e) not in self.where]
        order = hits + misses
        waves = [order[i:i + self.C] for i in range(0, len(order), self.C)]
        prev = set()
        out = []
        for w, wave in enumerate(waves):
            cur = []
            for e in wave:
                if (layer, e) in self.where:
                    s = self.where[(layer, e)]
                    self.trace.append((call, layer, e, s, self.gen[s], TRACE_HIT, w))
                    if s in self.prefetched:
                        self.prefetch_hits += 1
                        self.prefetched.discard(s)
                else:
                    s = self._victim((prev if self.pin_previous else set()) | set(cur))
                    self._load(call, layer, e, s, TRACE_STAGE, w)
                cur.append(s)
            for s in cur:                                   # the wave is consumed
                self.tick += 1
                self.last_use[s] = self.tick
            out.append(list(zip(wave, cur)))
            prev = set(cur)
        if predict is not None:                             # the prefetch bank
            nl, counts = predict
            cand = [e for e in range(len(counts)) if counts[e] > 0 and (nl, e) not in self.where]
            cand.sort(key=lambda e: (-int(counts[e]), e))
            bank = sorted(cand[:self.C])
            kept = {self.where[(nl, e)] for e in range(len(counts))
                    if counts[e] > 0 and (nl, e) in self.where}
            cur = []
            for e in bank:
                s = self._victim((prev if self.pin_previous else set()) | kept | set(cur))
                if s is None:
                    break
                self._load(call, nl, e, s, TRACE_PREFETCH, len(waves))
                self.last_use[s] = self.tick
                self.prefetched.add(s)
                cur.append(s)
            self.prefetches += len(cur)
        return out

    def slot_table(self, layer: int, E: int):
        """(slot_of_expert [E] with -1 when absent, generation_of_expert [E])."""
        st = np.full(E, -1, dtype=np.int64)
        gt = np.zeros(E, dtype=np.int64)
        for (l, e), s in self.where.items():
            if l == layer:
                st[e] = s
                gt[e] = self.gen[s]
        return st, gt
