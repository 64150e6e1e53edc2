/*
 * msi.h -- C ABI of the slot-addressed MoE layer forward for GB300 (sm_103a).
 *
 * The library runs the data-parallel hot path of storage-backed MoE inference
 * from "Memory-Sovereign Inference: Output-Exact Execution Beyond Full
 * Residency": a Plan maps each logical (layer, expert) object to a byte extent
 * in pinned host windows and to a reusable GPU slot with a stable address and
 * a generation (Sec. "A Shared Cross-Adapter Plan Core"); experts are staged
 * window -> slot asynchronously and published per generation (Sec. "Stable
 * Slots and Bundle Publication"; Sec. "Implementation", "Scheduling and
 * copies"); the layer forward routes tokens (fp32 router, softmax, top-k),
 * groups them per expert, runs each selected expert's complete gate, up and
 * down projections from its slot, and combines the weighted results
 * (Sec. "Output-Exact Execution Beyond the Full-Residency Envelope").  A
 * generation mismatch fails closed: nothing stale becomes visible
 * (Sec. "Lifetime Is Part of Correctness").
 *
 * Conventions
 *  - Every call returns msi_status; nothing is thrown across the ABI.
 *  - The caller owns every device and pinned host buffer passed in (slot pool,
 *    host windows, hidden rows, outputs, route-event buffers, workspace).  A
 *    plan owns only host metadata, CUDA events and a few device words per slot
 *    (the published generation and object of each slot).
 *  - Streams are cudaStream_t values passed as msi_stream; 0 is the legacy
 *    default stream.  Calls on one plan must come from one host thread at a
 *    time; forwards of one plan are meant to be issued on one compute stream.
 *  - Layouts: hidden rows bf16 row-major [T, H]; router weight fp32 [E, H];
 *    a bf16 expert extent is W13 [2I, H] (rows 0..I-1 gate, I..2I-1 up, each
 *    row K-contiguous) followed by W2 [H, I] (K-contiguous); a 4-bit extent is
 *    W13 codes [2I, H/2] | W2 codes [H, I/2] | W13 fp16 scales [2I, H/32] |
 *    W2 fp16 scales [H, I/32], code q -> scale * (q - 8), even column in the
 *    low nibble.
 *  - Shape limits of the library: E <= 512, 1 <= k <= min(E, 32), H a multiple
 *    of 256, I a multiple of 128, T >= 0.  Other shapes return
 *    MSI_ERR_UNSUPPORTED.
 */
#ifndef MSI_H_
#define MSI_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* msi_stream; /* a cudaStream_t */

typedef enum {
  MSI_OK = 0,
  MSI_ERR_INVALID_ARG = 1,       /* bad pointer, index, size or shape */
  MSI_ERR_STALE_GENERATION = 2,  /* expected generation differs from the published one */
  MSI_ERR_WRONG_OBJECT = 3,      /* the slot holds a different (layer, expert) object */
  MSI_ERR_SLOT_BUSY = 4,         /* a live consumer still holds the slot */
  MSI_ERR_NOT_RESIDENT = 5,      /* a needed expert has no slot */
  MSI_ERR_TIMEOUT = 6,           /* a bounded host or device wait ran out */
  MSI_ERR_CUDA = 7,              /* a CUDA runtime call failed (see msi_last_cuda_error) */
  MSI_ERR_SHUT_DOWN = 8,         /* the plan is being destroyed */
  MSI_ERR_UNSUPPORTED = 9,       /* shape outside the library's limits */
  MSI_ERR_WORKSPACE = 10,        /* workspace missing, misaligned or too small */
  MSI_ERR_SOURCE = 11            /* a source extent failed (short read / I/O error); its
                                    bundle was not staged and nothing was published */
} msi_status;

enum { MSI_W_BF16 = 0, MSI_W_Q4G32 = 1 };

enum { MSI_TRACE_HIT = 0, MSI_TRACE_STAGE = 1, MSI_TRACE_EVICT = 2,
       MSI_TRACE_PREFETCH = 3 /* a stage of a predicted object (next-layer prefetch) */ };

/* GPU slot lifecycle states (Sec. "Separate Window and GPU-Slot Lifecycles"). */
enum {
  MSI_SLOT_VACANT = 0,        /* holds no object */
  MSI_SLOT_LOADING = 1,       /* copy enqueued, readiness event not yet reached */
  MSI_SLOT_DEVICE_READY = 2,  /* published, never consumed */
  MSI_SLOT_IN_USE = 3,        /* a consumer (forward or caller ticket) is live */
  MSI_SLOT_RECYCLABLE = 4     /* published and every consumer finished */
};

/* Host-side fault hooks (msi_fault_inject), one-shot per (layer, expert). */
enum {
  MSI_FAULT_SHORT_READ = 1,        /* the object's next source delivery is short: staging it
                                      (alone or inside a bundle) fails with MSI_ERR_SOURCE */
  MSI_FAULT_STALE_COMPLETION = 2,  /* the object's next publication carries the previous
                                      generation (a late stale completion) */
  MSI_FAULT_WRONG_OBJECT = 3,      /* the object's next publication names another object */
  MSI_FAULT_IO_ERROR = 4,          /* with a source attached: the object's next read completes
                                      with an I/O error (EIO); its bundle is not published */
  MSI_FAULT_STALE_EPOCH = 5,       /* with a source attached: the object's next read carries the
                                      previous request epoch (a completion from before a reset);
                                      it is rejected at completion, its bundle not published */
  MSI_FAULT_DEVICE_WAIT = 6        /* the next forward on `layer` (expert: any valid index,
                                      ignored) runs its tensor-core kernels (router, expert
                                      GEMMs) with one extra device wait on a barrier nothing
                                      arrives at: it runs out after the plan's wait limit, the
                                      kernel drains its copies and MMAs, frees TMEM and reports
                                      MSI_ERR_TIMEOUT; the combine writes no `out` row */
};

/* Forward flags. */
enum {
  MSI_FWD_RESIDUAL = 1,   /* out = x + moe(x), rounded once to bf16 (decode stacks) */
  MSI_FWD_SINGLE_CTA = 2, /* run every expert GEMM on single-CTA 128-row tiles; by default
                             bf16 launches whose groups average >= 1,024 rows use CTA-pair
                             256-row tiles (both accumulate in fp32 over the same K order
                             and meet the same output tolerance) */
  MSI_FWD_SHARED_UNGATED = 4, /* the shared expert's output is added with gate 1 instead of
                                 sigmoid(x . w_sg) (the other reading of its gate; no effect
                                 without a shared expert) */
  MSI_FWD_SPLIT_WAVES = 8     /* streamed calls: launch each bf16 wave's gate-up and down GEMMs
                                 as two kernels; by default both run in one launch, the down
                                 tiles after the gate-up tiles they read, on 256-row CTA-pair
                                 tiles once the wave's groups average >= 1,024 rows (else, or
                                 with MSI_FWD_SINGLE_CTA, 128-row tiles: then bit-identical
                                 to the split launches with MSI_FWD_SINGLE_CTA) */
};

/* Plan description (copied by msi_plan_create; pointers must outlive the plan). */
typedef struct {
  int n_layers;                 /* layers whose experts the plan manages (>= 1) */
  int n_experts;                /* E routed experts per layer */
  int top_k;                    /* k */
  int hidden;                   /* H */
  int inter;                    /* I, routed and shared expert intermediate size */
  int has_shared;               /* 1: one always-resident shared expert per layer */
  int wdtype;                   /* MSI_W_BF16 or MSI_W_Q4G32 (routed experts) */
  int n_slots;                  /* S >= 2 GPU slots */
  void* slot_pool;              /* device, S * extent_bytes, 128-byte aligned, caller-owned */
  uint64_t extent_bytes;        /* must equal msi_extent_bytes(hidden, inter, wdtype) */
  const void* host_windows;     /* pinned host memory holding the canonical extents */
  const uint64_t* extent_off;   /* host [n_layers * E] byte offset of object (l, e) in
                                   host_windows; NULL: (l * E + e) * extent_bytes */
  const void* shared_w;         /* device, n_layers bf16 extents of the shared experts,
                                   128-byte aligned (NULL when has_shared == 0) */
  const float* shared_gate_w;   /* device fp32 [n_layers, H] shared-expert gate vectors */
  int wave_capacity;            /* experts per LRU wave; 0: n_slots / 2 */
  double wait_timeout_s;        /* bound on host waits for held consumers; 0: 1.0 s */
} msi_plan_desc;

typedef struct msi_plan msi_plan; /* opaque, owned by the library */

/* Route event of one layer call (device buffers, caller-owned).  This is the
 * router's top-k output recorded per layer and graph evaluation (Sec.
 * "Output-Exact Execution Beyond the Full-Residency Envelope"). */
typedef struct {
  int32_t* ids;      /* [T, k] expert ids, descending logit, ties -> lower id */
  float* weights;    /* [T, k] softmax over the selected k logits (sum to 1) */
  int32_t* counts;   /* [E] routed rows per expert */
  float* gap;        /* [T] logit of rank k-1 minus logit of rank k (+inf if k == E); may be NULL */
} msi_route_event;

/* One slot-trace record (telemetry of cache events and generations, Sec.
 * "Implementation", "Telemetry").  call and wave are -1 for msi_slot_stage. */
typedef struct {
  uint64_t seq;
  int32_t call, layer, expert, slot;
  uint64_t generation;  /* new generation for STAGE; held generation for HIT and EVICT */
  int32_t kind;         /* MSI_TRACE_* */
  int32_t wave;
} msi_trace_rec;

/* Plan telemetry counters. */
typedef struct {
  uint64_t forwards, streamed_forwards, stages, hits, evicts;
  uint64_t h2d_bytes;            /* extent bytes copied window -> slot */
  uint64_t rejections;           /* host prechecks and device checks that failed closed */
  uint64_t prefetches;           /* objects staged by next-layer prediction (also in stages) */
  uint64_t prefetch_hits;        /* hits on a prefetched object before its first consumption */
} msi_counters;

/* Bytes of one expert extent for the given shape and weight type (0 on bad input). */
uint64_t msi_extent_bytes(int hidden, int inter, int wdtype);

/* Create a plan: validates the description, copies the manifest, creates the
 * per-slot generation words (all slots Vacant, generation 0) and the TMA
 * descriptors over the slot pool.  Needs a current CUDA device; the plan
 * belongs to it.  Every call that enqueues work (staging, forwards, reset)
 * must be made with that device current, else it returns
 * MSI_ERR_INVALID_ARG with nothing enqueued; msi_plan_destroy makes it
 * current itself while it releases the plan. */
msi_status msi_plan_create(const msi_plan_desc* desc, msi_plan** out);

/* Destroy a plan.  Fails with MSI_ERR_SLOT_BUSY (and destroys nothing) while a
 * caller-held consumer ticket is live; otherwise drains all staging and
 * forwards issued through the plan, then frees it (reset/shutdown drain,
 * Sec. "Separate Window and GPU-Slot Lifecycles"). */
msi_status msi_plan_destroy(msi_plan* plan);

/* Device workspace bytes msi_moe_forward / msi_moe_forward_streamed need for T
 * tokens.  The workspace is caller-owned, 256-byte aligned, and must not be
 * shared by forwards that may run concurrently. */
msi_status msi_workspace_size(const msi_plan* plan, int T, size_t* bytes);

/* Stage object (layer, expert) into `slot`, asynchronously on `stage`:
 * waits (on the GPU) for the slot's last consumer, invalidates the slot's
 * published generation, copies the extent from the host window, publishes the
 * new generation (old + 1) and records the slot's readiness event.  Returns
 * MSI_ERR_TIMEOUT with nothing enqueued if a caller-held consumer ticket on the
 * slot is not released within wait_timeout_s (no reuse before the last
 * consumer, Sec. "Separate Window and GPU-Slot Lifecycles"). */
msi_status msi_slot_stage(msi_plan* plan, int slot, int layer, int expert, msi_stream stage,
                          uint64_t* new_generation);

/* The plan's ledger for one layer: slot_of_expert[e] (-1 if not resident) and
 * the generation published there (0 if not resident).  Host arrays [E]. */
msi_status msi_slot_table(const msi_plan* plan, int layer, int32_t* slot_of_expert,
                          uint64_t* gen_of_expert);

/* Current lifecycle state of one slot (MSI_SLOT_*), derived from the ledger,
 * its readiness and consumer events and caller-held tickets. */
msi_status msi_slot_state(const msi_plan* plan, int slot, int* state);

/* Layer forward over caller-managed residency (every needed expert already
 * staged).  slot_table and expected_generations are host arrays [E]
 * (slot -1: not resident).  Host precheck: if some e with slot_table[e] >= 0
 * names a slot whose ledger object is not (layer, e) or whose generation is
 * not expected_generations[e], nothing is enqueued and WRONG_OBJECT /
 * STALE_GENERATION is returned for the lowest such e.  Device re-check: the
 * forward re-reads the published generation of every needed expert's slot;
 * on mismatch (or a needed expert without slot) no expert output and no `out`
 * row is written, and msi_forward_status reports the failure.  Route events
 * are always written (routing precedes the Plan).  Asynchronous on `compute`.
 * hidden: device bf16 [T, H]; router_w: device fp32 [E, H]; out: device bf16
 * [T, H]. */
msi_status msi_moe_forward(msi_plan* plan, int layer, const void* hidden, int T,
                           const float* router_w, const int32_t* slot_table,
                           const uint64_t* expected_generations, void* out,
                           const msi_route_event* ev, void* workspace, size_t workspace_bytes,
                           unsigned flags, msi_stream compute);

/* msi_moe_forward for callers that cannot allocate device memory (code inside
 * another runtime's memory budget without an allocator handle, plugins whose
 * host framework owns every allocation, loops that forbid allocation after
 * start-up).  The paper has no counterpart: this is a library convenience.
 * Same arguments and behaviour as msi_moe_forward minus the workspace, which
 * is a fixed 32 MiB device array inside the library, reserved on every GPU
 * that loads the library until exit.  Returns MSI_ERR_WORKSPACE, enqueueing
 * nothing, when msi_workspace_size(plan, T) exceeds 32 MiB (above 478 tokens
 * at the Qwen3-Next layer shape: 512 experts, top-10, hidden 2048,
 * intermediate 512, shared expert).  The first call on a device resolves the
 * array's address (make it before any stream capture); after a device reset
 * the process must restart before calling this again.  All calls share the
 * array: calls whose kernels overlap on the GPU race, so serialise them.  The
 * call itself allocates nothing. */
msi_status msi_moe_forward_static(msi_plan* plan, int layer, const void* hidden, int T,
                                  const float* router_w, const int32_t* slot_table,
                                  const uint64_t* expected_generations, void* out,
                                  const msi_route_event* ev, unsigned flags, msi_stream compute);

/* Layer forward with plan-managed residency (LRU waves).  Routes on `compute`,
 * reads the per-expert counts back to the host (one synchronisation), then
 * processes the needed experts as hits then misses in waves of wave_capacity:
 * misses are staged on `stage` into victims chosen by least-recent use (slots
 * of the current and previous wave pinned), each wave published by one event
 * and consumed by the grouped expert FFN on `compute` while the next wave is
 * staged.  Every hit, stage and eviction is appended to the slot trace.
 * Returns after enqueueing the last wave and the combine. */
msi_status msi_moe_forward_streamed(msi_plan* plan, int layer, const void* hidden, int T,
                                    const float* router_w, void* out, const msi_route_event* ev,
                                    void* workspace, size_t workspace_bytes, unsigned flags,
                                    msi_stream compute, msi_stream stage);

/* msi_moe_forward_streamed over a stack of layers layer0 .. layer0 + n - 1
 * in one call (a decode step): layer i (from 0) reads the previous layer's
 * output (`hidden` for i = 0) and writes out_a when i is even, out_b when i
 * is odd, so the stack's output is in out_a when n is odd and in out_b when
 * it is even; both [T, H] bf16, device, 16-byte aligned, distinct from
 * `hidden` and from each other.  router_w: n device pointers (host array),
 * the layers' routers; evs: n route events (host array of structs with
 * device buffers).  flags apply to every layer (a stack normally passes
 * MSI_FWD_RESIDUAL).  Each layer is exactly one msi_moe_forward_streamed
 * call, made by the library without returning to the caller in between.
 * Stops at the first layer that fails and returns its status; *done (may be
 * NULL) receives the number of layers completed. */
msi_status msi_moe_forward_streamed_stack(msi_plan* plan, int layer0, int n, const void* hidden, int T,
                                          const float* const* router_w, void* out_a, void* out_b,
                                          const msi_route_event* evs, void* workspace,
                                          size_t workspace_bytes, unsigned flags, msi_stream compute,
                                          msi_stream stage, int* done);

/* msi_moe_forward_streamed plus next-layer prediction and a two-bank prefetch
 * (the paper's protected LRU with two-bank next-layer prefetch, Sec.
 * "Evaluation", "Cache and storage state"; prediction and pinning share the
 * slot lifecycle, Sec. "A Shared Cross-Adapter Plan Core").  The call's rows
 * are also routed through layer + 1's router (`next_router_w`, fp32 [E, H],
 * device) on a plan-owned side stream while the call's own waves run; the
 * predicted route event (top-k ids, weights, gap and per-expert counts of
 * layer + 1 for these rows; same layouts as `ev`, caller-owned device
 * buffers) is written to `next_ev`.  After the call's last wave is enqueued,
 * the predicted objects of layer + 1 that are not resident, ranked by
 * predicted count (descending; ties: lower expert id) and capped at
 * wave_capacity, are staged on `stage` as one bundle in ascending expert
 * order: victims by the wave rule, with the slots of the last wave, of the
 * bundle itself and of every predicted object already resident pinned; the
 * bundle ends early when no slot is left.  A prefetched object's last-use
 * tick is the current tick; its stage is traced as MSI_TRACE_PREFETCH with
 * wave = the call's number of waves.  The prediction changes residency only:
 * the call's outputs and route event are those of msi_moe_forward_streamed.
 * A rejected source read in the bundle unwinds that bundle (its slots become
 * Vacant) and the call still returns MSI_OK: prediction is advisory.
 * Errors: as msi_moe_forward_streamed, plus MSI_ERR_INVALID_ARG when
 * layer + 1 >= n_layers, next_router_w or next_ev is NULL, or (T > 0)
 * next_ev's ids / weights / gap are NULL. */
msi_status msi_moe_forward_streamed_next(msi_plan* plan, int layer, const void* hidden, int T,
                                         const float* router_w, void* out,
                                         const msi_route_event* ev, const float* next_router_w,
                                         const msi_route_event* next_ev, void* workspace,
                                         size_t workspace_bytes, unsigned flags,
                                         msi_stream compute, msi_stream stage);

/* Pin (pinned = 1) or unpin (0) object (layer, expert): once resident, a
 * pinned object is never chosen as a victim by the plan's waves or prefetch
 * bundles (msi_slot_stage, where the caller names the slot, is not
 * affected).  At most n_slots - 2 * wave_capacity objects may be pinned at
 * once, so every wave and bundle finds victims; the default wave capacity
 * (n_slots / 2) leaves no room for pins.  Pins survive msi_plan_reset.
 * Errors: MSI_ERR_INVALID_ARG for a null plan or an index out of range,
 * MSI_ERR_SLOT_BUSY when the pin limit is reached (nothing changes). */
msi_status msi_plan_pin(msi_plan* plan, int layer, int expert, int pinned);

/* ---------------------------------------------------------------------------
 * End-to-end calls from and to host memory.  The same forwards as
 * msi_moe_forward / msi_moe_forward_streamed, with the token rows read from
 * and the outputs written to host buffers: hidden_host [T, H] bf16 in,
 * out_host [T, H] bf16 out, and (nullable) ids_host [T, k] int32 receiving the
 * route ids.  Pinned host memory gives the full host-link rate; pageable
 * memory is staged by the driver.  The route event still goes to the device
 * buffers of `ev`.  The rows are copied into the workspace on a plan-owned
 * copy stream forked from `compute` (the router waits for them), the route
 * ids are copied back beside the expert GEMMs, and the combine runs in row
 * chunks whose outputs are copied back while the next chunk is combined.  The
 * copy stream joins `compute` before the call returns, so out_host and
 * ids_host hold the results once `compute` has reached the point after the
 * call (synchronise it, or an event recorded on it).  The host buffers must
 * stay valid until then.  Workspace: msi_workspace_size_host (the device
 * workspace plus two [T, H] bf16 row buffers).  Errors: as the device-buffer
 * forwards; MSI_ERR_INVALID_ARG for a null hidden_host or out_host with T > 0. */
msi_status msi_workspace_size_host(const msi_plan* plan, int T, size_t* bytes);
msi_status msi_moe_forward_host(msi_plan* plan, int layer, const void* hidden_host, int T,
                                const float* router_w, const int32_t* slot_table,
                                const uint64_t* expected_generations, void* out_host,
                                int32_t* ids_host, const msi_route_event* ev, void* workspace,
                                size_t workspace_bytes, unsigned flags, msi_stream compute);
msi_status msi_moe_forward_streamed_host(msi_plan* plan, int layer, const void* hidden_host, int T,
                                         const float* router_w, void* out_host, int32_t* ids_host,
                                         const msi_route_event* ev, void* workspace,
                                         size_t workspace_bytes, unsigned flags,
                                         msi_stream compute, msi_stream stage);

/* Wait for the most recent forward of the plan and return its device-side
 * status (an msi_status value; MSI_OK when every needed expert passed the
 * generation re-check and every bounded device wait completed). */
msi_status msi_forward_status(msi_plan* plan, int* device_status);

/* Reset: fails with MSI_ERR_SLOT_BUSY while a caller-held ticket is live;
 * otherwise waits for every staging and forward issued through the plan,
 * invalidates every slot (Vacant; its published generation word cleared, so
 * no expectation from before the reset can pass a check), clears the LRU state
 * and advances the request epoch.  Generations keep increasing across resets
 * (Sec. "Separate Window and GPU-Slot Lifecycles": reset advances the epoch
 * after the outstanding-work checks; drain or invalidate outstanding
 * versions). */
msi_status msi_plan_reset(msi_plan* plan, uint64_t* new_epoch);

/* Deterministic fault hooks for lifecycle tests, applied on the host (no GPU
 * fault is ever raised): see MSI_FAULT_*.  The paper's fault cells (its table
 * of fault modes) check that a short or failed read publishes nothing and
 * that a stale completion or wrong object is rejected before visibility.
 * kind: one MSI_FAULT_* value; layer in [0, n_layers), expert in
 * [0, n_experts).  Arming the same object again replaces its pending fault.
 * Errors: MSI_ERR_INVALID_ARG for a null plan, an unknown kind or an index
 * out of range.  Nothing is allocated; msi_plan_reset does not disarm. */
msi_status msi_fault_inject(msi_plan* plan, int kind, int layer, int expert);

/* Optional early-staging buffer for streamed calls (a library convenience;
 * the paper's runtime copies each miss after its plan).  buf: caller-owned
 * device memory, 16-byte aligned, bytes >= extent_bytes (at most
 * wave_capacity extents of it are used); NULL detaches (after waiting for
 * the calls that used it).  A streamed call whose T * top_k >= 8 * n_experts
 * (every expert then almost surely needed) copies, on its stage stream and
 * while it routes, the extents of the layer's non-resident experts in
 * ascending order (the order the LRU-wave plan stages misses) into the
 * buffer (in a host-buffer call, after its rows have crossed); its waves
 * then copy those extents device to device into their slots instead of from
 * the host windows (a wave of at most 8 MB drawn wholly from the buffer in
 * one launch that also invalidates and publishes its slots' words).
 * Victims, generations, publication and the slot trace
 * are those of a call without the buffer; outputs are bit-identical.  Not
 * used with a source attached.  The buffer must stay allocated until it is
 * detached or the plan destroyed. */
msi_status msi_plan_set_bounce(msi_plan* plan, void* buf, size_t bytes);

/* Limit of every bounded device wait of the plan's kernels, in SM clock
 * cycles (clock64); cycles <= 0 restores the default of 4e9 (~2 s at GB300
 * clocks).  A wait that runs out raises MSI_ERR_TIMEOUT in the forward's
 * status word (msi_forward_status); the kernel still waits, with its own
 * ~10 ms bound, for the copies and MMAs it issued, frees its TMEM and returns,
 * so the context stays usable.  Applies to forwards enqueued after the call.
 * Library convenience (the paper's runtime has no device waits). */
msi_status msi_plan_set_wait_cycles(msi_plan* plan, int64_t cycles);

/* Host-side consumer tickets: a caller that reads slots outside a forward
 * holds the slot while reading.  Staging into a held slot waits, bounded. */
/* ---------------------------------------------------------------------------
 * Bounded source service (paper, Sec. "Bounded Source Service"; window
 * lifecycle Free -> Reading -> HostReady -> Copying -> Free, Sec. "Separate
 * Window and GPU-Slot Lifecycles").  Expert extents are read from a file into
 * a fixed set of aligned host windows: at most n_windows reads are in flight
 * and the streamed weights occupy at most n_windows * window_bytes of host
 * memory (the paper's M_source bound).  With direct = 1 the file is opened
 * with O_DIRECT and each extent is read by a covering read (the range rounded
 * out to `align`), so no copy of the payload accumulates in the page cache;
 * direct = 0 reads through the page cache.  A read is rejected, and nothing
 * of it is copied or published, on an I/O error, a short read (fewer bytes
 * than cover the extent), an extent past the end of the file, or a
 * completion that does not match its request (object, epoch, generation).
 * ------------------------------------------------------------------------- */
#define MSI_MAX_WINDOWS 64

typedef struct msi_source msi_source; /* opaque, owned by the library */

typedef struct {
  const char* path;      /* file holding the extents (read-only) */
  int direct;            /* 1: O_DIRECT covering reads; 0: buffered reads */
  uint32_t align;        /* covering-read alignment, a power of two; 0 means 4096 */
  int n_windows;         /* fixed window count = in-flight read limit, 1..MSI_MAX_WINDOWS */
  void* windows;         /* caller-owned host memory, n_windows * window_bytes; pinned for
                            asynchronous H2D copies; with direct = 1 aligned to `align` */
  uint64_t window_bytes; /* W; >= an extent's covering read (extent + 2 * align rounded
                            up to align for direct reads); with direct = 1 a multiple of align */
} msi_source_desc;

typedef struct {
  uint64_t reads;          /* completed reads */
  uint64_t rejected;       /* reads or submissions rejected */
  uint64_t logical_bytes;  /* extent bytes of accepted reads */
  uint64_t physical_bytes; /* covering-read bytes of accepted reads */
  uint64_t padding_bytes;  /* physical - logical */
  double read_seconds;     /* summed completion latency of completed reads */
  int max_in_flight;       /* peak reads in flight */
  int windows_busy;        /* windows not Free at the query (a copy still in flight counts) */
} msi_source_stats;

/* Open: the file is opened (O_RDONLY, plus O_DIRECT when direct = 1) and one
 * reader thread is started per window.  Errors: MSI_ERR_INVALID_ARG (null
 * pointers, alignment, sizes), MSI_ERR_UNSUPPORTED (the file system refuses
 * O_DIRECT), MSI_ERR_SOURCE (the file cannot be opened).
 * Close is the source's shutdown check: it refuses with MSI_ERR_SLOT_BUSY,
 * changing nothing, while a plan still has the source attached
 * (msi_plan_set_source; msi_plan_destroy detaches) or a caller still holds a
 * window from msi_source_read; otherwise it waits for every read in flight and
 * every window's copy, then frees the source. */
msi_status msi_source_open(const msi_source_desc* desc, msi_source** out);
msi_status msi_source_close(msi_source* src);
msi_status msi_source_stats_read(msi_source* src, msi_source_stats* out);

/* Synchronous read of one extent [file_off, file_off + bytes) into a free
 * window: on MSI_OK *data points at the extent's first byte inside window
 * *window, which stays HostReady (reserved) until msi_source_release.
 * MSI_ERR_SOURCE on a rejected read (nothing is left reserved). */
msi_status msi_source_read(msi_source* src, uint64_t file_off, uint64_t bytes, const void** data,
                           int* window);
msi_status msi_source_release(msi_source* src, int window);

/* Attach a source to a plan: from then on msi_slot_stage and the LRU waves of
 * msi_moe_forward_streamed read each missing extent (layer l, expert e) from
 * the file at file_off[l * n_experts + e] (extent_bytes long) through the
 * source's windows instead of the plan's host windows, submitting up to
 * n_windows reads ahead of the H2D copies.  A rejected read fails the call
 * with MSI_ERR_SOURCE: the failing bundle (the wave, and every later wave of
 * the call) is neither copied nor published, its slots are left Vacant, and
 * no output row of the call is written.  src = NULL detaches.  The source
 * stays attached until detached or until msi_plan_destroy, and refuses to
 * close meanwhile.  file_off is copied. */
msi_status msi_plan_set_source(msi_plan* plan, msi_source* src, const uint64_t* file_off);

msi_status msi_consumer_hold(msi_plan* plan, int slot);
msi_status msi_consumer_release(msi_plan* plan, int slot);

/* Copy up to `cap` trace records (oldest first) into buf; *n receives the
 * number copied.  msi_trace_clear empties the trace. */
msi_status msi_trace_read(const msi_plan* plan, msi_trace_rec* buf, size_t cap, size_t* n);
msi_status msi_trace_clear(msi_plan* plan);

msi_status msi_get_counters(const msi_plan* plan, msi_counters* out);

/* Kernel kinds for per-kernel timing. */
enum {
  MSI_K_UPLOAD = 0,        /* per-call tables / forward begin */
  MSI_K_ROUTER = 1,        /* fp32 logits + top-k + weights + block histogram */
  MSI_K_SCAN = 2,          /* column prefix over router blocks */
  MSI_K_SCATTER = 3,       /* stable permutation */
  MSI_K_SETUP = 4,         /* generation re-check + GEMM groups */
  MSI_K_GATEUP = 5,        /* routed gate-up GEMM with SwiGLU epilogue */
  MSI_K_DOWN = 6,          /* routed down GEMM */
  MSI_K_SHARED_GATEUP = 7, /* shared-expert gate-up GEMM */
  MSI_K_SHARED_DOWN = 8,   /* shared-expert down GEMM */
  MSI_K_COMBINE = 9,       /* weighted combine */
  MSI_K_PUBLISH = 10,      /* slot generation publication (staging stream) */
  MSI_K_FFN = 11,          /* one wave's gate-up and down GEMMs in one launch */
  MSI_K_COUNT = 12
};

/* Per-kernel timing: when enabled, every launch is bracketed by CUDA events on
 * its own stream.  msi_timing_read waits for the recorded launches and returns
 * per kind the summed milliseconds and launch counts (arrays [MSI_K_COUNT]);
 * reset != 0 clears the accumulators. */
msi_status msi_timing_enable(msi_plan* plan, int on);
msi_status msi_timing_read(msi_plan* plan, double* ms, uint64_t* launches, int reset);

/* Number of kernels the library launched since the plan was created. */
uint64_t msi_kernel_launches(const msi_plan* plan);

/* Text of a status code; text of the last CUDA error seen by the library. */
const char* msi_status_string(msi_status s);
const char* msi_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* MSI_H_ */
