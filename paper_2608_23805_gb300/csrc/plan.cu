// Host runtime of the C ABI: the Plan (immutable manifest + mutable slot
// ledger), slot staging with generation publication (from host windows or
// through the bounded source service), the LRU-wave residency driver with
// next-layer prediction, the two-bank prefetch and caller pins, the layer
// forwards (caller-managed residency, plan-managed waves, and their
// host-buffer variants), reset, shutdown and the host-side fault hooks.
//
// Paper basis:
//  - Plan = manifest (object -> extent, slot compatibility, stable device
//    addresses) + mutable state (object, generation, readiness event and
//    consumers per slot); replacement policy kept separate from the lifecycle
//    (Sec. "A Shared Cross-Adapter Plan Core").
//  - Slot lifecycle Vacant -> Loading -> DeviceReady -> InUse -> Recyclable ->
//    Vacant; no reuse before the last consumer finishes (Sec. "Separate Window
//    and GPU-Slot Lifecycles").
//  - Bundle publication: all components checked before one publication
//    transition; a device event publishes readiness; layer exit releases the
//    consumer ticket (Sec. "Stable Slots and Bundle Publication";
//    Sec. "Implementation", "Scheduling and copies").
//  - Telemetry: stages, cache events, generations, H2D bytes, rejections
//    (Sec. "Implementation", "Telemetry").
//  - Per-layer LRU over 64 slots, with a two-bank next-layer prefetch (Sec.
//    "Evaluation", "Cache and storage state").  The wave policy (hits then
//    misses, waves of half the pool, the previous wave pinned, least-recent
//    victim, lowest index on ties) and the prefetch bundle (the predicted
//    objects ranked by predicted count, placed after the last wave) are the
//    readings this library takes where the paper gives no rule.
//  - Reset advances the request epoch after the outstanding-work checks;
//    shutdown also checks the source's outstanding work (Sec. "Separate
//    Window and GPU-Slot Lifecycles"; the fault cells of the paper's fault
//    table).
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "kernels.cuh"
#include "source.h"

using namespace msi;

namespace {

thread_local std::string g_last_cuda = "no error";

msi_status cuda_fail(cudaError_t e, const char* what) {
  g_last_cuda = std::string(what) + ": " + cudaGetErrorString(e);
  return MSI_ERR_CUDA;
}

#define CK(call)                                               \
  do {                                                         \
    cudaError_t e_ = (call);                                   \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);        \
  } while (0)

// Launch one kernel of kind `kind` on `strm`, counted and (optionally) timed.
#define LAUNCH(plan, kind, strm, call)                                   \
  do {                                                                   \
    cudaEvent_t ea_ = nullptr, eb_ = nullptr;                            \
    if ((plan)->timer.on) {                                              \
      ea_ = (plan)->timer.get();                                         \
      eb_ = (plan)->timer.get();                                         \
      cudaEventRecord(ea_, (strm));                                      \
    }                                                                    \
    cudaError_t e_ = (call);                                             \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);                  \
    if (ea_ != nullptr) {                                                \
      cudaEventRecord(eb_, (strm));                                      \
      (plan)->timer.pending.push_back({(kind), ea_, eb_});               \
    }                                                                    \
    (plan)->launches++;                                                  \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor [rows, inner] (inner contiguous), box 64 x box_rows, 128-byte swizzle.
bool make_tmap(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr || rows == 0) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Byte-granular 2-D map over rows of `row_bytes` (4-bit codes): boxes of 32
// bytes (64 codes, one K block) x 128 rows, no swizzle.
bool make_tmap_codes(CUtensorMap* m, const void* base, uint64_t row_bytes, uint64_t rows) {
  auto fn = encode_fn();
  if (fn == nullptr || rows == 0) return false;
  cuuint64_t dims[2] = {row_bytes, rows};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {32, 128};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Reference-counted pool of CUDA events (readiness and consumer fences).
struct EventPool {
  std::vector<cudaEvent_t> ev;
  std::vector<int> refs;
  std::vector<int> freel;

  msi_status acquire(int* id) {
    if (freel.empty()) {
      cudaEvent_t e;
      CK(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
      ev.push_back(e);
      refs.push_back(0);
      freel.push_back((int)ev.size() - 1);
    }
    *id = freel.back();
    freel.pop_back();
    refs[*id] = 1;
    return MSI_OK;
  }
  void ref(int id) {
    if (id >= 0) refs[id]++;
  }
  void unref(int id) {
    if (id >= 0 && --refs[id] == 0) freel.push_back(id);
  }
  // true once the recorded work completed (or the event never recorded)
  bool done(int id) {
    if (id < 0) return true;
    const cudaError_t e = cudaEventQuery(ev[id]);
    if (e == cudaErrorNotReady) {
      (void)cudaGetLastError();  // "not ready" is a state, not an error to report later
      return false;
    }
    return true;
  }
};

struct Slot {
  int layer = -1, expert = -1;  // object held; -1: vacant
  uint64_t gen = 0;             // generation of the current object
  int ready = -1;               // event publishing the last stage
  int consumer = -1;            // event of the last consumer
  int64_t last_use = -1;        // LRU tick of the last consumption
  bool prefetched = false;      // staged by prediction, not yet consumed
};

struct WaveEntry {
  int expert, slot;
  bool miss;
  uint64_t gen;
};

struct WsLayout {
  size_t status, table, expected, groups, total, sh_group, sh_total, w3, cand_v, cand_i, bcount,
      bbase, offsets, perm, inv, sg, h, yp, hs, ys, ready, ready_n, bytes;
  int tm;  // tokens per router block
};

constexpr long long kDeviceWaitCycles = 4000000000LL;  // ~2 s at GB300 clocks

// Opt-in per-kernel timing: event pairs around each launch, resolved on read.
struct KernelTimer {
  bool on = false;
  std::vector<cudaEvent_t> freel;
  struct Rec { int kind; cudaEvent_t a, b; };
  std::vector<Rec> pending;
  double ms[MSI_K_COUNT] = {};
  uint64_t n[MSI_K_COUNT] = {};

  cudaEvent_t get() {
    if (!freel.empty()) {
      cudaEvent_t e = freel.back();
      freel.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  void resolve() {
    for (auto& r : pending) {
      float t = 0.f;
      cudaEventSynchronize(r.b);
      if (cudaEventElapsedTime(&t, r.a, r.b) == cudaSuccess) ms[r.kind] += t;
      n[r.kind]++;
      freel.push_back(r.a);
      freel.push_back(r.b);
    }
    pending.clear();
  }
  void destroy() {
    resolve();
    for (auto e : freel) cudaEventDestroy(e);
    freel.clear();
  }
};

}  // namespace

struct msi_plan {
  msi_plan_desc d{};
  // the device current at msi_plan_create: the plan's device memory, streams,
  // events and tensor maps belong to it, and every call that enqueues work
  // requires it to be current
  int dev = -1;
  std::vector<uint64_t> off;
  int sms = 0;
  std::vector<Slot> slots;
  std::vector<int> where;  // [L * E]: slot holding (l, e) or -1
  std::vector<std::atomic<int>> holds;
  GenWord* d_gen = nullptr;
  // blocks finished by the one-launch staging of early-staged waves (device
  // counter, never reset) and the host's running total of blocks launched
  unsigned long long* d_ticket = nullptr;
  unsigned long long ticket_total = 0;
  int* h_status = nullptr;
  int* h_counts = nullptr;
  EventPool pool;
  int fwd_ev = -1;
  CUtensorMap tm_w13{}, tm_w2{}, tm_sh13{}, tm_sh2{};
  CUtensorMap tm_q13{}, tm_q2{};  // 4-bit plans: packed codes of W13 / W2 over the pool
  std::vector<msi_trace_rec> trace;
  uint64_t seq = 0;
  msi_counters ctr{};
  uint64_t launches = 0;
  int64_t tick = 0;
  int calls = 0;
  int C = 1;
  bool dying = false;
  uint64_t epoch = 0;
  std::map<uint64_t, int> faults;  // one-shot host-side fault hooks by object key
  KernelTimer timer;
  // the shared expert of a resident forward runs on `side`, forked after the
  // forward's first kernel and joined before the combine (plans with a shared
  // expert only)
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // bounded source service: when attached, missing extents are read from its
  // file (src_off[l * E + e]) through its windows instead of host_windows
  msi_source* src = nullptr;
  std::vector<uint64_t> src_off;
  // next-layer prediction: a plan-owned stream and events (created on first
  // use) and the predicted counts read back to the host
  cudaStream_t pred = nullptr;
  cudaEvent_t ev_pfork = nullptr, ev_pjoin = nullptr;
  int* h_pred = nullptr;
  // host-buffer calls: a plan-owned copy stream and two events (compute ->
  // copy, copy -> compute), created on first use
  cudaStream_t io = nullptr;
  cudaEvent_t ev_io_a = nullptr, ev_io_b = nullptr;
  // caller pins by object [L * E]: never a victim of the plan's waves/bundles
  std::vector<char> pinned_obj;
  int n_pins = 0;
  // clock64 cycles each bounded device wait of the plan's kernels may take
  // before it gives up (msi_plan_set_wait_cycles)
  long long wait_cycles = kDeviceWaitCycles;
  // MSI_FAULT_DEVICE_WAIT: the next forward on this layer runs its tensor-core
  // kernels with one wait that nothing ends (-1: none armed)
  int stall_layer = -1;
  // early staging (msi_plan_set_bounce): a caller-owned device buffer of
  // bounce_cap extents; during a streamed call, the extents copied into it
  // while the call routes (spec_idx[e]: index in the buffer, -1 if none; for
  // layer spec_layer only), and an event after the call's last read of it
  char* bounce = nullptr;
  int bounce_cap = 0;
  int spec_layer = -1;
  std::vector<int> spec_idx;
  cudaEvent_t ev_bounce = nullptr;
  std::mutex mu;

  explicit msi_plan(int S) : holds(S) {
    for (auto& h : holds) h.store(0);
  }
};

namespace {

// The tensor-core router splits E into chunks of min(E, 128) experts (MMA N,
// a multiple of 16) and keeps k + 1 <= 32 candidates per chunk and token.
// Small layers (E <= 64 and E * H <= 32,768) take the FFMA router instead:
// sized for 64 experts, its blocks finish in a few microseconds, below the
// fixed cost of the tensor path's three launches (decode sizes).
bool tensor_router(const msi_plan_desc& d) {
  const int E = d.n_experts;
  if (E <= 64 && (long long)E * d.hidden <= 32768) return false;
  return E % 16 == 0 && (E <= kRouterChunk || E % kRouterChunk == 0) && d.top_k <= 31 &&
         E / std::min(E, kRouterChunk) * std::min(d.top_k + 1, std::min(E, kRouterChunk)) <= 160;
}

// A call that enqueues work must be made with the plan's device current: its
// kernels would otherwise launch on another GPU against this plan's memory.
msi_status check_device(const msi_plan* p) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  return dev == p->dev ? MSI_OK : MSI_ERR_INVALID_ARG;
}

bool shape_ok(const msi_plan_desc& d) {
  return d.n_experts >= 1 && d.n_experts <= kMaxExperts && d.top_k >= 1 &&
         d.top_k <= std::min(d.n_experts, kMaxTopK) && d.hidden >= 256 && d.hidden % 256 == 0 &&
         d.inter >= 128 && d.inter % 128 == 0 &&
         (d.wdtype == MSI_W_BF16 || d.wdtype == MSI_W_Q4G32);
}

WsLayout layout(const msi_plan* p, int T) {
  WsLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t r = o;
    o += (bytes + 255) & ~(size_t)255;
    return r;
  };
  const size_t E = p->d.n_experts, k = p->d.top_k, H = p->d.hidden, I = p->d.inter;
  L.tm = kRouterTM;  // both routers count ids per 32-token block
  const size_t nb = ((size_t)T + L.tm - 1) / L.tm, Tk = (size_t)T * k;
  L.status = take(4);
  L.table = take(4 * E);
  L.expected = take(8 * E);
  L.groups = take(sizeof(Group) * std::max<size_t>(E, kMaxWave));
  L.total = take(8);      // 128-row tiles, 256-row pair tiles
  L.sh_group = take(sizeof(Group));
  L.sh_total = take(8);
  L.w3 = tensor_router(p->d) ? take(3 * E * H * 2) : 0;
  if (tensor_router(p->d)) {
    const size_t ch = std::min<size_t>(E, kRouterChunk);
    const size_t ncand = (E / ch) * std::min<size_t>(k + 1, ch);
    L.cand_v = take(4 * (size_t)T * ncand);
    L.cand_i = take(4 * (size_t)T * ncand);
  }
  L.bcount = take(4 * nb * E);
  L.bbase = take(4 * nb * E);
  L.offsets = take(4 * (E + 1));
  L.perm = take(4 * Tk);
  L.inv = take(4 * Tk);
  L.sg = take(4 * (size_t)T);
  L.h = take(2 * Tk * I);
  L.yp = take(2 * Tk * H);
  // fused GEMMs: a counter per 128-row tile, two banks (consecutive waves
  // alternate; each wave's kernel zeroes the other bank for the next)
  L.ready_n = Tk / kBM + E + 1;
  L.ready = take(2 * 4 * L.ready_n);
  if (p->d.has_shared) {
    L.hs = take(2 * (size_t)T * I);
    L.ys = take(2 * (size_t)T * H);
  }
  L.bytes = o;
  return L;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

void add_trace(msi_plan* p, int call, int layer, int expert, int slot, uint64_t gen, int kind,
               int wave) {
  msi_trace_rec r;
  r.seq = p->seq++;
  r.call = call;
  r.layer = layer;
  r.expert = expert;
  r.slot = slot;
  r.generation = gen;
  r.kind = kind;
  r.wave = wave;
  p->trace.push_back(r);
}

// Occupy `s` with (layer, e): records the eviction, bumps the generation.
void ledger_stage(msi_plan* p, int s, int layer, int e, int call, int wave,
                  int kind = MSI_TRACE_STAGE) {
  Slot& sl = p->slots[s];
  const int E = p->d.n_experts;
  if (sl.layer >= 0) {
    add_trace(p, call, sl.layer, sl.expert, s, sl.gen, MSI_TRACE_EVICT, wave);
    p->where[(size_t)sl.layer * E + sl.expert] = -1;
    p->ctr.evicts++;
  }
  sl.gen += 1;
  sl.layer = layer;
  sl.expert = e;
  sl.prefetched = false;
  p->where[(size_t)layer * E + e] = s;
  add_trace(p, call, layer, e, s, sl.gen, kind, wave);
  p->ctr.stages++;
  p->ctr.h2d_bytes += p->d.extent_bytes;
}

// A slot whose content is no longer its ledger object (a staging call that
// failed after invalidating it): the object is evicted and the slot Vacant.
void ledger_vacate(msi_plan* p, int s, int call, int wave) {
  Slot& sl = p->slots[s];
  if (sl.layer < 0) return;
  add_trace(p, call, sl.layer, sl.expert, s, sl.gen, MSI_TRACE_EVICT, wave);
  p->where[(size_t)sl.layer * p->d.n_experts + sl.expert] = -1;
  p->ctr.evicts++;
  sl.layer = sl.expert = -1;
  sl.prefetched = false;
}

// Victim for a miss: the lowest-index vacant slot, else the least-recently
// used slot (ties: lowest index), among the slots not pinned by the current
// wave or bundle and not holding a caller-pinned object; -1 when none is left.
int pick_victim(const msi_plan* p, const std::vector<char>& pinned) {
  const int S = p->d.n_slots, E = p->d.n_experts;
  for (int c = 0; c < S; ++c)
    if (!pinned[c] && p->slots[c].layer < 0) return c;
  int victim = -1;
  for (int c = 0; c < S; ++c) {
    const Slot& sl = p->slots[c];
    if (pinned[c] || p->pinned_obj[(size_t)sl.layer * E + sl.expert]) continue;
    if (victim < 0 || sl.last_use < p->slots[victim].last_use) victim = c;
  }
  return victim;
}

// Wait on `stream` for every not-yet-complete event in ids (deduplicated).
msi_status wait_events(msi_plan* p, std::vector<int>& ids, cudaStream_t stream) {
  std::sort(ids.begin(), ids.end());
  ids.erase(std::unique(ids.begin(), ids.end()), ids.end());
  for (int id : ids)
    if (id >= 0 && !p->pool.done(id)) CK(cudaStreamWaitEvent(stream, p->pool.ev[id], 0));
  return MSI_OK;
}

// Make `stream` wait for the publication of every slot in `slots`.  A slot
// whose publication event has completed drops its reference to it, so later
// calls (a resident pool is read by every forward) skip the query.
msi_status wait_ready(msi_plan* p, const std::vector<int>& slots, cudaStream_t stream) {
  std::vector<int> pending, complete;
  auto has = [](const std::vector<int>& v, int id) {
    return std::find(v.begin(), v.end(), id) != v.end();
  };
  for (int s : slots) {
    Slot& sl = p->slots[s];
    const int id = sl.ready;
    if (id < 0 || has(pending, id)) continue;
    if (has(complete, id) || p->pool.done(id)) {
      if (!has(complete, id)) complete.push_back(id);
      sl.ready = -1;
      p->pool.unref(id);
    } else {
      pending.push_back(id);
    }
  }
  for (int id : pending) CK(cudaStreamWaitEvent(stream, p->pool.ev[id], 0));
  return MSI_OK;
}

// Write the slots' published words (generation, object) on `stage`, in
// stream order (the publication kernel).
msi_status write_words(msi_plan* p, const PublishParams& w, cudaStream_t stage) {
  LAUNCH(p, MSI_K_PUBLISH, stage, launch_publish(w, p->d_gen, stage));
  return MSI_OK;
}

// Largest wave (bytes) staged by one launch from the early-staging buffer
constexpr uint64_t kStageCopyMaxBytes = 8ull << 20;

// Enqueue the copies of `misses` on `stage` and publish them with one event.
msi_status stage_enqueue(msi_plan* p, int layer, const std::vector<WaveEntry>& misses,
                         cudaStream_t stage) {
  if (misses.empty()) return MSI_OK;
  std::vector<int> waits;
  for (const auto& m : misses) {
    waits.push_back(p->slots[m.slot].consumer);
    waits.push_back(p->slots[m.slot].ready);
  }
  msi_status st = wait_events(p, waits, stage);
  if (st != MSI_OK) return st;
  PublishParams inv{}, pub{};
  inv.n = pub.n = (int)misses.size();
  for (size_t i = 0; i < misses.size(); ++i) {
    inv.slot[i] = pub.slot[i] = misses[i].slot;
    inv.gen[i] = 0;
    inv.obj[i] = 0;
    pub.gen[i] = misses[i].gen;
    pub.obj[i] = obj_key(layer, misses[i].expert);
    auto f = p->faults.find(obj_key(layer, misses[i].expert));
    if (f != p->faults.end() && f->second == MSI_FAULT_STALE_COMPLETION) {
      pub.gen[i] = misses[i].gen - 1;  // a late completion of the previous version lands
      p->faults.erase(f);
    } else if (f != p->faults.end() && f->second == MSI_FAULT_WRONG_OBJECT) {
      pub.obj[i] = obj_key(layer, (misses[i].expert + 1) % p->d.n_experts);
      p->faults.erase(f);
    }
  }
  const uint64_t eb = p->d.extent_bytes;
  // A small wave whose extents were all copied early (decode-sized waves):
  // invalidation, device-to-device copies and publication in one launch.  A
  // large wave keeps the copy engine: a copy kernel would contend for the
  // SMs the waves' GEMMs hold.
  bool one_launch = p->src == nullptr && p->spec_layer == layer &&
                    (uint64_t)misses.size() * eb <= kStageCopyMaxBytes && eb % 16 == 0;
  for (size_t i = 0; i < misses.size() && one_launch; ++i) one_launch = p->spec_idx[misses[i].expert] >= 0;
  if (one_launch) {
    StageCopyArgs sa{};
    sa.pub = pub;
    for (size_t i = 0; i < misses.size(); ++i)
      sa.src[i] = p->bounce + (size_t)p->spec_idx[misses[i].expert] * eb;
    sa.pool = static_cast<char*>(p->d.slot_pool);
    sa.bytes = eb;
    sa.parts = (int)std::max<uint64_t>(1, std::min<uint64_t>(256, eb / 16384));  // 16 KB a block
    sa.ticket = p->d_ticket;
    sa.target = p->ticket_total + (unsigned long long)misses.size() * (unsigned long long)sa.parts;
    LAUNCH(p, MSI_K_PUBLISH, stage, launch_stage_copy(sa, p->d_gen, stage));
    p->ticket_total = sa.target;
  } else {
  st = write_words(p, inv, stage);
  if (st != MSI_OK) return st;
  auto src_of = [&](const WaveEntry& m) {
    return static_cast<const char*>(p->d.host_windows) +
           p->off[(size_t)layer * p->d.n_experts + m.expert];
  };
  auto dst_of = [&](const WaveEntry& m) {
    return static_cast<char*>(p->d.slot_pool) + (size_t)m.slot * eb;
  };
  if (p->src != nullptr) {
    // source path: up to n_windows reads ahead of the copies, each read
    // checked (identity, length, completion status) before its copy
    const int nw = source_windows(p->src);
    std::vector<int> win(misses.size(), -1);
    std::vector<SourceRequest> rq(misses.size());
    for (size_t i = 0; i < misses.size(); ++i) {
      SourceRequest& r = rq[i];
      r.object = obj_key(layer, misses[i].expert);
      r.epoch = p->epoch;
      r.generation = misses[i].gen;
      r.file_off = p->src_off[(size_t)layer * p->d.n_experts + misses[i].expert];
      r.bytes = eb;
      r.inject = kInjectNone;
      auto f = p->faults.find(r.object);
      if (f != p->faults.end() && (f->second == MSI_FAULT_IO_ERROR || f->second == MSI_FAULT_SHORT_READ)) {
        r.inject = f->second == MSI_FAULT_IO_ERROR ? kInjectIoError : kInjectShortRead;
        p->faults.erase(f);
      }
    }
    // the identity each completion must carry; a hooked read is submitted
    // with the previous epoch, as a read from before a reset would be
    std::vector<SourceRequest> expect(rq);
    for (size_t i = 0; i < misses.size(); ++i) {
      auto f = p->faults.find(rq[i].object);
      if (f != p->faults.end() && f->second == MSI_FAULT_STALE_EPOCH) {
        rq[i].epoch = p->epoch - 1;
        p->faults.erase(f);
      }
    }
    size_t next = 0;
    msi_status fail = MSI_OK;
    for (size_t i = 0; i < misses.size() && fail == MSI_OK; ++i) {
      while (next < misses.size() && next < i + (size_t)nw && fail == MSI_OK) {
        fail = source_submit(p->src, rq[next], &win[next]);
        ++next;
      }
      if (fail != MSI_OK) break;
      const void* data = nullptr;
      fail = source_wait(p->src, win[i], expect[i], &data);
      win[i] = fail == MSI_OK ? win[i] : -1;
      if (fail != MSI_OK) break;
      CK(cudaMemcpyAsync(dst_of(misses[i]), data, eb, cudaMemcpyHostToDevice, stage));
      st = source_copying(p->src, win[i], stage);
      if (st != MSI_OK) return st;
      win[i] = -1;
    }
    if (fail != MSI_OK) {
      // nothing more is copied and the bundle is not published: reads still
      // in flight land and their windows return to Free
      for (size_t i = 0; i < next; ++i)
        if (win[i] >= 0) source_release(p->src, win[i]);
      p->ctr.rejections++;
      return fail == MSI_ERR_SOURCE ? MSI_ERR_SOURCE : fail;
    }
  } else {
  // one copy per run of extents that continue each other in both the source
  // and the slot pool (consecutive experts into consecutive slots): large
  // copies reach the host link's rate, per-extent copies fall short.  An
  // extent already copied into the early-staging buffer during this call's
  // routing comes from there, device to device.
  auto early = [&](const WaveEntry& m) {
    return p->spec_layer == layer && p->spec_idx[m.expert] >= 0;
  };
  auto from_of = [&](const WaveEntry& m) -> const char* {
    return early(m) ? p->bounce + (size_t)p->spec_idx[m.expert] * eb : src_of(m);
  };
  for (size_t i = 0; i < misses.size();) {
    const bool dev = early(misses[i]);
    const char* src = from_of(misses[i]);
    char* dst = dst_of(misses[i]);
    uint64_t bytes = eb;
    size_t j = i + 1;
    while (j < misses.size() && early(misses[j]) == dev && from_of(misses[j]) == src + bytes &&
           dst_of(misses[j]) == dst + bytes) {
      bytes += eb;
      ++j;
    }
    CK(cudaMemcpyAsync(dst, src, bytes, dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, stage));
    i = j;
  }
  }
  st = write_words(p, pub, stage);
  if (st != MSI_OK) return st;
  }
  int ev;
  st = p->pool.acquire(&ev);
  if (st != MSI_OK) return st;
  CK(cudaEventRecord(p->pool.ev[ev], stage));
  for (const auto& m : misses) {
    p->pool.unref(p->slots[m.slot].ready);
    p->slots[m.slot].ready = ev;
    p->pool.ref(ev);
  }
  p->pool.unref(ev);
  return MSI_OK;
}

// Record a consumer event on `s` for the slots in `used`.
msi_status consumer_record(msi_plan* p, const std::vector<int>& used, cudaStream_t s) {
  if (used.empty()) return MSI_OK;
  int ev;
  msi_status st = p->pool.acquire(&ev);
  if (st != MSI_OK) return st;
  CK(cudaEventRecord(p->pool.ev[ev], s));
  for (int slot : used) {
    p->pool.unref(p->slots[slot].consumer);
    p->slots[slot].consumer = ev;
    p->pool.ref(ev);
  }
  p->pool.unref(ev);
  return MSI_OK;
}

struct FwdCtx {
  int layer, T;
  const void* x;
  const float* router_w;
  void* out;
  const msi_route_event* ev;
  void* ws;
  WsLayout L;
  unsigned flags;
  int stall;  // MSI_FAULT_DEVICE_WAIT armed for this call
  cudaStream_t cs;
  CUtensorMap tm_h, tm_x, tm_hs;
  // host-buffer calls: the rows land on the copy stream (x_ready, recorded
  // there); the route ids and the output rows go back on it
  cudaStream_t io = nullptr;
  cudaEvent_t x_ready = nullptr;
  void* out_host = nullptr;
  int32_t* ids_host = nullptr;
};

struct HostIO {
  cudaStream_t io;
  cudaEvent_t x_ready;  // null when there are no rows (T = 0)
  void* out_host;
  int32_t* ids_host;
};

void apply_io(FwdCtx& f, const HostIO* h) {
  if (h == nullptr) return;
  f.io = h->io;
  f.x_ready = h->x_ready;
  f.out_host = h->out_host;
  f.ids_host = h->ids_host;
}

msi_status validate_fwd(msi_plan* p, int layer, const void* x, int T, const float* rw, void* out,
                        const msi_route_event* ev, void* ws, size_t ws_bytes) {
  if (p == nullptr || ev == nullptr) return MSI_ERR_INVALID_ARG;
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  msi_status dst = check_device(p);
  if (dst != MSI_OK) return dst;
  if (layer < 0 || layer >= p->d.n_layers || T < 0) return MSI_ERR_INVALID_ARG;
  if (T > 0 && (x == nullptr || rw == nullptr || out == nullptr || ev->ids == nullptr ||
                ev->weights == nullptr))
    return MSI_ERR_INVALID_ARG;
  if (ev->counts == nullptr) return MSI_ERR_INVALID_ARG;
  if ((uintptr_t)x % 16 || (uintptr_t)out % 16) return MSI_ERR_INVALID_ARG;
  const WsLayout L = layout(p, T);
  if (ws == nullptr || (uintptr_t)ws % 256 || ws_bytes < L.bytes) return MSI_ERR_WORKSPACE;
  return MSI_OK;
}

// Router + histogram over the call's rows for router weight `rw`: the route
// event (ids, weights, gap) and per-expert counts go to `ev`.  first: the
// forward's own routing (its first kernel clears the status word and writes
// the shared group; the shared gate is computed, and the side stream may fork
// after it).  Otherwise a prediction pass: no status reset, no shared group,
// no gate; it reuses the router scratch of the workspace, so it must be
// ordered after the forward's own routing and scatter.
msi_status route_rows(msi_plan* p, FwdCtx& f, const float* rw, const msi_route_event* ev, bool first,
                      const TableParams& tp, cudaStream_t s, bool scan = true) {
  const auto& d = p->d;
  const int E = d.n_experts, k = d.top_k, H = d.hidden;
  void* ws = f.ws;
  const WsLayout& L = f.L;
  const int nb = (f.T + L.tm - 1) / L.tm;
  const float* wsg = first && d.has_shared && !(f.flags & MSI_FWD_SHARED_UNGATED)
                         ? d.shared_gate_w + (size_t)f.layer * H
                         : nullptr;
  if (tensor_router(d)) {
    __nv_bfloat16* w3 = at<__nv_bfloat16>(ws, L.w3);
    // a resident call's table goes to the workspace here, for the scatter's
    // generation re-check
    const bool tab = first && tp.E > 0;
    LAUNCH(p, MSI_K_ROUTER, s,
           launch_split3(rw, (long long)E * H, w3, first ? at<int>(ws, L.status) : nullptr,
                         first && d.has_shared ? at<Group>(ws, L.sh_group) : nullptr,
                         at<int>(ws, L.sh_total), f.T, tp.shared_slot, tab ? &tp : nullptr,
                         at<int>(ws, L.table), at<unsigned long long>(ws, L.expected), s));
  }
  // host-buffer calls: every reader of the rows (router, shared expert) comes
  // after they have landed
  if (f.x_ready != nullptr) CK(cudaStreamWaitEvent(s, f.x_ready, 0));
  // the forward has begun (status cleared, shared group written): the shared
  // expert may start on the side stream from here
  if (first && d.has_shared) CK(cudaEventRecord(p->ev_fork, s));
  if (tensor_router(d)) {
    __nv_bfloat16* w3 = at<__nv_bfloat16>(ws, L.w3);
    const int ch = std::min(E, kRouterChunk);
    CUtensorMap tm_w3;
    if (!make_tmap(&tm_w3, w3, H, (uint64_t)3 * E, (uint32_t)ch)) return MSI_ERR_CUDA;
    RouterTcArgs ra{};
    ra.x = static_cast<const __nv_bfloat16*>(f.x);
    ra.wsg = wsg;
    ra.T = f.T;
    ra.H = H;
    ra.E = E;
    ra.k = k;
    ra.chunk = ch;
    ra.nchunk = E / ch;
    ra.kp = std::min(k + 1, ch);
    int cols = 32;
    while (cols < ch) cols <<= 1;
    ra.tmem_cols = cols;
    ra.cand_v = at<float>(ws, L.cand_v);
    ra.cand_i = at<int>(ws, L.cand_i);
    ra.ids = ev->ids;
    ra.weights = ev->weights;
    ra.gap = ev->gap;
    ra.sg = at<float>(ws, L.sg);
    ra.bcount = at<int>(ws, L.bcount);
    ra.status = at<int>(ws, L.status);
    ra.wait_limit = p->wait_cycles;
    ra.stall = f.stall;
    LAUNCH(p, MSI_K_ROUTER, s, launch_router_tc(f.tm_x, tm_w3, ra, s));
    p->launches++;  // launch_router_tc starts two kernels (logits + top-k, merge)
  } else {
    RouterArgs ra{};
    ra.x = static_cast<const __nv_bfloat16*>(f.x);
    ra.wr = rw;
    ra.wsg = wsg;
    ra.T = f.T;
    ra.H = H;
    ra.E = E;
    ra.k = k;
    ra.ids = ev->ids;
    ra.weights = ev->weights;
    ra.gap = ev->gap;
    ra.sg = at<float>(ws, L.sg);
    ra.bcount = at<int>(ws, L.bcount);
    ra.status = first ? at<int>(ws, L.status) : nullptr;
    ra.sh = first && d.has_shared ? at<Group>(ws, L.sh_group) : nullptr;
    ra.sh_total = at<int>(ws, L.sh_total);
    ra.shared_slot = tp.shared_slot;
    LAUNCH(p, MSI_K_ROUTER, s, launch_router(ra, s));
  }
  // the column scan (per-block prefixes and counts); a small forward's
  // scatter takes it over (scan = false)
  if (scan) {
    ScanArgs sa{at<int>(ws, L.bcount), nb, E, at<int>(ws, L.bbase), ev->counts};
    LAUNCH(p, MSI_K_SCAN, s, launch_colscan(sa, s));
  }
  return MSI_OK;
}

// A streamed wave runs its gate-up and down in one launch (gemm_fused.cu,
// gemm_fused_pair.cu): a wave is too small to fill the SMs' last round of
// gate-up tiles, and the down tiles fill it.  bf16 waves always; 4-bit waves
// on CTA pairs, once their groups average >= 512 rows (smaller 4-bit waves
// keep the split single-CTA launches).
bool fused_wave(const msi_plan* p, const FwdCtx& f, long long rows, int ng) {
  if (f.flags & MSI_FWD_SPLIT_WAVES) return false;
  if (p->d.wdtype == MSI_W_BF16) return true;
  return !(f.flags & MSI_FWD_SINGLE_CTA) && ng > 0 && rows >= 512LL * ng;
}

// A resident bf16 forward fuses its two projections while neither would take
// pair tiles (groups averaging < 512 rows, e.g. 4,096 tokens over 512
// experts): there the down projection's first tiles then overlap the
// gate-up's last round.  Longer calls keep the pair-tile down projection.
bool fused_resident(const msi_plan* p, const FwdCtx& f, long long rows, int ng) {
  return p->d.wdtype == MSI_W_BF16 && !(f.flags & MSI_FWD_SPLIT_WAVES) && ng > 0 &&
         !(!(f.flags & MSI_FWD_SINGLE_CTA) && rows >= 512LL * ng);
}

// Counters in one bank of the fused GEMMs' per-m-tile counters.
int ready_bank(const FwdCtx& f) { return (int)(f.L.ready_n); }

// Forward begin + router + histogram + permutation.
msi_status front(msi_plan* p, FwdCtx& f, const TableParams& tp) {
  const auto& d = p->d;
  const int E = d.n_experts, k = d.top_k, H = d.hidden, I = d.inter;
  void* ws = f.ws;
  const WsLayout& L = f.L;
  // Both routers clear the status word and write the shared group in their
  // first kernel, and the scatter kernel builds the GEMM groups (resident
  // calls), so only a call without rows needs the upload kernel.
  if (f.T == 0)
    LAUNCH(p, MSI_K_UPLOAD, f.cs, launch_upload(tp, at<int>(ws, L.table), at<unsigned long long>(ws, L.expected),
                            at<int>(ws, L.status), d.has_shared ? at<Group>(ws, L.sh_group) : nullptr,
                            at<int>(ws, L.sh_total), f.cs));
  if (f.T == 0) {
    LAUNCH(p, MSI_K_UPLOAD, f.cs, launch_zero_counts(f.ev->counts, E, f.cs));
    return MSI_OK;
  }
  const int nb = (f.T + L.tm - 1) / L.tm;
  if (!make_tmap(&f.tm_x, f.x, H, f.T, 128)) return MSI_ERR_CUDA;
  if (d.has_shared) {
    if (!make_tmap(&f.tm_hs, at<char>(ws, L.hs), I, f.T, 128)) return MSI_ERR_CUDA;
  }
  // up to kScatterWarps router blocks: one scatter block covers them all and
  // takes over the column scan (one launch fewer for decode-sized calls)
  const bool fuse_scan = nb <= kScatterWarps;
  msi_status st = route_rows(p, f, f.router_w, f.ev, true, tp, f.cs, !fuse_scan);
  if (st != MSI_OK) return st;
  ScatterArgs xa{};
  xa.ids = f.ev->ids;
  xa.counts = f.ev->counts;
  xa.fuse_scan = fuse_scan ? 1 : 0;
  xa.bcount = at<int>(ws, L.bcount);
  xa.counts_out = f.ev->counts;
  xa.bbase = at<int>(ws, L.bbase);
  xa.T = f.T;
  xa.k = k;
  xa.E = E;
  xa.nb = nb;
  xa.tm = L.tm;
  xa.perm = at<int>(ws, L.perm);
  xa.inv = at<int>(ws, L.inv);
  xa.offsets = at<int>(ws, L.offsets);
  xa.genwords = p->d_gen;
  xa.groups = at<Group>(ws, L.groups);
  xa.total_mtiles = at<int>(ws, L.total);
  xa.status = at<int>(ws, L.status);
  if (tp.E > 0) {
    // resident call: the scatter re-checks the table's slots from global
    // memory (the weight split copied it; the FFMA router path copies it here)
    if (!tensor_router(d))
      LAUNCH(p, MSI_K_UPLOAD, f.cs, launch_upload(tp, at<int>(ws, L.table), at<unsigned long long>(ws, L.expected),
                              nullptr, nullptr, nullptr, f.cs));
    xa.tab_slot = at<int>(ws, L.table);
    xa.tab_expected = at<unsigned long long>(ws, L.expected);
    xa.layer = tp.layer;
    if (fused_resident(p, f, (long long)f.T * k, E)) {
      xa.ready = at<int>(ws, L.ready);
      xa.n_ready = ready_bank(f);
    }
  } else if (!(f.flags & MSI_FWD_SPLIT_WAVES)) {
    // streamed call: the first fused wave's bank (later waves' banks are
    // zeroed by the wave before them)
    xa.ready = at<int>(ws, L.ready);
    xa.n_ready = ready_bank(f);
  }
  LAUNCH(p, MSI_K_SCATTER, f.cs, launch_scatter(xa, f.cs));
  const size_t Tk = (size_t)f.T * k;
  if (f.ids_host != nullptr) {
    // the route ids go back beside the expert GEMMs
    CK(cudaEventRecord(p->ev_io_a, f.cs));
    CK(cudaStreamWaitEvent(f.io, p->ev_io_a, 0));
    CK(cudaMemcpyAsync(f.ids_host, f.ev->ids, Tk * sizeof(int32_t), cudaMemcpyDeviceToHost, f.io));
  }
  if (!make_tmap(&f.tm_h, at<char>(ws, L.h), I, Tk, 128)) return MSI_ERR_CUDA;
  return MSI_OK;
}

GemmArgs gateup_args(msi_plan* p, FwdCtx& f, const Group* groups, int ng, const int* total,
                     __nv_bfloat16* out) {
  const auto& d = p->d;
  GemmArgs g{};
  g.groups = groups;
  g.num_groups = ng;
  g.total_mtiles = total;
  g.nt = d.inter / 128;
  g.kblocks = d.hidden / kBK;
  g.b_rows_per_slot = 3 * d.inter;
  g.b_row_off = 0;
  g.up_off = d.inter;
  g.out_ld = d.inter;
  g.out = out;
  g.x = static_cast<const __nv_bfloat16*>(f.x);
  g.x_ld = d.hidden;
  g.perm = at<int>(f.ws, f.L.perm);
  g.top_k = d.top_k;
  g.status = at<int>(f.ws, f.L.status);
  g.wait_limit = p->wait_cycles;
  g.stall = f.stall;
  return g;
}

GemmArgs down_args(msi_plan* p, FwdCtx& f, const Group* groups, int ng, const int* total,
                   __nv_bfloat16* out) {
  const auto& d = p->d;
  GemmArgs g = gateup_args(p, f, groups, ng, total, out);
  g.nt = d.hidden / kBN;
  g.kblocks = d.inter / kBK;
  g.b_rows_per_slot = 3 * d.hidden;
  g.b_row_off = 2 * d.hidden;
  g.up_off = 0;
  g.out_ld = d.hidden;
  return g;
}

// CTA-pair (256-row) tiles run ~2-7 % faster than 128-row tiles once a
// launch's groups average >= 1,024 rows (long prefills, the shared expert);
// below that their coarser row padding and tile rounds lose (measured at
// ~680 rows per group: 90 us against 80 us).
constexpr long long kPairMinRows = 1024;
// The down projection (K = 512, output-stream heavy) gains from pair tiles
// already at ~640 rows per group (measured 4 %), the gate-up does not.
constexpr long long kPairMinRowsDown = 512;
bool pair_tiles(const FwdCtx& f, long long rows, int groups, long long min_rows = kPairMinRows) {
  return !(f.flags & MSI_FWD_SINGLE_CTA) && groups > 0 && rows >= min_rows * groups;
}

// 4-bit weights: a pair CTA dequantises half the B rows of a single-CTA tile
// per unit of tensor work, which pays once the groups fill 256-row tiles.
constexpr long long kPairMinRowsQ4 = 512;
// A fused wave (gate-up and down in one launch) takes 256-row pair tiles
// once its groups average >= 1,024 rows: at ~640 rows per group their row
// padding (a 256-row tile per ~128-row remainder) outweighs the smaller
// operand feed per SM (measured at 32K, waves of 32: 2.14 ms per step on
// pairs against 2.10 ms on single-CTA tiles).
constexpr long long kPairMinRowsFused = 1024;


// wave_mtiles >= 0: the expert FFN of one wave (wp, index wave) or of a
// resident call (wp null) may run fused; -1: split launches.
msi_status routed_ffn(msi_plan* p, FwdCtx& f, int ng, int grid1, int grid2, long long rows,
                      int wave_mtiles = -1, const WaveParams* wp = nullptr, int wave = 0) {
  const bool bf16 = p->d.wdtype == MSI_W_BF16;
  const bool pair_up = bf16 ? pair_tiles(f, rows, ng) : pair_tiles(f, rows, ng, kPairMinRowsQ4);
  const bool pair_down = pair_tiles(f, rows, ng, bf16 ? kPairMinRowsDown : kPairMinRowsQ4);
  const auto& d = p->d;
  const Group* groups = at<Group>(f.ws, f.L.groups);
  const int* total = at<int>(f.ws, f.L.total);
  // 4-bit extent: W13 codes [2I, H/2] | W2 codes [H, I/2] | W13 scales [2I, H/32] | W2 scales [H, I/32];
  // code rows through the byte maps: W13 rows of H/2 bytes, W2 rows of I/2
  // bytes (an extent is a whole number of either: 27 I / 8 and 27 H / 8)
  const long long HI = (long long)d.hidden * d.inter;
  const int q13_rows = (int)(d.extent_bytes / (d.hidden / 2));
  const int q2_rows = (int)(d.extent_bytes / (d.inter / 2));
  const int q2_off = (int)(HI / (d.inter / 2));
  if (wave_mtiles >= 0 && fused_wave(p, f, rows, ng)) {
    // one launch: the wave's gate-up tiles, then its down tiles
    FusedArgs fa{};
    fa.groups = groups;
    fa.num_groups = ng;
    fa.total_mtiles = total;
    fa.nt_up = d.inter / 128;
    fa.nt_dn = d.hidden / kBN;
    fa.kb_up = d.hidden / kBK;
    fa.kb_dn = d.inter / kBK;
    fa.sched_w = std::max(1, fa.kb_up / fa.kb_dn);  // a gate-up tile's K blocks per down tile's
    fa.w13_rows_per_slot = 3 * d.inter;
    fa.w13_up_off = d.inter;
    fa.w2_rows_per_slot = 3 * d.hidden;
    fa.w2_row_off = 2 * d.hidden;
    fa.h = at<__nv_bfloat16>(f.ws, f.L.h);
    fa.h_ld = d.inter;
    fa.y = at<__nv_bfloat16>(f.ws, f.L.yp);
    fa.y_ld = d.hidden;
    fa.x = static_cast<const __nv_bfloat16*>(f.x);
    fa.x_ld = d.hidden;
    fa.perm = at<int>(f.ws, f.L.perm);
    fa.top_k = d.top_k;
    int* bank0 = at<int>(f.ws, f.L.ready);
    int* bank1 = bank0 + f.L.ready_n;
    fa.ready = (wave & 1) ? bank1 : bank0;
    fa.status = at<int>(f.ws, f.L.status);
    fa.wait_limit = p->wait_cycles;
    fa.stall = f.stall;
    static const WaveParams no_wave{};
    if (wp != nullptr) {
      // the kernel re-checks the wave's slots and builds its groups itself,
      // and zeroes the other bank for the next wave
      fa.wave = 1;
      fa.counts = f.ev->counts;
      fa.offsets = at<int>(f.ws, f.L.offsets);
      fa.genwords = p->d_gen;
      fa.ready_clear = (wave & 1) ? bank0 : bank1;
      fa.n_ready_clear = (int)f.L.ready_n;
    }
    const WaveParams& wv = wp != nullptr ? *wp : no_wave;
    const long long tiles = (long long)wave_mtiles * (fa.nt_up + fa.nt_dn);
    // a wave's launch leaves one SM (a pair: two) to the staging stream: the
    // next wave's invalidation and publication kernels run there at once
    // instead of waiting for this persistent launch to end, which would hold
    // back the next wave's copies (measured at 32K: 14.5 against 16.0 ms per
    // step)
    const int spare = wp != nullptr ? 1 : 0;
    const int pairs = (int)std::min<long long>(p->sms / 2 - spare, std::max<long long>(1, tiles));
    if (!bf16) {
      // 4-bit waves: CTA pairs (fused_wave admits them from 512 rows per group)
      fa.q4_pool = static_cast<const uint8_t*>(d.slot_pool);
      fa.q4_extent = d.extent_bytes;
      fa.q13_rows_per_slot = q13_rows;
      fa.q2_rows_per_slot = q2_rows;
      fa.q2_row_off = q2_off;
      fa.q13_scale_off = 3 * HI / 2;
      fa.q13_scale_ld = d.hidden / 16;
      fa.q2_scale_off = 3 * HI / 2 + HI / 8;
      fa.q2_scale_ld = d.inter / 16;
      LAUNCH(p, MSI_K_FFN, f.cs, launch_fused_wave_pair_q4(p->tm_q13, p->tm_q2, fa, wv, pairs, f.cs));
      return MSI_OK;
    }
    if (pair_tiles(f, rows, ng, kPairMinRowsFused)) {
      LAUNCH(p, MSI_K_FFN, f.cs, launch_fused_wave_pair(p->tm_w13, p->tm_w2, fa, wv, pairs, f.cs));
      return MSI_OK;
    }
    const int grid = (int)std::min<long long>(p->sms - spare, std::max<long long>(1, tiles));
    LAUNCH(p, MSI_K_FFN, f.cs, launch_fused_wave(p->tm_w13, p->tm_w2, f.tm_h, fa, wv, grid, f.cs));
    return MSI_OK;
  }
  GemmArgs g1 = gateup_args(p, f, groups, ng, total, at<__nv_bfloat16>(f.ws, f.L.h));
  GemmArgs g2 = down_args(p, f, groups, ng, total, at<__nv_bfloat16>(f.ws, f.L.yp));
  if (d.wdtype == MSI_W_Q4G32) {
    for (GemmArgs* g : {&g1, &g2}) {
      g->q4_pool = static_cast<const uint8_t*>(d.slot_pool);
      g->q4_extent = d.extent_bytes;
    }
    g1.q4_rows_per_slot = q13_rows;
    g1.q4_row_off = 0;
    g1.q4_scale_off = 3 * HI / 2;
    g1.q4_scale_ld = d.hidden / 16;
    g2.q4_rows_per_slot = q2_rows;
    g2.q4_row_off = q2_off;
    g2.q4_scale_off = 3 * HI / 2 + HI / 8;
    g2.q4_scale_ld = d.inter / 16;
    if (pair_up)
      LAUNCH(p, MSI_K_GATEUP, f.cs,
             launch_gemm_pair(kGateUpGatherQ4, f.tm_h, p->tm_q13, g1, std::max(1, grid1 / 2), f.cs));
    else
      LAUNCH(p, MSI_K_GATEUP, f.cs, launch_gemm(kGateUpGatherQ4, f.tm_h, p->tm_q13, g1, grid1, f.cs));
    if (pair_down)
      LAUNCH(p, MSI_K_DOWN, f.cs,
             launch_gemm_pair(kDownQ4, f.tm_h, p->tm_q2, g2, std::max(1, grid2 / 2), f.cs));
    else
      LAUNCH(p, MSI_K_DOWN, f.cs, launch_gemm(kDownQ4, f.tm_h, p->tm_q2, g2, grid2, f.cs));
    return MSI_OK;
  }
  if (pair_up)
    LAUNCH(p, MSI_K_GATEUP, f.cs,
           launch_gemm_pair(kGateUpGather, p->tm_w13, p->tm_w13, g1, std::max(1, grid1 / 2), f.cs));
  else
    LAUNCH(p, MSI_K_GATEUP, f.cs, launch_gemm(kGateUpGather, p->tm_w13, p->tm_w13, g1, grid1, f.cs));
  if (pair_down)
    LAUNCH(p, MSI_K_DOWN, f.cs,
           launch_gemm_pair(kDown, f.tm_h, p->tm_w2, g2, std::max(1, grid2 / 2), f.cs));
  else
    LAUNCH(p, MSI_K_DOWN, f.cs, launch_gemm(kDown, f.tm_h, p->tm_w2, g2, grid2, f.cs));
  return MSI_OK;
}

msi_status shared_ffn(msi_plan* p, FwdCtx& f, cudaStream_t stream) {
  if (!p->d.has_shared || f.T == 0) return MSI_OK;
  const Group* g = at<Group>(f.ws, f.L.sh_group);
  const int* total = at<int>(f.ws, f.L.sh_total);
  const int mt = (f.T + kBM - 1) / kBM;
  GemmArgs s1 = gateup_args(p, f, g, 1, total, at<__nv_bfloat16>(f.ws, f.L.hs));
  GemmArgs s2 = down_args(p, f, g, 1, total, at<__nv_bfloat16>(f.ws, f.L.ys));
  // the shared expert's weights are bf16 whatever the routed experts' format
  if (pair_tiles(f, f.T, 1)) {
    const int pt = (f.T + 2 * kBM - 1) / (2 * kBM);
    LAUNCH(p, MSI_K_SHARED_GATEUP, stream,
           launch_gemm_pair(kGateUpTma, f.tm_x, p->tm_sh13, s1, pt * s1.nt, stream));
    LAUNCH(p, MSI_K_SHARED_DOWN, stream,
           launch_gemm_pair(kDown, f.tm_hs, p->tm_sh2, s2, pt * s2.nt, stream));
    return MSI_OK;
  }
  LAUNCH(p, MSI_K_SHARED_GATEUP, stream, launch_gemm(kGateUpTma, f.tm_x, p->tm_sh13, s1, std::min(p->sms, mt * s1.nt), stream));
  LAUNCH(p, MSI_K_SHARED_DOWN, stream, launch_gemm(kDown, f.tm_hs, p->tm_sh2, s2, std::min(p->sms, mt * s2.nt), stream));
  return MSI_OK;
}

msi_status finish(msi_plan* p, FwdCtx& f) {
  const auto& d = p->d;
  if (f.T > 0) {
    // host-buffer calls combine in row chunks; each chunk's rows go back
    // while the next chunk is combined (only the last chunk's copy is left
    // after the combine: eight chunks from 8,192 rows)
    const int H = d.hidden, k = d.top_k;
    const int nc = f.out_host == nullptr || f.T < 1024 ? 1 : (f.T < 8192 ? 4 : 8);
    for (int ci = 0; ci < nc; ++ci) {
      const long long t0 = (long long)f.T * ci / nc, t1 = (long long)f.T * (ci + 1) / nc;
      CombineArgs c{};
      c.yp = at<__nv_bfloat16>(f.ws, f.L.yp);
      c.weights = f.ev->weights + t0 * k;
      c.inv = at<int>(f.ws, f.L.inv) + t0 * k;
      c.sg = d.has_shared && !(f.flags & MSI_FWD_SHARED_UNGATED) ? at<float>(f.ws, f.L.sg) + t0
                                                                 : nullptr;
      c.ys = d.has_shared ? at<__nv_bfloat16>(f.ws, f.L.ys) + t0 * H : nullptr;
      c.x = (f.flags & MSI_FWD_RESIDUAL) ? static_cast<const __nv_bfloat16*>(f.x) + t0 * H : nullptr;
      c.out = static_cast<__nv_bfloat16*>(f.out) + t0 * H;
      c.T = (int)(t1 - t0);
      c.H = H;
      c.k = k;
      c.status = at<int>(f.ws, f.L.status);
      LAUNCH(p, MSI_K_COMBINE, f.cs, launch_combine(c, f.cs));
      if (f.out_host != nullptr) {
        CK(cudaEventRecord(p->ev_io_a, f.cs));
        CK(cudaStreamWaitEvent(f.io, p->ev_io_a, 0));
        CK(cudaMemcpyAsync(static_cast<char*>(f.out_host) + t0 * H * 2, c.out, (t1 - t0) * H * 2,
                           cudaMemcpyDeviceToHost, f.io));
      }
    }
  }
  CK(cudaMemcpyAsync(p->h_status, at<int>(f.ws, f.L.status), sizeof(int), cudaMemcpyDeviceToHost,
                     f.cs));
  int ev;
  msi_status st = p->pool.acquire(&ev);
  if (st != MSI_OK) return st;
  CK(cudaEventRecord(p->pool.ev[ev], f.cs));
  p->pool.unref(p->fwd_ev);
  p->fwd_ev = ev;
  return MSI_OK;
}

bool wait_unheld(msi_plan* p, int slot) {
  const double lim = p->d.wait_timeout_s > 0 ? p->d.wait_timeout_s : 1.0;
  const auto t0 = std::chrono::steady_clock::now();
  while (p->holds[slot].load() > 0) {
    const double el = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
    if (el > lim) return false;
    std::this_thread::sleep_for(std::chrono::microseconds(200));
  }
  return true;
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================
extern "C" {

uint64_t msi_extent_bytes(int hidden, int inter, int wdtype) {
  if (hidden <= 0 || inter <= 0) return 0;
  const uint64_t HI = (uint64_t)hidden * inter;
  if (wdtype == MSI_W_BF16) return 3 * HI * 2;
  if (wdtype == MSI_W_Q4G32) {
    if (hidden % 32 || inter % 32) return 0;
    return 3 * HI / 2 + 3 * HI / 32 * 2;
  }
  return 0;
}

const char* msi_status_string(msi_status s) {
  switch (s) {
    case MSI_OK: return "ok";
    case MSI_ERR_INVALID_ARG: return "invalid argument";
    case MSI_ERR_STALE_GENERATION: return "stale generation";
    case MSI_ERR_WRONG_OBJECT: return "wrong object in slot";
    case MSI_ERR_SLOT_BUSY: return "slot busy (live consumer)";
    case MSI_ERR_NOT_RESIDENT: return "needed expert not resident";
    case MSI_ERR_TIMEOUT: return "bounded wait timed out";
    case MSI_ERR_CUDA: return "CUDA error";
    case MSI_ERR_SHUT_DOWN: return "plan shut down";
    case MSI_ERR_UNSUPPORTED: return "unsupported shape";
    case MSI_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case MSI_ERR_SOURCE: return "source extent failed; nothing published";
  }
  return "unknown status";
}

const char* msi_last_cuda_error(void) { return g_last_cuda.c_str(); }

msi_status msi_plan_create(const msi_plan_desc* desc, msi_plan** out) {
  if (desc == nullptr || out == nullptr) return MSI_ERR_INVALID_ARG;
  *out = nullptr;
  const msi_plan_desc& d = *desc;
  if (d.n_layers < 1 || d.n_slots < 2 || d.slot_pool == nullptr || d.host_windows == nullptr)
    return MSI_ERR_INVALID_ARG;
  if (d.wdtype != MSI_W_BF16 && d.wdtype != MSI_W_Q4G32) return MSI_ERR_INVALID_ARG;
  if (!shape_ok(d)) return MSI_ERR_UNSUPPORTED;
  if (d.extent_bytes != msi_extent_bytes(d.hidden, d.inter, d.wdtype)) return MSI_ERR_INVALID_ARG;
  if ((uintptr_t)d.slot_pool % 128) return MSI_ERR_INVALID_ARG;
  if (d.has_shared && (d.shared_w == nullptr || d.shared_gate_w == nullptr ||
                       (uintptr_t)d.shared_w % 128 || (uintptr_t)d.shared_gate_w % 16))
    return MSI_ERR_INVALID_ARG;
  const int C = d.wave_capacity > 0 ? d.wave_capacity : d.n_slots / 2;
  if (C < 1 || 2 * C > d.n_slots || C > kMaxWave) return MSI_ERR_INVALID_ARG;

  msi_plan* p = new msi_plan(d.n_slots);
  p->d = d;
  p->C = C;
  const size_t nobj = (size_t)d.n_layers * d.n_experts;
  p->off.resize(nobj);
  for (size_t i = 0; i < nobj; ++i) p->off[i] = d.extent_off ? d.extent_off[i] : i * d.extent_bytes;
  p->slots.resize(d.n_slots);
  p->where.assign(nobj, -1);
  p->pinned_obj.assign(nobj, 0);
  auto fail = [&](msi_status s) {
    if (p->d_gen) cudaFree(p->d_gen);
    if (p->d_ticket) cudaFree(p->d_ticket);
    if (p->h_status) cudaFreeHost(p->h_status);
    if (p->h_counts) cudaFreeHost(p->h_counts);
    if (p->side) cudaStreamDestroy(p->side);
    if (p->ev_fork) cudaEventDestroy(p->ev_fork);
    if (p->ev_join) cudaEventDestroy(p->ev_join);
    delete p;
    return s;
  };
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  p->dev = dev;
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&p->sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaMalloc(&p->d_gen, sizeof(GenWord) * d.n_slots);
  if (e == cudaSuccess) e = cudaMemset(p->d_gen, 0, sizeof(GenWord) * d.n_slots);
  if (e == cudaSuccess) e = cudaMalloc(&p->d_ticket, sizeof(unsigned long long));
  if (e == cudaSuccess) e = cudaMemset(p->d_ticket, 0, sizeof(unsigned long long));
  if (e == cudaSuccess) e = cudaMallocHost(&p->h_status, sizeof(int));
  if (e == cudaSuccess) e = cudaMallocHost(&p->h_counts, sizeof(int) * d.n_experts);
  if (e == cudaSuccess && d.has_shared) e = cudaStreamCreateWithFlags(&p->side, cudaStreamNonBlocking);
  if (e == cudaSuccess && d.has_shared) e = cudaEventCreateWithFlags(&p->ev_fork, cudaEventDisableTiming);
  if (e == cudaSuccess && d.has_shared) e = cudaEventCreateWithFlags(&p->ev_join, cudaEventDisableTiming);
  if (e != cudaSuccess) return fail(cuda_fail(e, "msi_plan_create"));
  *p->h_status = 0;
  const uint64_t H = d.hidden, I = d.inter, S = d.n_slots;
  if (d.wdtype == MSI_W_BF16) {
    if (!make_tmap(&p->tm_w13, d.slot_pool, H, S * 3 * I, 128) ||
        !make_tmap(&p->tm_w2, d.slot_pool, I, S * 3 * H, 128))
      return fail(MSI_ERR_CUDA);
  }
  if (d.wdtype == MSI_W_Q4G32) {
    if (d.extent_bytes % (H / 2) || d.extent_bytes % (I / 2) ||
        !make_tmap_codes(&p->tm_q13, d.slot_pool, H / 2, S * (d.extent_bytes / (H / 2))) ||
        !make_tmap_codes(&p->tm_q2, d.slot_pool, I / 2, S * (d.extent_bytes / (I / 2))))
      return fail(MSI_ERR_CUDA);
  }
  if (d.has_shared) {
    if (!make_tmap(&p->tm_sh13, d.shared_w, H, (uint64_t)d.n_layers * 3 * I, 128) ||
        !make_tmap(&p->tm_sh2, d.shared_w, I, (uint64_t)d.n_layers * 3 * H, 128))
      return fail(MSI_ERR_CUDA);
  }
  *out = p;
  return MSI_OK;
}

msi_status msi_plan_destroy(msi_plan* p) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  {
    std::lock_guard<std::mutex> g(p->mu);
    for (auto& h : p->holds)
      if (h.load() > 0) return MSI_ERR_SLOT_BUSY;
    p->dying = true;
    // release everything with the plan's device current (the caller's current
    // device is restored afterwards)
    int cur = -1;
    const bool swap = cudaGetDevice(&cur) == cudaSuccess && cur != p->dev && cudaSetDevice(p->dev) == cudaSuccess;
    // drain: every readiness, consumer and forward event still referenced
    for (auto& s : p->slots) {
      if (s.ready >= 0) cudaEventSynchronize(p->pool.ev[s.ready]);
      if (s.consumer >= 0) cudaEventSynchronize(p->pool.ev[s.consumer]);
    }
    if (p->fwd_ev >= 0) cudaEventSynchronize(p->pool.ev[p->fwd_ev]);
    if (p->side) cudaStreamSynchronize(p->side);
    if (p->pred) cudaStreamSynchronize(p->pred);
    source_attach(p->src, -1);  // every window copy of this plan has completed
    p->src = nullptr;
    p->timer.destroy();
    for (auto ev : p->pool.ev) cudaEventDestroy(ev);
    cudaFree(p->d_gen);
    cudaFree(p->d_ticket);
    cudaFreeHost(p->h_status);
    cudaFreeHost(p->h_counts);
    if (p->side) cudaStreamDestroy(p->side);
    if (p->ev_fork) cudaEventDestroy(p->ev_fork);
    if (p->ev_join) cudaEventDestroy(p->ev_join);
    if (p->pred) cudaStreamDestroy(p->pred);
    if (p->ev_pfork) cudaEventDestroy(p->ev_pfork);
    if (p->ev_pjoin) cudaEventDestroy(p->ev_pjoin);
    if (p->h_pred) cudaFreeHost(p->h_pred);
    if (p->io) {
      cudaStreamSynchronize(p->io);
      cudaStreamDestroy(p->io);
    }
    if (p->ev_io_a) cudaEventDestroy(p->ev_io_a);
    if (p->ev_io_b) cudaEventDestroy(p->ev_io_b);
    if (p->ev_bounce) {
      cudaEventSynchronize(p->ev_bounce);
      cudaEventDestroy(p->ev_bounce);
    }
    if (swap) cudaSetDevice(cur);
  }
  delete p;
  return MSI_OK;
}

}  // extern "C"

int msi::plan_device(const msi_plan* p) { return p->dev; }

extern "C" {

msi_status msi_workspace_size(const msi_plan* p, int T, size_t* bytes) {
  if (p == nullptr || bytes == nullptr || T < 0) return MSI_ERR_INVALID_ARG;
  *bytes = layout(p, T).bytes;
  return MSI_OK;
}

msi_status msi_slot_stage(msi_plan* p, int slot, int layer, int expert, msi_stream stage,
                          uint64_t* new_generation) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  msi_status dst = check_device(p);
  if (dst != MSI_OK) return dst;
  const auto& d = p->d;
  if (slot < 0 || slot >= d.n_slots || layer < 0 || layer >= d.n_layers || expert < 0 ||
      expert >= d.n_experts)
    return MSI_ERR_INVALID_ARG;
  const int cur = p->where[(size_t)layer * d.n_experts + expert];
  if (cur >= 0 && cur != slot) return MSI_ERR_INVALID_ARG;  // one slot per object
  if (p->src == nullptr) {
    auto f = p->faults.find(obj_key(layer, expert));
    if (f != p->faults.end() && f->second == MSI_FAULT_SHORT_READ) {
      p->faults.erase(f);  // the source delivered less than the extent: nothing is staged
      p->ctr.rejections++;
      return MSI_ERR_SOURCE;
    }
  }
  if (!wait_unheld(p, slot)) {
    p->ctr.rejections++;
    return MSI_ERR_TIMEOUT;
  }
  Slot& sl = p->slots[slot];
  const uint64_t gen = sl.gen + 1;
  std::vector<WaveEntry> m{{expert, slot, true, gen}};
  msi_status st = stage_enqueue(p, layer, m, reinterpret_cast<cudaStream_t>(stage));
  if (st == MSI_ERR_SOURCE) {
    // the slot's published word was invalidated before the read failed: the
    // object it held is gone
    ledger_vacate(p, slot, -1, -1);
    return st;
  }
  if (st != MSI_OK) return st;
  ledger_stage(p, slot, layer, expert, -1, -1);
  if (new_generation) *new_generation = sl.gen;
  return MSI_OK;
}

msi_status msi_slot_table(const msi_plan* cp, int layer, int32_t* slot_of, uint64_t* gen_of) {
  msi_plan* p = const_cast<msi_plan*>(cp);
  if (p == nullptr || slot_of == nullptr || gen_of == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (layer < 0 || layer >= p->d.n_layers) return MSI_ERR_INVALID_ARG;
  const int E = p->d.n_experts;
  for (int e = 0; e < E; ++e) {
    const int s = p->where[(size_t)layer * E + e];
    slot_of[e] = s;
    gen_of[e] = s >= 0 ? p->slots[s].gen : 0;
  }
  return MSI_OK;
}

msi_status msi_slot_state(const msi_plan* cp, int slot, int* state) {
  msi_plan* p = const_cast<msi_plan*>(cp);
  if (p == nullptr || state == nullptr || slot < 0 || slot >= p->d.n_slots)
    return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  const Slot& s = p->slots[slot];
  if (s.layer < 0) *state = MSI_SLOT_VACANT;
  else if (!p->pool.done(s.ready)) *state = MSI_SLOT_LOADING;
  else if (p->holds[slot].load() > 0 || !p->pool.done(s.consumer)) *state = MSI_SLOT_IN_USE;
  else if (s.consumer < 0) *state = MSI_SLOT_DEVICE_READY;
  else *state = MSI_SLOT_RECYCLABLE;
  return MSI_OK;
}

namespace {

msi_status forward_resident(msi_plan* p, int layer, const void* x, int T, const float* rw,
                            const int32_t* table, const uint64_t* expected, void* out,
                            const msi_route_event* ev, void* ws, size_t ws_bytes, unsigned flags,
                            msi_stream compute, const HostIO* hio) {
  msi_status st = validate_fwd(p, layer, x, T, rw, out, ev, ws, ws_bytes);
  if (st != MSI_OK) return st;
  if (table == nullptr || expected == nullptr) return MSI_ERR_INVALID_ARG;
  const auto& d = p->d;
  const int E = d.n_experts;
  // host precheck: nothing is enqueued when a named slot does not hold the
  // requested object and version
  std::vector<int> used;
  for (int e = 0; e < E; ++e) {
    const int s = table[e];
    if (s < -1 || s >= d.n_slots) return MSI_ERR_INVALID_ARG;
    if (s < 0) continue;
    const Slot& sl = p->slots[s];
    if (sl.layer != layer || sl.expert != e) {
      p->ctr.rejections++;
      return MSI_ERR_WRONG_OBJECT;
    }
    if (sl.gen != expected[e]) {
      p->ctr.rejections++;
      return MSI_ERR_STALE_GENERATION;
    }
    used.push_back(s);
  }
  FwdCtx f{};
  f.layer = layer;
  f.T = T;
  f.x = x;
  f.router_w = rw;
  f.out = out;
  f.ev = ev;
  f.ws = ws;
  f.L = layout(p, T);
  f.flags = flags;
  f.stall = p->stall_layer == layer;
  if (f.stall) p->stall_layer = -1;  // one-shot
  f.cs = reinterpret_cast<cudaStream_t>(compute);
  apply_io(f, hio);
  // readiness: the compute stream waits for every pending publication it reads
  st = wait_ready(p, used, f.cs);
  if (st != MSI_OK) return st;
  static thread_local TableParams tp;
  tp.E = E;
  tp.layer = layer;
  tp.T = T;
  tp.shared_slot = d.has_shared ? layer : -1;
  for (int e = 0; e < E; ++e) {
    tp.slot[e] = table[e];
    tp.expected[e] = expected[e];
  }
  st = front(p, f, tp);
  if (st != MSI_OK) return st;
  const bool fork = d.has_shared && T > 0;
  if (fork) {
    // the shared expert needs no routing: it runs on the side stream while
    // the router, scan and scatter leave most SMs idle, and joins before the
    // combine
    CK(cudaStreamWaitEvent(p->side, p->ev_fork, 0));
    st = shared_ffn(p, f, p->side);
    if (st != MSI_OK) return st;
    CK(cudaEventRecord(p->ev_join, p->side));
  }
  if (T > 0) {
    // the scatter kernel has re-checked the slots' generations and built the
    // GEMM groups (`tp` carries the table)
    const long long mt_max = ((long long)T * d.top_k + kBM - 1) / kBM + E;
    const int g1 = (int)std::min<long long>(p->sms, mt_max * (d.inter / 128));
    const int g2 = (int)std::min<long long>(p->sms, mt_max * (d.hidden / kBN));
    st = routed_ffn(p, f, E, g1, g2, (long long)T * d.top_k,
                    fused_resident(p, f, (long long)T * d.top_k, E) ? (int)mt_max : -1);
    if (st != MSI_OK) return st;
    st = consumer_record(p, used, f.cs);
    if (st != MSI_OK) return st;
  }
  if (fork) CK(cudaStreamWaitEvent(f.cs, p->ev_join, 0));
  st = finish(p, f);
  if (st != MSI_OK) return st;
  p->ctr.forwards++;
  return MSI_OK;
}

}  // namespace

msi_status msi_moe_forward(msi_plan* p, int layer, const void* x, int T, const float* rw,
                           const int32_t* table, const uint64_t* expected, void* out,
                           const msi_route_event* ev, void* ws, size_t ws_bytes, unsigned flags,
                           msi_stream compute) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  return forward_resident(p, layer, x, T, rw, table, expected, out, ev, ws, ws_bytes, flags, compute,
                          nullptr);
}

namespace {

// Plan-owned prediction stream, its fork/join events and the host copy of
// the predicted counts (created on the first predicting call).
msi_status prediction_resources(msi_plan* p) {
  if (p->pred != nullptr) return MSI_OK;
  // created into locals and kept only all together, so that a failure
  // leaves nothing half-made behind for the next call
  int* h = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  cudaStream_t s = nullptr;
  cudaError_t e = cudaMallocHost(&h, sizeof(int) * p->d.n_experts);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&join, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
  if (e != cudaSuccess) {
    if (h) cudaFreeHost(h);
    if (fork) cudaEventDestroy(fork);
    if (join) cudaEventDestroy(join);
    if (s) cudaStreamDestroy(s);
    return cuda_fail(e, "prediction stream");
  }
  p->h_pred = h;
  p->ev_pfork = fork;
  p->ev_pjoin = join;
  p->pred = s;
  return MSI_OK;
}

// The prefetch bundle for layer `nl` after call `call`'s last wave (slots
// `last`): predicted objects not resident, ranked by predicted count
// (descending; ties: lower id), at most C, staged in ascending expert order;
// the last wave's slots, the bundle's own and those of predicted objects
// already resident are pinned.  A rejected read unwinds the bundle only.
msi_status prefetch_bundle(msi_plan* p, int nl, int call, int wave, const std::vector<int>& last,
                           cudaStream_t ss) {
  const int E = p->d.n_experts;
  const int* cnt = p->h_pred;
  std::vector<char> pinned(p->d.n_slots, 0);
  for (int sl : last) pinned[sl] = 1;
  std::vector<int> cand;
  for (int e = 0; e < E; ++e) {
    if (cnt[e] <= 0) continue;
    const int r = p->where[(size_t)nl * E + e];
    if (r >= 0)
      pinned[r] = 1;
    else
      cand.push_back(e);
  }
  std::stable_sort(cand.begin(), cand.end(), [&](int a, int b) { return cnt[a] > cnt[b]; });
  if ((int)cand.size() > p->C) cand.resize(p->C);
  std::sort(cand.begin(), cand.end());
  // host windows: a source known to be short is refused before anything is
  // planned (the bundle is dropped; the call itself is unaffected)
  for (int e : cand) {
    if (p->src != nullptr) break;
    auto f = p->faults.find(obj_key(nl, e));
    if (f != p->faults.end() && f->second == MSI_FAULT_SHORT_READ) {
      p->faults.erase(f);
      p->ctr.rejections++;
      return MSI_OK;
    }
  }
  std::vector<WaveEntry> bundle;
  for (int e : cand) {
    const int sl = pick_victim(p, pinned);
    if (sl < 0) break;
    ledger_stage(p, sl, nl, e, call, wave, MSI_TRACE_PREFETCH);
    p->slots[sl].last_use = p->tick;  // prefetching is not consumption
    p->slots[sl].prefetched = true;
    pinned[sl] = 1;
    p->ctr.prefetches++;
    bundle.push_back({e, sl, true, p->slots[sl].gen});
  }
  if (bundle.empty()) return MSI_OK;
  const msi_status r = stage_enqueue(p, nl, bundle, ss);
  if (r == MSI_ERR_SOURCE) {
    for (const auto& we : bundle) ledger_vacate(p, we.slot, call, wave);
    return MSI_OK;
  }
  return r;
}

msi_status forward_streamed(msi_plan* p, int layer, const void* x, int T, const float* rw, void* out,
                            const msi_route_event* ev, const float* next_rw,
                            const msi_route_event* next_ev, void* ws, size_t ws_bytes,
                            unsigned flags, msi_stream compute, msi_stream stage,
                            const HostIO* hio = nullptr) {
  msi_status st = validate_fwd(p, layer, x, T, rw, out, ev, ws, ws_bytes);
  if (st != MSI_OK) return st;
  const bool predict = next_rw != nullptr;
  if (predict) {
    if (layer + 1 >= p->d.n_layers || next_ev == nullptr || next_ev->counts == nullptr ||
        (T > 0 && (next_ev->ids == nullptr || next_ev->weights == nullptr || next_ev->gap == nullptr)))
      return MSI_ERR_INVALID_ARG;
    st = prediction_resources(p);
    if (st != MSI_OK) return st;
  }
  const auto& d = p->d;
  const int E = d.n_experts;
  FwdCtx f{};
  f.layer = layer;
  f.T = T;
  f.x = x;
  f.router_w = rw;
  f.out = out;
  f.ev = ev;
  f.ws = ws;
  f.L = layout(p, T);
  f.flags = flags;
  f.stall = p->stall_layer == layer;
  if (f.stall) p->stall_layer = -1;  // one-shot
  f.cs = reinterpret_cast<cudaStream_t>(compute);
  apply_io(f, hio);
  cudaStream_t ss = reinterpret_cast<cudaStream_t>(stage);
  // Early staging: when the call is long enough that every expert is almost
  // surely needed (T k >= 8 E), the extents of the first misses the waves
  // would stage (the non-resident experts, ascending, as the LRU-wave plan
  // orders misses) are copied into the caller's early-staging buffer while
  // the call routes; the waves then copy them device to device.  Residency,
  // victims, publication and the trace are decided by the plan as always;
  // an extent copied early but not needed is simply not used.
  struct SpecEnd {
    msi_plan* p;
    cudaStream_t ss;
    bool on = false;
    ~SpecEnd() {
      if (!on) return;
      cudaEventRecord(p->ev_bounce, ss);  // after every read of the buffer in this call
      p->spec_layer = -1;
    }
  } spec_end{p, ss};
  if (p->bounce != nullptr && p->src == nullptr && T > 0 && (long long)T * d.top_k >= 8LL * E) {
    std::fill(p->spec_idx.begin(), p->spec_idx.end(), -1);
    CK(cudaStreamWaitEvent(ss, p->ev_bounce, 0));  // the previous call's reads of the buffer
    // a host-buffer call's rows cross the host link first (routing waits on them)
    if (f.x_ready != nullptr) CK(cudaStreamWaitEvent(ss, f.x_ready, 0));
    const uint64_t eb = d.extent_bytes;
    int n = 0;
    for (int e = 0; e < E && n < p->bounce_cap; ++e)
      if (p->where[(size_t)layer * E + e] < 0) p->spec_idx[e] = n++;
    for (int e = 0; e < E;) {
      if (p->spec_idx[e] < 0) {
        ++e;
        continue;
      }
      // runs of experts that continue each other in the host windows
      const char* src = static_cast<const char*>(d.host_windows) + p->off[(size_t)layer * E + e];
      uint64_t bytes = eb;
      int j = e + 1;
      while (j < E && p->spec_idx[j] == p->spec_idx[j - 1] + 1 &&
             static_cast<const char*>(d.host_windows) + p->off[(size_t)layer * E + j] == src + bytes) {
        bytes += eb;
        ++j;
      }
      CK(cudaMemcpyAsync(p->bounce + (size_t)p->spec_idx[e] * eb, src, bytes, cudaMemcpyHostToDevice, ss));
      e = j;
    }
    p->spec_layer = layer;
    spec_end.on = true;
  }
  static thread_local TableParams tp;
  tp.E = 0;
  tp.layer = layer;
  tp.T = T;
  tp.shared_slot = d.has_shared ? layer : -1;
  st = front(p, f, tp);
  if (st != MSI_OK) return st;
  // counts back to the host: the needed set decides the staging
  CK(cudaMemcpyAsync(p->h_counts, ev->counts, sizeof(int) * E, cudaMemcpyDeviceToHost, f.cs));
  int cev;
  st = p->pool.acquire(&cev);
  if (st != MSI_OK) return st;
  CK(cudaEventRecord(p->pool.ev[cev], f.cs));
  if (predict) {
    // layer + 1's router over the same rows, on the prediction stream while
    // this call's waves run; it reuses the router scratch, so it forks after
    // the scatter, and the compute stream joins it before the call ends
    CK(cudaEventRecord(p->ev_pfork, f.cs));
    CK(cudaStreamWaitEvent(p->pred, p->ev_pfork, 0));
    if (T == 0) {
      LAUNCH(p, MSI_K_UPLOAD, p->pred, launch_zero_counts(next_ev->counts, E, p->pred));
    } else {
      st = route_rows(p, f, next_rw, next_ev, false, tp, p->pred);
      if (st != MSI_OK) return st;
    }
    CK(cudaMemcpyAsync(p->h_pred, next_ev->counts, sizeof(int) * E, cudaMemcpyDeviceToHost, p->pred));
    CK(cudaEventRecord(p->ev_pjoin, p->pred));
  }
  // every return from here on (an error included) leaves the compute stream
  // joined to the prediction, which reads the router scratch the next call
  // overwrites
  struct PredJoin {
    cudaStream_t cs;
    cudaEvent_t ev;
    ~PredJoin() {
      if (ev != nullptr) cudaStreamWaitEvent(cs, ev, 0);
    }
  } pred_join{f.cs, predict ? p->ev_pjoin : nullptr};
  // The shared expert needs no residency.  A call that will stage at least
  // two waves of misses (T k >= 8 E: every expert almost surely needed)
  // runs it on the compute stream right after its first miss wave's GEMMs,
  // where that stream would otherwise wait for the next wave's copies;
  // ahead of the hit waves it would hold back their GEMMs and with them the
  // consumer tickets the next copies wait for.  Other calls run it here,
  // beside the host's planning.
  int resident_now = 0;
  for (int e = 0; e < E; ++e) resident_now += p->where[(size_t)layer * E + e] >= 0;
  bool late_shared = d.has_shared && T > 0 && (long long)T * d.top_k >= 8LL * E &&
                           E - resident_now >= 2 * p->C;
  if (!late_shared) {
    st = shared_ffn(p, f, f.cs);
    if (st != MSI_OK) return st;
  }
  const cudaError_t se = cudaEventSynchronize(p->pool.ev[cev]);
  p->pool.unref(cev);
  if (se != cudaSuccess) return cuda_fail(se, "counts readback");

  // held slots: wait (bounded) before planning so the plan never picks them
  for (int s = 0; s < d.n_slots; ++s)
    if (!wait_unheld(p, s)) {
      p->ctr.rejections++;
      return MSI_ERR_TIMEOUT;
    }

  // host windows: every miss's source must be whole before any bundle is
  // planned or published (with a source attached, reads are checked as they
  // complete and a failure unwinds the call's remaining bundles)
  for (int e = 0; e < E && p->src == nullptr; ++e) {
    if (p->h_counts[e] <= 0 || p->where[(size_t)layer * E + e] >= 0) continue;
    auto f = p->faults.find(obj_key(layer, e));
    if (f != p->faults.end() && f->second == MSI_FAULT_SHORT_READ) {
      p->faults.erase(f);
      p->ctr.rejections++;
      return MSI_ERR_SOURCE;
    }
  }

  // ---- LRU-wave plan (host ledger; identical rules to the slot simulator) ----
  const int call = p->calls++;
  std::vector<int> hits, misses;
  for (int e = 0; e < E; ++e) {
    if (p->h_counts[e] <= 0) continue;
    (p->where[(size_t)layer * E + e] >= 0 ? hits : misses).push_back(e);
  }
  std::vector<int> order(hits);
  order.insert(order.end(), misses.begin(), misses.end());
  // Waves are planned one at a time, just before they are staged: the rules
  // (and so the trace) are those of planning them all up front, and a bundle
  // whose read is rejected leaves no later wave planned.
  const size_t n_waves = (order.size() + p->C - 1) / p->C;
  std::vector<std::vector<WaveEntry>> waves;
  std::vector<char> pinned(d.n_slots, 0);
  std::vector<int> prev;
  auto plan_wave = [&]() -> msi_status {
    const int w = (int)waves.size();
    const size_t w0 = (size_t)w * p->C;
    std::vector<WaveEntry> wave;
    std::fill(pinned.begin(), pinned.end(), 0);
    for (int s : prev) pinned[s] = 1;
    for (size_t i = w0; i < std::min(order.size(), w0 + p->C); ++i) {
      const int e = order[i];
      int s = p->where[(size_t)layer * E + e];
      bool miss = false;
      if (s >= 0) {
        add_trace(p, call, layer, e, s, p->slots[s].gen, MSI_TRACE_HIT, w);
        p->ctr.hits++;
        if (p->slots[s].prefetched) {
          p->ctr.prefetch_hits++;
          p->slots[s].prefetched = false;
        }
      } else {
        s = pick_victim(p, pinned);
        if (s < 0) return MSI_ERR_SLOT_BUSY;  // excluded by the pin limit
        ledger_stage(p, s, layer, e, call, w);
        miss = true;
      }
      pinned[s] = 1;
      wave.push_back({e, s, miss, p->slots[s].gen});
    }
    prev.clear();
    for (const auto& we : wave) {
      p->tick += 1;
      p->slots[we.slot].last_use = p->tick;
      prev.push_back(we.slot);
    }
    waves.push_back(std::move(wave));
    return MSI_OK;
  };

  // ---- issue: plan + stage(w + 1) overlaps compute(w) ----
  auto stage_wave = [&](size_t w) -> msi_status {
    const msi_status pw = plan_wave();
    if (pw != MSI_OK) return pw;
    std::vector<WaveEntry> m;
    for (const auto& we : waves[w])
      if (we.miss) m.push_back(we);
    msi_status r = stage_enqueue(p, layer, m, ss);
    if (r == MSI_ERR_SOURCE) {
      // a rejected read: this bundle is not published and no later one is
      // planned; the bundle's slots hold nothing (each was invalidated before
      // its copies) and become Vacant in the ledger
      for (const auto& we : waves[w])
        if (we.miss) ledger_vacate(p, we.slot, call, (int)w);
    }
    return r;
  };
  if (n_waves > 0) {
    st = stage_wave(0);
    if (st != MSI_OK) return st;
  }
  static thread_local WaveParams wp;
  for (size_t w = 0; w < n_waves; ++w) {
    if (w + 1 < n_waves) {
      st = stage_wave(w + 1);
      if (st != MSI_OK) return st;
    }
    std::vector<int> used;
    int mtiles = 0;
    long long wave_rows = 0;
    wp.n = (int)waves[w].size();
    wp.layer = layer;
    for (int i = 0; i < wp.n; ++i) {
      const WaveEntry& we = waves[w][i];
      used.push_back(we.slot);
      wp.slot[i] = we.slot;
      wp.expert[i] = we.expert;
      wp.expected[i] = we.gen;
      mtiles += (p->h_counts[we.expert] + kBM - 1) / kBM;
      wave_rows += p->h_counts[we.expert];
    }
    st = wait_ready(p, used, f.cs);
    if (st != MSI_OK) return st;
    const bool fused = fused_wave(p, f, wave_rows, wp.n);
    if (!fused) {
      // split launches: the setup kernel re-checks the wave's slots and
      // builds its groups (a fused wave's kernel does both itself)
      SetupArgs sa{};
      sa.counts = ev->counts;
      sa.offsets = at<int>(ws, f.L.offsets);
      sa.genwords = p->d_gen;
      sa.E = E;
      sa.layer = layer;
      sa.groups = at<Group>(ws, f.L.groups);
      sa.total_mtiles = at<int>(ws, f.L.total);
      sa.status = at<int>(ws, f.L.status);
      LAUNCH(p, MSI_K_SETUP, f.cs, launch_setup_wave(sa, wp, f.cs));
    }
    const int g1 = std::max(1, std::min(p->sms, mtiles * (d.inter / 128)));
    const int g2 = std::max(1, std::min(p->sms, mtiles * (d.hidden / kBN)));
    st = routed_ffn(p, f, wp.n, g1, g2, wave_rows, fused ? mtiles : -1, fused ? &wp : nullptr, (int)w);
    if (st != MSI_OK) return st;
    st = consumer_record(p, used, f.cs);
    if (st != MSI_OK) return st;
    if (late_shared) {
      bool any_miss = false;
      for (const auto& we : waves[w]) any_miss = any_miss || we.miss;
      if (any_miss || w + 1 == n_waves) {
        st = shared_ffn(p, f, f.cs);
        if (st != MSI_OK) return st;
        late_shared = false;
      }
    }
  }
  if (predict) {
    // the predicted counts (the prediction ran beside the waves' GEMMs), then
    // the prefetch bundle on the stage stream, overlapping those GEMMs
    const cudaError_t pe = cudaEventSynchronize(p->ev_pjoin);
    if (pe != cudaSuccess) return cuda_fail(pe, "predicted counts readback");
    st = prefetch_bundle(p, layer + 1, call, (int)n_waves, prev, ss);
    if (st != MSI_OK) return st;
    CK(cudaStreamWaitEvent(f.cs, p->ev_pjoin, 0));
    pred_join.ev = nullptr;
  }
  st = finish(p, f);
  if (st != MSI_OK) return st;
  p->ctr.forwards++;
  p->ctr.streamed_forwards++;
  return MSI_OK;
}

}  // namespace

msi_status msi_moe_forward_streamed(msi_plan* p, int layer, const void* x, int T, const float* rw,
                                    void* out, const msi_route_event* ev, void* ws, size_t ws_bytes,
                                    unsigned flags, msi_stream compute, msi_stream stage) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  return forward_streamed(p, layer, x, T, rw, out, ev, nullptr, nullptr, ws, ws_bytes, flags, compute,
                          stage);
}

msi_status msi_moe_forward_streamed_stack(msi_plan* p, int layer0, int n, const void* x, int T,
                                          const float* const* rw, void* out_a, void* out_b,
                                          const msi_route_event* evs, void* ws, size_t ws_bytes,
                                          unsigned flags, msi_stream compute, msi_stream stage, int* done) {
  if (done != nullptr) *done = 0;
  if (p == nullptr || n < 0 || (n > 0 && (rw == nullptr || evs == nullptr)) || out_a == nullptr ||
      out_b == nullptr || out_a == out_b || out_a == x || out_b == x)
    return MSI_ERR_INVALID_ARG;
  if (layer0 < 0 || (long long)layer0 + n > p->d.n_layers) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  const void* in = x;
  for (int i = 0; i < n; ++i) {
    void* out = (i & 1) ? out_b : out_a;
    const msi_status st = forward_streamed(p, layer0 + i, in, T, rw[i], out, &evs[i], nullptr, nullptr, ws,
                                           ws_bytes, flags, compute, stage);
    if (st != MSI_OK) return st;
    if (done != nullptr) *done = i + 1;
    in = out;
  }
  return MSI_OK;
}

msi_status msi_moe_forward_streamed_next(msi_plan* p, int layer, const void* x, int T, const float* rw,
                                         void* out, const msi_route_event* ev, const float* next_rw,
                                         const msi_route_event* next_ev, void* ws, size_t ws_bytes,
                                         unsigned flags, msi_stream compute, msi_stream stage) {
  if (p == nullptr || next_rw == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  return forward_streamed(p, layer, x, T, rw, out, ev, next_rw, next_ev, ws, ws_bytes, flags, compute,
                          stage);
}

namespace {

size_t rows_bytes(const msi_plan* p, int T) {
  return ((size_t)T * p->d.hidden * 2 + 255) / 256 * 256;
}

// Host-buffer call, first half: the rows go into the workspace tail on the
// copy stream (forked from `compute`); x_dev / out_dev are the device row
// buffers the forward then uses with h (x_ready, out_host) set.
msi_status host_begin(msi_plan* p, int T, const void* hidden_host, void* out_host, void* ws,
                      size_t ws_bytes, cudaStream_t cs, HostIO* h, void** x_dev, void** out_dev) {
  if (T < 0 || (T > 0 && (hidden_host == nullptr || out_host == nullptr))) return MSI_ERR_INVALID_ARG;
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  msi_status dst = check_device(p);
  if (dst != MSI_OK) return dst;
  const size_t base = layout(p, T).bytes, rb = rows_bytes(p, T);
  if (ws == nullptr || (uintptr_t)ws % 256 || ws_bytes < base + 2 * rb) return MSI_ERR_WORKSPACE;
  if (p->io == nullptr) {
    // created into locals and kept only all together (see prediction_resources)
    cudaStream_t s = nullptr;
    cudaEvent_t ea = nullptr, eb = nullptr;
    cudaError_t e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ea, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&eb, cudaEventDisableTiming);
    if (e != cudaSuccess) {
      if (s) cudaStreamDestroy(s);
      if (ea) cudaEventDestroy(ea);
      if (eb) cudaEventDestroy(eb);
      return cuda_fail(e, "copy stream");
    }
    p->io = s;
    p->ev_io_a = ea;
    p->ev_io_b = eb;
  }
  *x_dev = static_cast<char*>(ws) + base;
  *out_dev = static_cast<char*>(ws) + base + rb;
  *h = HostIO{p->io, nullptr, T > 0 ? out_host : nullptr, nullptr};
  CK(cudaEventRecord(p->ev_io_a, cs));
  CK(cudaStreamWaitEvent(p->io, p->ev_io_a, 0));
  if (T > 0) {
    CK(cudaMemcpyAsync(*x_dev, hidden_host, (size_t)T * p->d.hidden * 2, cudaMemcpyHostToDevice, p->io));
    CK(cudaEventRecord(p->ev_io_b, p->io));
    h->x_ready = p->ev_io_b;
  }
  return MSI_OK;
}

// Second half: the copy stream joins `compute` (also after a failed forward,
// so that no copy outlives the call's place in the compute stream).
msi_status host_end(msi_plan* p, cudaStream_t cs, msi_status st) {
  CK(cudaEventRecord(p->ev_io_b, p->io));
  CK(cudaStreamWaitEvent(cs, p->ev_io_b, 0));
  return st;
}

}  // namespace

msi_status msi_workspace_size_host(const msi_plan* p, int T, size_t* bytes) {
  if (p == nullptr || bytes == nullptr || T < 0) return MSI_ERR_INVALID_ARG;
  *bytes = layout(p, T).bytes + 2 * rows_bytes(p, T);
  return MSI_OK;
}

msi_status msi_moe_forward_host(msi_plan* p, int layer, const void* hidden_host, int T,
                                const float* rw, const int32_t* table, const uint64_t* expected,
                                void* out_host, int32_t* ids_host, const msi_route_event* ev,
                                void* ws, size_t ws_bytes, unsigned flags, msi_stream compute) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(compute);
  HostIO h{};
  void *x = nullptr, *out = nullptr;
  msi_status st = host_begin(p, T, hidden_host, out_host, ws, ws_bytes, cs, &h, &x, &out);
  if (st != MSI_OK) return st;
  h.ids_host = T > 0 ? ids_host : nullptr;
  st = forward_resident(p, layer, x, T, rw, table, expected, out, ev, ws, ws_bytes, flags, compute, &h);
  return host_end(p, cs, st);
}

msi_status msi_moe_forward_streamed_host(msi_plan* p, int layer, const void* hidden_host, int T,
                                         const float* rw, void* out_host, int32_t* ids_host,
                                         const msi_route_event* ev, void* ws, size_t ws_bytes,
                                         unsigned flags, msi_stream compute, msi_stream stage) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(compute);
  HostIO h{};
  void *x = nullptr, *out = nullptr;
  msi_status st = host_begin(p, T, hidden_host, out_host, ws, ws_bytes, cs, &h, &x, &out);
  if (st != MSI_OK) return st;
  h.ids_host = T > 0 ? ids_host : nullptr;
  st = forward_streamed(p, layer, x, T, rw, out, ev, nullptr, nullptr, ws, ws_bytes, flags, compute,
                        stage, &h);
  return host_end(p, cs, st);
}

msi_status msi_plan_pin(msi_plan* p, int layer, int expert, int pinned) {
  if (p == nullptr || layer < 0 || expert < 0) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (layer >= p->d.n_layers || expert >= p->d.n_experts) return MSI_ERR_INVALID_ARG;
  char& o = p->pinned_obj[(size_t)layer * p->d.n_experts + expert];
  const bool on = pinned != 0;
  if (on == (o != 0)) return MSI_OK;
  if (on && p->n_pins + 1 > p->d.n_slots - 2 * p->C) return MSI_ERR_SLOT_BUSY;
  o = on ? 1 : 0;
  p->n_pins += on ? 1 : -1;
  return MSI_OK;
}

msi_status msi_forward_status(msi_plan* p, int* device_status) {
  if (p == nullptr || device_status == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (p->fwd_ev < 0) {
    *device_status = MSI_OK;
    return MSI_OK;
  }
  CK(cudaEventSynchronize(p->pool.ev[p->fwd_ev]));
  *device_status = *p->h_status;
  if (*device_status != MSI_OK) p->ctr.rejections++;
  return MSI_OK;
}

msi_status msi_plan_reset(msi_plan* p, uint64_t* new_epoch) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  msi_status dst = check_device(p);
  if (dst != MSI_OK) return dst;
  for (auto& h : p->holds)
    if (h.load() > 0) return MSI_ERR_SLOT_BUSY;
  // drain: every outstanding stage, consumer and forward
  for (auto& sl : p->slots) {
    if (sl.ready >= 0) CK(cudaEventSynchronize(p->pool.ev[sl.ready]));
    if (sl.consumer >= 0) CK(cudaEventSynchronize(p->pool.ev[sl.consumer]));
  }
  if (p->fwd_ev >= 0) CK(cudaEventSynchronize(p->pool.ev[p->fwd_ev]));
  // invalidate: nothing published before the reset can pass a check after it
  CK(cudaMemset(p->d_gen, 0, sizeof(GenWord) * p->d.n_slots));
  const int E = p->d.n_experts;
  for (int s = 0; s < p->d.n_slots; ++s) {
    Slot& sl = p->slots[s];
    if (sl.layer >= 0) {
      add_trace(p, -1, sl.layer, sl.expert, s, sl.gen, MSI_TRACE_EVICT, -1);
      p->where[(size_t)sl.layer * E + sl.expert] = -1;
      p->ctr.evicts++;
    }
    sl.layer = sl.expert = -1;
    sl.last_use = -1;
    sl.prefetched = false;
    p->pool.unref(sl.ready);
    p->pool.unref(sl.consumer);
    sl.ready = sl.consumer = -1;
  }
  p->tick = 0;
  p->epoch++;
  if (new_epoch) *new_epoch = p->epoch;
  return MSI_OK;
}

msi_status msi_plan_set_source(msi_plan* p, msi_source* src, const uint64_t* file_off) {
  if (p == nullptr || (src != nullptr && file_off == nullptr)) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  if (p->src != src) {
    source_attach(p->src, -1);
    source_attach(src, +1);
  }
  p->src = src;
  p->src_off.clear();
  if (src != nullptr)
    p->src_off.assign(file_off, file_off + (size_t)p->d.n_layers * p->d.n_experts);
  return MSI_OK;
}

msi_status msi_fault_inject(msi_plan* p, int kind, int layer, int expert) {
  if (p == nullptr || layer < 0 || layer >= p->d.n_layers || expert < 0 ||
      expert >= p->d.n_experts)
    return MSI_ERR_INVALID_ARG;
  if (kind != MSI_FAULT_SHORT_READ && kind != MSI_FAULT_STALE_COMPLETION &&
      kind != MSI_FAULT_WRONG_OBJECT && kind != MSI_FAULT_IO_ERROR && kind != MSI_FAULT_STALE_EPOCH &&
      kind != MSI_FAULT_DEVICE_WAIT)
    return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (kind == MSI_FAULT_DEVICE_WAIT)
    p->stall_layer = layer;
  else
    p->faults[obj_key(layer, expert)] = kind;
  return MSI_OK;
}

msi_status msi_plan_set_bounce(msi_plan* p, void* buf, size_t bytes) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  if (buf == nullptr) {
    // the caller may free the buffer once the calls that used it completed
    if (p->ev_bounce != nullptr) CK(cudaEventSynchronize(p->ev_bounce));
    p->bounce = nullptr;
    p->bounce_cap = 0;
    return MSI_OK;
  }
  if ((uintptr_t)buf % 16 || bytes < p->d.extent_bytes) return MSI_ERR_INVALID_ARG;
  msi_status dst = check_device(p);
  if (dst != MSI_OK) return dst;
  if (p->ev_bounce == nullptr) {
    cudaEvent_t e = nullptr;
    CK(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
    p->ev_bounce = e;
  } else {
    CK(cudaEventSynchronize(p->ev_bounce));
  }
  p->bounce = static_cast<char*>(buf);
  p->bounce_cap = (int)std::min<uint64_t>(bytes / p->d.extent_bytes, (uint64_t)p->C);
  p->spec_idx.assign(p->d.n_experts, -1);
  return MSI_OK;
}

msi_status msi_plan_set_wait_cycles(msi_plan* p, int64_t cycles) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  p->wait_cycles = cycles > 0 ? (long long)cycles : kDeviceWaitCycles;
  return MSI_OK;
}

msi_status msi_consumer_hold(msi_plan* p, int slot) {
  if (p == nullptr || slot < 0 || slot >= p->d.n_slots) return MSI_ERR_INVALID_ARG;
  if (p->dying) return MSI_ERR_SHUT_DOWN;
  p->holds[slot].fetch_add(1);
  return MSI_OK;
}

msi_status msi_consumer_release(msi_plan* p, int slot) {
  if (p == nullptr || slot < 0 || slot >= p->d.n_slots) return MSI_ERR_INVALID_ARG;
  int cur = p->holds[slot].load();
  while (cur > 0 && !p->holds[slot].compare_exchange_weak(cur, cur - 1)) {
  }
  return cur > 0 ? MSI_OK : MSI_ERR_INVALID_ARG;
}

msi_status msi_trace_read(const msi_plan* cp, msi_trace_rec* buf, size_t cap, size_t* n) {
  msi_plan* p = const_cast<msi_plan*>(cp);
  if (p == nullptr || n == nullptr || (buf == nullptr && cap > 0)) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  const size_t m = std::min(cap, p->trace.size());
  if (m) std::memcpy(buf, p->trace.data(), m * sizeof(msi_trace_rec));
  *n = m;
  return MSI_OK;
}

msi_status msi_trace_clear(msi_plan* p) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  p->trace.clear();
  return MSI_OK;
}

msi_status msi_get_counters(const msi_plan* cp, msi_counters* out) {
  msi_plan* p = const_cast<msi_plan*>(cp);
  if (p == nullptr || out == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  *out = p->ctr;
  return MSI_OK;
}

uint64_t msi_kernel_launches(const msi_plan* p) { return p ? p->launches : 0; }

msi_status msi_timing_enable(msi_plan* p, int on) {
  if (p == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  p->timer.on = on != 0;
  return MSI_OK;
}

msi_status msi_timing_read(msi_plan* p, double* ms, uint64_t* launches, int reset) {
  if (p == nullptr || ms == nullptr || launches == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(p->mu);
  p->timer.resolve();
  for (int k = 0; k < MSI_K_COUNT; ++k) {
    ms[k] = p->timer.ms[k];
    launches[k] = p->timer.n[k];
    if (reset) {
      p->timer.ms[k] = 0.0;
      p->timer.n[k] = 0;
    }
  }
  return MSI_OK;
}

}  // extern "C"
