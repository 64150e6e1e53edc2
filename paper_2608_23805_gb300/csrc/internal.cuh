// Internal declarations shared by the library's translation units: limits,
// the generation word and GEMM group, the grouped GEMM's argument block,
// tiling and launchers, and the PTX wrappers for sm_103a (mbarrier, TMA,
// tcgen05, cp.async).  The other kernels' argument blocks and launchers are
// in kernels.cuh.  Nothing here is part of the public C ABI (include/msi.h).
#pragma once

#include <atomic>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/msi.h"

namespace msi {

// Raise a kernel's dynamic shared-memory limit once per device (the attribute
// belongs to the device's context); `done` holds one bit per device ordinal.
template <typename K>
inline cudaError_t smem_attr_once(K* kernel, int bytes, std::atomic<unsigned long long>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = dev < 64 ? 1ull << dev : 0ull;
  if (bit != 0 && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit != 0) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// ---------------------------------------------------------------------------
// Limits of the kernels
// ---------------------------------------------------------------------------
constexpr int kMaxExperts = 512;
constexpr int kMaxTopK = 32;
constexpr int kMaxWave = 256;

// After an expired wait (abort), a CTA still waits for the TMA loads and MMAs
// it issued before releasing shared memory and TMEM.  Those always complete
// within microseconds, so that drain has its own bound (~10 ms at 2 GHz),
// independent of the wait limit that expired (which may be short).
constexpr long long kDrainCycles = 20000000LL;

// ---------------------------------------------------------------------------
// Device-side records
// ---------------------------------------------------------------------------

// Published identity of one slot: written on the staging stream after the
// extent copy (obj = 0 while a copy is in flight or the slot is vacant).
struct GenWord {
  unsigned long long gen;
  unsigned long long obj;  // ((layer + 1) << 32) | expert
};

__host__ __device__ inline unsigned long long obj_key(int layer, int expert) {
  return ((unsigned long long)(layer + 1) << 32) | (unsigned)expert;
}

// One expert group of a grouped GEMM launch.
struct Group {
  int row_begin;   // first permuted row
  int row_count;   // rows routed to the expert
  int slot;        // weight block index in the B tensor maps
  int mt_begin;    // prefix of 128-row tiles over the preceding groups
  int ok;          // generation re-check passed
  int expert;
  int pt_begin;    // prefix of 256-row (CTA-pair) tiles over the preceding groups
  int pad1;
};

// ---------------------------------------------------------------------------
// Grouped GEMM argument block (the other kernels' blocks: kernels.cuh)
// ---------------------------------------------------------------------------
struct GemmArgs {
  const Group* groups;
  int num_groups;
  const int* total_mtiles;  // device: [0] 128-row tiles, [1] 256-row pair tiles
  int nt;                   // N tiles per group
  int kblocks;              // K / 64
  int b_rows_per_slot;      // rows of one weight block in the B tensor map
  int b_row_off;            // row offset of the operand inside the block
  int up_off;               // gate-up: row offset of the up rows (I)
  int out_ld;               // output row length (elements)
  __nv_bfloat16* out;
  const __nv_bfloat16* x;   // gather source rows [T, H]
  int x_ld;
  const int* perm;          // permuted row -> t*k + j
  int top_k;
  int* status;
  long long wait_limit;     // clock64 cycles per bounded wait
  // non-zero: the epilogue's first thread also waits on a barrier nothing
  // arrives at (a host-armed test of the expiry path: the wait runs out after
  // wait_limit, the CTA aborts, drains and reports MSI_ERR_TIMEOUT)
  int stall;
  // 4-bit weights (q4 modes): codes and fp16 scales read from the slot pool
  const uint8_t* q4_pool;
  unsigned long long q4_extent;  // bytes per slot
  int q4_rows_per_slot;          // rows of the code tensor map per slot (extent / row bytes)
  int q4_row_off;                // first code row of this operand inside a slot
  long long q4_scale_off;        // byte offset of this operand's scales in an extent
  int q4_scale_ld;               // bytes per weight row of scales (K / 16)
};

enum GemmMode { kGateUpGather = 0, kGateUpTma = 1, kDown = 2, kGateUpGatherQ4 = 3, kDownQ4 = 4 };

// One LRU wave's experts: slot, expert id and the generation each must hold
// (kernel parameter, by value).
struct WaveParams {
  int n;
  int layer;
  int slot[kMaxWave];
  int expert[kMaxWave];
  unsigned long long expected[kMaxWave];
};

// One wave's gate-up and down projections in one launch (gemm_fused.cu).
struct FusedArgs {
  const Group* groups;
  int num_groups;
  const int* total_mtiles;  // device: [0] 128-row tiles
  int nt_up, nt_dn;         // column tiles: I / 128 (h), H / 256 (y)
  int kb_up, kb_dn;         // K blocks: H / 64, I / 64
  int w13_rows_per_slot;    // rows of one slot in the W13 map (3 I); gate rows at n * 128
  int w13_up_off;           // up rows after the gate rows (I)
  int w2_rows_per_slot;     // rows of one slot in the W2 map (3 H)
  int w2_row_off;           // W2 after W13 inside a slot (2 H rows of I)
  __nv_bfloat16* h;         // [T k, I]
  int h_ld;
  __nv_bfloat16* y;         // [T k, H]
  int y_ld;
  const __nv_bfloat16* x;   // [T, H]
  int x_ld;
  const int* perm;          // permuted row -> t k + j
  int top_k;
  int* ready;               // [m-tiles] finished gate-up tiles per 128-row tile (zero at launch)
  int* status;
  long long wait_limit;
  int stall;                // as GemmArgs::stall
  // wave mode (wave != 0): the kernel builds the wave's groups itself from the
  // call's counts and offsets and the WaveParams (the generation re-check of
  // every slot, fail closed), and zeroes ready_clear[0, n_ready_clear) for the
  // next wave (the counters of the previous one); groups / total_mtiles unused
  int wave;
  const int* counts;        // [E] rows per expert
  const int* offsets;       // [E + 1] first permuted row per expert
  const GenWord* genwords;  // published (generation, object) per slot
  int* ready_clear;
  int n_ready_clear;
  int sched_w;              // FusedSched: down tiles one gate-up tile is worth (>= 1)
  // 4-bit waves (gemm_fused_pair.cu, Q4): codes by TMA through the code maps,
  // fp16 scales read from the slot pool
  const uint8_t* q4_pool;
  unsigned long long q4_extent;   // bytes per slot
  int q13_rows_per_slot;          // W13 code rows (H / 2 bytes each) per slot
  int q2_rows_per_slot;           // W2 code rows (I / 2 bytes each) per slot
  int q2_row_off;                 // first W2 code row inside a slot
  long long q13_scale_off;        // byte offset of the W13 scales in an extent
  int q13_scale_ld;               // bytes of scales per W13 row (H / 16)
  long long q2_scale_off;         // byte offset of the W2 scales in an extent
  int q2_scale_ld;                // bytes of scales per W2 row (I / 16)
};

// ---------------------------------------------------------------------------
// Launchers (return cudaError_t of the launch)
// ---------------------------------------------------------------------------
cudaError_t launch_gemm(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                        const GemmArgs& a, int grid, cudaStream_t s);
// CTA-pair variant (tcgen05 cta_group::2, 256 x 256 tiles) of kGateUpGather,
// kGateUpTma and kDown; `max_pairs` bounds the pairs launched.
cudaError_t launch_gemm_pair(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                             const GemmArgs& a, int max_pairs, cudaStream_t s);
// Gate-up and down of one wave in one cooperative launch of `grid` CTAs
// (at most one per SM); tmW13 / tmW2 as the pool maps of the two projections.
cudaError_t launch_fused_wave(const CUtensorMap& tmW13, const CUtensorMap& tmW2, const CUtensorMap& tmH,
                              const FusedArgs& a, const WaveParams& w, int grid, cudaStream_t s);
// The same on CTA pairs (256-row tiles, gemm_fused_pair.cu); at most
// `max_pairs` pairs, never more than can be resident at once.
cudaError_t launch_fused_wave_pair(const CUtensorMap& tmW13, const CUtensorMap& tmW2,
                                   const FusedArgs& a, const WaveParams& w, int max_pairs, cudaStream_t s);
// 4-bit waves on CTA pairs (tmQ13 / tmQ2: the byte-granular code maps).
cudaError_t launch_fused_wave_pair_q4(const CUtensorMap& tmQ13, const CUtensorMap& tmQ2,
                                      const FusedArgs& a, const WaveParams& w, int max_pairs, cudaStream_t s);

// GEMM tiling
constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kBK = 64;
constexpr int kStages = 4;
constexpr int kABytes = kBM * kBK * 2;
constexpr int kBBytes = kBN * kBK * 2;

// ---------------------------------------------------------------------------
// PTX wrappers (device)
// ---------------------------------------------------------------------------
#if defined(__CUDACC__)

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// explicit shared-space accesses for the dequant warps' operand writes and
// code reads (a generic access to shared memory takes the generic path)
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

__device__ __forceinline__ uint2 ld_shared_v2(uint32_t addr) {
  uint2 v;
  asm volatile("ld.shared.v2.b32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Static tile schedule of the fused kernels.  U gate-up tiles (indices
// 0..U-1) then D down tiles (U..U+D-1) over P workers (CTAs, or CTA pairs).
// Gate-up tiles go round-robin: worker c takes c, c + P, ...; the first
// U mod P workers get one more than the rest.  A gate-up tile is worth w
// down tiles, so the down tiles first make up that difference (phase A: the
// first w * (P - U mod P) down tiles round-robin over the workers with one
// gate-up tile fewer), then go round-robin over all workers (phase B).
// Every tile has exactly one worker, and every worker runs its gate-up
// tiles first and then its down tiles, each in increasing index order.
struct FusedSched {
  int U, D, P, c, n_hi, n_lo, DA;
  __host__ __device__ __forceinline__ FusedSched(int U_, int D_, int P_, int c_, int w)
      : U(U_), D(D_), P(P_), c(c_) {
    n_hi = U % P;
    n_lo = P - n_hi;
    DA = n_hi > 0 ? (D < w * n_lo ? D : w * n_lo) : 0;
  }
  // the worker's first down tile, or -1
  __host__ __device__ __forceinline__ int down_first() const {
    if (c >= n_hi && c - n_hi < DA) return U + (c - n_hi);
    const int i = DA + c;
    return i < D ? U + i : -1;
  }
  __host__ __device__ __forceinline__ int first() const { return c < U ? c : down_first(); }
  // the worker's tile after t, or -1
  __host__ __device__ __forceinline__ int next(int t) const {
    if (t < U) return t + P < U ? t + P : down_first();
    const int i = t - U;
    if (i < DA) {
      if (i + n_lo < DA) return t + n_lo;
      return DA + c < D ? U + DA + c : -1;
    }
    return i + P < D ? t + P : -1;
  }
};

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and raises the CTA's abort flag) when the wait
// exceeds `limit` clock64 cycles or another role already aborted.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) {
      *abort_flag = 1;
      return false;
    }
  }
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_prefetch(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// 2-D tiled TMA load global -> shared, completion counted on `bar` (bytes).
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int c0,
                                            int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
// Arrive on `bar` (counted as one expected arrival) once all of this thread's
// earlier cp.async copies have completed.
__device__ __forceinline__ void cp_async_arrive_noinc(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// --- tcgen05 (5th-generation tensor cores, accumulators in TMEM) ---
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// --- clusters of two CTAs (tcgen05 cta_group::2) ---
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// shared::cluster address of the object at `saddr` (shared::cta) in CTA `rank`
__device__ __forceinline__ uint32_t mapa_shared(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
// Arrive on a barrier of a CTA of this cluster (shared::cluster address).
// Default semantics (release, CTA scope), as for a local arrive: the pair
// protocol orders data through the barriers' own completion mechanisms (TMA
// transaction counts, tcgen05.commit), so no cluster-wide fence is needed on
// the per-stage path.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// Every thread of both CTAs of the cluster.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Issued by one warp in each CTA of the pair.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// Pair MMA, issued by the even CTA: A rows and B rows (N) come half from each
// CTA's shared memory at the same offsets; each CTA's TMEM receives its rows.
__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on the barrier at `bar`'s offset in both CTAs when all earlier
// pair MMAs of this thread complete.
__device__ __forceinline__ void umma_commit_pair(uint64_t* bar) {
  const uint16_t mask = 3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
      "[%0], %1;" ::"r"(smem_u32(bar)),
      "h"(mask)
      : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once all previously issued tcgen05 ops of this thread complete.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns; the wait carries the registers so
// that no use can be scheduled before the load completes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, "
      "%30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
// Wait for this thread's TMEM loads; the registers pass through the wait so
// that no use is scheduled before it.
template <int N>
__device__ __forceinline__ void tmem_wait_regs(uint32_t (&r)[N]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+r"(r[i]));
}
// 32-byte global store (one full sector), 32-byte aligned address.
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t* v) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(v[0]),
               "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
               : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes grouped in 8-row (1024-byte) atoms.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4)      // start address
         | ((uint64_t)1 << 16)                    // leading byte offset (unused for SW128 K-major)
         | ((uint64_t)(1024 >> 4) << 32)          // stride byte offset: 8 rows x 128 B
         | ((uint64_t)1 << 46)                    // descriptor version (sm_100 family)
         | ((uint64_t)2 << 61);                   // swizzle mode: 128 B
}

// Instruction descriptor of kind::f16: D fp32, A and B bf16, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Epilogue of one accumulator tile for the thread's token row, output
// columns [c0, c1): TMEM columns at tb to bf16 at dst (32-byte aligned),
// stored when `valid`.
//   gate-up: TMEM columns 0-127 hold x.Wg^T and 128-255 x.Wu^T of the same
//            128 intermediate units; h = silu(g) * u = g * u / (1 + e^-g);
//            c0, c1 are h columns (multiples of 32, <= 128).
//   down:    output column c is TMEM column c (multiples of 64, <= 256).
// TMEM is read 64 columns per wait and each store fills a 32-byte sector.
template <bool GATEUP>
__device__ __forceinline__ void epilogue_cols(uint32_t tb, __nv_bfloat16* dst, bool valid, int c0,
                                              int c1) {
  if (GATEUP) {
#pragma unroll 1
    for (int c = c0; c < c1; c += 32) {
      uint32_t g[32], u[32];
      tmem_ld32(tb + c, g);
      tmem_ld32(tb + 128 + c, u);
      tmem_wait_regs(g);
      tmem_wait_regs(u);
      uint32_t p[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
        const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
        // approximate divide (2 ulp): far below the bf16 rounding of h; an
        // infinite e^-g (g < -88) gives 0, the limit of silu
        p[i] = pack_bf16x2(__fdividef(g0 * u0, 1.0f + __expf(-g0)),
                           __fdividef(g1 * u1, 1.0f + __expf(-g1)));
      }
      if (valid) {
        st_global_v8(dst + c, p);
        st_global_v8(dst + c + 16, p + 8);
      }
    }
  } else {
#pragma unroll 1
    for (int c = c0; c < c1; c += 64) {
      uint32_t v[32], w[32];
      tmem_ld32(tb + c, v);
      tmem_ld32(tb + c + 32, w);
      tmem_wait_regs(v);
      tmem_wait_regs(w);
      uint32_t p[32];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        p[i] = pack_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
        p[16 + i] = pack_bf16x2(__uint_as_float(w[2 * i]), __uint_as_float(w[2 * i + 1]));
      }
      if (valid) {
#pragma unroll
        for (int q = 0; q < 4; ++q) st_global_v8(dst + c + 16 * q, p + 8 * q);
      }
    }
  }
}

// The whole tile for the thread's row.
template <bool GATEUP>
__device__ __forceinline__ void epilogue_tile(uint32_t tb, __nv_bfloat16* dst, bool valid) {
  epilogue_cols<GATEUP>(tb, dst, valid, 0, GATEUP ? 128 : 256);
}

// Store 32 rows of RB bytes each, held one row per lane (16-byte words in p),
// through the warp's shared-memory staging buffer (32 x RB bytes, chunks
// XOR-swizzled by row): read back eight lanes per 128 bytes of a row, so each
// global store instruction covers whole rows (RB = 128: four rows of 128 B;
// RB = 64: eight rows of 64 B) instead of one 16-32 B piece of 32 rows.
// The swizzle key of row r is (r >> log2(8 / Q)) mod Q (Q chunks a row): the
// eight lanes that share one 16-byte store wavefront then reach eight
// different 16-byte bank groups, in the row-per-lane writes as in the
// row-major reads.
// Rows >= nvalid (past the expert's segment) are not stored.
template <int RB>
__device__ __forceinline__ void store_rows_staged(const uint32_t* p, uint8_t* stg,
                                                  __nv_bfloat16* row0, size_t ld, int nvalid,
                                                  int lane) {
  constexpr int Q = RB / 16;  // 16-byte chunks per row
  static_assert(Q == 2 || Q == 4 || Q == 8, "staged rows of 32, 64 or 128 bytes");
  constexpr int kShift = Q == 2 ? 2 : (Q == 4 ? 1 : 0);
  const int key = (lane >> kShift) & (Q - 1);
#pragma unroll
  for (int q = 0; q < Q; ++q)
    *reinterpret_cast<uint4*>(stg + lane * RB + ((q ^ key) << 4)) =
        make_uint4(p[4 * q], p[4 * q + 1], p[4 * q + 2], p[4 * q + 3]);
  __syncwarp();
#pragma unroll
  for (int it = 0; it < Q; ++it) {
    const int idx = it * 32 + lane;
    const int row = idx / Q, q = idx % Q;
    const uint4 v = *reinterpret_cast<const uint4*>(stg + row * RB + ((q ^ ((row >> kShift) & (Q - 1))) << 4));
    if (row < nvalid)
      *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(row0 + (size_t)row * ld) + q * 16) = v;
  }
  __syncwarp();
}

// Whole-tile epilogue of one warp (32 token rows, TMEM lanes of the warp's
// quarter) with staged, row-coalesced stores.  row0: output of the warp's
// first row at the tile's first column; nvalid: rows of the 32 inside the
// expert's segment; stg: the warp's 4 KB staging buffer.
template <bool GATEUP>
__device__ __forceinline__ void epilogue_tile_staged(uint32_t tb, __nv_bfloat16* row0, size_t ld,
                                                     int nvalid, uint8_t* stg, int lane) {
  if (GATEUP) {
#pragma unroll 1
    for (int c = 0; c < 128; c += 32) {
      uint32_t g[32], u[32];
      tmem_ld32(tb + c, g);
      tmem_ld32(tb + 128 + c, u);
      tmem_wait_regs(g);
      tmem_wait_regs(u);
      uint32_t p[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
        const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
        p[i] = pack_bf16x2(__fdividef(g0 * u0, 1.0f + __expf(-g0)),
                           __fdividef(g1 * u1, 1.0f + __expf(-g1)));
      }
      store_rows_staged<64>(p, stg, row0 + c, ld, nvalid, lane);
    }
  } else {
#pragma unroll 1
    for (int c = 0; c < 256; c += 64) {
      uint32_t v[32], w[32];
      tmem_ld32(tb + c, v);
      tmem_ld32(tb + c + 32, w);
      tmem_wait_regs(v);
      tmem_wait_regs(w);
      uint32_t p[32];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        p[i] = pack_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
        p[16 + i] = pack_bf16x2(__uint_as_float(w[2 * i]), __uint_as_float(w[2 * i + 1]));
      }
      store_rows_staged<128>(p, stg, row0 + c, ld, nvalid, lane);
    }
  }
}

// The staged epilogue of one warp's 32 rows, TMEM read 16 columns at a time
// (the 4-bit modes' thread count leaves 72 registers a thread;
// CTA-pair kernels).
template <bool GATEUP>
__device__ __forceinline__ void epilogue_tile_staged_lean(uint32_t tb, __nv_bfloat16* row0, size_t ld,
                                                          int nvalid, uint8_t* stg, int lane) {
  if (GATEUP) {
#pragma unroll 1
    for (int c = 0; c < 128; c += 16) {
      uint32_t g[16], u[16];
      tmem_ld16(tb + c, g);
      tmem_ld16(tb + 128 + c, u);
      tmem_ld_wait(g);
      tmem_ld_wait(u);
      uint32_t p[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
        const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
        p[i] = pack_bf16x2(__fdividef(g0 * u0, 1.0f + __expf(-g0)),
                           __fdividef(g1 * u1, 1.0f + __expf(-g1)));
      }
      store_rows_staged<32>(p, stg, row0 + c, ld, nvalid, lane);
    }
  } else {
#pragma unroll 1
    for (int c = 0; c < kBN; c += 16) {
      uint32_t v[16];
      tmem_ld16(tb + c, v);
      tmem_ld_wait(v);
      uint32_t p[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) p[i] = pack_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
      store_rows_staged<32>(p, stg, row0 + c, ld, nvalid, lane);
    }
  }
}

// ---------------------------------------------------------------------------
// 4-bit weights (both GEMM kernels)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  uint64_t v;
  asm("mov.b64 %0, {%1, %2};" : "=l"(v) : "r"(__float_as_uint(lo)), "r"(__float_as_uint(hi)));
  return v;
}

// Eight 4-bit codes of one 32-bit word (code 2i in the low nibble of byte i,
// code 2i+1 in its high nibble) -> eight bf16 weights scale * (q - 8), the
// 16-byte chunk of one K-major row.  Each code becomes the float 128 + q by
// placing its byte under the exponent byte 0x43 (one byte permute; q < 16
// fills the top mantissa bits); one fused multiply-add per two values then
// gives (128 + q) * s - 136 * s = (q - 8) * s exactly (the product needs at
// most 8 + 11 bits and the fp16-exact scale times 136 is exact in fp32), and
// each weight is rounded once to bf16.  nbias2 holds -136 * s twice.
__device__ __forceinline__ uint4 dequant8(uint32_t w, uint64_t scale2, uint64_t nbias2) {
  const uint32_t lo = w & 0x0F0F0F0Fu, hi = (w >> 4) & 0x0F0F0F0Fu;
  uint32_t o[4];
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    uint32_t el, eh;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(el) : "r"(lo), "r"(0x43000000u), "r"(0x7044u + (b << 8)));
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(eh) : "r"(hi), "r"(0x43000000u), "r"(0x7044u + (b << 8)));
    uint64_t v;
    asm("mov.b64 %0, {%1, %2};" : "=l"(v) : "r"(el), "r"(eh));
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(v) : "l"(v), "l"(scale2), "l"(nbias2));
    uint32_t vl, vh;
    asm("mov.b64 {%0, %1}, %2;" : "=r"(vl), "=r"(vh) : "l"(v));
    // the first operand lands in the upper half: (odd column, even column)
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(o[b]) : "r"(vh), "r"(vl));
  }
  return make_uint4(o[0], o[1], o[2], o[3]);
}

// Shared-memory group table of a fused launch, read by every role: tile
// prefix s_mt[0..ng] (s_mt[ng] = tiles), slot, first permuted row and rows
// per group.  Wave mode builds it from the wave (the generation re-check of
// each slot: a group whose slot does not hold the expected object and
// version gets no tiles, and CTA 0 records the lowest such expert's status,
// fail closed); otherwise it is read from the groups in global memory.
// tile_rows: 128 (single-CTA tiles) or 256 (pair tiles).  Every thread of the
// CTA calls it (blockDim >= kMaxWave); returns the number of groups.
__device__ __forceinline__ int fused_group_table(const FusedArgs& a, const WaveParams& w, int tile_rows,
                                                 bool record, int* s_mt, int* s_slot, int* s_rb,
                                                 int* s_cnt, int* s_tmp) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (!a.wave) {
    for (int g = tid; g < a.num_groups; g += blockDim.x) {
      const Group G = a.groups[g];
      s_mt[g] = tile_rows == kBM ? G.mt_begin : G.pt_begin;
      s_slot[g] = G.slot;
      s_rb[g] = G.row_begin;
      s_cnt[g] = G.row_count;
    }
    if (tid == 0) s_mt[a.num_groups] = __ldg(a.total_mtiles + (tile_rows == kBM ? 0 : 1));
    return a.num_groups;
  }
  const int n = w.n;
  int e = 0, cnt = 0, slot = 0, code = 0;
  if (tid < n) {
    e = w.expert[tid];
    cnt = __ldg(&a.counts[e]);
    slot = w.slot[tid];
    if (cnt > 0) {
      if (slot < 0) {
        code = MSI_ERR_NOT_RESIDENT;
      } else {
        const unsigned long long obj = a.genwords[slot].obj;
        const unsigned long long gen = a.genwords[slot].gen;
        if (obj != obj_key(w.layer, e)) code = MSI_ERR_WRONG_OBJECT;
        else if (gen != w.expected[tid]) code = MSI_ERR_STALE_GENERATION;
      }
    }
  }
  const int mt = (tid < n && code == 0) ? (cnt + tile_rows - 1) / tile_rows : 0;
  // exclusive scan of mt over the block; lowest failing expert
  int incl = mt;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  int key = code ? (e << 4) | code : 0x7fffffff;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) key = min(key, __shfl_xor_sync(0xffffffffu, key, off));
  if (lane == 31) s_tmp[warp] = incl;
  if (lane == 0) s_tmp[32 + warp] = key;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  int base = 0, total = 0, kmin = 0x7fffffff;
  for (int q = 0; q < nw; ++q) {
    if (q < warp) base += s_tmp[q];
    total += s_tmp[q];
    kmin = min(kmin, s_tmp[32 + q]);
  }
  if (tid < n) {
    s_mt[tid] = base + incl - mt;
    s_slot[tid] = slot < 0 ? 0 : slot;
    s_rb[tid] = __ldg(&a.offsets[e]);
    s_cnt[tid] = code == 0 ? cnt : 0;
  }
  if (tid == 0) {
    s_mt[n] = total;
    if (record && kmin != 0x7fffffff) atomicCAS(a.status, 0, kmin & 15);
  }
  return n;
}

#endif  // __CUDACC__

}  // namespace msi
