// One LRU wave's complete expert FFN in a single persistent launch on CTA
// pairs (tcgen05 cta_group::2, sm_103a).
//
// The work is that of gemm_fused.cu (each selected expert's gate, up and down
// projections over its routed rows, paper Sec. "Output-Exact Execution Beyond
// the Full-Residency Envelope", weights read from the slot the Plan published
// for it, Sec. "Stable Slots and Bundle Publication"), tiled as in
// gemm_pair.cu: two CTAs on neighbouring SMs share one 256 x 256 output tile,
// each holding 128 of its A rows and 128 of its B rows, so per unit of tensor
// work an SM receives a third less operand data than with single-CTA tiles.
//
// Tiles (FusedSched over the pairs: gate-up tiles round-robin, down tiles
// weighted to even out the pairs' work):
//   t <  n_up: gate-up pair tile (g, m2, n): h[256 rows, 128 n .. 128 n + 128)
//              (the even CTA holds the gate rows of B, the odd CTA the up rows);
//   t >= n_up: down pair tile (g, m2, n): y[256 rows, 256 n .. 256 n + 256)
//              (CTA r holds B rows 256 n + 128 r .. + 128 of W2).
// A down tile reads the h rows of its 256-row tile, written by the gate-up
// epilogues of both CTAs of every gate-up tile of that m-tile: each publishes
// on the m-tile's counter (stores, a gpu-scope fence, a release add) and the
// down tile's A loads wait until the counter reaches 2 * (I / 128).  Every
// pair processes all its gate-up tiles before its down tiles, so a pair
// waiting on a down tile waits only for gate-up tiles, which their pairs
// reach without waiting; the grid never exceeds the clusters that can be
// resident at once.
//
// Synchronisation within a pair is that of gemm_pair.cu: each CTA's loads
// complete on its own `full` barrier, the odd CTA's relay forwards completed
// stages to the even CTA, the even CTA issues the pair MMAs and commits to
// `empty` and `tfull` of both CTAs, the epilogue warps of both CTAs free an
// accumulator on the even CTA's `tempty`.  Every wait is bounded; on expiry a
// CTA raises its abort flag, its roles drain and the kernel reports
// MSI_ERR_TIMEOUT.
//
// Roles per CTA: warps 0-3 epilogue, warp 4 MMA issue (even CTA) or stage
// relay (odd CTA) and TMEM allocation, warp 5 TMA producer (B), warps 6-9 the
// CTA's 128 A rows by cp.async (x rows through the permutation for gate-up
// tiles, h rows for down tiles).
//
// 4-bit weights (Q4): the producer loads each stage's packed codes of the
// CTA's 128 B rows (one 128 x 32-byte box of the code maps over the slot
// pool) into a three-stage ring, and sixteen dequant warps convert them into
// the bf16 B stage as in gemm_pair.cu (a quarter row per thread: 16 codes
// under one fp16 scale, w = s * (q - 8) exact in fp32, rounded once to bf16),
// with the W13 or W2 scales of the tile's rows.  The epilogue reads TMEM 16
// columns at a time so that the 832 threads fit the register file.
#include <algorithm>

#include <cuda_fp16.h>

#include "internal.cuh"

namespace msi {

namespace {

constexpr int kQRows = 2 * kBM;       // 256 token rows per pair tile
constexpr int kQStages = 6;
constexpr int kQA = kBM * kBK * 2;    // 16 KB: this CTA's 128 A rows of one K step
constexpr int kQB = 128 * kBK * 2;    // 16 KB: this CTA's 128 B rows of one K step
constexpr uint32_t kQIdesc = idesc_bf16(kQRows, kBN);
constexpr int kQEpiWarps = 4;
constexpr int kQGatherWarps = 4;
constexpr int kQGatherWarp0 = 6;
constexpr int kQRawRow = 32;          // 64 codes of one B row per stage (one TMA box row)
constexpr int kQRaw = 3;              // 4-bit: code stages in flight
constexpr int kQDq = 16;              // 4-bit: dequant warps

template <bool Q4>
struct QCfg {
  static constexpr int kThreads = (kQGatherWarp0 + kQGatherWarps + (Q4 ? kQDq : 0)) * 32;
  // own gather threads + (bf16) the producer's expect_tx or (4-bit) each dequant warp
  static constexpr int kFullLocal = kQGatherWarps * 32 + (Q4 ? kQDq : 1);
  static constexpr int kRawBytes = Q4 ? kQRaw * 128 * kQRawRow : 0;
  // group table: tile prefix, slot, first row, rows, scan scratch (4-bit
  // launches are waves only, at most kMaxWave groups)
  static constexpr int kGroups = Q4 ? kMaxWave : kMaxExperts;
  static constexpr int kSmem = 1024 + kQStages * (kQA + kQB) + kRawBytes + 256 + kQEpiWarps * 4096 +
                               (4 * kGroups + 1 + 64) * 4;
};

struct QTile {
  int up;  // 1: gate-up tile, 0: down tile
  int g, m2, n;
};

// Pair tile t -> (kind, group, 256-row tile, column tile) from the
// shared-memory table of the groups' 256-row tile prefix.
__device__ __forceinline__ QTile qdecode(const FusedArgs& a, int ng, const int* s_pt, int t) {
  const int n_up = s_pt[ng] * a.nt_up;
  QTile c;
  c.up = t < n_up;
  const int nt = c.up ? a.nt_up : a.nt_dn;
  const int tt = c.up ? t : t - n_up;
  int lo = 0, hi = ng - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_pt[mid] * nt <= tt) lo = mid; else hi = mid - 1;
  }
  const int mt2 = s_pt[lo + 1] - s_pt[lo];
  const int local = tt - s_pt[lo] * nt;
  c.g = lo;
  c.n = local / mt2;
  c.m2 = local - c.n * mt2;
  return c;
}

__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_release_gpu_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void epilogue_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

}  // namespace

template <bool Q4>
__global__ void __launch_bounds__(QCfg<Q4>::kThreads, 1)
    fused_wave_pair_kernel(const __grid_constant__ CUtensorMap tmW13,
                           const __grid_constant__ CUtensorMap tmW2, const FusedArgs a,
                           const __grid_constant__ WaveParams w) {
  using C = QCfg<Q4>;
  extern __shared__ uint8_t smem_raw[];
  // the same offsets in both CTAs: the pair MMA addresses the peer's operands
  // through the even CTA's descriptors
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kQStages * kQA;
  uint8_t* raw_codes = sB + kQStages * kQB;  // 4-bit: [kQRaw][128][32]
  uint64_t* full = reinterpret_cast<uint64_t*>(raw_codes + C::kRawBytes);
  uint64_t* empty = full + kQStages;
  uint64_t* tfull = empty + kQStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* never = drain + 1;  // no thread ever arrives here
  uint64_t* raw_full = never + 1;            // 4-bit: code stage landed (TMA bytes)
  uint64_t* raw_empty = raw_full + kQRaw;    // 4-bit: code stage converted by every dequant warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(raw_empty + kQRaw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint8_t* epi_stage = reinterpret_cast<uint8_t*>(full) + 256;  // 4 KB per epilogue warp
  int* s_pt = reinterpret_cast<int*>(epi_stage + kQEpiWarps * 4096);  // [groups + 1] tile prefix
  int* s_slot = s_pt + C::kGroups + 1;                                // [groups]
  int* s_rb = s_slot + C::kGroups;                                    // [groups] first row
  int* s_cnt = s_rb + C::kGroups;                                     // [groups] rows
  int* s_tmp = s_cnt + C::kGroups;                                    // [64]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kQStages; ++s) {
      mbar_init(&full[s], C::kFullLocal + (leader ? 1 : 0));  // + the peer's relay
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 2 * kQEpiWarps);  // the epilogue warps of both CTAs
    }
    mbar_init(drain, 1);
    mbar_init(never, 1);
    for (int r = 0; r < kQRaw && Q4; ++r) {
      mbar_init(&raw_full[r], 1);
      mbar_init(&raw_empty[r], kQDq);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4) {
    tmem_alloc_pair(tmem_slot, 512);
    tmem_relinquish_pair();
  }
  if (warp == 5 && lane == 0) {
    tma_prefetch(&tmW13);
    tma_prefetch(&tmW2);
  }
  // the previous wave's counters, zeroed for the next wave
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < a.n_ready_clear; r += gridDim.x * blockDim.x)
    a.ready_clear[r] = 0;
  const int ng = fused_group_table(a, w, kQRows, blockIdx.x == 0, s_pt, s_slot, s_rb, s_cnt, s_tmp);
  tc_fence_before();
  cluster_sync_all();  // both CTAs' barriers initialised before any cross-CTA arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int pair = blockIdx.x >> 1;
  const int npairs = gridDim.x >> 1;
  const FusedSched sc(s_pt[ng] * a.nt_up, s_pt[ng] * a.nt_dn, npairs, pair, a.sched_w);
  const long long lim = a.wait_limit;

  if (warp == 5) {
    // ------------------------------------------------------------- TMA producer (B)
    if (lane == 0 && !Q4) {
      uint32_t it = 0;
      for (int t = sc.first(); t >= 0; t = sc.next(t)) {
        const QTile tc = qdecode(a, ng, s_pt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        // gate-up: the even CTA holds 128 gate rows, the odd CTA the matching
        // up rows; down: CTA r holds W2 rows 256 n + 128 r .. + 128
        const int brow = tc.up ? s_slot[tc.g] * a.w13_rows_per_slot + (rank ? a.w13_up_off : 0) + tc.n * 128
                               : s_slot[tc.g] * a.w2_rows_per_slot + a.w2_row_off + tc.n * kBN + (int)rank * 128;
        const CUtensorMap* map = tc.up ? &tmW13 : &tmW2;
        bool ok = true;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kQStages;
          const uint32_t ph = (it / kQStages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], kQB);
          tma_load_2d(sB + s * kQB, map, &full[s], kb * kBK, brow);
        }
        if (!ok) break;
      }
      // On abort, wait (bounded) for the loads this thread armed to land
      // before the CTA's shared memory is released.
      if (*abort_flag) {
        for (int d = 0; d < kQStages && it > 0; ++d) {
          const uint32_t j = it - 1 - d;
          if ((int)j < 0) break;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % kQStages], (j / kQStages) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
      }
    } else if (lane == 0) {
      // 4-bit: the CTA's 128 code rows of each stage into the raw ring
      // (gate-up: gate rows in the even CTA, up rows in the odd one; down:
      // W2 rows 256 n + 128 r)
      uint32_t it = 0;
      for (int t = sc.first(); t >= 0; t = sc.next(t)) {
        const QTile tc = qdecode(a, ng, s_pt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        const int qrow = tc.up ? s_slot[tc.g] * a.q13_rows_per_slot + (rank ? a.w13_up_off : 0) + tc.n * 128
                               : s_slot[tc.g] * a.q2_rows_per_slot + a.q2_row_off + tc.n * kBN + (int)rank * 128;
        const CUtensorMap* map = tc.up ? &tmW13 : &tmW2;
        bool ok = true;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int r = it % kQRaw;
          if (!mbar_wait(&raw_empty[r], ((it / kQRaw) & 1) ^ 1, abort_flag, lim)) { ok = false; break; }
          mbar_arrive_expect_tx(&raw_full[r], 128 * kQRawRow);
          tma_load_2d(raw_codes + r * (128 * kQRawRow), map, &raw_full[r], kb * kQRawRow, qrow);
        }
        if (!ok) break;
      }
      if (*abort_flag) {
        for (int d = 0; d < kQRaw && it > 0; ++d) {
          const uint32_t j = it - 1 - d;
          if ((int)j < 0) break;
          const long long t0 = clock64();
          while (!mbar_try_wait(&raw_full[j % kQRaw], (j / kQRaw) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
      }
    }
  } else if (warp == 4) {
    if (lane == 0 && leader) {
      // ----------------------------------------------------------- MMA issuer
      uint32_t it = 0, jt = 0;
      for (int t = sc.first(); t >= 0; t = sc.next(t), ++jt) {
        const QTile tc = qdecode(a, ng, s_pt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1, abort_flag, lim)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kBN;
        bool ok = true;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kQStages;
          const uint32_t ph = (it / kQStages) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
          // this CTA's A rows were written by cp.async (generic proxy); the
          // relay fenced the peer's before forwarding its stage
          fence_proxy_async_smem();
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * kQA));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * kQB));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) umma_bf16_pair(d, ad + 2 * k, bd + 2 * k, kQIdesc, (kb | k) != 0);
          umma_commit_pair(&empty[s]);
        }
        if (!ok) break;
        umma_commit_pair(&tfull[acc]);
      }
      umma_commit_pair(drain);
    } else if (lane == 0) {
      // ------------------------------------------------------ stage relay (odd)
      uint32_t it = 0;
      bool ok = true;
      for (int t = sc.first(); t >= 0 && ok; t = sc.next(t)) {
        const QTile tc = qdecode(a, ng, s_pt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kQStages;
          const uint32_t ph = (it / kQStages) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
          fence_proxy_async_smem();
          mbar_arrive_remote(mapa_shared(smem_u32(&full[s]), 0));
        }
      }
    }
    if (lane == 0) {
      // every pair MMA that reads this CTA's shared memory or writes its TMEM
      // has completed before either is released
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0) && clock64() - t0 < kDrainCycles) {
      }
    }
  } else if (warp < kQEpiWarps) {
    // ------------------------------------------------------------- epilogue
    uint32_t jt = 0;
    const uint32_t lead_tempty[2] = {mapa_shared(smem_u32(&tempty[0]), 0),
                                     mapa_shared(smem_u32(&tempty[1]), 0)};
    if (a.stall && threadIdx.x == 0) mbar_wait(never, 0, abort_flag, lim);  // runs out: abort
    for (int t = sc.first(); t >= 0; t = sc.next(t), ++jt) {
      const QTile tc = qdecode(a, ng, s_pt, t);
      const int cnt = s_cnt[tc.g];
      const size_t rb = (size_t)s_rb[tc.g];
      const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
      if (!mbar_wait(&tfull[acc], aph, abort_flag, lim)) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16) + acc * kBN;
      const int row_w = tc.m2 * kQRows + (int)rank * kBM + warp * 32;  // warp's first row in the group
      if (tc.up) {
        if (Q4)
          epilogue_tile_staged_lean<true>(tb, a.h + (rb + row_w) * a.h_ld + tc.n * 128, a.h_ld, cnt - row_w,
                                          epi_stage + warp * 4096, lane);
        else
          epilogue_tile_staged<true>(tb, a.h + (rb + row_w) * a.h_ld + tc.n * 128, a.h_ld, cnt - row_w,
                                     epi_stage + warp * 4096, lane);
        // publish this CTA's half of the tile: every epilogue thread's h
        // stores, then one release add on the 256-row tile's counter
        __threadfence();
        epilogue_bar();
        if (threadIdx.x == 0) red_release_gpu_add(&a.ready[s_pt[tc.g] + tc.m2], 1);
      } else if (Q4) {
        epilogue_tile_staged_lean<false>(tb, a.y + (rb + row_w) * a.y_ld + tc.n * kBN, a.y_ld, cnt - row_w,
                                         epi_stage + warp * 4096, lane);
      } else {
        epilogue_tile_staged<false>(tb, a.y + (rb + row_w) * a.y_ld + tc.n * kBN, a.y_ld, cnt - row_w,
                                    epi_stage + warp * 4096, lane);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(lead_tempty[acc]);
    }
  } else if (warp < kQGatherWarp0 + kQGatherWarps) {
    // ------------------------------------------------------------- A rows
    const int gt = threadIdx.x - kQGatherWarp0 * 32;  // 0..127
    const int chunk = gt & 7;                         // 16-byte chunk of a 128-byte row slice
    const int r0 = gt >> 3;                           // rows r0 + 16 i of this CTA's 128
    uint32_t it = 0;
    bool ok = true;
    // this thread's eight A rows of tile t: a gate-up tile's permutation
    // entries (token * k + j), a down tile's h rows; -1 past the group's
    // segment.  Loaded one tile ahead and first used at that tile's start.
    auto tile_rows = [&](int t, int (&pr)[8]) {
      const QTile tc = qdecode(a, ng, s_pt, t);
      const int cnt = s_cnt[tc.g];
      const int rb = s_rb[tc.g];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = tc.m2 * kQRows + (int)rank * kBM + r0 + 16 * i;
        pr[i] = rr >= cnt ? -1 : (tc.up ? __ldg(&a.perm[rb + rr]) : rb + rr);
      }
    };
    int pr[8], pr_next[8];
    const int t_first = sc.first();
    if (t_first >= 0) tile_rows(t_first, pr);
    for (int t = t_first; t >= 0 && ok; t = sc.next(t)) {
      const int t_next = sc.next(t);
      const bool has_next = t_next >= 0;
      if (has_next) tile_rows(t_next, pr_next);
      const QTile tc = qdecode(a, ng, s_pt, t);
      const int kb_n = tc.up ? a.kb_up : a.kb_dn;
      if (!tc.up) {
        // both CTAs of every gate-up tile of this 256-row tile have published
        const int* rdy = a.ready + s_pt[tc.g] + tc.m2;
        bool seen = true;
        if (lane == 0) {
          const long long t0 = clock64();
          while (ld_acquire_gpu(rdy) < 2 * a.nt_up) {
            if (*abort_flag) { seen = false; break; }
            if (clock64() - t0 > lim) {
              *abort_flag = 1;
              seen = false;
              break;
            }
          }
        }
        seen = __shfl_sync(0xffffffffu, seen, 0);
        __syncwarp();
        if (!seen) { ok = false; break; }
      }
      const __nv_bfloat16* src_base = tc.up ? a.x : a.h;
      const size_t ld = tc.up ? (size_t)a.x_ld : (size_t)a.h_ld;
      const __nv_bfloat16* src[8];
      uint32_t nbytes[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (pr[i] >= 0) {
          src[i] = src_base + (size_t)(tc.up ? pr[i] / a.top_k : pr[i]) * ld + chunk * 8;
          nbytes[i] = 16;
        } else {
          src[i] = src_base;
          nbytes[i] = 0;  // zero-fill rows past the group's segment
        }
      }
      for (int kb = 0; kb < kb_n; ++kb, ++it) {
        const int s = it % kQStages;
        const uint32_t ph = (it / kQStages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
        uint8_t* dstA = sA + s * kQA;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int rr = r0 + 16 * i;
          cp_async16(dstA + rr * 128 + ((chunk ^ (rr & 7)) << 4), src[i] + kb * kBK, nbytes[i]);
        }
        cp_async_arrive_noinc(&full[s]);  // arrives when this thread's copies land
      }
      if (has_next) {
#pragma unroll
        for (int i = 0; i < 8; ++i) pr[i] = pr_next[i];
      }
    }
    cp_async_wait<0>();
  } else if (Q4) {
    // ------------------------------------------------------------- 4-bit dequant
    // a warp takes 8 of the CTA's 128 B rows, four lanes to a row (a quarter
    // row of 16 codes under one scale); its code reads cover 256 contiguous
    // bytes and its SW128 writes reach every bank group once per 8 lanes
    const int d = (warp - kQGatherWarp0 - kQGatherWarps) * 8 + (lane >> 2);  // B row, 0..127
    const int qt = lane & 3;                                                 // codes 16 qt .. 16 qt + 15
    // this thread's scale row of tile t (W13 rows for a gate-up tile, W2
    // rows for a down tile); scales of a stage pair are one 8-byte load
    auto scale_row = [&](int t) -> const uint8_t* {
      const QTile tc = qdecode(a, ng, s_pt, t);
      const uint8_t* ext = a.q4_pool + (unsigned long long)s_slot[tc.g] * a.q4_extent;
      return tc.up ? ext + a.q13_scale_off + (size_t)((rank ? a.w13_up_off : 0) + tc.n * 128 + d) * a.q13_scale_ld
                   : ext + a.q2_scale_off + (size_t)(tc.n * kBN + (int)rank * 128 + d) * a.q2_scale_ld;
    };
    uint32_t it = 0;
    bool ok = true;
    // the next stage pair's scales are loaded one pair ahead, across tiles
    const int t_first = sc.first();
    uint2 nxt = t_first >= 0 ? __ldg(reinterpret_cast<const uint2*>(scale_row(t_first))) : make_uint2(0, 0);
    for (int t = t_first; t >= 0 && ok; t = sc.next(t)) {
      const QTile tc = qdecode(a, ng, s_pt, t);
      const int kb_n = tc.up ? a.kb_up : a.kb_dn;  // even (K a multiple of 128)
      const uint8_t* srow = scale_row(t);
      const int t_next = sc.next(t);
      const uint8_t* srow_next = t_next >= 0 ? scale_row(t_next) : nullptr;
      uint2 cur = make_uint2(0, 0);
      for (int kb = 0; kb < kb_n; ++kb, ++it) {
        if ((kb & 1) == 0) {
          cur = nxt;
          if (kb + 2 < kb_n) nxt = __ldg(reinterpret_cast<const uint2*>(srow + (kb + 2) * 4));
          else if (srow_next != nullptr) nxt = __ldg(reinterpret_cast<const uint2*>(srow_next));
        }
        const int r = it % kQRaw;
        if (!mbar_wait(&raw_full[r], (it / kQRaw) & 1, abort_flag, lim)) { ok = false; break; }
        const int s = it % kQStages;
        const uint32_t ph = (it / kQStages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
        const uint2 cw = ld_shared_v2(smem_u32(raw_codes + r * (128 * kQRawRow) + d * kQRawRow + qt * 8));
        const uint32_t sc = (kb & 1) ? cur.y : cur.x;
        const float sv = __half2float(__ushort_as_half((unsigned short)(qt >= 2 ? sc >> 16 : sc & 0xFFFFu)));
        const uint64_t sx2 = f32x2(sv, sv), nx2 = f32x2(-136.0f * sv, -136.0f * sv);
        const uint32_t dst_row = smem_u32(sB + s * kQB + d * 128);
        const int c0 = qt * 2;  // 16-byte chunks c0, c0 + 1 of the 128-byte row
        st_shared_v4(dst_row + ((c0 ^ (d & 7)) << 4), dequant8(cw.x, sx2, nx2));
        st_shared_v4(dst_row + (((c0 + 1) ^ (d & 7)) << 4), dequant8(cw.y, sx2, nx2));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&full[s]);
          mbar_arrive(&raw_empty[r]);  // the warp's rows of this code stage are consumed
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while the other may still reach it
  if (warp == 4) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, 512);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicCAS(a.status, 0, (int)MSI_ERR_TIMEOUT);
}

template <bool Q4>
static cudaError_t launch_pair(const CUtensorMap& tmW13, const CUtensorMap& tmW2, const FusedArgs& a,
                               const WaveParams& w, int max_pairs, cudaStream_t s) {
  static std::atomic<unsigned long long> attr_done{0};
  static std::atomic<int> max_clusters[64] = {};
  auto kernel = fused_wave_pair_kernel<Q4>;
  cudaError_t e = smem_attr_once(kernel, QCfg<Q4>::kSmem, attr_done);
  if (e != cudaSuccess) return e;
  if (max_pairs < 1) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(QCfg<Q4>::kThreads, 1, 1);
  cfg.dynamicSmemBytes = QCfg<Q4>::kSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  // the grid never exceeds the pairs that can be resident at once: a pair
  // waiting on another pair's gate-up tile never holds an SM that pair needs
  int mc = dev < 64 ? max_clusters[dev].load() : 0;
  if (mc <= 0) {
    cfg.gridDim = dim3(2, 1, 1);
    e = cudaOccupancyMaxActiveClusters(&mc, kernel, &cfg);
    if (e != cudaSuccess) return e;
    if (mc <= 0) return cudaErrorInvalidConfiguration;
    if (dev < 64) max_clusters[dev].store(mc);
  }
  const int pairs = std::max(1, std::min(mc, max_pairs));
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  return cudaLaunchKernelEx(&cfg, kernel, tmW13, tmW2, a, w);
}

cudaError_t launch_fused_wave_pair(const CUtensorMap& tmW13, const CUtensorMap& tmW2,
                                   const FusedArgs& a, const WaveParams& w, int max_pairs, cudaStream_t s) {
  return launch_pair<false>(tmW13, tmW2, a, w, max_pairs, s);
}

cudaError_t launch_fused_wave_pair_q4(const CUtensorMap& tmQ13, const CUtensorMap& tmQ2,
                                      const FusedArgs& a, const WaveParams& w, int max_pairs, cudaStream_t s) {
  if (!a.wave) return cudaErrorInvalidValue;  // 4-bit fused launches are waves (group table of kMaxWave)
  return launch_pair<true>(tmQ13, tmQ2, a, w, max_pairs, s);
}

}  // namespace msi
