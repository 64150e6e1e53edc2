// One LRU wave's complete expert FFN in a single persistent launch (sm_103a).
//
// Each selected expert runs its complete gate, up and down projections
// (paper, Sec. "Output-Exact Execution Beyond the Full-Residency Envelope")
// on weights read from the stable slot address the Plan published for it
// (Sec. "Stable Slots and Bundle Publication").  In a streamed call the pool
// holds one wave of experts at a time (Sec. "Evaluation", "Cache and storage
// state": LRU64), so a wave has only ~640 tiles of gate-up work for 152 SMs:
// launched as two kernels, each pays a partly empty last round of tiles and
// its own ramp.  Here one launch takes the wave's gate-up tiles first and its
// down tiles after them, and the small down tiles (K = I) fill the SMs the
// last gate-up round leaves idle.
//
// Tiles (128 rows x 256 columns x 64 K per stage, 4-stage ring, two TMEM
// accumulators of 256 columns, as in gemm.cu):
//   gate-up tile (g, m, n), t <  n_up:  h[rows, 128 n .. 128 n + 128) =
//       silu(x Wg^T) * (x Wu^T) over 128 routed rows of group g, A rows
//       gathered from x through the permutation;
//   down tile (g, m, n),    t >= n_up:  y[rows, 256 n .. 256 n + 256) = h W2^T,
//       A rows read from h.
// A down tile needs every gate-up tile of its m-tile (the whole h row): the
// gate-up epilogue publishes each finished tile on a per-m-tile counter
// (stores, a gpu-scope fence, a release add), and the producer acquires that
// counter, orders the h writes before its async-proxy reads
// (fence.proxy.async.global) and loads the down tile's A rows from h by TMA.
//
// Progress: tiles follow a static schedule (FusedSched: gate-up tiles
// round-robin, down tiles weighted to even out the CTAs' work), in which
// every CTA runs its gate-up tiles before its down tiles.  A CTA waiting on
// a down tile waits for gate-up tiles, which their CTAs reach without
// waiting on anything (no down tile comes before a gate-up tile in any CTA's
// sequence).  The launch is cooperative, so every CTA is resident.
//
// Roles: warps 0-3 epilogue, warp 4 MMA issue + TMEM allocation, warp 5 TMA
// producer (B: W13 or W2 rows of the group's slot; A of a down tile: h
// rows), warps 6-9 the gate-up tiles' A rows (x rows through the
// permutation) by cp.async into the 128-byte-swizzled layout, arriving on the
// stage barrier as their copies land (on a down tile's stages they only
// arrive).  Every wait is bounded; on expiry the CTA raises its
// abort flag, all roles drain and the kernel reports MSI_ERR_TIMEOUT.
#include "internal.cuh"

namespace msi {

namespace {

constexpr int kFEpiWarps = 4;
constexpr int kFGatherWarps = 4;
constexpr int kFGatherWarp0 = 6;
constexpr int kFThreads = (kFGatherWarp0 + kFGatherWarps) * 32;
constexpr int kFStages = kStages;
constexpr int kFFullCount = 1 + kFGatherWarps * 32;  // producer (expect_tx) + each gather thread
constexpr uint32_t kFIdesc = idesc_bf16(kBM, kBN);
// + the group table: tile prefix, slot, first row, rows, scan scratch
constexpr int kFSmem = 1024 + kFStages * (kABytes + kBBytes) + 256 + kFEpiWarps * 4096 +
                       (4 * kMaxExperts + 1 + 64) * 4;

struct FTile {
  int up;  // 1: gate-up tile, 0: down tile
  int g, m, n;
};

// Tile t -> (kind, group, 128-row tile, column tile) from the shared-memory
// table of the groups' 128-row tile prefix (s_mt[num_groups] = m-tiles).
__device__ __forceinline__ FTile fdecode(const FusedArgs& a, int ng, const int* s_mt, int t) {
  const int n_up = s_mt[ng] * a.nt_up;
  FTile c;
  c.up = t < n_up;
  const int nt = c.up ? a.nt_up : a.nt_dn;
  const int tt = c.up ? t : t - n_up;
  int lo = 0, hi = ng - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_mt[mid] * nt <= tt) lo = mid; else hi = mid - 1;
  }
  const int mt = s_mt[lo + 1] - s_mt[lo];
  const int local = tt - s_mt[lo] * nt;
  c.g = lo;
  c.n = local / mt;
  c.m = local - c.n * mt;
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

// Generic-proxy writes to global memory (observed through an acquire) before
// this thread's later async-proxy (TMA) reads.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// One arrival counting for `count` expected arrivals.
__device__ __forceinline__ void mbar_arrive_n(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// The four epilogue warps (128 threads) only.
__device__ __forceinline__ void epilogue_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

}  // namespace

__global__ void __launch_bounds__(kFThreads, 1)
    fused_wave_kernel(const __grid_constant__ CUtensorMap tmW13,
                      const __grid_constant__ CUtensorMap tmW2, const __grid_constant__ CUtensorMap tmH,
                      const FusedArgs a, const __grid_constant__ WaveParams w) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kFStages * kABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + kFStages * kBBytes);
  uint64_t* empty = full + kFStages;
  uint64_t* tfull = empty + kFStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* never = drain + 1;  // no thread ever arrives here
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(never + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint8_t* epi_stage = reinterpret_cast<uint8_t*>(full) + 256;  // 4 KB per epilogue warp
  int* s_mt = reinterpret_cast<int*>(epi_stage + kFEpiWarps * 4096);  // [groups + 1] tile prefix
  int* s_slot = s_mt + kMaxExperts + 1;                                // [groups]
  int* s_rb = s_slot + kMaxExperts;                                    // [groups] first row
  int* s_cnt = s_rb + kMaxExperts;                                     // [groups] rows
  int* s_tmp = s_cnt + kMaxExperts;                                    // [64]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFStages; ++s) {
      mbar_init(&full[s], kFFullCount);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kFEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(never, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  if (warp == 5 && lane == 0) {
    tma_prefetch(&tmW13);
    tma_prefetch(&tmW2);
    tma_prefetch(&tmH);
  }
  // the previous wave's counters, zeroed for the next wave
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < a.n_ready_clear; r += gridDim.x * blockDim.x)
    a.ready_clear[r] = 0;
  const int ng = fused_group_table(a, w, kBM, blockIdx.x == 0, s_mt, s_slot, s_rb, s_cnt, s_tmp);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const FusedSched sc(s_mt[ng] * a.nt_up, s_mt[ng] * a.nt_dn, gridDim.x, blockIdx.x, a.sched_w);
  const long long lim = a.wait_limit;

  if (warp == 5) {
    // ------------------------------------------------------------- TMA producer (B)
    if (lane == 0) {
      uint32_t it = 0;
      for (int t = sc.first(); t >= 0; t = sc.next(t)) {
        const FTile tc = fdecode(a, ng, s_mt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        const int r0 = tc.up ? s_slot[tc.g] * a.w13_rows_per_slot + tc.n * 128
                             : s_slot[tc.g] * a.w2_rows_per_slot + a.w2_row_off + tc.n * kBN;
        const int r1 = tc.up ? r0 + a.w13_up_off : r0 + 128;
        const CUtensorMap* map = tc.up ? &tmW13 : &tmW2;
        bool ok = true;
        if (!tc.up) {
          // every gate-up tile of this m-tile has published its h columns
          const int* rdy = a.ready + s_mt[tc.g] + tc.m;
          const long long t0 = clock64();
          while (ld_acquire_gpu(rdy) < a.nt_up) {
            if (*abort_flag) { ok = false; break; }
            if (clock64() - t0 > lim) {
              *abort_flag = 1;
              ok = false;
              break;
            }
          }
          if (!ok) break;
          fence_proxy_async_global();
        }
        // the down tile's A: its 128 h rows (rows past the group's segment
        // are the next group's or the tensor's zero fill; their outputs are
        // not stored)
        const int arow = s_rb[tc.g] + tc.m * kBM;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kFStages;
          const uint32_t ph = (it / kFStages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], tc.up ? kBBytes : kBBytes + kABytes);
          uint8_t* b = sB + s * kBBytes;
          tma_load_2d(b, map, &full[s], kb * kBK, r0);
          tma_load_2d(b + kBBytes / 2, map, &full[s], kb * kBK, r1);
          if (!tc.up) tma_load_2d(sA + s * kABytes, &tmH, &full[s], kb * kBK, arow);
        }
        if (!ok) break;
      }
      // On abort, wait (bounded) for the loads this thread armed to land
      // before the CTA's shared memory is released.
      if (*abort_flag) {
        for (int d = 0; d < kFStages && it > 0; ++d) {
          const uint32_t j = it - 1 - d;
          if ((int)j < 0) break;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % kFStages], (j / kFStages) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
      }
    }
  } else if (warp == 4) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t it = 0, jt = 0;
      for (int t = sc.first(); t >= 0; t = sc.next(t), ++jt) {
        const FTile tc = fdecode(a, ng, s_mt, t);
        const int kb_n = tc.up ? a.kb_up : a.kb_dn;
        const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1, abort_flag, lim)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kBN;
        bool ok = true;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kFStages;
          const uint32_t ph = (it / kFStages) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
          // cp.async (generic proxy) wrote A: order those writes before this
          // thread's tensor-core (async proxy) reads
          fence_proxy_async_smem();
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * kABytes));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * kBBytes));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) umma_bf16(d, ad + 2 * k, bd + 2 * k, kFIdesc, (kb | k) != 0);
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
      }
      // every MMA this thread issued has completed before TMEM is released
      umma_commit(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0) && clock64() - t0 < kDrainCycles) {
      }
    }
  } else if (warp < kFEpiWarps) {
    // ------------------------------------------------------------- epilogue
    uint32_t jt = 0;
    if (a.stall && threadIdx.x == 0) mbar_wait(never, 0, abort_flag, lim);  // runs out: abort
    for (int t = sc.first(); t >= 0; t = sc.next(t), ++jt) {
      const FTile tc = fdecode(a, ng, s_mt, t);
      const int cnt = s_cnt[tc.g];
      const size_t rb = (size_t)s_rb[tc.g];
      const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
      if (!mbar_wait(&tfull[acc], aph, abort_flag, lim)) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16) + acc * kBN;
      const int row_w = tc.m * kBM + warp * 32;  // the warp's first row inside the group
      if (tc.up) {
        epilogue_tile_staged<true>(tb, a.h + (rb + row_w) * a.h_ld + tc.n * 128, a.h_ld, cnt - row_w,
                                   epi_stage + warp * 4096, lane);
        // publish the tile: every epilogue thread's h stores, then one release
        // add on the m-tile's counter
        __threadfence();
        epilogue_bar();
        if (threadIdx.x == 0) red_release_gpu_add(&a.ready[s_mt[tc.g] + tc.m], 1);
      } else {
        epilogue_tile_staged<false>(tb, a.y + (rb + row_w) * a.y_ld + tc.n * kBN, a.y_ld, cnt - row_w,
                                    epi_stage + warp * 4096, lane);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  } else {
    // ------------------------------------------------------------- A rows
    const int gt = threadIdx.x - kFGatherWarp0 * 32;  // 0..127
    const int chunk = gt & 7;                         // 16-byte chunk of a 128-byte row slice
    const int r0 = gt >> 3;                           // rows r0 + 16 i
    uint32_t it = 0;
    bool ok = true;
    // this thread's eight permutation entries of gate-up tile t (routed row
    // token * k + j; -1 past the group's segment), loaded one tile ahead and
    // first used at that tile's start, so the loads' latency is not waited
    // for at the start of the current tile
    auto tile_rows = [&](int t, int (&pr)[8]) {
      const FTile tc = fdecode(a, ng, s_mt, t);
      const int cnt = s_cnt[tc.g];
      const int rb = s_rb[tc.g];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = tc.m * kBM + r0 + 16 * i;
        pr[i] = (!tc.up || rr >= cnt) ? -1 : __ldg(&a.perm[rb + rr]);
      }
    };
    int pr[8], pr_next[8];
    const int t_first = sc.first();
    if (t_first >= 0) tile_rows(t_first, pr);
    for (int t = t_first; t >= 0 && ok; t = sc.next(t)) {
      const int t_next = sc.next(t);
      const bool has_next = t_next >= 0;
      if (has_next) tile_rows(t_next, pr_next);
      const FTile tc = fdecode(a, ng, s_mt, t);
      const int kb_n = tc.up ? a.kb_up : a.kb_dn;
      if (!tc.up) {
        // the producer loads a down tile's A by TMA: each warp only arrives
        // (for its 32 threads) once the stage is free
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kFStages;
          const uint32_t ph = (it / kFStages) & 1;
          bool free_stage = true;
          if (lane == 0) free_stage = mbar_wait(&empty[s], ph ^ 1, abort_flag, lim);
          free_stage = __shfl_sync(0xffffffffu, free_stage, 0);
          if (!free_stage) { ok = false; break; }
          if (lane == 0) mbar_arrive_n(&full[s], 32);
          __syncwarp();
        }
      } else {
        const __nv_bfloat16* src[8];
        uint32_t nbytes[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (pr[i] >= 0) {
            src[i] = a.x + (size_t)(pr[i] / a.top_k) * a.x_ld + chunk * 8;
            nbytes[i] = 16;
          } else {
            src[i] = a.x;
            nbytes[i] = 0;  // zero-fill rows past the group's segment
          }
        }
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = it % kFStages;
          const uint32_t ph = (it / kFStages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
          uint8_t* dstA = sA + s * kABytes;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int rr = r0 + 16 * i;
            cp_async16(dstA + rr * 128 + ((chunk ^ (rr & 7)) << 4), src[i] + kb * kBK, nbytes[i]);
          }
          cp_async_arrive_noinc(&full[s]);  // arrives when this thread's copies land
        }
      }
      if (has_next) {
#pragma unroll
        for (int i = 0; i < 8; ++i) pr[i] = pr_next[i];
      }
    }
    cp_async_wait<0>();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicCAS(a.status, 0, (int)MSI_ERR_TIMEOUT);
}

cudaError_t launch_fused_wave(const CUtensorMap& tmW13, const CUtensorMap& tmW2, const CUtensorMap& tmH,
                              const FusedArgs& a, const WaveParams& w, int grid, cudaStream_t s) {
  static std::atomic<unsigned long long> attr_done{0};
  cudaError_t e = smem_attr_once(fused_wave_kernel, kFSmem, attr_done);
  if (e != cudaSuccess) return e;
  if (grid < 1) return cudaSuccess;
  // cooperative: every CTA resident, so a CTA waiting on another's gate-up
  // tile never waits for an SM that CTA cannot get
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kFThreads, 1, 1);
  cfg.dynamicSmemBytes = kFSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fused_wave_kernel, tmW13, tmW2, tmH, a, w);
}

}  // namespace msi
