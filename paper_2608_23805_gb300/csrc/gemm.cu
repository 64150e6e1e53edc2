// Grouped expert GEMMs on tcgen05 tensor cores (sm_103a).
//
// Each selected expert runs its complete gate, up and down projections
// (paper, Sec. "Output-Exact Execution Beyond the Full-Residency Envelope"),
// reading its weights from the stable address of the GPU slot the Plan
// published for it (Sec. "Stable Slots and Bundle Publication").
//
// One persistent kernel per projection pair:
//   gate-up (kGateUpGather / kGateUpTma / kGateUpGatherQ4):  h = silu(x Wg^T) * (x Wu^T) -> bf16
//   down    (kDown / kDownQ4):                                y = h W2^T                  -> bf16
// The q4 modes read 4-bit weights (one fp16 scale per 32 weights of a row)
// from the slot and dequantise them to bf16 in shared memory inside the
// producer: eight warps prefetch codes and scales with cp.async into a
// three-stage raw ring and each thread converts its own B row
// (w = scale * (q - 8), exact in fp32 and rounded once to bf16, two values
// per packed f32x2 instruction) into the swizzled layout the MMA reads, so the
// weights cross HBM at 0.5625 bytes each.
// Tile: 128 token rows x 256 weight rows x 64 K per stage, 4-stage smem ring,
// fp32 accumulators double-buffered in TMEM (2 x 256 columns).  Weights (B)
// come by TMA from the slot pool viewed as one 2-D tensor per operand; the
// routed token rows (A) of the gate-up GEMM are gathered through the
// permutation with cp.async into the same 128-byte-swizzled layout TMA
// writes, each thread arriving on the stage barrier when its copies land
// (cp.async.mbarrier.arrive.noinc); the down GEMM's A (h, already in permuted
// order) comes by TMA.
//
// Roles (warp-specialised):  warps 0-3 epilogue (TMEM -> registers -> global,
// one token row per thread), warp 4 MMA issue + TMEM allocation, warp 5 TMA
// producer, warps 6-9 row gather (gather modes), then eight dequant warps
// (q4 modes).  Every wait is bounded;
// on expiry the CTA raises its abort flag, all roles drain and the kernel
// reports MSI_ERR_TIMEOUT in the status word.
#include <cuda_fp16.h>

#include "internal.cuh"

namespace msi {

namespace {

constexpr int kEpiWarps = 4;
constexpr int kGatherWarps = 4;
constexpr uint32_t kIdesc = idesc_bf16(kBM, kBN);

constexpr int kRawRowBytes = 32;  // 64 codes of one B row per stage (one TMA box row)

template <int MODE>
struct Cfg {
  static constexpr bool kQ4 = (MODE == kGateUpGatherQ4 || MODE == kDownQ4);
  static constexpr bool kGather = (MODE == kGateUpGather || MODE == kGateUpGatherQ4);
  static constexpr bool kGateUp = (MODE == kGateUpGather || MODE == kGateUpTma || MODE == kGateUpGatherQ4);
  static constexpr bool kTmaA = !kGather;
  static constexpr bool kTmaB = !kQ4;
  static constexpr bool kTmaAny = kTmaA || kTmaB;
  static constexpr int kGatherWarp0 = 6;
  static constexpr int kDqWarp0 = 6 + (kGather ? kGatherWarps : 0);
  // q4: sixteen dequant warps, one thread per half B row (256 rows x 2)
  static constexpr int kDq = kQ4 ? 16 : 0;
  static constexpr int kThreads = (kDqWarp0 + kDq) * 32;
  static constexpr uint32_t kTxBytes = (kTmaB ? kBBytes : 0) + (kTmaA ? kABytes : 0);
  // gather threads arrive one by one as their copies land (cp.async ... arrive.noinc)
  static constexpr int kFullCount = (kTmaAny ? 1 : 0) + (kGather ? kGatherWarps * 32 : 0) + kDq;
  // operand ring depth and, in the q4 modes, the ring of packed code stages
  // that the producer fills by TMA ahead of the conversion
  static constexpr int kStg = kStages;
  static constexpr int kRaw = kQ4 ? 3 : 1;
  static constexpr int kRawBytes = kQ4 ? kRaw * kBN * kRawRowBytes : 0;
  static constexpr uint32_t kRawTx = kBN * kRawRowBytes;
  // bf16 modes stage each epilogue warp's rows in shared memory (4 KB per
  // warp) for row-coalesced stores; the q4 raw ring leaves no room for it
  static constexpr bool kStagedEpi = !kQ4;
  // the groups' 128-row tile prefix and slot, read once per launch so that
  // tile lookups (every role, every tile) stay in shared memory
  static constexpr int kGroupTableBytes = (2 * kMaxExperts + 2) * 4;
  static constexpr int kSmem = 1024 + kStg * (kABytes + kBBytes) + kRawBytes + 256 +
                               (kStagedEpi ? kEpiWarps * 4096 : 0) + kGroupTableBytes;
};

struct TileCoord {
  int g, m, n;
};

// Tile t -> (group, 128-row tile, column tile) from the shared-memory table
// of the groups' tile prefix (s_mt[num_groups] = total tiles).
__device__ __forceinline__ TileCoord decode_tile(const GemmArgs& a, const int* s_mt, int t) {
  int lo = 0, hi = a.num_groups - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_mt[mid] * a.nt <= t) lo = mid; else hi = mid - 1;
  }
  const int mt = s_mt[lo + 1] - s_mt[lo];
  const int local = t - s_mt[lo] * a.nt;
  TileCoord c;
  c.g = lo;
  c.n = local / mt;
  c.m = local - c.n * mt;
  return c;
}

// q4 epilogue: TMEM read 16 columns at a time, so that the kernel's many
// dequant threads fit the register file (one 32-byte store per chunk).
template <bool GATEUP>
__device__ __forceinline__ void epilogue_tile_lean(uint32_t tb, __nv_bfloat16* dst, bool valid) {
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
      if (valid) st_global_v8(dst + c, p);
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
      if (valid) st_global_v8(dst + c, p);
    }
  }
}

}  // namespace

template <int MODE>
__global__ void __launch_bounds__(Cfg<MODE>::kThreads, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const GemmArgs a) {
  using C = Cfg<MODE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::kStg * kABytes;
  uint8_t* raw_codes = sB + C::kStg * kBBytes;                    // q4: [C::kRaw][256][32]
  uint64_t* full = reinterpret_cast<uint64_t*>(raw_codes + C::kRawBytes);
  uint64_t* empty = full + C::kStg;
  uint64_t* tfull = empty + C::kStg;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* raw_full = drain + 1;           // q4: code stage landed (TMA bytes)
  uint64_t* raw_empty = raw_full + C::kRaw;  // q4: code stage converted by every dequant warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(raw_empty + C::kRaw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* never = reinterpret_cast<uint64_t*>(tmem_slot + 2);  // no thread ever arrives here
  uint8_t* epi_stage = reinterpret_cast<uint8_t*>(full) + 256;  // kEpiWarps x 4 KB (bf16 modes)
  // group table after the epilogue staging (bf16 modes) or the barriers (q4)
  int* s_mt = reinterpret_cast<int*>(reinterpret_cast<uint8_t*>(full) + 256 +
                                     (C::kStagedEpi ? kEpiWarps * 4096 : 0));  // [num_groups + 1]
  int* s_slot = s_mt + kMaxExperts + 1;                                       // [num_groups]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStg; ++s) {
      mbar_init(&full[s], C::kFullCount);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(never, 1);
    for (int r = 0; r < C::kRaw && C::kQ4; ++r) {
      mbar_init(&raw_full[r], 1);
      mbar_init(&raw_empty[r], C::kDq);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  if (warp == 5 && lane == 0) {
    if (C::kTmaB || C::kQ4) tma_prefetch(&tmB);
    if (C::kTmaA) tma_prefetch(&tmA);
  }
  for (int g = threadIdx.x; g < a.num_groups; g += blockDim.x) {
    s_mt[g] = __ldg(&a.groups[g].mt_begin);
    s_slot[g] = __ldg(&a.groups[g].slot);
  }
  if (threadIdx.x == 0) s_mt[a.num_groups] = __ldg(a.total_mtiles);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total = s_mt[a.num_groups] * a.nt;
  const long long lim = a.wait_limit;

  if (warp == 5) {
    // ------------------------------------------------------------- TMA producer
    if (lane == 0 && (C::kTmaAny || C::kQ4)) {
      uint32_t it = 0, raw_issued = 0;
      // the next tile's first A row is loaded one tile ahead (its latency
      // hides behind this tile's stages instead of stalling the ring)
      int rb_next = blockIdx.x < total ? __ldg(&a.groups[decode_tile(a, s_mt, blockIdx.x).g].row_begin) : 0;
      for (int t = blockIdx.x; t < total; t += gridDim.x) {
        const TileCoord tc = decode_tile(a, s_mt, t);
        const int brow = s_slot[tc.g] * a.b_rows_per_slot + a.b_row_off;
        const int arow = rb_next + tc.m * kBM;
        // q4: the tile's two 128-row blocks of packed codes (gate: n * 128 and
        // up: up_off + n * 128; down: n * 256 and n * 256 + 128)
        const int qbase = s_slot[tc.g] * a.q4_rows_per_slot + a.q4_row_off;
        const int qrow0 = qbase + (C::kGateUp ? tc.n * 128 : tc.n * kBN);
        const int qrow1 = C::kGateUp ? qbase + a.up_off + tc.n * 128 : qrow0 + 128;
        if (t + (int)gridDim.x < total)
          rb_next = __ldg(&a.groups[decode_tile(a, s_mt, t + gridDim.x).g].row_begin);
        bool ok = true;
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          if (C::kQ4) {
            const int r = it % C::kRaw;
            if (!mbar_wait(&raw_empty[r], ((it / C::kRaw) & 1) ^ 1, abort_flag, lim)) { ok = false; break; }
            mbar_arrive_expect_tx(&raw_full[r], C::kRawTx);
            uint8_t* q = raw_codes + r * (kBN * kRawRowBytes);
            tma_load_2d(q, &tmB, &raw_full[r], kb * kRawRowBytes, qrow0);
            tma_load_2d(q + 128 * kRawRowBytes, &tmB, &raw_full[r], kb * kRawRowBytes, qrow1);
            ++raw_issued;
            if (!C::kTmaAny) continue;
          }
          const int s = it % C::kStg;
          const uint32_t ph = (it / C::kStg) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], C::kTxBytes);
          uint8_t* b = sB + s * kBBytes;
          if (C::kTmaB && C::kGateUp) {
            tma_load_2d(b, &tmB, &full[s], kb * kBK, brow + tc.n * 128);
            tma_load_2d(b + kBBytes / 2, &tmB, &full[s], kb * kBK, brow + a.up_off + tc.n * 128);
          } else if (C::kTmaB) {
            tma_load_2d(b, &tmB, &full[s], kb * kBK, brow + tc.n * kBN);
            tma_load_2d(b + kBBytes / 2, &tmB, &full[s], kb * kBK, brow + tc.n * kBN + 128);
          }
          if (C::kTmaA) tma_load_2d(sA + s * kABytes, &tmA, &full[s], kb * kBK, arow);
        }
        if (!ok) break;
      }
      // On abort, wait (bounded) for the copies this thread armed to land
      // before the CTA's shared memory is released.
      if (*abort_flag) {
        for (int d = 0; d < C::kStg && it > 0 && C::kTmaAny; ++d) {
          const uint32_t j = it - 1 - d;
          if ((int)j < 0) break;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % C::kStg], (j / C::kStg) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
        for (int d = 0; d < C::kRaw && C::kQ4; ++d) {
          if ((int)raw_issued - 1 - d < 0) break;
          const uint32_t j = raw_issued - 1 - d;
          const long long t0 = clock64();
          while (!mbar_try_wait(&raw_full[j % C::kRaw], (j / C::kRaw) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
      }
    }
  } else if (warp == 4) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t it = 0, jt = 0;
      for (int t = blockIdx.x; t < total; t += gridDim.x, ++jt) {
        const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1, abort_flag, lim)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kBN;
        bool ok = true;
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          const int s = it % C::kStg;
          const uint32_t ph = (it / C::kStg) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
          // cp.async (generic proxy) wrote A in the gather modes: order those
          // writes before this thread's tensor-core (async proxy) reads
          if (C::kGather) fence_proxy_async_smem();
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * kABytes));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * kBBytes));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            // advance 16 bf16 (32 bytes) along K inside the 128-byte swizzle atom
            umma_bf16(d, ad + 2 * k, bd + 2 * k, kIdesc, (kb | k) != 0);
          }
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
  } else if (warp < kEpiWarps) {
    // ------------------------------------------------------------- epilogue
    uint32_t jt = 0;
    const int r = warp * 32 + lane;
    if (a.stall && threadIdx.x == 0) mbar_wait(never, 0, abort_flag, lim);  // runs out: abort
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++jt) {
      const TileCoord tc = decode_tile(a, s_mt, t);
      const Group* G = &a.groups[tc.g];
      const int cnt = __ldg(&G->row_count);
      const bool valid = tc.m * kBM + r < cnt;
      const size_t orow = (size_t)__ldg(&G->row_begin) + (size_t)tc.m * kBM + r;
      const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
      if (!mbar_wait(&tfull[acc], aph, abort_flag, lim)) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16) + acc * kBN;
      const int ncol0 = tc.n * (C::kGateUp ? 128 : kBN);
      if (C::kStagedEpi) {
        const int row_w = tc.m * kBM + warp * 32;  // the warp's first row inside the group
        epilogue_tile_staged<C::kGateUp>(
            tb, a.out + ((size_t)__ldg(&G->row_begin) + row_w) * a.out_ld + ncol0, a.out_ld,
            cnt - row_w, epi_stage + warp * 4096, lane);
      } else {
        epilogue_tile_lean<C::kGateUp>(tb, a.out + orow * a.out_ld + ncol0, valid);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  } else if (C::kGather && warp < C::kGatherWarp0 + kGatherWarps) {
    // ------------------------------------------------------------- row gather
    const int gt = threadIdx.x - C::kGatherWarp0 * 32;  // 0..127
    const int chunk = gt & 7;             // 16-byte chunk of a 128-byte row slice
    const int r0 = gt >> 3;               // rows r0 + 16 i
    uint32_t it = 0;
    bool ok = true;
    // permuted-row entries (t*k + j, or -1 past the expert's segment) of this
    // thread's eight rows, loaded one tile ahead so that the next tile's first
    // copies do not wait on the group and permutation loads
    auto tile_rows = [&](int t, int (&pr)[8]) {
      const TileCoord tc = decode_tile(a, s_mt, t);
      const Group* G = &a.groups[tc.g];
      const int cnt = __ldg(&G->row_count);
      const int rb = __ldg(&G->row_begin);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = tc.m * kBM + r0 + 16 * i;
        pr[i] = rr < cnt ? __ldg(&a.perm[rb + rr]) : -1;
      }
    };
    int pr[8], pr_next[8];
    if (blockIdx.x < total) tile_rows(blockIdx.x, pr);
    for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
      const bool has_next = t + (int)gridDim.x < total;
      if (has_next) tile_rows(t + gridDim.x, pr_next);
      const __nv_bfloat16* src[8];
      uint32_t nbytes[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (pr[i] >= 0) {
          src[i] = a.x + (size_t)(pr[i] / a.top_k) * a.x_ld + chunk * 8;
          nbytes[i] = 16;
        } else {
          src[i] = a.x;
          nbytes[i] = 0;  // zero-fill rows past the expert's segment
        }
      }
      for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
        const int s = it % C::kStg;
        const uint32_t ph = (it / C::kStg) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
        uint8_t* dstA = sA + s * kABytes;
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
  } else if (C::kQ4) {
    // ------------------------------------------------------------- q4 dequant
    // a warp takes 16 rows, two lanes to a row: its code reads cover 512
    // contiguous bytes and its SW128 writes hit distinct banks
    const int d = (warp - C::kDqWarp0) * 16 + (lane >> 1);  // B row of this thread, 0..255
    const int half = lane & 1;                               // codes 32 half .. 32 half + 31 of each stage
    const uint32_t my_tiles =
        (uint32_t)blockIdx.x < (uint32_t)total ? (total - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    const uint32_t nstages = my_tiles * a.kblocks;
    // this thread's scale row for tile ordinal j, from the shared-memory group
    // table (a search in global memory would stall the row's pipeline)
    uint32_t srow_tile = 0xFFFFFFFFu;
    const uint8_t* srow = nullptr;
    auto scales_of = [&](uint32_t st) -> uint2 {  // the two stages st, st + 1 (st even)
      const uint32_t j = st / a.kblocks;
      if (j != srow_tile) {
        const int t = blockIdx.x + j * gridDim.x;
        int lo = 0, hi = a.num_groups - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (s_mt[mid] * a.nt <= t) lo = mid; else hi = mid - 1;
        }
        const int mt = s_mt[lo + 1] - s_mt[lo];
        const int n = (t - s_mt[lo] * a.nt) / mt;
        int row;
        if (C::kGateUp) row = d < 128 ? n * 128 + d : a.up_off + n * 128 + (d - 128);
        else row = n * kBN + d;
        srow = a.q4_pool + (unsigned long long)s_slot[lo] * a.q4_extent + a.q4_scale_off +
               (size_t)row * a.q4_scale_ld;
        srow_tile = j;
      }
      // 4 fp16 scales, 8-byte aligned (row stride K / 16 bytes, K a multiple of 128)
      return __ldg(reinterpret_cast<const uint2*>(srow + (st % a.kblocks) * 4));
    };
    // scales of a stage pair are loaded one pair ahead (kblocks is even)
    uint2 sc_cur = nstages > 0 ? scales_of(0) : make_uint2(0, 0);
    uint2 sc_nxt = nstages > 2 ? scales_of(2) : make_uint2(0, 0);
    bool ok = true;
    for (uint32_t it = 0; it < nstages; ++it) {
      if (it > 0 && (it & 1) == 0) {
        sc_cur = sc_nxt;
        if (it + 2 < nstages) sc_nxt = scales_of(it + 2);
      }
      const int r = it % C::kRaw;
      if (!mbar_wait(&raw_full[r], (it / C::kRaw) & 1, abort_flag, lim)) { ok = false; break; }
      const int s = it % C::kStg;
      const uint32_t ph = (it / C::kStg) & 1;
      if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
      // this thread's half row: 32 codes (16 bytes) under one group scale
      const uint4 cw = ld_shared_v4(smem_u32(raw_codes + r * (kBN * kRawRowBytes) + d * kRawRowBytes + half * 16));
      const uint32_t sc = (it & 1) ? sc_cur.y : sc_cur.x;
      const float sv = __half2float(__ushort_as_half((unsigned short)(half ? sc >> 16 : sc & 0xFFFFu)));
      const uint64_t sx2 = f32x2(sv, sv), nx2 = f32x2(-136.0f * sv, -136.0f * sv);
      const uint32_t dst_row = smem_u32(sB + s * kBBytes + d * 128);
      const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = half * 4 + j;  // 16-byte chunk of the 128-byte row
        st_shared_v4(dst_row + ((c ^ (d & 7)) << 4), dequant8(words[j], sx2, nx2));
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&full[s]);
        mbar_arrive(&raw_empty[r]);  // the warp's rows of this code stage are consumed
      }
    }
    (void)ok;
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

template <int MODE>
static cudaError_t launch_mode(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& a,
                               int grid, cudaStream_t s) {
  static std::atomic<unsigned long long> attr_done{0};
  const int smem = Cfg<MODE>::kSmem;
  {
    cudaError_t e = smem_attr_once(grouped_gemm_kernel<MODE>, smem, attr_done);
    if (e != cudaSuccess) return e;
  }
  grouped_gemm_kernel<MODE><<<grid, Cfg<MODE>::kThreads, smem, s>>>(tmA, tmB, a);
  return cudaGetLastError();
}

cudaError_t launch_gemm(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& a,
                        int grid, cudaStream_t s) {
  switch (mode) {
    case kGateUpGather: return launch_mode<kGateUpGather>(tmA, tmB, a, grid, s);
    case kGateUpTma: return launch_mode<kGateUpTma>(tmA, tmB, a, grid, s);
    case kDown: return launch_mode<kDown>(tmA, tmB, a, grid, s);
    case kGateUpGatherQ4: return launch_mode<kGateUpGatherQ4>(tmA, tmB, a, grid, s);
    case kDownQ4: return launch_mode<kDownQ4>(tmA, tmB, a, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace msi
