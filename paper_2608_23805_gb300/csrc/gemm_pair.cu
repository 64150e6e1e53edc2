// Grouped expert GEMMs on CTA pairs (tcgen05 cta_group::2, sm_103a).
//
// Same projections as the single-CTA kernel in gemm.cu (paper, Sec.
// "Output-Exact Execution Beyond the Full-Residency Envelope": each selected
// expert's gate, up and down projections over its routed rows, weights read
// from the stable slot address the Plan published), for groups large enough
// to fill 256-row tiles, as in a long prefill.
//
// Two CTAs on neighbouring SMs form a cluster and share one 256 x 256 output
// tile.  CTA r holds A rows [128 r, 128 r + 128) of the tile and B rows
// (output columns) [128 r, 128 r + 128) in its own shared memory; the even
// CTA issues the pair MMA, which reads both halves of A and B at the same
// shared-memory offsets and accumulates each CTA's 128 rows into that CTA's
// TMEM.  Per K step of 64 each SM therefore fills 32 KB of shared memory for
// 128 x 256 x 64 multiply-adds, against 48 KB in the single-CTA tile: the
// reduction that lets the tensor pipe outrun the L2 -> SM feed.
//
// Tile: 256 token rows x 256 output columns x 64 K per stage, 6-stage ring per
// CTA, fp32 accumulators double-buffered in TMEM (2 x 256 columns).
//
// Synchronisation (all waits bounded; on expiry the CTA raises its abort flag,
// the roles drain and the status word reports MSI_ERR_TIMEOUT):
//   * each CTA's TMA loads and row-gather copies complete on that CTA's own
//     `full` barrier; in the odd CTA a relay thread forwards each completed
//     stage to the even CTA's `full` barrier, so no copy ever signals a
//     barrier in the other CTA (an aborted CTA never receives a late
//     transaction count);
//   * the even CTA's MMA thread waits its `full` barrier (own stage + relayed
//     peer stage), issues four pair MMAs and commits to `empty` of both CTAs
//     (multicast), and to `tfull` of both CTAs at the end of a tile;
//   * the epilogue warps of both CTAs read their own TMEM and arrive on the
//     even CTA's `tempty` barrier (eight arrivals free an accumulator);
//   * teardown: the MMA issuer's final commit reaches `drain` in both CTAs,
//     each CTA waits it, then a cluster barrier, then both release TMEM.
// Cross-CTA arrivals are plain (CTA-scope release) remote arrives: a
// cluster-scope release or acquire on every K step serialises the pipeline
// behind a cluster-wide fence (measured: 1.5-1.9x slower).
//
// Roles per CTA: warps 0-3 epilogue, warp 4 MMA issue (even CTA) or stage
// relay (odd CTA) and TMEM allocation, warp 5 TMA producer, warps 6-9 row
// gather (gate-up over routed rows), and in the 4-bit modes sixteen dequant
// warps.
//
// 4-bit modes: each CTA converts only its own 128 B rows (half of the pair
// tile's 256), so per unit of tensor work a CTA dequantises half as many
// weights as a single-CTA tile does.  The producer loads the CTA's 128 rows of
// packed codes per stage by TMA into a three-stage raw ring; each dequant
// thread converts a quarter row (16 codes under one group scale) into the
// CTA's SW128 B stage and arrives on its own `full` barrier, which the relay
// forwards as in the bf16 modes.
#include <algorithm>

#include "internal.cuh"

namespace msi {

namespace {

constexpr int kPairRows = 2 * kBM;         // 256 token rows per pair tile
constexpr int kPStages = 6;
constexpr int kPA = kBM * kBK * 2;         // 16 KB: this CTA's 128 A rows of one K step
constexpr int kPB = 128 * kBK * 2;         // 16 KB: this CTA's 128 B rows of one K step
constexpr uint32_t kPIdesc = idesc_bf16(kPairRows, kBN);
constexpr int kPEpiWarps = 4;
constexpr int kPGatherWarps = 4;
constexpr int kPRawRow = 32;               // 64 codes of one B row per stage (one TMA box row)

template <int MODE>
struct PCfg {
  static constexpr bool kQ4 = (MODE == kGateUpGatherQ4 || MODE == kDownQ4);
  static constexpr bool kGather = (MODE == kGateUpGather || MODE == kGateUpGatherQ4);
  static constexpr bool kGateUp = (MODE == kGateUpGather || MODE == kGateUpTma || MODE == kGateUpGatherQ4);
  static constexpr int kGatherWarp0 = 6;
  static constexpr int kDqWarp0 = kGatherWarp0 + (kGather ? kPGatherWarps : 0);
  static constexpr int kDq = kQ4 ? 16 : 0;  // dequant warps (one thread per quarter B row)
  static constexpr int kThreads = (kDqWarp0 + kDq) * 32;
  // the producer arms `full` when it loads an operand by TMA (B in the bf16
  // modes, A whenever the rows are not gathered)
  static constexpr bool kProducerFull = !kQ4 || !kGather;
  static constexpr uint32_t kTx = (kQ4 ? 0 : kPB) + (kGather ? 0 : kPA);
  // own producer (expect_tx) + own gather threads (one arrival each as their
  // copies land) + own dequant warps
  static constexpr int kFullLocal = (kProducerFull ? 1 : 0) + (kGather ? kPGatherWarps * 32 : 0) + kDq;
  static constexpr int kRaw = kQ4 ? 3 : 1;
  static constexpr int kRawBytes = kQ4 ? kRaw * 128 * kPRawRow : 0;
  static constexpr uint32_t kRawTx = 128 * kPRawRow;
  // + the groups' 256-row tile prefix and slot (shared-memory tile lookups)
  static constexpr int kSmem = 1024 + kPStages * (kPA + kPB) + kRawBytes + 256 + kPEpiWarps * 4096 +
                               (2 * kMaxExperts + 2) * 4;
};

struct PairTile {
  int g, m2, n;
};

// Pair tile t -> (group, 256-row tile, column tile) from the shared-memory
// table of the groups' pair-tile prefix (s_pt[num_groups] = total).
__device__ __forceinline__ PairTile decode_pair(const GemmArgs& a, const int* s_pt, int t) {
  int lo = 0, hi = a.num_groups - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_pt[mid] * a.nt <= t) lo = mid; else hi = mid - 1;
  }
  const int mt2 = s_pt[lo + 1] - s_pt[lo];
  const int local = t - s_pt[lo] * a.nt;
  PairTile c;
  c.g = lo;
  c.n = local / mt2;
  c.m2 = local - c.n * mt2;
  return c;
}

}  // namespace

template <int MODE>
__global__ void __launch_bounds__(PCfg<MODE>::kThreads, 1)
    grouped_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA,
                             const __grid_constant__ CUtensorMap tmB, const GemmArgs a) {
  using C = PCfg<MODE>;
  extern __shared__ uint8_t smem_raw[];
  // the same offsets in both CTAs: the pair MMA addresses the peer's operands
  // through the even CTA's descriptors
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kPStages * kPA;
  uint8_t* raw_codes = sB + kPStages * kPB;  // q4: [C::kRaw][128][32]
  uint64_t* full = reinterpret_cast<uint64_t*>(raw_codes + C::kRawBytes);
  uint64_t* empty = full + kPStages;
  uint64_t* tfull = empty + kPStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* raw_full = drain + 1;            // q4: code stage landed (TMA bytes)
  uint64_t* raw_empty = raw_full + C::kRaw;  // q4: code stage converted by every dequant warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(raw_empty + C::kRaw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* never = reinterpret_cast<uint64_t*>(tmem_slot + 2);  // no thread ever arrives here
  uint8_t* epi_stage = reinterpret_cast<uint8_t*>(full) + 256;  // 4 KB per epilogue warp
  int* s_pt = reinterpret_cast<int*>(epi_stage + kPEpiWarps * 4096);  // [num_groups + 1]
  int* s_slot = s_pt + kMaxExperts + 1;                               // [num_groups]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPStages; ++s) {
      mbar_init(&full[s], C::kFullLocal + (leader ? 1 : 0));  // + the peer's relay
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 2 * kPEpiWarps);  // the epilogue warps of both CTAs
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
    tmem_alloc_pair(tmem_slot, 512);
    tmem_relinquish_pair();
  }
  if (warp == 5 && lane == 0) {
    tma_prefetch(&tmB);
    if (!C::kGather) tma_prefetch(&tmA);
  }
  for (int g = threadIdx.x; g < a.num_groups; g += blockDim.x) {
    s_pt[g] = __ldg(&a.groups[g].pt_begin);
    s_slot[g] = __ldg(&a.groups[g].slot);
  }
  if (threadIdx.x == 0) s_pt[a.num_groups] = __ldg(a.total_mtiles + 1);
  tc_fence_before();
  cluster_sync_all();  // both CTAs' barriers initialised before any cross-CTA arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total = s_pt[a.num_groups] * a.nt;
  const int pair = blockIdx.x >> 1;
  const int npairs = gridDim.x >> 1;
  const long long lim = a.wait_limit;

  if (warp == 5) {
    // ------------------------------------------------------------- TMA producer
    if (lane == 0) {
      uint32_t it = 0, raw_issued = 0;
      // the next tile's first A row is loaded one tile ahead
      int rb_next = pair < total ? __ldg(&a.groups[decode_pair(a, s_pt, pair).g].row_begin) : 0;
      for (int t = pair; t < total; t += npairs) {
        const PairTile tc = decode_pair(a, s_pt, t);
        const int rb = rb_next;
        if (t + npairs < total) rb_next = __ldg(&a.groups[decode_pair(a, s_pt, t + npairs).g].row_begin);
        const int brow0 = s_slot[tc.g] * a.b_rows_per_slot + a.b_row_off;
        // gate-up: the even CTA holds 128 gate rows, the odd CTA the matching up rows
        const int brow = C::kGateUp ? brow0 + (rank ? a.up_off : 0) + tc.n * 128
                                    : brow0 + tc.n * kBN + (int)rank * 128;
        const int arow = rb + tc.m2 * kPairRows + (int)rank * kBM;
        // q4: this CTA's 128 rows of packed codes (gate-up: gate rows in the
        // even CTA, up rows in the odd one, as for the bf16 rows)
        const int qbase = s_slot[tc.g] * a.q4_rows_per_slot + a.q4_row_off;
        const int qrow = C::kGateUp ? qbase + (rank ? a.up_off : 0) + tc.n * 128
                                    : qbase + tc.n * kBN + (int)rank * 128;
        bool ok = true;
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          if (C::kQ4) {
            const int r = it % C::kRaw;
            if (!mbar_wait(&raw_empty[r], ((it / C::kRaw) & 1) ^ 1, abort_flag, lim)) { ok = false; break; }
            mbar_arrive_expect_tx(&raw_full[r], C::kRawTx);
            tma_load_2d(raw_codes + r * (128 * kPRawRow), &tmB, &raw_full[r], kb * kPRawRow, qrow);
            ++raw_issued;
            if (!C::kProducerFull) continue;
          }
          const int s = it % kPStages;
          const uint32_t ph = (it / kPStages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[s], C::kTx);
          if (!C::kQ4) tma_load_2d(sB + s * kPB, &tmB, &full[s], kb * kBK, brow);
          if (!C::kGather) tma_load_2d(sA + s * kPA, &tmA, &full[s], kb * kBK, arow);
        }
        if (!ok) break;
      }
      // On abort, wait (bounded) for the copies this thread armed to land
      // before the CTA's shared memory is released.
      if (*abort_flag) {
        for (int d = 0; d < kPStages && it > 0 && C::kProducerFull; ++d) {
          const uint32_t j = it - 1 - d;
          if ((int)j < 0) break;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % kPStages], (j / kPStages) & 1) && clock64() - t0 < kDrainCycles) {
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
    if (lane == 0 && leader) {
      // ----------------------------------------------------------- MMA issuer
      uint32_t it = 0, jt = 0;
      for (int t = pair; t < total; t += npairs, ++jt) {
        const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1, abort_flag, lim)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kBN;
        bool ok = true;
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          const int s = it % kPStages;
          const uint32_t ph = (it / kPStages) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
          // this CTA's gathered rows were written by cp.async (generic proxy);
          // the relay fenced the peer's before forwarding its stage
          if (C::kGather) fence_proxy_async_smem();
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(sA + s * kPA));
          const uint64_t bd = sw128_desc(smem_u32(sB + s * kPB));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            umma_bf16_pair(d, ad + 2 * k, bd + 2 * k, kPIdesc, (kb | k) != 0);
          }
          umma_commit_pair(&empty[s]);
        }
        if (!ok) break;
        umma_commit_pair(&tfull[acc]);
      }
      umma_commit_pair(drain);
    } else if (lane == 0) {
      // ------------------------------------------------------ stage relay (odd)
      const uint32_t my_tiles = pair < total ? (uint32_t)((total - 1 - pair) / npairs + 1) : 0u;
      const uint32_t nst = my_tiles * (uint32_t)a.kblocks;
      for (uint32_t it = 0; it < nst; ++it) {
        const int s = it % kPStages;
        const uint32_t ph = (it / kPStages) & 1;
        if (!mbar_wait(&full[s], ph, abort_flag, lim)) break;
        if (C::kGather) fence_proxy_async_smem();
        mbar_arrive_remote(mapa_shared(smem_u32(&full[s]), 0));
      }
    }
    if (lane == 0) {
      // every pair MMA that reads this CTA's shared memory or writes its TMEM
      // has completed before either is released
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0) && clock64() - t0 < kDrainCycles) {
      }
    }
  } else if (warp < kPEpiWarps) {
    // ------------------------------------------------------------- epilogue
    uint32_t jt = 0;
    const uint32_t lead_tempty[2] = {mapa_shared(smem_u32(&tempty[0]), 0),
                                     mapa_shared(smem_u32(&tempty[1]), 0)};
    if (a.stall && threadIdx.x == 0) mbar_wait(never, 0, abort_flag, lim);  // runs out: abort
    for (int t = pair; t < total; t += npairs, ++jt) {
      const PairTile tc = decode_pair(a, s_pt, t);
      const Group* G = &a.groups[tc.g];
      const int cnt = __ldg(&G->row_count);
      const uint32_t acc = jt & 1, aph = (jt >> 1) & 1;
      if (!mbar_wait(&tfull[acc], aph, abort_flag, lim)) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16) + acc * kBN;
      const int row_w = tc.m2 * kPairRows + (int)rank * kBM + warp * 32;  // warp's first row in the group
      __nv_bfloat16* row0 =
          a.out + ((size_t)__ldg(&G->row_begin) + row_w) * a.out_ld + tc.n * (C::kGateUp ? 128 : kBN);
      if (C::kQ4)
        epilogue_tile_staged_lean<C::kGateUp>(tb, row0, a.out_ld, cnt - row_w, epi_stage + warp * 4096, lane);
      else
        epilogue_tile_staged<C::kGateUp>(tb, row0, a.out_ld, cnt - row_w, epi_stage + warp * 4096, lane);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(lead_tempty[acc]);
    }
  } else if (C::kGather && warp < C::kGatherWarp0 + kPGatherWarps) {
    // ------------------------------------------------------------- row gather
    const int gt = threadIdx.x - C::kGatherWarp0 * 32;  // 0..127
    const int chunk = gt & 7;             // 16-byte chunk of a 128-byte row slice
    const int r0 = gt >> 3;               // rows r0 + 16 i of this CTA's 128
    uint32_t it = 0;
    bool ok = true;
    // permuted-row entries of this thread's eight rows, one tile ahead
    auto tile_rows = [&](int t, int (&pr)[8]) {
      const PairTile tc = decode_pair(a, s_pt, t);
      const Group* G = &a.groups[tc.g];
      const int cnt = __ldg(&G->row_count);
      const int rb = __ldg(&G->row_begin);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = tc.m2 * kPairRows + (int)rank * kBM + r0 + 16 * i;
        pr[i] = rr < cnt ? __ldg(&a.perm[rb + rr]) : -1;
      }
    };
    int pr[8], pr_next[8];
    if (pair < total) tile_rows(pair, pr);
    for (int t = pair; t < total && ok; t += npairs) {
      const bool has_next = t + npairs < total;
      if (has_next) tile_rows(t + npairs, pr_next);
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
        const int s = it % kPStages;
        const uint32_t ph = (it / kPStages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) { ok = false; break; }
        uint8_t* dstA = sA + s * kPA;
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
  } else if (C::kQ4 && warp >= C::kDqWarp0) {
    // ------------------------------------------------------------- q4 dequant
    // a warp takes 8 rows, four lanes to a row: its code reads cover 256
    // contiguous bytes and its SW128 writes hit distinct banks
    const int d = (warp - C::kDqWarp0) * 8 + (lane >> 2);  // this CTA's B row, 0..127
    const int qt = lane & 3;                                // codes 16 qt .. 16 qt + 15 of each stage
    const uint32_t my_tiles = pair < total ? (uint32_t)((total - 1 - pair) / npairs + 1) : 0u;
    const uint32_t nstages = my_tiles * (uint32_t)a.kblocks;
    // this thread's scale row for tile ordinal j (shared-memory group table)
    uint32_t srow_tile = 0xFFFFFFFFu;
    const uint8_t* srow = nullptr;
    auto scales_of = [&](uint32_t st) -> uint2 {  // stages st, st + 1 (st even)
      const uint32_t j = st / a.kblocks;
      if (j != srow_tile) {
        const PairTile tc = decode_pair(a, s_pt, pair + (int)j * npairs);
        const int row = C::kGateUp ? (rank ? a.up_off : 0) + tc.n * 128 + d
                                   : tc.n * kBN + (int)rank * 128 + d;
        srow = a.q4_pool + (unsigned long long)s_slot[tc.g] * a.q4_extent + a.q4_scale_off +
               (size_t)row * a.q4_scale_ld;
        srow_tile = j;
      }
      // 4 fp16 scales, 8-byte aligned (row stride K / 16 bytes, K a multiple of 128)
      return __ldg(reinterpret_cast<const uint2*>(srow + (st % a.kblocks) * 4));
    };
    uint2 sc_cur = nstages > 0 ? scales_of(0) : make_uint2(0, 0);
    uint2 sc_nxt = nstages > 2 ? scales_of(2) : make_uint2(0, 0);
    for (uint32_t it = 0; it < nstages; ++it) {
      if (it > 0 && (it & 1) == 0) {
        sc_cur = sc_nxt;
        if (it + 2 < nstages) sc_nxt = scales_of(it + 2);
      }
      const int r = it % C::kRaw;
      if (!mbar_wait(&raw_full[r], (it / C::kRaw) & 1, abort_flag, lim)) break;
      const int s = it % kPStages;
      const uint32_t ph = (it / kPStages) & 1;
      if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) break;
      const uint2 cw = ld_shared_v2(smem_u32(raw_codes + r * (128 * kPRawRow) + d * kPRawRow + qt * 8));
      const uint32_t sc = (it & 1) ? sc_cur.y : sc_cur.x;
      const float sv = __half2float(__ushort_as_half((unsigned short)(qt >= 2 ? sc >> 16 : sc & 0xFFFFu)));
      const uint64_t sx2 = f32x2(sv, sv), nx2 = f32x2(-136.0f * sv, -136.0f * sv);
      const uint32_t dst_row = smem_u32(sB + s * kPB + d * 128);
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

namespace {

struct PairLaunchInfo {
  std::atomic<unsigned long long> attr_done{0};
  std::atomic<int> max_clusters[64] = {};
};

template <int MODE>
cudaError_t launch_pair_mode(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& a,
                             int max_pairs, cudaStream_t s) {
  static PairLaunchInfo info;
  const int smem = PCfg<MODE>::kSmem;
  auto kernel = grouped_gemm_pair_kernel<MODE>;
  cudaError_t e = smem_attr_once(kernel, smem, info.attr_done);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(PCfg<MODE>::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  // pairs that can be resident at once (a persistent grid never waits for a
  // pair to finish before another can start)
  int mc = dev < 64 ? info.max_clusters[dev].load() : 0;
  if (mc <= 0) {
    cfg.gridDim = dim3(2, 1, 1);
    e = cudaOccupancyMaxActiveClusters(&mc, kernel, &cfg);
    if (e != cudaSuccess) return e;
    if (mc <= 0) return cudaErrorInvalidConfiguration;
    if (dev < 64) info.max_clusters[dev].store(mc);
  }
  const int pairs = std::max(1, std::min(mc, max_pairs));
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  return cudaLaunchKernelEx(&cfg, kernel, tmA, tmB, a);
}

}  // namespace

cudaError_t launch_gemm_pair(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                             const GemmArgs& a, int max_pairs, cudaStream_t s) {
  switch (mode) {
    case kGateUpGather: return launch_pair_mode<kGateUpGather>(tmA, tmB, a, max_pairs, s);
    case kGateUpTma: return launch_pair_mode<kGateUpTma>(tmA, tmB, a, max_pairs, s);
    case kDown: return launch_pair_mode<kDown>(tmA, tmB, a, max_pairs, s);
    case kGateUpGatherQ4: return launch_pair_mode<kGateUpGatherQ4>(tmA, tmB, a, max_pairs, s);
    case kDownQ4: return launch_pair_mode<kDownQ4>(tmA, tmB, a, max_pairs, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace msi
