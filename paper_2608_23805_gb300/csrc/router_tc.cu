// Router on tcgen05 tensor cores with fp32-exact products: fp32 logits,
// top-k, softmax weights, shared-expert gate and the per-block expert
// histogram in one kernel (the logits stay in TMEM).
//
// The router's top-k output is the route event recorded per layer and graph
// evaluation (paper, Sec. "Output-Exact Execution Beyond the Full-Residency
// Envelope").  Readings: weights are the softmax over the selected k logits;
// equal logits rank the lower expert id first.
//
// Exact split: every fp32 weight w equals hi + mid + lo with hi = bf16(w),
// mid = bf16(w - hi), lo = bf16(w - hi - mid) (each difference is exact in
// fp32 and the last remainder has at most 8 significant bits).  The hidden
// rows are bf16, so every product x * plane is exact in fp32 and
// logits = x Wr^T is three bf16 MMAs accumulating in fp32 -- the same value as
// an fp32 GEMM up to accumulation order.
//
// One CTA = 128 tokens x all E experts (E <= 512 fp32 accumulators per row in
// TMEM, in chunks of <= 256 columns).  Stage = 64 K of one plane of one
// expert chunk: x tile (TMA, 16 KB) + 256 weight rows (TMA, 32 KB), 4 stages.
// Warps 0-3: epilogue (one token row per thread: top-(k+1) insertion over the
// row's E logits in ascending id order, weights, gap, histogram, shared gate),
// warp 4: MMA + TMEM, warp 5: TMA producer.  All waits are bounded.
#include "internal.cuh"

namespace msi {

namespace {

constexpr int NTH = 192;
constexpr int RT_STAGES = 4;
constexpr int RT_A = 128 * 64 * 2;
constexpr int RT_B = 256 * 64 * 2;
constexpr int RT_SMEM = 1024 + RT_STAGES * (RT_A + RT_B) + 256 + kMaxExperts * 4;
constexpr int RT_LLD = kMaxExperts + 1;  // padded logits row (floats)
static_assert(64 * RT_LLD * 4 <= RT_STAGES * (RT_A + RT_B), "logits half does not fit");

__global__ void split3_kernel(const float* __restrict__ w, long long n, __nv_bfloat16* __restrict__ out) {
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const float v = w[i];
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(hi);
    const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
    const float r2 = r1 - __bfloat162float(mid);
    out[i] = hi;
    out[n + i] = mid;
    out[2 * n + i] = __float2bfloat16_rn(r2);
  }
}

__global__ void __launch_bounds__(NTH, 1)
    router_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                     const RouterTcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + RT_STAGES * RT_A;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + RT_STAGES * RT_B);
  uint64_t* empty = full + RT_STAGES;
  uint64_t* tfull = empty + RT_STAGES;
  uint64_t* drain = tfull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* hist = reinterpret_cast<int*>(reinterpret_cast<uint8_t*>(full) + 256);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, k = a.k;
  const int nchunk = (E + 255) / 256;
  const int kblocks = a.H / 64;
  const int nstage = nchunk * kblocks * 3;
  const int m0 = blockIdx.x * 128;
  const long long lim = a.wait_limit;

  for (int e = threadIdx.x; e < E; e += NTH) hist[e] = 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < RT_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, a.tmem_cols);
    tmem_relinquish();
  }
  if (warp == 5 && lane == 0) {
    tma_prefetch(&tmX);
    tma_prefetch(&tmW);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 5) {
    if (lane == 0) {
      int it = 0;
      for (; it < nstage; ++it) {
        const int s = it % RT_STAGES;
        const uint32_t ph = (it / RT_STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) break;
        const int c = it / (kblocks * 3);
        const int rem = it - c * kblocks * 3;
        const int kb = rem / 3, plane = rem - kb * 3;
        mbar_arrive_expect_tx(&full[s], RT_A + RT_B);
        tma_load_2d(sA + s * RT_A, &tmX, &full[s], kb * 64, m0);
        tma_load_2d(sB + s * RT_B, &tmW, &full[s], kb * 64, plane * E + c * 256);
      }
      if (*abort_flag) {
        for (int d = 0; d < RT_STAGES && it - 1 - d >= 0; ++d) {
          const int j = it - 1 - d;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % RT_STAGES], (j / RT_STAGES) & 1) && clock64() - t0 < lim) {
          }
        }
      }
    }
  } else if (warp == 4) {
    if (lane == 0) {
      bool ok = true;
      for (int it = 0; it < nstage; ++it) {
        const int s = it % RT_STAGES;
        const uint32_t ph = (it / RT_STAGES) & 1;
        if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
        tc_fence_after();
        const int c = it / (kblocks * 3);
        const int rem = it - c * kblocks * 3;
        const int n_c = min(256, E - c * 256);
        const uint32_t idesc = idesc_bf16(128, n_c);
        const uint64_t ad = sw128_desc(smem_u32(sA + s * RT_A));
        const uint64_t bd = sw128_desc(smem_u32(sB + s * RT_B));
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          umma_bf16(tmem_base + c * 256, ad + 2 * kk, bd + 2 * kk, idesc, (rem | kk) != 0);
        umma_commit(&empty[s]);
      }
      if (ok) umma_commit(tfull);
      umma_commit(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0) && clock64() - t0 < lim) {
      }
    }
  } else {
    // ------------------------------------------------------------- epilogue
    // Logits TMEM -> shared memory (the stage buffers are free once the MMA
    // loop is done), 64 rows at a time, rows padded to LLD floats so that the
    // 32 lanes' column writes fall into distinct banks; then one warp per
    // token picks the top k+1 by warp-shuffle argmax (logit desc, id asc).
    const bool ready = __all_sync(0xffffffffu, mbar_wait(tfull, 0, abort_flag, lim));
    tc_fence_after();
    float* L = reinterpret_cast<float*>(smem);
    const int tid = threadIdx.x;  // 0..127
    const int per_lane = (E + 31) >> 5;
    for (int half = 0; half < 2; ++half) {
      if (ready && (warp >> 1) == half) {
        const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16);
        float* row = L + (size_t)((warp & 1) * 32 + lane) * RT_LLD;
        for (int e0 = 0; e0 < E; e0 += 16) {
          uint32_t v[16];
          tmem_ld16(tb + e0, v);
          tmem_ld_wait(v);
#pragma unroll
          for (int j = 0; j < 16; ++j) row[e0 + j] = __uint_as_float(v[j]);
        }
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (ready) {
        for (int q = 0; q < 16; ++q) {
          const int rl = warp * 16 + q;           // row within this half
          const int t = m0 + half * 64 + rl;
          if (t >= a.T) break;
          const float* row = L + (size_t)rl * RT_LLD;
          float v[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int e = lane + 32 * i;
            v[i] = (i < per_lane && e < E) ? row[e] : -INFINITY;
          }
          uint32_t removed = 0;
          float my_v = -INFINITY, next_v = -INFINITY;
          int my_i = 0;
          const int rounds = min(k + 1, E);
          for (int rr = 0; rr < rounds; ++rr) {
            float bv = -INFINITY;
            int bi = 0x7fffffff;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int e = lane + 32 * i;
              if (i < per_lane && e < E && !((removed >> i) & 1u)) {
                if (v[i] > bv || (v[i] == bv && e < bi)) { bv = v[i]; bi = e; }
              }
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
              const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
              const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
              if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
            }
            if ((bi & 31) == lane) removed |= 1u << (bi >> 5);
            if (rr == lane) { my_v = bv; my_i = bi; }
            if (rr == k) next_v = bv;
          }
          const float l0 = __shfl_sync(0xffffffffu, my_v, 0);
          const float ex = (lane < k) ? expf(my_v - l0) : 0.f;
          float sum = ex;
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
          if (lane < k) {
            a.ids[(size_t)t * k + lane] = my_i;
            a.weights[(size_t)t * k + lane] = ex / sum;
            atomicAdd(&hist[my_i], 1);
          }
          if (a.gap != nullptr) {
            const float lk1 = __shfl_sync(0xffffffffu, my_v, k - 1);
            if (lane == 0) a.gap[t] = (k < E) ? (lk1 - next_v) : INFINITY;
          }
        }
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
    }
    tc_fence_before();
    if (a.wsg != nullptr) {
      // shared-expert gate: warp w computes x . w_sg for rows w*32 .. w*32+31
      for (int q = 0; q < 32; ++q) {
        const int tt = m0 + warp * 32 + q;
        if (tt >= a.T) break;
        const __nv_bfloat16* xr = a.x + (size_t)tt * a.H;
        float s = 0.f;
#pragma unroll 8
        for (int h = lane * 8; h < a.H; h += 256) {
          const uint4 xv = __ldg(reinterpret_cast<const uint4*>(xr + h));
          const float4 w0 = __ldg(reinterpret_cast<const float4*>(a.wsg + h));
          const float4 w1 = __ldg(reinterpret_cast<const float4*>(a.wsg + h + 4));
          s = fmaf(bf16_lo(xv.x), w0.x, s);
          s = fmaf(bf16_hi(xv.x), w0.y, s);
          s = fmaf(bf16_lo(xv.y), w0.z, s);
          s = fmaf(bf16_hi(xv.y), w0.w, s);
          s = fmaf(bf16_lo(xv.z), w1.x, s);
          s = fmaf(bf16_hi(xv.z), w1.y, s);
          s = fmaf(bf16_lo(xv.w), w1.z, s);
          s = fmaf(bf16_hi(xv.w), w1.w, s);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
        if (lane == 0) a.sg[tt] = 1.0f / (1.0f + expf(-s));
      }
    }
    // histogram of this block's routed ids -> bcount[block][e]
    for (int e = tid; e < E; e += 128) a.bcount[(size_t)blockIdx.x * E + e] = hist[e];
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, a.tmem_cols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicCAS(a.status, 0, (int)MSI_ERR_TIMEOUT);
}

}  // namespace

cudaError_t launch_split3(const float* w, long long n, __nv_bfloat16* out, cudaStream_t s) {
  const long long want = (n + 255) / 256;
  const int grid = (int)(want < 152 * 8 ? want : 152 * 8);
  split3_kernel<<<grid, 256, 0, s>>>(w, n, out);
  return cudaGetLastError();
}

cudaError_t launch_router_tc(const CUtensorMap& tmX, const CUtensorMap& tmW, const RouterTcArgs& a,
                             cudaStream_t s) {
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(router_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         RT_SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int nb = (a.T + 127) / 128;
  if (nb == 0) return cudaSuccess;
  router_tc_kernel<<<nb, NTH, RT_SMEM, s>>>(tmX, tmW, a);
  return cudaGetLastError();
}

}  // namespace msi
