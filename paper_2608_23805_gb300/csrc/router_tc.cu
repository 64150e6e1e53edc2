// Router on tcgen05 tensor cores with fp32-exact products: fp32 logits,
// top-k, softmax weights, shared-expert gate and the per-block expert
// histogram (the logits never reach HBM).
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
// Two kernels:
//  1. router_tc_kernel, one CTA per (128 tokens, chunk of <= 128 experts):
//     logits of the chunk in TMEM (per stage one x tile and the chunk's rows
//     of all three planes, by TMA, feeding 12 MMAs), then each token's
//     top-(k+1) candidates within the chunk by warp-shuffle argmax (logit
//     desc, id asc) from shared memory, four rows at a time per warp.
//  2. router_merge_kernel, one CTA per 32 tokens (sixteen warps, two tokens
//     each): the top-(k+1) of the union of the chunks' candidates (it contains
//     the global top-(k+1)), weights, gap, the block's expert histogram for
//     the permutation and the shared-expert gate sigmoid(x . w_sg).
// Warps 0-3 move the logits from TMEM to shared memory, warp 4 MMA + TMEM,
// warp 5 TMA producer (one lane each for the single-thread roles; every role
// claims its whole warp); then all eight warps select.  All waits are bounded.
#include "kernels.cuh"

namespace msi {

namespace {

constexpr int NTH = 256;  // 8 warps: all of them select top-k once the logits are in smem
constexpr int RT_STAGES = 3;
constexpr int RT_A = 128 * 64 * 2;                   // x tile (64 K)
constexpr int RT_B = kRouterChunk * 64 * 2;          // one plane's chunk weight rows (64 K)
constexpr int RT_STAGE = RT_A + 3 * RT_B;            // x tile + the three planes
constexpr int RT_LLD = kRouterChunk + 1;             // padded logits row (floats)
constexpr int RT_SMEM = 1024 + RT_STAGES * RT_STAGE + 256;
static_assert(128 * RT_LLD * 4 <= RT_STAGES * RT_STAGE, "logits tile does not fit");

__device__ __forceinline__ void split3_body(const float* __restrict__ w, long long n,
                                            __nv_bfloat16* __restrict__ out, int* status, Group* sh,
                                            int* sh_total, int T, int shared_slot) {
  // the forward's first kernel (status null: a prediction pass)
  if (blockIdx.x == 0 && threadIdx.x == 0 && status != nullptr)
    forward_begin(status, sh, sh_total, T, shared_slot);
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

__global__ void split3_kernel(const float* __restrict__ w, long long n, __nv_bfloat16* __restrict__ out,
                              int* status, Group* sh, int* sh_total, int T, int shared_slot) {
  split3_body(w, n, out, status, sh, sh_total, T, shared_slot);
}

// The same, plus the resident call's table copied to global memory: the
// first warp of each block takes 32 entries, so the argument's entries are
// read through many SMs' constant caches at once.
__global__ void split3_table_kernel(const float* __restrict__ w, long long n,
                                    __nv_bfloat16* __restrict__ out, int* status, Group* sh,
                                    int* sh_total, int T, int shared_slot, const TableParams tp,
                                    int* __restrict__ tab_slot,
                                    unsigned long long* __restrict__ tab_expected) {
  if (threadIdx.x < 32) {
    for (int g = blockIdx.x * 32 + threadIdx.x; g < tp.E; g += gridDim.x * 32) {
      tab_slot[g] = tp.slot[g];
      tab_expected[g] = tp.expected[g];
    }
  }
  split3_body(w, n, out, status, sh, sh_total, T, shared_slot);
}

// Selection order of the route event: logit descending, then expert id
// ascending.  A logit maps to a 32-bit key with the same order (-0 counted as
// +0), so a warp finds the best head of its lanes with one redux.sync max and
// breaks a tie with one redux.sync min over the ids holding that key.
__device__ __forceinline__ uint32_t logit_key(float v) {
  uint32_t b = __float_as_uint(v);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_logit(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// Sort one lane's N (key, id) pairs: key descending, id ascending.
template <int N>
__device__ __forceinline__ void sort_desc(uint32_t (&k)[N], int (&id)[N]) {
#pragma unroll
  for (int i = 1; i < N; ++i) {
#pragma unroll
    for (int j = i; j > 0; --j) {
      const bool sw = k[j] > k[j - 1] || (k[j] == k[j - 1] && id[j] < id[j - 1]);
      const uint32_t tk = sw ? k[j - 1] : k[j];
      const int ti = sw ? id[j - 1] : id[j];
      k[j - 1] = sw ? k[j] : k[j - 1];
      id[j - 1] = sw ? id[j] : id[j - 1];
      k[j] = tk;
      id[j] = ti;
    }
  }
}

// One selection round over the lanes' sorted heads: returns the winning key
// and id (same in every lane); the lane that held it drops its head.
template <int N>
__device__ __forceinline__ void take_best(uint32_t (&k)[N], int (&id)[N], uint32_t& bk, int& bi) {
  bk = __reduce_max_sync(0xffffffffu, k[0]);
  bi = __reduce_min_sync(0xffffffffu, k[0] == bk ? id[0] : 0x7fffffff);
  if (id[0] == bi && k[0] == bk) {
#pragma unroll
    for (int i = 0; i + 1 < N; ++i) {
      k[i] = k[i + 1];
      id[i] = id[i + 1];
    }
    k[N - 1] = 0u;  // below every logit's key
    id[N - 1] = 0x7fffffff;
  }
}

__global__ void __launch_bounds__(NTH, 1)
    router_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                     const RouterTcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + RT_STAGES * RT_STAGE);
  uint64_t* empty = full + RT_STAGES;
  uint64_t* tfull = empty + RT_STAGES;
  uint64_t* drain = tfull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* ready_flag = const_cast<int*>(abort_flag) + 1;
  uint64_t* never = reinterpret_cast<uint64_t*>(tmem_slot + 4);  // no thread ever arrives here

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E;
  const int ch = a.chunk;                 // experts per chunk
  // the chunks of one token tile are neighbours in launch order, so the x
  // tile is read from HBM once and from L2 by the other chunks
  const int c = (int)(blockIdx.x % (unsigned)a.nchunk);  // chunk index
  const int kblocks = a.H / 64;
  const int nstage = kblocks;
  const int m0 = (int)(blockIdx.x / (unsigned)a.nchunk) * 128;
  const long long lim = a.wait_limit;

  if (threadIdx.x == 0) {
    for (int s = 0; s < RT_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(drain, 1);
    mbar_init(never, 1);
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
    // ------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int it = 0;
      for (; it < nstage; ++it) {
        const int s = it % RT_STAGES;
        const uint32_t ph = (it / RT_STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, lim)) break;
        uint8_t* st = smem + s * RT_STAGE;
        // x box: 128 rows of 64 bf16; weight boxes: `ch` rows of 64 bf16 per plane
        mbar_arrive_expect_tx(&full[s], RT_A + 3 * ch * 128);
        tma_load_2d(st, &tmX, &full[s], it * 64, m0);
#pragma unroll
        for (int plane = 0; plane < 3; ++plane)
          tma_load_2d(st + RT_A + plane * RT_B, &tmW, &full[s], it * 64, plane * E + c * ch);
      }
      if (*abort_flag) {
        for (int d = 0; d < RT_STAGES && it - 1 - d >= 0; ++d) {
          const int j = it - 1 - d;
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[j % RT_STAGES], (j / RT_STAGES) & 1) && clock64() - t0 < kDrainCycles) {
          }
        }
      }
    }
  } else if (warp == 4) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      bool ok = true;
      const uint32_t idesc = idesc_bf16(128, ch);
      for (int it = 0; it < nstage; ++it) {
        const int s = it % RT_STAGES;
        const uint32_t ph = (it / RT_STAGES) & 1;
        if (!mbar_wait(&full[s], ph, abort_flag, lim)) { ok = false; break; }
        tc_fence_after();
        const uint8_t* st = smem + s * RT_STAGE;
        const uint64_t ad = sw128_desc(smem_u32(st));
#pragma unroll
        for (int plane = 0; plane < 3; ++plane) {
          const uint64_t bd = sw128_desc(smem_u32(st + RT_A + plane * RT_B));
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            umma_bf16(tmem_base, ad + 2 * kk, bd + 2 * kk, idesc, (it | plane | kk) != 0);
        }
        umma_commit(&empty[s]);
      }
      if (ok) umma_commit(tfull);
      umma_commit(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0) && clock64() - t0 < kDrainCycles) {
      }
    }
  } else if (warp < 4) {
    // ------------------------------------------------------------- epilogue
    // Chunk logits TMEM -> shared memory (the stage buffers are free once the
    // MMA loop is done; rows padded so the 32 lanes' column writes fall into
    // distinct banks).
    if (a.stall && threadIdx.x == 0) mbar_wait(never, 0, abort_flag, lim);  // runs out: abort
    const bool ready = __all_sync(0xffffffffu, mbar_wait(tfull, 0, abort_flag, lim)) && !*abort_flag;
    tc_fence_after();
    float* L = reinterpret_cast<float*>(smem);
    if (ready) {
      const uint32_t tb = tmem_base + ((uint32_t)(warp * 32) << 16);
      float* row = L + (size_t)(warp * 32 + lane) * RT_LLD;
      for (int e0 = 0; e0 < ch; e0 += 16) {
        uint32_t v[16];
        tmem_ld16(tb + e0, v);
        tmem_ld_wait(v);
#pragma unroll
        for (int j = 0; j < 16; ++j) row[e0 + j] = __uint_as_float(v[j]);
      }
    }
    if (threadIdx.x == 0) *ready_flag = ready ? 1 : 0;
  }

  tc_fence_before();
  __syncthreads();
  if (*ready_flag) {
    // ------------------------------------------------------------- top-k
    // every warp: its 16 tokens' top k+1 in the chunk, four tokens at a time
    const float* L = reinterpret_cast<const float*>(smem);
    const int kp = a.kp;  // candidates per chunk: min(k + 1, chunk)
    constexpr int NL = kRouterChunk / 32;  // logits per lane and token
    for (int q0 = warp * 16; q0 < warp * 16 + 16; q0 += 4) {
      uint32_t kk[4][NL];
      int id[4][NL];
      float my_v[4];
      int my_i[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float* row = L + (size_t)(q0 + u) * RT_LLD;
#pragma unroll
        for (int i = 0; i < NL; ++i) {
          const int e = lane + 32 * i;
          kk[u][i] = e < ch ? logit_key(row[e]) : 0u;
          id[u][i] = e < ch ? e : 0x7fffffff;
        }
        sort_desc(kk[u], id[u]);
        my_v[u] = -INFINITY;
        my_i[u] = 0x7fffffff;
      }
      for (int rr = 0; rr < kp; ++rr) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          uint32_t bk;
          int bi;
          take_best(kk[u], id[u], bk, bi);
          if (rr == lane) {
            my_v[u] = key_logit(bk);
            my_i[u] = c * ch + bi;  // global expert id
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int t = m0 + q0 + u;
        if (lane < kp && t < a.T) {
          const size_t o = ((size_t)t * a.nchunk + c) * kp + lane;
          a.cand_v[o] = my_v[u];
          a.cand_i[o] = my_i[u];
        }
      }
    }
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

// One CTA per 32-token block (sixteen warps, two tokens each, selected
// together): top-(k+1) of the union of the chunks' candidates, the route
// event (ids, weights, gap), the block's expert histogram (one row of bcount
// for the permutation) and, when the layer has a shared expert, its gate
// sigmoid(x . w_sg).
constexpr int kMergeTPW = 2;                     // tokens per warp
constexpr int kMergeThreads = 32 / kMergeTPW * 32;  // one CTA per 32-token block

__global__ void __launch_bounds__(kMergeThreads) router_merge_kernel(const RouterTcArgs a) {
  constexpr int U = kMergeTPW;
  __shared__ int hist[kMaxExperts];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, k = a.k;
  const int ncand = a.nchunk * a.kp;  // <= 160
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[e] = 0;
  __syncthreads();
  const int tw = blockIdx.x * 32 + warp * U;  // this warp's first token
  {
    uint32_t kk[U][5];
    int id[U][5];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = tw + u;
#pragma unroll
      for (int i = 0; i < 5; ++i) {
        const int j = lane + 32 * i;
        const bool in = t < a.T && j < ncand;
        const int cid = in ? a.cand_i[(size_t)t * ncand + j] : -1;
        const bool real = cid >= 0 && cid < E;  // an aborted router leaves no valid candidate
        kk[u][i] = real ? logit_key(a.cand_v[(size_t)t * ncand + j]) : 0u;
        id[u][i] = real ? cid : 0x7fffffff;
      }
      sort_desc(kk[u], id[u]);
    }
    float my_v[U], next_v[U];
    int my_i[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      my_v[u] = -INFINITY;
      next_v[u] = -INFINITY;
      my_i[u] = 0;
    }
    const int rounds = min(k + 1, E);
    for (int rr = 0; rr < rounds; ++rr) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        uint32_t bk;
        int bi;
        take_best(kk[u], id[u], bk, bi);
        const float bv = bk == 0u ? -INFINITY : key_logit(bk);
        if (rr == lane) {
          my_v[u] = bv;
          my_i[u] = bi;
        }
        if (rr == k) next_v[u] = bv;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = tw + u;
      const float l0 = __shfl_sync(0xffffffffu, my_v[u], 0);
      const float ex = (lane < k) ? expf(my_v[u] - l0) : 0.f;
      float sum = ex;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      const float lk1 = __shfl_sync(0xffffffffu, my_v[u], k - 1);
      if (t < a.T) {
        if (lane < k) {
          // an aborted router leaves no valid candidate: expert 0 stands in,
          // counted like any id, so that the permutation stays a bijection
          // (the status word already fails the call)
          const bool real = my_i[u] >= 0 && my_i[u] < E;
          const int id = real ? my_i[u] : 0;
          a.ids[(size_t)t * k + lane] = id;
          a.weights[(size_t)t * k + lane] = ex / sum;
          atomicAdd(&hist[id], 1);
        }
        if (a.gap != nullptr && lane == 0) a.gap[t] = (k < E) ? (lk1 - next_v[u]) : INFINITY;
      }
    }
  }
  if (a.wsg != nullptr) {
    // shared-expert gate of the warp's tokens, dot products interleaved
    float sum[U];
#pragma unroll
    for (int u = 0; u < U; ++u) sum[u] = 0.f;
#pragma unroll 4
    for (int h = lane * 8; h < a.H; h += 256) {
      const float4 w0 = __ldg(reinterpret_cast<const float4*>(a.wsg + h));
      const float4 w1 = __ldg(reinterpret_cast<const float4*>(a.wsg + h + 4));
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (tw + u >= a.T) continue;
        const uint4 xv = __ldg(reinterpret_cast<const uint4*>(a.x + (size_t)(tw + u) * a.H + h));
        float s = sum[u];
        s = fmaf(bf16_lo(xv.x), w0.x, s);
        s = fmaf(bf16_hi(xv.x), w0.y, s);
        s = fmaf(bf16_lo(xv.y), w0.z, s);
        s = fmaf(bf16_hi(xv.y), w0.w, s);
        s = fmaf(bf16_lo(xv.z), w1.x, s);
        s = fmaf(bf16_hi(xv.z), w1.y, s);
        s = fmaf(bf16_lo(xv.w), w1.z, s);
        s = fmaf(bf16_hi(xv.w), w1.w, s);
        sum[u] = s;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float s = sum[u];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (lane == 0 && tw + u < a.T) a.sg[tw + u] = 1.0f / (1.0f + expf(-s));
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) a.bcount[(size_t)blockIdx.x * E + e] = hist[e];
}

}  // namespace

cudaError_t launch_split3(const float* w, long long n, __nv_bfloat16* out, int* status, Group* sh,
                          int* sh_total, int T, int shared_slot, const TableParams* tp,
                          int* tab_slot, unsigned long long* tab_expected, cudaStream_t s) {
  const long long want = (n + 255) / 256;
  const int grid = (int)(want < 152 * 8 ? want : 152 * 8);
  if (tp != nullptr)
    split3_table_kernel<<<grid, 256, 0, s>>>(w, n, out, status, sh, sh_total, T, shared_slot, *tp,
                                             tab_slot, tab_expected);
  else
    split3_kernel<<<grid, 256, 0, s>>>(w, n, out, status, sh, sh_total, T, shared_slot);
  return cudaGetLastError();
}

cudaError_t launch_router_tc(const CUtensorMap& tmX, const CUtensorMap& tmW, const RouterTcArgs& a,
                             cudaStream_t s) {
  static std::atomic<unsigned long long> attr_done{0};
  {
    cudaError_t e = smem_attr_once(router_tc_kernel, RT_SMEM, attr_done);
    if (e != cudaSuccess) return e;
  }
  const int nb = (a.T + 127) / 128;
  if (nb == 0) return cudaSuccess;
  router_tc_kernel<<<(unsigned)nb * (unsigned)a.nchunk, NTH, RT_SMEM, s>>>(tmX, tmW, a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  router_merge_kernel<<<(a.T + 31) / 32, kMergeThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace msi
