// Router: fp32 logits, top-k, softmax weights, shared-expert gate and the
// per-block expert histogram, fused in one kernel (logits never reach HBM).
//
// The router's top-k output is the route event the paper records once per
// layer and graph evaluation, before any Plan action (Sec. "Output-Exact
// Execution Beyond the Full-Residency Envelope").  Readings where the paper is
// silent: weights are the softmax over the selected k logits (they sum to 1);
// equal logits rank the lower expert id first.
//
// Block = 32 tokens x all E (<= 512) experts, 256 threads.  Each thread owns
// an 8-token x (EP / 64)-expert fp32 register tile (experts strided by 64 so
// a warp reads 32 consecutive expert rows); EP, the experts a block covers, is
// 64 for E <= 64 (eight times less work and staging for small layers) and
// 512 otherwise.  K is staged 32 at a time with cp.async:
// x as bf16 [32 tok][32 k]; Wr as fp32 [512 e][32 k] with the eight 16-byte
// chunks of each row XOR-swizzled by (e & 7), so a warp's 16-byte reads of
// one k-quad hit all 32 banks once per 8 lanes.  Accumulation runs over h in
// ascending order.  Top-k: one warp per token, k+1 rounds of a warp-shuffle
// argmax over (logit desc, id asc).
#include "kernels.cuh"

namespace msi {

namespace {
constexpr int TM = kRouterTM;
constexpr int BK = 32;
constexpr int NTH = 256;
constexpr int XS_BYTES = TM * BK * 2;        // 2 KB

// Shared-memory plan for EP experts per block (the logits and ids reuse the
// stages): EP = 512, two 66 KB stages; EP = 64, eight 10 KB stages, so that a
// small layer's whole K (H <= 256) is in flight at once.
template <int EP>
struct RCfg {
  static constexpr int WS_BYTES = EP * BK * 4;
  static constexpr int STAGE_BYTES = XS_BYTES + WS_BYTES;
  static constexpr int NSTAGE = EP <= 64 ? 8 : 2;
  static constexpr int LLD = EP + 4;         // logits row stride (floats)
  static constexpr int SMEM = NSTAGE * STAGE_BYTES;
  static constexpr int J = EP / 64;          // experts per thread
  static_assert(TM * LLD * 4 + TM * kMaxTopK * 4 <= SMEM, "logits do not fit");
};

template <int EP>
__device__ __forceinline__ void load_stage(const RouterArgs& a, uint8_t* st, int t0, int kb) {
  const int tid = threadIdx.x;
  uint8_t* xs = st;
  uint8_t* ws = st + XS_BYTES;
  if (tid < TM * 4) {
    const int tok = tid >> 2, c = tid & 3;
    const bool v = (t0 + tok) < a.T;
    const __nv_bfloat16* src = a.x + (size_t)(v ? t0 + tok : 0) * a.H + kb * BK + c * 8;
    cp_async16(xs + tok * 64 + c * 16, src, v ? 16u : 0u);
  }
#pragma unroll
  for (int i = 0; i < (EP * 8) / NTH; ++i) {
    const int idx = tid + NTH * i;
    const int e = idx >> 3, c = idx & 7;
    const bool v = e < a.E;
    const float* src = a.wr + (size_t)(v ? e : 0) * a.H + kb * BK + c * 4;
    cp_async16(ws + e * 128 + ((c ^ (e & 7)) << 4), src, v ? 16u : 0u);
  }
}

// Top-k, softmax weights, gap and shared gate of the block's tokens from the
// logits L[TM][lld] in shared memory (each warp TM / warps tokens), then the
// block's expert histogram.  ids_s: shared scratch [TM * k].  NV: logits per
// lane (E <= 32 NV).
template <int NV>
__device__ __forceinline__ void select_and_count(const RouterArgs& a, const float* L, int lld, int* ids_s,
                                                 int t0) {
  const int tid = threadIdx.x;
  // top-k: warp w handles tokens w*tpw .. w*tpw+tpw-1
  const int warp = tid >> 5, lane = tid & 31;
  const int nvalid = min(TM, a.T - t0);
  const int k = a.k;
  const int per_lane = (a.E + 31) >> 5;  // <= 16
  const int tpw = TM / (int)(blockDim.x >> 5);  // tokens per warp
  for (int q = 0; q < tpw; ++q) {
    const int tok = warp * tpw + q;
    if (tok >= nvalid) break;
    float v[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int e = lane + 32 * i;
      v[i] = (i < per_lane && e < a.E) ? L[tok * lld + e] : -INFINITY;
    }
    uint32_t removed = 0;
    float my_v = -INFINITY;
    int my_i = 0;
    float next_v = -INFINITY;  // logit of rank k (when k < E)
    const int rounds = min(k + 1, a.E);
    for (int r = 0; r < rounds; ++r) {
      float bv = -INFINITY;
      int bi = 0x7fffffff;
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        const int e = lane + 32 * i;
        if (i < per_lane && e < a.E && !((removed >> i) & 1u)) {
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
      if (r == lane) { my_v = bv; my_i = bi; }
      if (r == k) next_v = bv;
    }
    const float l0 = __shfl_sync(0xffffffffu, my_v, 0);
    float ex = (lane < k) ? expf(my_v - l0) : 0.f;
    float sum = ex;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    const size_t t = (size_t)t0 + tok;
    if (lane < k) {
      a.ids[t * k + lane] = my_i;
      a.weights[t * k + lane] = ex / sum;
      ids_s[tok * k + lane] = my_i;
    }
    if (a.gap != nullptr) {
      const float lk1 = __shfl_sync(0xffffffffu, my_v, k - 1);
      if (lane == 0) a.gap[t] = (k < a.E) ? (lk1 - next_v) : INFINITY;
    }
    if (a.wsg != nullptr) {
      const __nv_bfloat16* xr = a.x + t * a.H;
      float s = 0.f;
      for (int h = lane * 8; h < a.H; h += 256) {
        const uint4 xv = *reinterpret_cast<const uint4*>(xr + h);
        const float4 w0 = *reinterpret_cast<const float4*>(a.wsg + h);
        const float4 w1 = *reinterpret_cast<const float4*>(a.wsg + h + 4);
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
      if (lane == 0) a.sg[t] = 1.0f / (1.0f + expf(-s));
    }
  }
  __syncthreads();

  // per-block histogram of the routed ids (deterministic, no atomics)
  const int nids = nvalid * k;
  for (int e = tid; e < a.E; e += NTH) {
    int c = 0;
    for (int i = 0; i < nids; ++i) c += (ids_s[i] == e);
    a.bcount[(size_t)blockIdx.x * a.E + e] = c;
  }
}

template <int EP>
__global__ void __launch_bounds__(NTH, 1) router_kernel(const RouterArgs a) {
  using C = RCfg<EP>;
  constexpr int STAGE_BYTES = C::STAGE_BYTES, LLD = C::LLD, J = C::J, NSTAGE = C::NSTAGE;
  // the forward's first kernel (status null: a prediction pass)
  if (blockIdx.x == 0 && threadIdx.x == 0 && a.status != nullptr)
    forward_begin(a.status, a.sh, a.sh_total, a.T, a.shared_slot);
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x;
  const int t0 = blockIdx.x * TM;
  const int tg = tid >> 6;   // token group: tokens tg*8 .. tg*8+7
  const int el = tid & 63;   // experts el + 64 j
  float acc[8][J];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < J; ++j) acc[i][j] = 0.f;

  const int nk = a.H / BK;
  // NSTAGE - 1 stages ahead; each iteration refills the slot the previous one
  // consumed, then waits for its own stage
#pragma unroll
  for (int i = 0; i < NSTAGE - 1; ++i) {
    if (i < nk) load_stage<EP>(a, smem + i * STAGE_BYTES, t0, i);
    cp_async_commit();
  }
  for (int kb = 0; kb < nk; ++kb) {
    const int nx = kb + NSTAGE - 1;
    if (nx < nk) load_stage<EP>(a, smem + (nx % NSTAGE) * STAGE_BYTES, t0, nx);
    cp_async_commit();
    cp_async_wait<NSTAGE - 1>();
    __syncthreads();
    const uint8_t* xs = smem + (kb % NSTAGE) * STAGE_BYTES;
    const uint8_t* ws = xs + XS_BYTES;
#pragma unroll
    for (int kq = 0; kq < BK / 4; ++kq) {
      float4 w[J];
#pragma unroll
      for (int j = 0; j < J; ++j) {
        const int e = el + 64 * j;
        w[j] = *reinterpret_cast<const float4*>(ws + e * 128 + ((kq ^ (e & 7)) << 4));
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const uint2 xv = *reinterpret_cast<const uint2*>(xs + (tg * 8 + i) * 64 + kq * 8);
        const float x0 = bf16_lo(xv.x), x1 = bf16_hi(xv.x), x2 = bf16_lo(xv.y), x3 = bf16_hi(xv.y);
#pragma unroll
        for (int j = 0; j < J; ++j) {
          float s = acc[i][j];
          s = fmaf(x0, w[j].x, s);
          s = fmaf(x1, w[j].y, s);
          s = fmaf(x2, w[j].z, s);
          s = fmaf(x3, w[j].w, s);
          acc[i][j] = s;
        }
      }
    }
    __syncthreads();
  }

  // logits -> shared memory [TM][LLD]
  float* L = reinterpret_cast<float*>(smem);
  int* ids_s = reinterpret_cast<int*>(smem + TM * LLD * 4);
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < J; ++j) L[(tg * 8 + i) * LLD + el + 64 * j] = acc[i][j];
  __syncthreads();

  select_and_count<16>(a, L, LLD, ids_s, t0);
}

// Layers of at most 32 experts: one lane per expert, EL lanes per token
// (EL = 16 for at most 16 experts, two tokens a warp; else 32), the block's
// 32 tokens at once.  A lane computes its (token, expert) logit as one fp32
// fmaf chain over h in ascending order (the tiled kernel's value), four h at
// a time from a chunk of Wr staged in shared memory as [h / 4][EL][4] (one
// 16-byte read per lane) and the token's x row (one 8-byte broadcast).  The
// tiled kernel would spend a block of 256 threads and 64 expert columns on
// them.
constexpr int kSmallHC = 256;                  // h per staged chunk
constexpr int kSmallLLD = 36;                  // logits row stride (floats)
template <int EL>
struct SmallCfg {
  static constexpr int kWarps = TM * EL / 32;
  static constexpr int kThreads = kWarps * 32;
  static constexpr int kWT = kSmallHC * EL * 4;    // Wr chunk [HC / 4][EL][4] fp32
  static constexpr int kXS = TM * kSmallHC * 2;    // x chunk [TM][HC] bf16
  static constexpr int kSmem = kWT + kXS + TM * kSmallLLD * 4 + TM * kMaxTopK * 4;
};

template <int EL>
__global__ void __launch_bounds__(SmallCfg<EL>::kThreads, 1) router_small_kernel(const RouterArgs a) {
  using C = SmallCfg<EL>;
  // the forward's first kernel (status null: a prediction pass)
  if (blockIdx.x == 0 && threadIdx.x == 0 && a.status != nullptr)
    forward_begin(a.status, a.sh, a.sh_total, a.T, a.shared_slot);
  extern __shared__ __align__(128) uint8_t smem[];
  float4* wt = reinterpret_cast<float4*>(smem);
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(smem + C::kWT);
  float* L = reinterpret_cast<float*>(smem + C::kWT + C::kXS);
  int* ids_s = reinterpret_cast<int*>(smem + C::kWT + C::kXS + TM * kSmallLLD * 4);
  const int tid = threadIdx.x;
  const int tok = tid / EL, e = tid % EL;  // this lane's token (in the block) and expert
  const int t0 = blockIdx.x * TM;
  const int nvalid = min(TM, a.T - t0);
  float acc = 0.f;
  for (int h0 = 0; h0 < a.H; h0 += kSmallHC) {
    const int hc = min(kSmallHC, a.H - h0);
    const int nq = hc / 4;  // h quads of this chunk
    for (int i = tid; i < a.E * nq; i += C::kThreads) {
      const int ee = i % a.E, q = i / a.E;
      wt[q * EL + ee] = __ldg(reinterpret_cast<const float4*>(a.wr + (size_t)ee * a.H + h0) + q);
    }
    const int nc = hc / 8;  // 16-byte chunks of a token's row in this chunk
    for (int i = tid; i < TM * nc; i += C::kThreads) {
      const int tk = i / nc, c = i - tk * nc;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (tk < nvalid) v = __ldg(reinterpret_cast<const uint4*>(a.x + (size_t)(t0 + tk) * a.H + h0) + c);
      reinterpret_cast<uint4*>(xs + tk * kSmallHC)[c] = v;
    }
    __syncthreads();
    if (e < a.E) {
      const uint2* xr = reinterpret_cast<const uint2*>(xs + tok * kSmallHC);
      for (int q = 0; q < nq; ++q) {
        const float4 w = wt[q * EL + e];
        const uint2 xv = xr[q];
        acc = fmaf(bf16_lo(xv.x), w.x, acc);
        acc = fmaf(bf16_hi(xv.x), w.y, acc);
        acc = fmaf(bf16_lo(xv.y), w.z, acc);
        acc = fmaf(bf16_hi(xv.y), w.w, acc);
      }
    }
    __syncthreads();
  }
  L[tok * kSmallLLD + e] = acc;
  __syncthreads();
  select_and_count<1>(a, L, kSmallLLD, ids_s, t0);
}

}  // namespace

template <int EP>
static cudaError_t launch_ep(const RouterArgs& a, cudaStream_t s) {
  static std::atomic<unsigned long long> attr_done{0};
  {
    cudaError_t e = smem_attr_once(router_kernel<EP>, RCfg<EP>::SMEM, attr_done);
    if (e != cudaSuccess) return e;
  }
  const int nb = (a.T + TM - 1) / TM;
  if (nb == 0) return cudaSuccess;
  router_kernel<EP><<<nb, NTH, RCfg<EP>::SMEM, s>>>(a);
  return cudaGetLastError();
}

template <int EL>
static cudaError_t launch_small(const RouterArgs& a, cudaStream_t s) {
  using C = SmallCfg<EL>;
  static std::atomic<unsigned long long> attr_done{0};
  {
    cudaError_t e = smem_attr_once(router_small_kernel<EL>, C::kSmem, attr_done);
    if (e != cudaSuccess) return e;
  }
  const int nb = (a.T + TM - 1) / TM;
  if (nb == 0) return cudaSuccess;
  router_small_kernel<EL><<<nb, C::kThreads, C::kSmem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_router(const RouterArgs& a, cudaStream_t s) {
  if (a.E <= 16) return launch_small<16>(a, s);
  if (a.E <= 32) return launch_small<32>(a, s);
  return a.E <= 64 ? launch_ep<64>(a, s) : launch_ep<512>(a, s);
}

}  // namespace msi
