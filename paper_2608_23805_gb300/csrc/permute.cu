// Token grouping (histogram, scan, stable permutation), the per-call table
// upload, the generation re-check that builds the GEMM groups, the slot
// generation publication, and the weighted combine.
//
// Permutation: row r in [offsets[e], offsets[e+1]) holds the (t, j) pairs
// routed to expert e in (t, j) order; perm[r] = t*k + j, inv[t*k + j] = r.
// Atomic-free: per-router-block counts (written by the router kernel) ->
// column prefix over blocks -> per-warp stable ranks from __match_any_sync.
//
// Generation re-check (fail closed): a published version must denote the
// requested object and version, and a mismatch is rejected before any
// consumer reads the slot (paper, Sec. "Lifetime Is Part of Correctness";
// Sec. "Stable Slots and Bundle Publication").
#include "kernels.cuh"

namespace msi {

namespace {

// ---- column prefix over router blocks: bbase[b][e], counts[e] ----
__global__ void __launch_bounds__(1024) colscan_kernel(const ScanArgs a) {
  __shared__ int part[32][33];
  const int tx = threadIdx.x, ty = threadIdx.y;
  const int e = blockIdx.x * 32 + tx;
  const int sz = (a.nb + 31) / 32;
  const int b0 = min(a.nb, ty * sz), b1 = min(a.nb, b0 + sz);
  int sum = 0;
  if (e < a.E)
#pragma unroll 8
    for (int b = b0; b < b1; ++b) sum += a.bcount[(size_t)b * a.E + e];
  part[ty][tx] = sum;
  __syncthreads();
  int run = 0;
  for (int y = 0; y < ty; ++y) run += part[y][tx];
  if (e < a.E) {
#pragma unroll 8
    for (int b = b0; b < b1; ++b) {
      const int v = a.bcount[(size_t)b * a.E + e];
      a.bbase[(size_t)b * a.E + e] = run;
      run += v;
    }
    if (ty == 31) a.counts[e] = run;
  }
}

__device__ __forceinline__ int check_code(const GenWord* gw, int slot, int layer, int e,
                                          unsigned long long expected) {
  if (slot < 0) return MSI_ERR_NOT_RESIDENT;
  const unsigned long long obj = gw[slot].obj;
  const unsigned long long gen = gw[slot].gen;
  if (obj != obj_key(layer, e)) return MSI_ERR_WRONG_OBJECT;
  if (gen != expected) return MSI_ERR_STALE_GENERATION;
  return 0;
}

// ---- scatter: one warp per router block ----

// Exclusive scan over the block of four values per thread (128 threads);
// returns the thread's base and leaves the block total in *total.
__device__ __forceinline__ int scan4(const int (&v)[4], int* wsum, int* total) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = v[0] + v[1] + v[2] + v[3];
  int incl = s;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  int base = incl - s, tot = 0;
  for (int w = 0; w < kScatterWarps; ++w) {
    if (w < warp) base += wsum[w];
    tot += wsum[w];
  }
  *total = tot;
  __syncthreads();
  return base;
}

// Setup block of the scatter, resident call: the generation re-check of every
// routed expert's slot (fail closed) and the GEMM groups with their 128- and
// 256-row tile prefixes.
__device__ void scatter_setup(const ScatterArgs& a, const int* offs,
                              const int* s_cnt) {
  __shared__ int wsum[kScatterWarps];
  __shared__ int kmin[kScatterWarps];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (a.ready != nullptr)  // fused GEMMs: counters of the call's first launch
    for (int r = tid; r < a.n_ready; r += blockDim.x) a.ready[r] = 0;
  if (a.tab_slot == nullptr) return;  // streamed call: the groups are built per wave
  int cnt[4], code[4], mt[4], pt[4];
  int key = 0x7fffffff;
  int slot[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = tid * 4 + i;
    cnt[i] = code[i] = mt[i] = pt[i] = 0;
    slot[i] = -1;
    if (e < a.E) {
      cnt[i] = s_cnt[e];
      slot[i] = a.tab_slot[e];
      if (cnt[i] > 0) code[i] = check_code(a.genwords, slot[i], a.layer, e, a.tab_expected[e]);
      if (code[i] == 0) {
        mt[i] = (cnt[i] + kBM - 1) / kBM;
        pt[i] = (cnt[i] + 2 * kBM - 1) / (2 * kBM);
      } else {
        key = min(key, (e << 4) | code[i]);
      }
    }
  }
  int mtot = 0, ptot = 0;
  int mb = scan4(mt, wsum, &mtot);
  int pb = scan4(pt, wsum, &ptot);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = tid * 4 + i;
    if (e < a.E) {
      Group g;
      g.row_begin = offs[e];
      g.row_count = cnt[i];
      g.slot = slot[i] < 0 ? 0 : slot[i];
      g.mt_begin = mb;
      g.ok = code[i] == 0;
      g.expert = e;
      g.pt_begin = pb;
      g.pad1 = 0;
      a.groups[e] = g;
    }
    mb += mt[i];
    pb += pt[i];
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) key = min(key, __shfl_xor_sync(0xffffffffu, key, off));
  if (lane == 0) kmin[warp] = key;
  __syncthreads();
  if (tid == 0) {
    int m = kmin[0];
    for (int w = 1; w < kScatterWarps; ++w) m = min(m, kmin[w]);
    a.total_mtiles[0] = mtot;
    a.total_mtiles[1] = ptot;
    if (m != 0x7fffffff) atomicCAS(a.status, 0, m & 15);
  }
}

__global__ void __launch_bounds__(kScatterWarps * 32) scatter_kernel(const ScatterArgs a) {
  __shared__ int offs[kMaxExperts + 1];
  __shared__ int s_cnt[kMaxExperts];
  __shared__ int run[kScatterWarps][kMaxExperts];
  __shared__ int wsum[kScatterWarps];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // exclusive scan of counts (E <= 512, 128 threads x 4 values); with
  // fuse_scan the counts are the column sums of the router blocks' counts
  int v[4], s = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = tid * 4 + i;
    int c = 0;
    if (e < a.E) {
      if (a.fuse_scan) {
        for (int b = 0; b < a.nb; ++b) c += a.bcount[(size_t)b * a.E + e];
      } else {
        c = a.counts[e];
      }
      s_cnt[e] = c;
    }
    v[i] = c;
    s += v[i];
  }
  int incl = s;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  int base = incl - s;
  for (int w = 0; w < warp; ++w) base += wsum[w];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = tid * 4 + i;
    if (e <= a.E) offs[e] = base;
    base += v[i];
  }
  if (tid == kScatterWarps * 32 - 1 && a.E == kMaxExperts) offs[kMaxExperts] = base;
  __syncthreads();
  // the last block (one past the scatter blocks) writes the offsets and runs
  // the resident setup, in parallel with the scatter
  if (blockIdx.x == gridDim.x - 1) {
    for (int e = tid; e <= a.E; e += blockDim.x) a.offsets[e] = offs[e];
    if (a.fuse_scan)
      for (int e = tid; e < a.E; e += blockDim.x) a.counts_out[e] = s_cnt[e];
    scatter_setup(a, offs, s_cnt);
    return;
  }

  const int b = blockIdx.x * kScatterWarps + warp;
  if (b >= a.nb) return;
  for (int e = lane; e < a.E; e += 32) run[warp][e] = 0;
  __syncwarp();
  const int f0 = b * a.tm * a.k;
  const int f1 = min(a.T, (b + 1) * a.tm) * a.k;
  const unsigned lt = (1u << lane) - 1u;
  // eight steps of 32 ids at a time: their ids and block bases are loaded
  // together (independent loads), then ranked in order
  constexpr int kAhead = 8;
  for (int fc = f0; fc < f1; fc += 32 * kAhead) {
    int ev[kAhead], pre[kAhead];
#pragma unroll
    for (int j = 0; j < kAhead; ++j) {
      const int f = fc + 32 * j + lane;
      ev[j] = f < f1 ? a.ids[f] : -1;
    }
#pragma unroll
    for (int j = 0; j < kAhead; ++j) {
      pre[j] = 0;  // this expert's ids in the router blocks before b
      if (ev[j] >= 0) {
        if (a.fuse_scan) {
          for (int bb = 0; bb < b; ++bb) pre[j] += a.bcount[(size_t)bb * a.E + ev[j]];
        } else {
          pre[j] = a.bbase[(size_t)b * a.E + ev[j]];
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kAhead; ++j) {
      if (fc + 32 * j >= f1) break;  // uniform across the warp
      const int f = fc + 32 * j + lane;
      const int e = ev[j];
      const bool valid = e >= 0;
      const unsigned mask = __match_any_sync(0xffffffffu, e);
      int before = 0;
      if (valid) {
        before = run[warp][e];
        const int pos = offs[e] + pre[j] + before + __popc(mask & lt);
        a.perm[pos] = f;
        a.inv[f] = pos;
      }
      __syncwarp();
      if (valid && lane == 31 - __clz(mask)) run[warp][e] = before + __popc(mask);
      __syncwarp();
    }
  }
}

// ---- per-call table upload + forward begin ----
__global__ void upload_kernel(const TableParams p, int* table, unsigned long long* expected,
                              int* status, Group* sh, int* sh_total) {
  for (int e = threadIdx.x; e < p.E; e += blockDim.x) {
    table[e] = p.slot[e];
    expected[e] = p.expected[e];
  }
  if (threadIdx.x == 0 && status != nullptr) forward_begin(status, sh, sh_total, p.T, p.shared_slot);
}

// ---- generation re-check + GEMM groups (one block) ----
__device__ __forceinline__ int block_excl_scan(int v, int* tmp, int* total) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int incl = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) tmp[warp] = incl;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  int base = 0, tot = 0;
  for (int w = 0; w < nw; ++w) {
    if (w < warp) base += tmp[w];
    tot += tmp[w];
  }
  *total = tot;
  return base + incl - v;
}

__device__ __forceinline__ int block_min(int v, int* tmp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, off));
  __syncthreads();
  if (lane == 0) tmp[warp] = v;
  __syncthreads();
  int m = 0x7fffffff;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = min(m, tmp[w]);
  return m;
}

// One LRU wave of a streamed call: re-check the wave's slots and build its
// GEMM groups (the resident call does this in the scatter kernel).
__global__ void __launch_bounds__(kMaxExperts) setup_kernel(const SetupArgs a, const WaveParams w) {
  __shared__ int tmp[32];
  const int i = threadIdx.x;
  const int n = w.n;
  int e = -1, cnt = 0, slot = -1, code = 0;
  if (i < n) {
    e = w.expert[i];
    cnt = a.counts[e];
    slot = w.slot[i];
    if (cnt > 0) code = check_code(a.genwords, slot, a.layer, e, w.expected[i]);
  }
  const int mt = (i < n && code == 0) ? (cnt + kBM - 1) / kBM : 0;
  const int pt = (i < n && code == 0) ? (cnt + 2 * kBM - 1) / (2 * kBM) : 0;
  int total = 0, ptotal = 0;
  const int mt_begin = block_excl_scan(mt, tmp, &total);
  __syncthreads();
  const int pt_begin = block_excl_scan(pt, tmp, &ptotal);
  if (i < n) {
    Group g;
    g.row_begin = a.offsets[e];
    g.row_count = cnt;
    g.slot = slot < 0 ? 0 : slot;
    g.mt_begin = mt_begin;
    g.ok = code == 0;
    g.expert = e;
    g.pt_begin = pt_begin;
    g.pad1 = 0;
    a.groups[i] = g;
  }
  if (a.ready != nullptr)
    for (int r = i; r < a.n_ready; r += blockDim.x) a.ready[r] = 0;
  const int key = code ? (e << 4) | code : 0x7fffffff;
  const int m = block_min(key, tmp);
  if (i == 0) {
    a.total_mtiles[0] = total;
    a.total_mtiles[1] = ptotal;
    if (m != 0x7fffffff) atomicCAS(a.status, 0, m & 15);
  }
}

__global__ void publish_kernel(const PublishParams p, GenWord* gw) {
  const int i = threadIdx.x;
  if (i < p.n) {
    GenWord g;
    g.gen = p.gen[i];
    g.obj = p.obj[i];
    gw[p.slot[i]] = g;
  }
}

// Block b copies part b % parts of extent b / parts.  Its first thread
// invalidates the extent's slot word and makes that visible before the
// block's copies; every block makes its copies visible before it takes a
// ticket, and the block that takes the launch's last ticket publishes.
__global__ void stage_copy_kernel(const StageCopyArgs a, GenWord* gw) {
  const int i = blockIdx.x / a.parts, part = blockIdx.x % a.parts;
  const int slot = a.pub.slot[i];
  if (threadIdx.x == 0) {
    GenWord z;
    z.gen = 0;
    z.obj = 0;
    gw[slot] = z;
    __threadfence();
  }
  __syncthreads();
  const uint4* src = reinterpret_cast<const uint4*>(a.src[i]);
  uint4* dst = reinterpret_cast<uint4*>(a.pool + (size_t)slot * a.bytes);
  const unsigned long long n16 = a.bytes / 16;
  const unsigned long long per = (n16 + a.parts - 1) / a.parts;
  const unsigned long long b0 = per * part, b1 = min(n16, b0 + per);
  // four 16-byte loads in flight per thread before their stores
  for (unsigned long long k = b0 + threadIdx.x; k < b1; k += 4ull * blockDim.x) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const unsigned long long kk = k + (unsigned long long)u * blockDim.x;
      if (kk < b1) v[u] = __ldg(src + kk);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const unsigned long long kk = k + (unsigned long long)u * blockDim.x;
      if (kk < b1) dst[kk] = v[u];
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0 && atomicAdd(a.ticket, 1ull) + 1ull == a.target) {
    __threadfence();
    for (int j = 0; j < a.pub.n; ++j) {
      GenWord g;
      g.gen = a.pub.gen[j];
      g.obj = a.pub.obj[j];
      gw[a.pub.slot[j]] = g;
    }
  }
}

// ---- combine: out[t] = sum_j w[t,j] yp[inv[t*k+j]] (+ sg[t] ys[t]) (+ x[t]) ----
__device__ __forceinline__ void fma8(float (&acc)[8], float w, const uint4& y) {
  acc[0] = fmaf(w, bf16_lo(y.x), acc[0]);
  acc[1] = fmaf(w, bf16_hi(y.x), acc[1]);
  acc[2] = fmaf(w, bf16_lo(y.y), acc[2]);
  acc[3] = fmaf(w, bf16_hi(y.y), acc[3]);
  acc[4] = fmaf(w, bf16_lo(y.z), acc[4]);
  acc[5] = fmaf(w, bf16_hi(y.z), acc[5]);
  acc[6] = fmaf(w, bf16_lo(y.w), acc[6]);
  acc[7] = fmaf(w, bf16_hi(y.w), acc[7]);
}

// One block per token; the token's k row indices and weights are read once
// into shared memory, and up to eight expert rows are loaded before they are
// summed (still in j order, fp32), so each thread keeps eight 16-byte loads
// in flight.
__global__ void __launch_bounds__(256) combine_kernel(const CombineArgs a) {
  if (*a.status != 0) return;  // fail closed: nothing stale becomes visible
  __shared__ int s_row[kMaxTopK];
  __shared__ float s_w[kMaxTopK];
  const int t = blockIdx.x;
  if (threadIdx.x < a.k) {
    s_row[threadIdx.x] = __ldg(&a.inv[(size_t)t * a.k + threadIdx.x]);
    s_w[threadIdx.x] = __ldg(&a.weights[(size_t)t * a.k + threadIdx.x]);
  }
  __syncthreads();
  const int nchunk = a.H >> 3;
  for (int c = threadIdx.x; c < nchunk; c += blockDim.x) {
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    int j = 0;
    for (; j + 8 <= a.k; j += 8) {
      uint4 y[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        y[u] = __ldg(reinterpret_cast<const uint4*>(a.yp + (size_t)s_row[j + u] * a.H) + c);
#pragma unroll
      for (int u = 0; u < 8; ++u) fma8(acc, s_w[j + u], y[u]);
    }
    if (j + 4 <= a.k) {
      uint4 y[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        y[u] = __ldg(reinterpret_cast<const uint4*>(a.yp + (size_t)s_row[j + u] * a.H) + c);
#pragma unroll
      for (int u = 0; u < 4; ++u) fma8(acc, s_w[j + u], y[u]);
      j += 4;
    }
    for (; j < a.k; ++j)
      fma8(acc, s_w[j], __ldg(reinterpret_cast<const uint4*>(a.yp + (size_t)s_row[j] * a.H) + c));
    if (a.ys != nullptr)  // gate sigmoid(x . w_sg), or 1 for an ungated shared expert
      fma8(acc, a.sg != nullptr ? a.sg[t] : 1.0f,
           __ldg(reinterpret_cast<const uint4*>(a.ys + (size_t)t * a.H) + c));
    if (a.x != nullptr) {
      const uint4 y = __ldg(reinterpret_cast<const uint4*>(a.x + (size_t)t * a.H) + c);
      acc[0] += bf16_lo(y.x);
      acc[1] += bf16_hi(y.x);
      acc[2] += bf16_lo(y.y);
      acc[3] += bf16_hi(y.y);
      acc[4] += bf16_lo(y.z);
      acc[5] += bf16_hi(y.z);
      acc[6] += bf16_lo(y.w);
      acc[7] += bf16_hi(y.w);
    }
    uint4 o;
    o.x = pack_bf16x2(acc[0], acc[1]);
    o.y = pack_bf16x2(acc[2], acc[3]);
    o.z = pack_bf16x2(acc[4], acc[5]);
    o.w = pack_bf16x2(acc[6], acc[7]);
    reinterpret_cast<uint4*>(a.out + (size_t)t * a.H)[c] = o;
  }
}

__global__ void zero_kernel(int* p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0;
}

}  // namespace

cudaError_t launch_colscan(const ScanArgs& a, cudaStream_t s) {
  colscan_kernel<<<(a.E + 31) / 32, dim3(32, 32), 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_scatter(const ScatterArgs& a, cudaStream_t s) {
  const int grid = (a.nb + kScatterWarps - 1) / kScatterWarps + 1;  // + the setup block
  scatter_kernel<<<grid, kScatterWarps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_upload(const TableParams& p, int* table, unsigned long long* expected, int* status,
                          Group* shared_group, int* shared_total, cudaStream_t s) {
  upload_kernel<<<1, 512, 0, s>>>(p, table, expected, status, shared_group, shared_total);
  return cudaGetLastError();
}


cudaError_t launch_setup_wave(const SetupArgs& a, const WaveParams& w, cudaStream_t s) {
  setup_kernel<<<1, kMaxExperts, 0, s>>>(a, w);
  return cudaGetLastError();
}

cudaError_t launch_publish(const PublishParams& p, GenWord* genwords, cudaStream_t s) {
  if (p.n == 0) return cudaSuccess;
  publish_kernel<<<1, kMaxWave, 0, s>>>(p, genwords);
  return cudaGetLastError();
}

cudaError_t launch_stage_copy(const StageCopyArgs& a, GenWord* genwords, cudaStream_t s) {
  if (a.pub.n == 0) return cudaSuccess;
  stage_copy_kernel<<<a.pub.n * a.parts, 256, 0, s>>>(a, genwords);
  return cudaGetLastError();
}

cudaError_t launch_combine(const CombineArgs& a, cudaStream_t s) {
  if (a.T == 0) return cudaSuccess;
  const int nthreads = min(256, a.H / 8);
  combine_kernel<<<a.T, nthreads, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_zero_counts(int* counts, int E, cudaStream_t s) {
  zero_kernel<<<1, 256, 0, s>>>(counts, E);
  return cudaGetLastError();
}

}  // namespace msi
