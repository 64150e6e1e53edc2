// Argument blocks and launchers of the non-GEMM kernels (routers,
// histogram scan, scatter, wave setup, publication, combine) and the helper
// with which a forward's first kernel begins it.  The grouped GEMMs see only
// internal.cuh.
#pragma once

#include "internal.cuh"

namespace msi {

constexpr int kRouterTM = 32;  // tokens per fp32 FFMA router block
constexpr int kRouterChunk = 128;  // experts per tensor-core router CTA
constexpr int kScatterWarps = 4;   // scatter warps per block, one per router block

// The device that was current when the plan was created (plan.cu).
int plan_device(const msi_plan* p);

struct RouterArgs {
  const __nv_bfloat16* x;  // [T, H]
  const float* wr;         // [E, H]
  const float* wsg;        // [H] or nullptr
  int T, H, E, k;
  int* ids;                // [T, k]
  float* weights;          // [T, k]
  float* gap;              // [T] or nullptr
  float* sg;               // [T] (when wsg)
  int* bcount;             // [nb, E] routed ids per router block and expert
  // the forward's first kernel: status cleared and the shared group written
  // by block 0 (status null: a prediction pass, which begins nothing)
  int* status;
  Group* sh;               // or nullptr
  int* sh_total;
  int shared_slot;
};

struct RouterTcArgs {
  const __nv_bfloat16* x;  // [T, H] (shared-gate dot products)
  const float* wsg;        // [H] or nullptr
  int T, H, E, k;
  int chunk;               // experts per router CTA (<= kRouterChunk)
  int nchunk;              // E / chunk
  int kp;                  // candidates per chunk: min(k + 1, chunk)
  int tmem_cols;           // power of two >= max(32, chunk)
  float* cand_v;           // [T, nchunk, kp] candidate logits
  int* cand_i;             // [T, nchunk, kp] candidate expert ids
  int* ids;                // [T, k]
  float* weights;          // [T, k]
  float* gap;              // [T] or nullptr
  float* sg;               // [T]
  int* bcount;             // [ceil(T/32), E]
  int* status;
  long long wait_limit;
  int stall;               // as GemmArgs::stall
};

struct ScanArgs {
  const int* bcount;
  int nb, E;
  int* bbase;    // [nb, E] exclusive prefix over blocks within each expert
  int* counts;   // [E]
};

struct ScatterArgs {
  const int* ids;     // [T*k]
  const int* counts;  // [E]
  const int* bbase;   // [nb, E]
  // fuse_scan (nb <= kScatterWarps: one block's warps cover every router
  // block): counts and block prefixes are taken from bcount here, and the
  // last block writes the counts to counts_out (no column-scan launch)
  int fuse_scan;
  const int* bcount;  // [nb, E]
  int* counts_out;    // [E]
  int T, k, E, nb;
  int tm;             // tokens per router block
  int* perm;          // [T*k]
  int* inv;           // [T*k]
  int* offsets;       // [E+1]
  // an extra last block writes the offsets and, for a resident call, re-checks
  // the named slots' generations and builds the GEMM groups
  const GenWord* genwords;
  Group* groups;
  int* total_mtiles;   // [0]: 128-row tiles, [1]: 256-row pair tiles
  int* status;
  // resident call: the call's table, copied to global memory by an earlier
  // kernel of the forward (weight split or upload); null for a streamed call
  const int* tab_slot;                    // [E]
  const unsigned long long* tab_expected;  // [E]
  int layer;
  // fused resident GEMMs: per-m-tile counters zeroed by the setup block (or nullptr)
  int* ready;
  int n_ready;
};

// Per-call tables uploaded by value (kernel parameters, < 32 KB).
struct TableParams {
  int E;
  int layer;
  int T;
  int shared_slot;                 // shared-expert weight block (layer) or -1
  int slot[kMaxExperts];
  unsigned long long expected[kMaxExperts];
};

struct PublishParams {
  int n;
  int slot[kMaxWave];
  unsigned long long gen[kMaxWave];
  unsigned long long obj[kMaxWave];
};

struct SetupArgs {
  const int* counts;
  const int* offsets;
  const GenWord* genwords;
  int E, layer;
  Group* groups;
  int* total_mtiles;   // [0]: 128-row tiles, [1]: 256-row pair tiles
  int* status;
  int* ready;          // fused wave: per-m-tile counters, zeroed here (or nullptr)
  int n_ready;
};

struct CombineArgs {
  const __nv_bfloat16* yp;   // [T*k, H]
  const float* weights;      // [T, k]
  const int* inv;            // [T*k]
  const float* sg;           // [T]; nullptr: gate 1 (with ys)
  const __nv_bfloat16* ys;   // [T, H] or nullptr
  const __nv_bfloat16* x;    // residual or nullptr
  __nv_bfloat16* out;        // [T, H]
  int T, H, k;
  const int* status;
};

// ---------------------------------------------------------------------------
// Launchers (asynchronous on the given stream; return the launch error)
// ---------------------------------------------------------------------------
cudaError_t launch_router(const RouterArgs& a, cudaStream_t s);
// Also begins the forward (its first kernel): clears the status word and,
// when sh is not null, writes the shared-expert group of T rows in block
// `shared_slot` and its tile counts.  With tp not null it also copies the
// call's slot table and expected generations to tab_slot / tab_expected
// (the entries are read from the kernel argument by many blocks at once;
// one block reading all of them serialises on its constant cache).
cudaError_t launch_split3(const float* w, long long n, __nv_bfloat16* out, int* status, Group* sh,
                          int* sh_total, int T, int shared_slot, const TableParams* tp,
                          int* tab_slot, unsigned long long* tab_expected, cudaStream_t s);
cudaError_t launch_router_tc(const CUtensorMap& tmX, const CUtensorMap& tmW, const RouterTcArgs& a,
                             cudaStream_t s);
cudaError_t launch_colscan(const ScanArgs& a, cudaStream_t s);
cudaError_t launch_scatter(const ScatterArgs& a, cudaStream_t s);
// Copies the call's table to global memory and, when status is not null,
// begins the forward (as the first kernel of a call without rows).
cudaError_t launch_upload(const TableParams& p, int* table, unsigned long long* expected,
                          int* status, Group* shared_group, int* shared_total, cudaStream_t s);
cudaError_t launch_setup_wave(const SetupArgs& a, const WaveParams& w, cudaStream_t s);
cudaError_t launch_publish(const PublishParams& p, GenWord* genwords, cudaStream_t s);
// One launch for a wave whose extents all come from the early-staging buffer:
// each slot's published word is invalidated before any byte of its extent is
// copied (device to device), and the last block to finish publishes the
// wave's words.  ticket counts finished blocks across launches; target is its
// value once this launch's blocks have finished.
struct StageCopyArgs {
  PublishParams pub;
  const char* src[kMaxWave];     // extents in the early-staging buffer
  char* pool;                    // slot pool base
  unsigned long long bytes;      // extent bytes (a multiple of 16)
  unsigned long long* ticket;
  unsigned long long target;
  int parts;                     // blocks per extent
};
cudaError_t launch_stage_copy(const StageCopyArgs& a, GenWord* genwords, cudaStream_t s);
cudaError_t launch_combine(const CombineArgs& a, cudaStream_t s);
cudaError_t launch_zero_counts(int* counts, int E, cudaStream_t s);

#ifdef __CUDACC__
// The forward's start, written by its first kernel (one thread): the status
// word cleared and, with a shared expert, its single group over all T rows
// (slot = its weight block) with the 128-row and 256-row tile counts.
__device__ __forceinline__ void forward_begin(int* status, Group* sh, int* sh_total, int T,
                                              int shared_slot) {
  *status = 0;
  if (sh != nullptr) {
    Group g;
    g.row_begin = 0;
    g.row_count = T;
    g.slot = shared_slot;
    g.mt_begin = 0;
    g.ok = 1;
    g.expert = -1;
    g.pt_begin = g.pad1 = 0;
    *sh = g;
    sh_total[0] = (T + kBM - 1) / kBM;
    sh_total[1] = (T + 2 * kBM - 1) / (2 * kBM);
  }
}
#endif

}  // namespace msi
