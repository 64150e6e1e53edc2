// msi_moe_forward_static: the resident layer forward for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc or use an allocator at all: code running
// inside another runtime's memory budget with no allocator handle, plugins
// whose host framework owns every allocation, and hard real-time or
// safety-critical loops that forbid allocation after start-up.  This entry
// point needs no caller workspace: its scratch is one file-scope device array
// of fixed size, reserved on every GPU that loads this library until the
// process exits.
//
// Contract:
//  - Scratch limit kStaticScratchBytes (32 MiB).  A call whose
//    msi_workspace_size(plan, T) exceeds it returns MSI_ERR_WORKSPACE and
//    enqueues nothing: up to 478 tokens a call at the Qwen3-Next layer shape
//    (512 experts, top-10, hidden 2048, intermediate 512, shared expert),
//    21,502 at hidden 256 / intermediate 128 / 16 experts / top-2.
//  - The call must be made with the plan's device current (the device that
//    was current at msi_plan_create); otherwise MSI_ERR_INVALID_ARG, nothing
//    enqueued.
//  - The device address of the array is resolved with cudaGetSymbolAddress on
//    the first call on each device (with that device current) and cached;
//    make that first call before any stream capture.  The cache is not
//    invalidated: after a device reset (cudaDeviceReset, or the primary
//    context released and re-created) the process must restart before it
//    calls this entry point again.
//  - Every call on a device shares the one array, which keeps the previous
//    call's contents.  The forward writes every scratch word it reads before
//    reading it (the status word is cleared by the forward's first kernel), so
//    nothing has to start at zero.  Calls whose kernels overlap on the GPU
//    (two streams, or two plans) race on the array: serialise them.
//  - The call allocates nothing itself: no cudaMalloc, cudaFree or allocating
//    library routine.
#include <mutex>

#include "kernels.cuh"

namespace {

constexpr size_t kStaticScratchBytes = 32ull << 20;
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

}  // namespace

extern "C" msi_status msi_moe_forward_static(msi_plan* plan, int layer, const void* hidden, int T,
                                             const float* router_w, const int32_t* slot_table,
                                             const uint64_t* expected_generations, void* out,
                                             const msi_route_event* ev, unsigned flags,
                                             msi_stream compute) {
  if (plan == nullptr || T < 0) return MSI_ERR_INVALID_ARG;
  size_t need = 0;
  msi_status st = msi_workspace_size(plan, T, &need);
  if (st != MSI_OK) return st;
  if (need > kStaticScratchBytes) return MSI_ERR_WORKSPACE;
  // the scratch must be the plan's device's array: the plan's kernels run there
  const int dev = msi::plan_device(plan);
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess) return MSI_ERR_CUDA;
  if (cur != dev) return MSI_ERR_INVALID_ARG;
  if (dev < 0 || dev >= kMaxDevices) return MSI_ERR_CUDA;
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> g(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
        return MSI_ERR_CUDA;
      g_scratch_addr[dev] = p;
    }
    scratch = g_scratch_addr[dev];
  }
  return msi_moe_forward(plan, layer, hidden, T, router_w, slot_table, expected_generations, out,
                         ev, scratch, kStaticScratchBytes, flags, compute);
}
