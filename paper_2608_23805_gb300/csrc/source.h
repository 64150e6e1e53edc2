// Internal interface of the bounded source service (source.cpp) used by the
// plan's staging path.  Not part of the public C ABI (include/msi.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/msi.h"

namespace msi {

// Host-side fault injection carried by a request (one-shot hooks of the plan).
constexpr int kInjectNone = 0;
constexpr int kInjectIoError = 1;    // the read completes with EIO
constexpr int kInjectShortRead = 2;  // the read delivers one byte less than the extent

// One extent read: the identity present at submission travels with it and is
// compared at completion.
struct SourceRequest {
  uint64_t object;      // ((layer + 1) << 32) | expert
  uint64_t epoch;       // the plan's request epoch at submission
  uint64_t generation;  // the slot generation the read will publish
  uint64_t file_off;
  uint64_t bytes;
  int inject;
};

// Submit a covering read into a free window (waits for the oldest window
// copy when none is free).  MSI_ERR_SOURCE on extent overflow.
msi_status source_submit(msi_source* s, const SourceRequest& rq, int* window);
// Wait for the window's read and check it against `expect`; on MSI_OK the
// window is HostReady and *data points at the extent.  A rejected read frees
// the window and returns MSI_ERR_SOURCE.
msi_status source_wait(msi_source* s, int window, const SourceRequest& expect, const void** data);
// The window's H2D copy has been enqueued on `stream`: Copying until an event
// recorded there completes.
msi_status source_copying(msi_source* s, int window, cudaStream_t stream);
// Return a window (its read, if in flight, lands first) without copying it.
msi_status source_release(msi_source* s, int window);
int source_windows(const msi_source* s);
// A plan attaches (+1) or detaches (-1); an attached source refuses to close.
void source_attach(msi_source* s, int delta);

}  // namespace msi
