// Bounded source service (paper, Sec. "Bounded Source Service"; the window
// lifecycle of Sec. "Separate Window and GPU-Slot Lifecycles").
//
// Expert extents are read from a file into a fixed set of N_w aligned host
// windows, so the host memory the stream of weights can occupy is bounded by
// N_w * W (the paper's M_source bound) and, with O_DIRECT, no second copy of
// the payload accumulates in the page cache.  Each window moves
// Free -> Reading -> HostReady -> Copying -> Free:
//   * submit: a covering read of the extent (the aligned range containing it)
//     goes to one reader thread per window; at most N_w reads are in flight;
//   * completion: the result is rejected on a negative completion (I/O
//     error), a short read (fewer bytes than cover the extent) or a request
//     that does not match the one submitted (object, epoch, generation);
//     extent overflow (past the end of the file) and oversize extents are
//     rejected at submission;
//   * the caller enqueues the H2D copy out of the window and hands the window
//     an event recorded after it; the window is free again once that event
//     has completed.
// Statistics: reads, rejections, logical bytes, physical bytes, padding
// (physical - logical), summed completion latency, peak reads in flight.
#include "source.h"

#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <cerrno>
#include <chrono>
#include <condition_variable>
#include <cstring>
#include <deque>
#include <mutex>
#include <thread>
#include <vector>

struct msi_source {
  enum State { kFree, kReading, kHostReady, kCopying };
  struct Win {
    State st = kFree;
    msi::SourceRequest req{};
    uint64_t cov_off = 0, cov_len = 0, lead = 0;
    int64_t got = 0;  // bytes delivered by the covering read
    int err = 0;      // errno of a failed read
    double secs = 0.0;
    cudaEvent_t ev = nullptr;  // recorded after the window's H2D copy
  };
  int fd = -1;
  bool direct = false;
  uint64_t align = 4096;
  uint64_t fsize = 0;
  uint8_t* base = nullptr;
  uint64_t wbytes = 0;
  std::vector<Win> w;
  std::mutex mu;
  std::condition_variable cv_job, cv_done;
  std::deque<int> jobs;
  std::vector<std::thread> th;
  bool stop = false;
  msi_source_stats st{};
  int in_flight = 0;
  int attached = 0;  // plans staging through this source

  void worker() {
    for (;;) {
      int i;
      {
        std::unique_lock<std::mutex> l(mu);
        cv_job.wait(l, [&] { return stop || !jobs.empty(); });
        if (stop && jobs.empty()) return;
        i = jobs.front();
        jobs.pop_front();
      }
      Win& x = w[i];
      const auto t0 = std::chrono::steady_clock::now();
      int64_t got = 0;
      int err = 0;
      if (x.req.inject == msi::kInjectIoError) {
        err = EIO;
      } else {
        uint8_t* dst = base + (size_t)i * wbytes;
        while ((uint64_t)got < x.cov_len) {
          const ssize_t r = pread(fd, dst + got, x.cov_len - got, (off_t)(x.cov_off + got));
          if (r < 0) {
            if (errno == EINTR) continue;
            err = errno;
            break;
          }
          if (r == 0) break;  // end of file
          got += r;
        }
        if (x.req.inject == msi::kInjectShortRead && err == 0) {
          // the source delivers one byte less than the extent needs
          const int64_t need = (int64_t)(x.lead + x.req.bytes);
          if (got >= need) got = need - 1;
        }
      }
      const double secs = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
      {
        std::lock_guard<std::mutex> l(mu);
        x.got = got;
        x.err = err;
        x.secs = secs;
        x.st = kHostReady;
        in_flight--;
      }
      cv_done.notify_all();
    }
  }

  // A window whose copy has completed returns to Free.
  bool reclaim(int i) {
    Win& x = w[i];
    if (x.st != kCopying) return x.st == kFree;
    if (x.ev != nullptr) {
      const cudaError_t e = cudaEventQuery(x.ev);
      if (e == cudaErrorNotReady) {
        (void)cudaGetLastError();
        return false;
      }
    }
    x.st = kFree;
    return true;
  }
};

namespace msi {

msi_status source_submit(msi_source* s, const SourceRequest& rq, int* window) {
  if (s == nullptr || window == nullptr || rq.bytes == 0) return MSI_ERR_INVALID_ARG;
  // extent overflow: the extent must lie inside the file
  if (rq.file_off > s->fsize || rq.bytes > s->fsize - rq.file_off) {
    std::lock_guard<std::mutex> l(s->mu);
    s->st.rejected++;
    return MSI_ERR_SOURCE;
  }
  const uint64_t a = s->direct ? s->align : 1;
  const uint64_t cov_off = rq.file_off / a * a;
  const uint64_t lead = rq.file_off - cov_off;
  const uint64_t cov_len = (lead + rq.bytes + a - 1) / a * a;
  if (cov_len > s->wbytes) return MSI_ERR_INVALID_ARG;  // the extent does not fit a window
  // a free window: Free, or Copying with its copy completed; else wait for the
  // oldest copy still in flight (an H2D copy always completes)
  int i = -1;
  {
    std::lock_guard<std::mutex> l(s->mu);
    for (int c = 0; c < (int)s->w.size() && i < 0; ++c)
      if (s->reclaim(c)) i = c;
  }
  if (i < 0) {
    for (int c = 0; c < (int)s->w.size() && i < 0; ++c) {
      if (s->w[c].st == msi_source::kCopying && s->w[c].ev != nullptr) {
        if (cudaEventSynchronize(s->w[c].ev) != cudaSuccess) return MSI_ERR_CUDA;
        std::lock_guard<std::mutex> l(s->mu);
        if (s->reclaim(c)) i = c;
      }
    }
  }
  if (i < 0) return MSI_ERR_SLOT_BUSY;  // every window is Reading or HostReady (caller-held)
  {
    std::lock_guard<std::mutex> l(s->mu);
    msi_source::Win& x = s->w[i];
    x.req = rq;
    x.cov_off = cov_off;
    x.cov_len = cov_len;
    x.lead = lead;
    x.got = 0;
    x.err = 0;
    x.st = msi_source::kReading;
    s->jobs.push_back(i);
    s->in_flight++;
    if (s->in_flight > s->st.max_in_flight) s->st.max_in_flight = s->in_flight;
  }
  s->cv_job.notify_one();
  *window = i;
  return MSI_OK;
}

msi_status source_wait(msi_source* s, int i, const SourceRequest& expect, const void** data) {
  if (s == nullptr || i < 0 || i >= (int)s->w.size()) return MSI_ERR_INVALID_ARG;
  std::unique_lock<std::mutex> l(s->mu);
  msi_source::Win& x = s->w[i];
  s->cv_done.wait(l, [&] { return x.st != msi_source::kReading; });
  if (x.st != msi_source::kHostReady) return MSI_ERR_INVALID_ARG;
  s->st.reads++;
  s->st.read_seconds += x.secs;
  const bool neg = x.err != 0;
  const bool shortr = x.got < (int64_t)(x.lead + x.req.bytes);
  const bool mismatch = x.req.object != expect.object || x.req.epoch != expect.epoch ||
                        x.req.generation != expect.generation || x.req.bytes != expect.bytes;
  if (neg || shortr || mismatch) {
    s->st.rejected++;
    x.st = msi_source::kFree;  // nothing of this read becomes host-ready for a copy
    return MSI_ERR_SOURCE;
  }
  s->st.logical_bytes += x.req.bytes;
  s->st.physical_bytes += x.cov_len;
  s->st.padding_bytes += x.cov_len - x.req.bytes;
  if (data) *data = s->base + (size_t)i * s->wbytes + x.lead;
  return MSI_OK;
}

msi_status source_copying(msi_source* s, int i, cudaStream_t stream) {
  if (s == nullptr || i < 0 || i >= (int)s->w.size()) return MSI_ERR_INVALID_ARG;
  msi_source::Win& x = s->w[i];
  if (x.ev == nullptr && cudaEventCreateWithFlags(&x.ev, cudaEventDisableTiming) != cudaSuccess)
    return MSI_ERR_CUDA;
  if (cudaEventRecord(x.ev, stream) != cudaSuccess) return MSI_ERR_CUDA;
  std::lock_guard<std::mutex> l(s->mu);
  x.st = msi_source::kCopying;
  return MSI_OK;
}

msi_status source_release(msi_source* s, int i) {
  if (s == nullptr || i < 0 || i >= (int)s->w.size()) return MSI_ERR_INVALID_ARG;
  std::unique_lock<std::mutex> l(s->mu);
  msi_source::Win& x = s->w[i];
  s->cv_done.wait(l, [&] { return x.st != msi_source::kReading; });  // a read in flight lands first
  if (x.st == msi_source::kHostReady) x.st = msi_source::kFree;
  return MSI_OK;
}

int source_windows(const msi_source* s) { return s ? (int)s->w.size() : 0; }

void source_attach(msi_source* s, int delta) {
  if (s == nullptr) return;
  std::lock_guard<std::mutex> l(s->mu);
  s->attached += delta;
}

}  // namespace msi

extern "C" {

msi_status msi_source_open(const msi_source_desc* d, msi_source** out) {
  if (d == nullptr || out == nullptr || d->path == nullptr || d->windows == nullptr) return MSI_ERR_INVALID_ARG;
  *out = nullptr;
  const uint64_t align = d->align ? d->align : 4096;
  if ((align & (align - 1)) != 0 || d->n_windows < 1 || d->n_windows > MSI_MAX_WINDOWS ||
      d->window_bytes == 0)
    return MSI_ERR_INVALID_ARG;
  if (d->direct && ((uintptr_t)d->windows % align || d->window_bytes % align)) return MSI_ERR_INVALID_ARG;
  const int fd = open(d->path, O_RDONLY | (d->direct ? O_DIRECT : 0));
  if (fd < 0) return errno == EINVAL ? MSI_ERR_UNSUPPORTED : MSI_ERR_SOURCE;
  struct stat sb;
  if (fstat(fd, &sb) != 0) {
    close(fd);
    return MSI_ERR_SOURCE;
  }
  msi_source* s = new msi_source();
  s->fd = fd;
  s->direct = d->direct != 0;
  s->align = align;
  s->fsize = (uint64_t)sb.st_size;
  s->base = static_cast<uint8_t*>(d->windows);
  s->wbytes = d->window_bytes;
  s->w.resize(d->n_windows);
  for (int i = 0; i < d->n_windows; ++i) s->th.emplace_back([s] { s->worker(); });
  *out = s;
  return MSI_OK;
}

msi_status msi_source_close(msi_source* s) {
  if (s == nullptr) return MSI_ERR_INVALID_ARG;
  {
    std::unique_lock<std::mutex> l(s->mu);
    // shutdown check: no plan may still stage through the source and no
    // caller may still hold a window it read
    if (s->attached > 0) return MSI_ERR_SLOT_BUSY;
    s->cv_done.wait(l, [&] {
      for (const auto& x : s->w)
        if (x.st == msi_source::kReading) return false;
      return true;
    });
    for (const auto& x : s->w)
      if (x.st == msi_source::kHostReady) return MSI_ERR_SLOT_BUSY;
    s->stop = true;
  }
  s->cv_job.notify_all();
  for (auto& t : s->th) t.join();  // every read in flight has landed
  for (auto& x : s->w) {
    if (x.ev != nullptr) {
      cudaEventSynchronize(x.ev);
      cudaEventDestroy(x.ev);
    }
  }
  close(s->fd);
  delete s;
  return MSI_OK;
}

msi_status msi_source_stats_read(msi_source* s, msi_source_stats* out) {
  if (s == nullptr || out == nullptr) return MSI_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> l(s->mu);
  *out = s->st;
  out->windows_busy = 0;
  for (int i = 0; i < (int)s->w.size(); ++i)
    if (!s->reclaim(i)) out->windows_busy++;
  return MSI_OK;
}

msi_status msi_source_read(msi_source* s, uint64_t file_off, uint64_t bytes, const void** data,
                           int* window) {
  msi::SourceRequest rq{};
  rq.file_off = file_off;
  rq.bytes = bytes;
  msi_status st = msi::source_submit(s, rq, window);
  if (st != MSI_OK) return st;
  st = msi::source_wait(s, *window, rq, data);
  if (st != MSI_OK) *window = -1;
  return st;
}

msi_status msi_source_release(msi_source* s, int window) { return msi::source_release(s, window); }

}  // extern "C"
