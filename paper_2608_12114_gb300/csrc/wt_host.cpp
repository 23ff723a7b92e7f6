// Host side of the wt library: the C ABI of include/wt.h.
//
//   open     parallel per-file open / fstat / pread index / validate / mmap
//            (Algorithm 1's guarded shared read-only map), then the device
//            route for each mapping (Sec. 7.3: registration and direct read are
//            probed separately; GB300 reads pageable memory through the host
//            page tables, so a registration is optional there)
//   adopt    batches tensors into launches of the gather kernel (or copy-engine
//            copies, or the staged pinned ring) and records one event per
//            batch: contract C3 (order on the GPU), Table "tab:contract"
//   pass     plans one persistent GEMV launch per group of descriptors sharing
//            a wait event; plans are cached and uploaded stream-ordered
//   close    waits on the handle's own events, unregisters, unmaps
#include <fcntl.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cerrno>
#include <condition_variable>
#include <deque>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <list>
#include <mutex>
#include <new>
#include <string>
#include <string_view>
#include <thread>
#include <unordered_map>
#include <unordered_set>
#include <memory>
#include <vector>

#include <cuda.h>  // CUtensorMap and its encoder's signature (resolved through the runtime)
#include <cuda_runtime.h>

#include "../../include/wt.h"
#include "../../include/wt_dlpack.h"
#include "wt_fnv.h"
#include "wt_kernels.h"
#include "wt_q8rows.h"

#ifndef MADV_POPULATE_READ
#define MADV_POPULATE_READ 22
#endif

namespace {

thread_local std::string t_err;

int set_err(int code, const char *fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  t_err = buf;
  return code;
}

int cuda_err(cudaError_t e, const char *what) {
  cudaGetLastError();  // clear the sticky-free error so later calls start clean
  return set_err(WT_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define CU(call)                                        \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return cuda_err(e_, #call);  \
  } while (0)

// Live objects of the library (wt_live): handles, launch plans, CUDA events, and the device
// and pinned host bytes the library itself allocated.  Every create/allocate below goes
// through these helpers so that a leak shows up as a count that does not return.
std::atomic<int64_t> g_live_handles{0}, g_live_plans{0}, g_live_events{0}, g_dev_bytes{0}, g_pinned_bytes{0};

cudaError_t ev_create(cudaEvent_t *ev, unsigned flags) {
  const cudaError_t e = cudaEventCreateWithFlags(ev, flags);
  if (e == cudaSuccess) g_live_events++;
  return e;
}

void ev_destroy(cudaEvent_t ev) {
  if (ev && cudaEventDestroy(ev) == cudaSuccess) g_live_events--;
}

cudaError_t dev_alloc(void **p, size_t n) {
  const cudaError_t e = cudaMalloc(p, n);
  if (e == cudaSuccess) g_dev_bytes += (int64_t)n;
  return e;
}

void dev_free(void *p, size_t n) {
  if (p && cudaFree(p) == cudaSuccess) g_dev_bytes -= (int64_t)n;
}

cudaError_t pinned_alloc(void **p, size_t n) {
  const cudaError_t e = cudaHostAlloc(p, n, cudaHostAllocDefault);
  if (e == cudaSuccess) g_pinned_bytes += (int64_t)n;
  return e;
}


// ------------------------------------------------------------------ block cache
// A handle's own device and pinned allocations (its status word, plan tables and their pinned
// staging copies, split-K workspaces) come from a per-device cache of power-of-two blocks, kept
// when the handle closes and handed to the next one.  A fresh handle then makes no cudaMalloc,
// cudaHostAlloc or cudaFree call: on GB300 those cost tens of microseconds each (cudaFree also
// waits for the device), which was most of the host time of a small checkpoint's file -> first
// use.  Blocks of 256 B .. 64 MiB are cached, up to kCapBytes per device and kind; larger
// blocks, and frees beyond the cap, go to the driver as before.  wt_live counts the bytes
// handed out (device_bytes, pinned_bytes) apart from the bytes the cache holds.
std::atomic<int64_t> g_dev_cached{0}, g_pinned_cached{0};

struct BlockCache {
  static constexpr int kMinLog2 = 8, kMaxLog2 = 26;
  static constexpr int64_t kCapBytes = 256ll << 20;
  std::mutex mu;
  std::vector<void *> free_blocks[kMaxLog2 + 1];
  int64_t cached = 0;
  // status words: 256-byte device blocks that are zero (cleared by the closing handle, after
  // its work has completed), so an open takes one without a memset
  std::vector<int *> clean_status;
  cudaStream_t stream = nullptr;  // clears status words
};
BlockCache g_dev_cache[64], g_pin_cache[64];

int block_log2(size_t n) {
  int c = BlockCache::kMinLog2;
  while (c <= BlockCache::kMaxLog2 && ((size_t)1 << c) < n) ++c;
  return c;  // kMaxLog2 + 1: not cached
}

cudaError_t cached_alloc(bool pinned, int dev, void **p, size_t n) {
  *p = nullptr;
  const int c = block_log2(n);
  if (dev >= 0 && dev < 64 && c <= BlockCache::kMaxLog2) {
    BlockCache &bc = pinned ? g_pin_cache[dev] : g_dev_cache[dev];
    std::lock_guard<std::mutex> g(bc.mu);
    if (!bc.free_blocks[c].empty()) {
      *p = bc.free_blocks[c].back();
      bc.free_blocks[c].pop_back();
      bc.cached -= (int64_t)1 << c;
      (pinned ? g_pinned_cached : g_dev_cached) -= (int64_t)1 << c;
      (pinned ? g_pinned_bytes : g_dev_bytes) += (int64_t)n;
      return cudaSuccess;
    }
  }
  const size_t sz = c <= BlockCache::kMaxLog2 ? (size_t)1 << c : n;
  const cudaError_t e = pinned ? cudaHostAlloc(p, sz, cudaHostAllocDefault) : cudaMalloc(p, sz);
  if (e == cudaSuccess) (pinned ? g_pinned_bytes : g_dev_bytes) += (int64_t)n;
  return e;
}

// p must no longer be in use by any enqueued work.
void cached_free(bool pinned, int dev, void *p, size_t n) {
  if (!p) return;
  (pinned ? g_pinned_bytes : g_dev_bytes) -= (int64_t)n;
  const int c = block_log2(n);
  if (dev >= 0 && dev < 64 && c <= BlockCache::kMaxLog2) {
    BlockCache &bc = pinned ? g_pin_cache[dev] : g_dev_cache[dev];
    std::lock_guard<std::mutex> g(bc.mu);
    if (bc.cached + ((int64_t)1 << c) <= BlockCache::kCapBytes) {
      bc.free_blocks[c].push_back(p);
      bc.cached += (int64_t)1 << c;
      (pinned ? g_pinned_cached : g_dev_cached) += (int64_t)1 << c;
      return;
    }
  }
  if (pinned) cudaFreeHost(p);
  else cudaFree(p);
}

// Clears a status word on the cache's own stream and waits for that alone (not the device).
// Called with bc.mu held.
cudaError_t status_clear(BlockCache &bc, int *p) {
  cudaError_t e = bc.stream ? cudaSuccess : cudaStreamCreateWithFlags(&bc.stream, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaMemsetAsync(p, 0, 256, bc.stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(bc.stream);
  return e;
}

// A zeroed 256-byte status word on device `dev` (the current device).
cudaError_t status_take(int dev, int **p) {
  *p = nullptr;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  BlockCache &bc = g_dev_cache[dev];
  std::lock_guard<std::mutex> g(bc.mu);
  if (!bc.clean_status.empty()) {
    *p = bc.clean_status.back();
    bc.clean_status.pop_back();
    bc.cached -= 256;
    g_dev_cached -= 256;
    g_dev_bytes += 256;
    return cudaSuccess;
  }
  cudaError_t e = cudaMalloc(reinterpret_cast<void **>(p), 256);
  if (e != cudaSuccess) return e;
  e = status_clear(bc, *p);
  if (e != cudaSuccess) {
    cudaFree(*p);
    *p = nullptr;
    return e;
  }
  g_dev_bytes += 256;
  return cudaSuccess;
}

// Returns a status word once every kernel that could write it has completed: it is cleared
// and kept for the next handle (freed if the clear fails or the cache is full).
void status_give(int dev, int *p) {
  if (!p) return;
  g_dev_bytes -= 256;
  if (dev >= 0 && dev < 64) {
    BlockCache &bc = g_dev_cache[dev];
    std::lock_guard<std::mutex> g(bc.mu);
    if (bc.cached + 256 <= BlockCache::kCapBytes && status_clear(bc, p) == cudaSuccess) {
      bc.clean_status.push_back(p);
      bc.cached += 256;
      g_dev_cached += 256;
      return;
    }
    cudaGetLastError();
  }
  cudaFree(p);
}

constexpr uint64_t kAlign = 64;
constexpr int kMaxDims = 4;

int elem_bytes(int dtype) {
  switch (dtype) {
    case WT_F32: return 4;
    case WT_BF16: case WT_F16: return 2;
    case WT_I8: case WT_U8: return 1;
    default: return 0;
  }
}

// ------------------------------------------------------------------ small thread pool
class Pool {
 public:
  explicit Pool(int n) {
    for (int i = 0; i < n; ++i) th_.emplace_back([this] { run(); });
  }
  ~Pool() {
    {
      std::lock_guard<std::mutex> g(m_);
      stop_ = true;
    }
    cv_.notify_all();
    for (auto &t : th_) t.join();
  }
  int size() const { return (int)th_.size(); }
  // Runs fn(i) for i in [0, n) on the pool and the calling thread; returns when all are done.
  void parallel_for(size_t n, const std::function<void(size_t)> &fn) {
    if (n == 0) return;
    std::lock_guard<std::mutex> one_at_a_time(call_mu_);
    if (th_.empty() || n == 1) {
      for (size_t i = 0; i < n; ++i) fn(i);
      return;
    }
    std::atomic<size_t> next{0};
    std::atomic<size_t> done{0};
    auto body = [&] {
      size_t i;
      while ((i = next.fetch_add(1)) < n) {
        fn(i);
        done.fetch_add(1);
      }
    };
    {
      std::lock_guard<std::mutex> g(m_);
      job_ = body;
      gen_++;
    }
    cv_.notify_all();
    body();
    std::unique_lock<std::mutex> lk(m_);
    done_cv_.wait(lk, [&] { return done.load() == n && active_ == 0; });
    job_ = nullptr;
  }

 private:
  void run() {
    uint64_t seen = 0;
    for (;;) {
      std::function<void()> job;
      {
        std::unique_lock<std::mutex> lk(m_);
        cv_.wait(lk, [&] { return stop_ || (gen_ != seen && job_); });
        if (stop_) return;
        seen = gen_;
        job = job_;
        active_++;
      }
      job();
      {
        std::lock_guard<std::mutex> g(m_);
        active_--;
      }
      done_cv_.notify_all();
    }
  }
  std::vector<std::thread> th_;
  std::mutex call_mu_;
  std::mutex m_;
  std::condition_variable cv_, done_cv_;
  std::function<void()> job_;
  uint64_t gen_ = 0;
  int active_ = 0;
  bool stop_ = false;
};

Pool &host_pool() {
  static Pool p([] {
    unsigned n = std::thread::hardware_concurrency();
    return (int)std::min(15u, n > 1 ? n - 1 : 0u);
  }());
  return p;
}

// ------------------------------------------------------------------ handle
struct Tensor {
  std::string name;
  int dtype = 0;
  int ndim = 0;
  uint64_t shape[kMaxDims] = {0, 0, 0, 0};
  uint64_t nbytes = 0;
  uint64_t offset = 0;
};

struct File {
  std::string path;
  uint8_t *base = nullptr;  // mapping (nullptr: opened with WT_OPEN_NOMAP, or small under MAP_LARGE)
  size_t size = 0;
  bool small = false;       // WT_OPEN_MAP_LARGE left it unmapped: adopted through the pinned ring
  int64_t index_ns = 0, map_ns = 0;  // host time wt_open spent parsing and mapping it
  // identity at wt_open: a WT_OPEN_NOMAP file is opened again by a staged adopt, which checks
  // that the path still names the file whose index was validated
  uint64_t st_dev = 0, st_ino = 0;
  int64_t mtime_ns = 0;
  unsigned route = WT_ROUTE_NONE;
  bool registered = false;
  unsigned reg_flags = 0;        // cudaHostRegister flags the registration holds (0: none)
  bool populated = false;        // page-table entries already filled (registered files)
  const uint8_t *dev = nullptr;  // device-readable address of base
  std::vector<Tensor> tensors;
};

struct Plan {
  std::vector<uint8_t> key;
  struct Launch {
    int dtype;
    int grid;
    size_t mats, pieces, begin;  // byte offsets in the table
    size_t maps = SIZE_MAX;      // multi-column launches: tensor maps (128-byte aligned)
    bool umma = false;           // multi-column launch on tcgen05 (wt_umma.cu)
    bool q8rows = false;         // int8 multi-column launch on the row-owner kernel (wt_q8rows.cu)
    bool mapped_cols = false;    // map endpoint with T columns
    int nt = 0;                  // warp-MMA multi-column launches: 8-column tiles (1 or 2)
    uint32_t nmat = 0, ntiles = 0;
  };
  struct Generic {
    int dtype;
    const uint8_t *W, *x;
    float *y;
    uint64_t M, K;
    const uint8_t *scale;
    uint32_t cols;
  };
  struct Zero {
    float *y;
    uint64_t M;
  };
  struct Group {
    size_t first = 0;  // index of the group's first descriptor (its wait_event is read per call)
    std::vector<Launch> launches;
    std::vector<Launch> mapped;  // W read in place from a file mapping (map endpoint)
    std::vector<Launch> cols;    // multi-column kernel (tensor cores)
    size_t reduce = 0;           // SegReduce table of this group's column-segmented matrices
    int n_reduce = 0;
    uint32_t reduce_rows = 0;
    std::vector<Generic> generic;
    std::vector<Zero> zero;
    uint64_t wbytes = 0;         // weight bytes the group streams (timeline records)
  };
  std::vector<Group> groups;
  std::vector<uint8_t> table;
  uint8_t *host = nullptr;  // pinned copy of table
  uint8_t *dev = nullptr;
  cudaEvent_t uploaded = nullptr;
  std::vector<std::pair<cudaStream_t, cudaEvent_t>> last;  // (stream, its latest run's completion)
  bool sent = false;
  cudaStream_t sent_on = nullptr;
  bool pinned = false;  // used inside a captured CUDA graph: kept until wt_close
  size_t table_bytes = 0;  // size of `host` and `dev`
  float *ws = nullptr;  // split-K segment partials (device), ws_floats floats
  size_t ws_floats = 0;
  std::vector<std::pair<size_t, size_t>> ws_patches;  // (table byte offset of a pointer, ws float offset)
  uint64_t launches = 0;
  int device = -1;  // its blocks' cache
};

// The staged arm's pinned ring: one per device for the whole process (pinning host memory
// costs far more than a first use of a small checkpoint, so it is paid once), allocated by
// the first staged adopt on the device and kept until the process exits.  Staged adopts on
// one device take turns on it (its mutex); a slot is refilled once the device has read it.
struct Ring {
  static constexpr int kSlots = 4;
  static constexpr size_t kSlotBytes = 64ull << 20;
  std::mutex mu;
  bool ready = false;
  cudaStream_t stream = nullptr;  // the staged half of a mixed adopt (WT_OPEN_MAP_LARGE)
  uint8_t *slot[kSlots] = {nullptr, nullptr, nullptr, nullptr};
  cudaEvent_t done[kSlots] = {nullptr, nullptr, nullptr, nullptr};
  bool used[kSlots] = {false, false, false, false};
  int next = 0;
};

Ring g_ring[64];

}  // namespace

struct wt_handle {
  std::vector<File> files;
  std::vector<std::pair<uintptr_t, uint32_t>> by_base;  // (mapping start, file), sorted: address lookups
  std::vector<std::pair<uint32_t, uint32_t>> order;  // global tensor index -> (file, entry)
  bool host_only = false;
  bool prefaulted = false;
  // WT_OPEN_TIMELINE: timing events around every ingest batch and every GEMV group, read
  // back (and released) by wt_trace
  struct TraceEv {
    int kind;
    uint64_t index, bytes;
    cudaEvent_t begin, end;
    bool own_end;       // an ingest batch's end event is its ready event, owned by `events`
    cudaEvent_t event;  // ingest: the batch's ready event; GEMV: the event the group waited on
  };
  bool timeline = false;
  std::vector<TraceEv> trace;
  std::atomic<uint64_t> n_batches{0};
  uint64_t n_groups = 0;
  // WT_OPEN_STAMPS: one-column GEMV launches run the stamping kernel into stamp_dev
  // (stamp_cap CTAs of wt::kStampFields words); stamp_ctas is the grid of the latest one
  bool stamping = false;
  uint64_t *stamp_dev = nullptr;
  size_t stamp_cap = 0;
  int stamp_ctas = 0;
  int device = -1;
  int *status = nullptr;
  std::vector<cudaEvent_t> events;
  std::list<Plan *> plans;
  std::atomic<uint64_t> kernel_launches{0};
  wt_open_phases open_times{};
  std::mutex mu;
  // events and trace records: a mixed adopt (WT_OPEN_MAP_LARGE) adds them from two threads
  std::mutex ev_mu;

  const Tensor &tensor(size_t i) const {
    return files[order[i].first].tensors[order[i].second];
  }
};

namespace {

// ------------------------------------------------------------------ index parser
struct Reader {
  const uint8_t *p;
  size_t n, pos = 0;
  bool need(size_t k) const { return pos <= n && k <= n - pos; }
  uint64_t le(int k) {
    uint64_t v = 0;
    for (int i = 0; i < k; ++i) v |= (uint64_t)p[pos + i] << (8 * i);
    pos += k;
    return v;
  }
};

int parse_file(File &f, int fd, uint64_t fsize) {
  const char *path = f.path.c_str();
  if (fsize < 16) return set_err(WT_EFORMAT, "%s: shorter than the 16-byte header", path);
  uint8_t hdr[16];
  if (wt::fault_injected("pread")) return set_err(WT_EIO, "%s: pread header: injected fault", path);
  if (pread(fd, hdr, 16, 0) != 16) return set_err(WT_EIO, "%s: pread header: %s", path, strerror(errno));
  if (memcmp(hdr, "WTCKPT01", 8) != 0) return set_err(WT_EFORMAT, "%s: bad magic", path);
  Reader h{hdr, 16, 8};
  const uint64_t ilen = h.le(8);
  if (ilen < 4 || ilen > fsize - 16) return set_err(WT_EFORMAT, "%s: index length outside the file", path);
  std::vector<uint8_t> ix(ilen);
  if ((uint64_t)pread(fd, ix.data(), ilen, 16) != ilen)
    return set_err(WT_EIO, "%s: pread index: %s", path, strerror(errno));
  Reader r{ix.data(), ix.size()};
  const uint64_t count = r.le(4);
  constexpr uint64_t kMinEntry = 2 + 1 + 1 + 1 + 8 + 8 + 8;
  if (count > (ilen - 4) / kMinEntry) return set_err(WT_EFORMAT, "%s: entry count exceeds the index", path);
  f.tensors.resize(count);
  const uint64_t first_blob = 16 + ilen;
  uint64_t end_prev = first_blob;
  std::unordered_set<std::string> names;
  for (uint64_t i = 0; i < count; ++i) {
    Tensor &t = f.tensors[i];
    if (!r.need(2)) return set_err(WT_EFORMAT, "%s: entry %llu: index ends inside the name length", path, (unsigned long long)i);
    const uint64_t nl = r.le(2);
    if (nl == 0) return set_err(WT_EFORMAT, "%s: entry %llu: empty name", path, (unsigned long long)i);
    if (!r.need(nl + 2)) return set_err(WT_EFORMAT, "%s: entry %llu: index ends inside the name", path, (unsigned long long)i);
    t.name.assign(reinterpret_cast<const char *>(r.p + r.pos), nl);
    r.pos += nl;
    if (t.name.find('\0') != std::string::npos)
      return set_err(WT_EFORMAT, "%s: entry %llu: NUL byte in name", path, (unsigned long long)i);
    t.dtype = (int)r.le(1);
    t.ndim = (int)r.le(1);
    const int es = elem_bytes(t.dtype);
    if (es == 0) return set_err(WT_EFORMAT, "%s: entry %llu: unknown dtype %d", path, (unsigned long long)i, t.dtype);
    if (t.ndim < 1 || t.ndim > kMaxDims)
      return set_err(WT_EFORMAT, "%s: entry %llu: ndim %d outside 1..4", path, (unsigned long long)i, t.ndim);
    if (!r.need(8ull * t.ndim + 16)) return set_err(WT_EFORMAT, "%s: entry %llu: index ends inside the shape", path, (unsigned long long)i);
    unsigned __int128 elems = 1;
    for (int d = 0; d < t.ndim; ++d) {
      t.shape[d] = r.le(8);
      elems *= t.shape[d];
      if (elems > ((unsigned __int128)1 << 64)) elems = ((unsigned __int128)1 << 64) + 1;  // saturate
    }
    const unsigned __int128 bytes = elems * (unsigned)es;
    t.offset = r.le(8);
    t.nbytes = r.le(8);
    if (bytes > UINT64_MAX) return set_err(WT_EFORMAT, "%s: entry %llu: shape product overflows", path, (unsigned long long)i);
    if ((unsigned __int128)t.nbytes != bytes)
      return set_err(WT_EFORMAT, "%s: entry %llu: nbytes %llu != prod(shape) * %d", path, (unsigned long long)i,
                     (unsigned long long)t.nbytes, es);
    if (t.offset % kAlign) return set_err(WT_EFORMAT, "%s: entry %llu: offset %llu not 64-byte aligned", path, (unsigned long long)i, (unsigned long long)t.offset);
    if (t.offset < first_blob) return set_err(WT_EFORMAT, "%s: entry %llu: blob overlaps the header/index", path, (unsigned long long)i);
    if (t.offset > fsize || t.nbytes > fsize - t.offset)
      return set_err(WT_EFORMAT, "%s: entry %llu: blob runs past the end of the file", path, (unsigned long long)i);
    if (t.offset < end_prev) return set_err(WT_EFORMAT, "%s: entry %llu: blob overlaps the previous blob", path, (unsigned long long)i);
    end_prev = t.offset + t.nbytes;
    if (!names.insert(t.name).second) return set_err(WT_EFORMAT, "%s: entry %llu: duplicate name '%s'", path, (unsigned long long)i, t.name.c_str());
  }
  if (r.pos != ilen) return set_err(WT_EFORMAT, "%s: index length does not match its entries", path);
  return WT_OK;
}

void unmap_file(File &f) {
  if (f.registered) {
    cudaHostUnregister(f.base);
    f.registered = false;
  }
  if (f.base) {
    munmap(f.base, f.size);
    f.base = nullptr;
  }
}

// open, parse and map one file (not with `nomap`, nor when it is smaller than `map_min`
// bytes); closes the fd on every path.
int64_t now_ns() {
  return std::chrono::duration_cast<std::chrono::nanoseconds>(std::chrono::steady_clock::now().time_since_epoch())
      .count();
}

int open_one(File &f, bool nomap, uint64_t map_min) {
  const int64_t t0 = now_ns();
  if (wt::fault_injected("open")) return set_err(WT_EIO, "%s: open: injected fault", f.path.c_str());
  const int fd = open(f.path.c_str(), O_RDONLY | O_CLOEXEC);
  if (fd < 0) return set_err(WT_EIO, "%s: open: %s", f.path.c_str(), strerror(errno));
  struct stat st;
  if (fstat(fd, &st) != 0) {
    int e = errno;
    close(fd);
    return set_err(WT_EIO, "%s: fstat: %s", f.path.c_str(), strerror(e));
  }
  int rc = parse_file(f, fd, (uint64_t)st.st_size);
  f.st_dev = (uint64_t)st.st_dev;
  f.st_ino = (uint64_t)st.st_ino;
  f.mtime_ns = (int64_t)st.st_mtim.tv_sec * 1000000000ll + st.st_mtim.tv_nsec;
  const bool skip = nomap || (uint64_t)st.st_size < map_min;
  f.small = !nomap && skip;
  const int64_t t1 = now_ns();
  f.index_ns = t1 - t0;
  if (rc == WT_OK && skip) f.size = (size_t)st.st_size;
  if (rc == WT_OK && !skip) {
    f.size = (size_t)st.st_size;
    const bool injected = wt::fault_injected("mmap");
    void *p = injected ? MAP_FAILED : mmap(nullptr, f.size, PROT_READ, MAP_SHARED, fd, 0);
    if (p == MAP_FAILED) rc = set_err(WT_EIO, "%s: mmap: %s", f.path.c_str(), injected ? "injected fault" : strerror(errno));
    else f.base = static_cast<uint8_t *>(p);
    f.map_ns = now_ns() - t1;
  }
  close(fd);  // Algorithm 1: the mapping outlives the descriptor
  return rc;
}

void prefault(const uint8_t *p, size_t n) {
  if (n == 0) return;
  const uintptr_t pg = (uintptr_t)sysconf(_SC_PAGESIZE);
  const uintptr_t a = reinterpret_cast<uintptr_t>(p) & ~(pg - 1);
  const uintptr_t b = (reinterpret_cast<uintptr_t>(p) + n + pg - 1) & ~(pg - 1);
  if (madvise(reinterpret_cast<void *>(a), b - a, MADV_POPULATE_READ) != 0) {
    // older kernels: touch one byte per page
    volatile uint8_t sink = 0;
    for (uintptr_t q = a; q < b; q += pg) sink ^= *reinterpret_cast<const volatile uint8_t *>(q);
    (void)sink;
  }
}

std::vector<bool> g_prepared(64, false);
std::mutex g_prep_mu;

int prepare_device(int dev) {
  std::lock_guard<std::mutex> g(g_prep_mu);
  if (dev < 0 || dev >= 64) return set_err(WT_ECUDA, "device index %d out of range", dev);
  if (!g_prepared[dev]) {
    CU(wt::gemv_prepare());
    CU(wt::gemm_cols_prepare());
    CU(wt::gemm_cols_umma_prepare());
    CU(wt::gemm_q8_rows_prepare());
    g_prepared[dev] = true;
  }
  return WT_OK;
}

// Mappings never overlap, so sorted by start, a range [a, b) meets a mapping iff it meets the
// last mapping starting before b.
bool inside_mapping(const wt_handle *h, const void *p, uint64_t n) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p), b = a + (n ? n : 1);
  auto it = std::lower_bound(h->by_base.begin(), h->by_base.end(), std::make_pair(b, (uint32_t)0));
  if (it == h->by_base.begin()) return false;
  const File &f = h->files[std::prev(it)->second];
  const uintptr_t s = reinterpret_cast<uintptr_t>(f.base), e = s + f.size;
  return a < e && b > s;
}

int new_event(wt_handle *h, cudaEvent_t *ev) {
  CU(ev_create(ev, h->timeline ? cudaEventDefault : cudaEventDisableTiming));
  std::lock_guard<std::mutex> g(h->ev_mu);
  h->events.push_back(*ev);
  return WT_OK;
}

// A timing event recorded on s now, kept for wt_trace (WT_OPEN_TIMELINE handles only).
int trace_mark(cudaStream_t s, cudaEvent_t *ev) {
  CU(ev_create(ev, cudaEventDefault));
  const cudaError_t e = cudaEventRecord(*ev, s);
  if (e != cudaSuccess) {
    ev_destroy(*ev);
    *ev = nullptr;
    return cuda_err(e, "cudaEventRecord (timeline)");
  }
  return WT_OK;
}

void trace_push(wt_handle *h, const wt_handle::TraceEv &t) {
  std::lock_guard<std::mutex> g(h->ev_mu);
  h->trace.push_back(t);
}

// ------------------------------------------------------------------ adopt
struct Range {
  size_t tensor;  // position in the caller's list
  uint32_t file;  // file index and byte offset of the source (pread of WT_OPEN_NOMAP files)
  uint64_t foff;
  const uint8_t *src_host;  // nullptr for a WT_OPEN_NOMAP file
  const uint8_t *src_dev;
  uint8_t *dst;
  uint64_t n;
  bool populated;  // source page-table entries already filled
};

// One process-wide thread fills page tables ahead of the ingest launches (MADV_POPULATE_READ
// on the mapped sources of batch after batch).  A thread of its own per wt_adopt call cost a
// spawn and a join on every call; one thread for all of them keeps the populate calls from
// contending on the address-space lock, which made the many-small checkpoint's adopt three
// times slower when the whole host pool populated (6.6 -> 20 ms for 2506 files).
class Populator {
 public:
  Populator() : th_([this] { run(); }) {}
  ~Populator() {
    {
      std::lock_guard<std::mutex> g(mu_);
      stop_ = true;
    }
    cv_.notify_all();
    th_.join();
  }
  // Queues job for the thread and returns its ticket; the caller must wait(ticket) before
  // anything the job refers to goes away.
  uint64_t post(std::function<void()> job) {
    std::lock_guard<std::mutex> g(mu_);
    q_.push_back(std::move(job));
    cv_.notify_all();
    return ++posted_;
  }
  void wait(uint64_t ticket) {
    std::unique_lock<std::mutex> lk(mu_);
    done_cv_.wait(lk, [&] { return done_ >= ticket; });
  }

 private:
  void run() {
    for (;;) {
      std::function<void()> job;
      {
        std::unique_lock<std::mutex> lk(mu_);
        cv_.wait(lk, [&] { return stop_ || !q_.empty(); });
        if (q_.empty()) return;
        job = std::move(q_.front());
        q_.pop_front();
      }
      job();
      {
        std::lock_guard<std::mutex> g(mu_);
        ++done_;
      }
      done_cv_.notify_all();
    }
  }
  std::mutex mu_;
  std::condition_variable cv_, done_cv_;
  std::deque<std::function<void()>> q_;
  uint64_t posted_ = 0, done_ = 0;
  bool stop_ = false;
  std::thread th_;
};

Populator &populator() {
  static Populator p;
  return p;
}

int adopt_device(wt_handle *h, const std::vector<Range> &rs, unsigned mode, cudaStream_t s,
                 void **ready) {
  // Batches of 256 MiB: each batch is one gather launch and one event, and a gather kernel's
  // ramp and tail idle part of the link (a 64 MiB batch ran at a median 204 GB/s of the
  // link's 210, a 128 MiB one at 207).  Callers that allocate segment by segment make several
  // smaller calls, which keep full batches too.  Measured with the allocation inside the run:
  // batches of at least 2 MiB -> 64 MiB took the mid decoder from 188 to 194 GB/s; 64 -> 128
  // MiB the large decoder from 197.9 to 198.6 and the mid decoder from 195.5 to 196.8 GB/s;
  // 128 -> 256 MiB the large decoder from 198.3 to 199.9 and the mid from 196.6 to 197.9 GB/s,
  // with many-small unchanged.
  const uint64_t target = 256ull << 20;
  // When the stream has nothing in flight the link is idle until the first batch lands, and
  // that batch waits for its own page tables first: batches then start at 4 MiB and double up
  // to the target, so the first launch follows the population of 4 MiB instead of 64.  A call
  // that finds its stream busy (a later segment of a first use) keeps full batches.
  const cudaError_t q = cudaStreamQuery(s);
  if (q != cudaSuccess && q != cudaErrorNotReady) cudaGetLastError();
  uint64_t cap = q == cudaSuccess ? std::min<uint64_t>(target, 4ull << 20) : target;
  // One gather CTA per SM: the link runs at 207 GB/s with 2, 1 or a third of a CTA per SM.
  // An event-gated GEMV group shares the SMs with the next batch's gather and advances at
  // about the gather's pace (a 200 MB group in ~1 ms instead of ~30 us alone); 48 or 64
  // gather CTAs leave it almost untouched, but file -> first use measured 86-97 ms with
  // them against 78 ms here, so the link-bound whole keeps the wide grid.
  const int grid_cap = wt::num_sms();
  // Ranges are cut into pieces that fill each batch to its size (cuts at multiples of 64 KiB
  // from the range's start, so each piece keeps its range's alignment): page-table population
  // and transfer then pipeline inside a large tensor.  A tensor's event is the event of the
  // batch holding its last piece.
  std::vector<Range> ps;
  ps.reserve(rs.size());
  std::vector<std::pair<size_t, size_t>> batches;
  size_t b0 = 0;
  uint64_t bbytes = 0;
  for (const Range &r : rs) {
    uint64_t o = 0;
    do {
      if (ps.size() > b0 && (bbytes >= cap || ps.size() - b0 >= (size_t)wt::kMaxGather)) {
        batches.push_back({b0, ps.size()});
        b0 = ps.size();
        bbytes = 0;
        cap = std::min<uint64_t>(target, cap * 2);
      }
      uint64_t take = r.n - o;
      if (take > cap - bbytes) take = std::min(take, std::max<uint64_t>((cap - bbytes) & ~((1ull << 16) - 1), 1ull << 16));
      ps.push_back({r.tensor, r.file, r.foff + o, r.src_host ? r.src_host + o : nullptr,
                    r.src_dev ? r.src_dev + o : nullptr, r.dst + o, take, r.populated});
      bbytes += take;
      o += take;
    } while (o < r.n);
  }
  if (ps.size() > b0) batches.push_back({b0, ps.size()});
  // The populator fills the page-table entries of batch after batch; batch b is enqueued once
  // its sources are populated, so this host work (about 1 TB/s for large ranges, a few
  // microseconds per small mapping) overlaps the transfer of earlier batches.
  std::vector<std::vector<std::pair<const uint8_t *, size_t>>> work(batches.size());
  bool any = false;
  for (size_t b = 0; b < batches.size(); ++b)
    for (size_t k = batches[b].first; k < batches[b].second; ++k)
      if (!ps[k].populated && ps[k].src_host)
        for (uint64_t o = 0; o < ps[k].n; o += 16ull << 20) {
          work[b].push_back({ps[k].src_host + o, (size_t)std::min<uint64_t>(16ull << 20, ps[k].n - o)});
          any = true;
        }
  std::mutex mu;
  std::condition_variable cv;
  size_t populated = any ? 0 : batches.size();
  std::atomic<bool> stop{false};
  uint64_t ticket = 0;
  if (any) {
    // the first batch is populated here, on the calling thread: its launch then waits for no
    // handoff to the populator and back; the populator starts at the second batch meanwhile
    for (const auto &w : work[0]) prefault(w.first, w.second);
    populated = 1;
  }
  if (any && batches.size() > 1) {
    ticket = populator().post([&] {
      for (size_t b = 1; b < batches.size() && !stop.load(); ++b) {
        for (const auto &w : work[b]) prefault(w.first, w.second);
        {
          std::lock_guard<std::mutex> g(mu);
          populated = b + 1;
        }
        cv.notify_one();
      }
    });
  }
  struct Joiner {  // the job refers to this frame: wait for it on every way out
    uint64_t ticket;
    std::atomic<bool> &stop;
    ~Joiner() {
      stop.store(true);
      if (ticket) populator().wait(ticket);
    }
  } joiner{ticket, stop};
  for (size_t b = 0; b < batches.size(); ++b) {
    if (any) {
      std::unique_lock<std::mutex> lk(mu);
      cv.wait(lk, [&] { return populated > b; });
    }
    const size_t i = batches[b].first, j = batches[b].second;
    cudaEvent_t tb = nullptr;
    if (h->timeline) {
      int rc = trace_mark(s, &tb);
      if (rc) return rc;
    }
    if (mode == WT_ADOPT_GATHER) {
      wt::GatherBatch gb;
      memset(&gb, 0, sizeof gb);
      uint64_t chunks = 0;
      for (size_t k = i; k < j; ++k) {
        const uint32_t q = gb.n++;
        gb.chunk_prefix[q] = chunks;
        gb.src[q] = ps[k].src_dev;
        gb.dst[q] = ps[k].dst;
        gb.nbytes[q] = ps[k].n;
        chunks += (ps[k].n + (1ull << wt::kGatherChunkLog2) - 1) >> wt::kGatherChunkLog2;
      }
      gb.chunk_prefix[gb.n] = chunks;
      if (chunks) {
        CU(wt::launch_gather(gb, (int)std::min<uint64_t>(chunks, (uint64_t)grid_cap), s));
        h->kernel_launches++;
      }
    } else {
      for (size_t k = i; k < j; ++k)
        if (ps[k].n) CU(cudaMemcpyAsync(ps[k].dst, ps[k].src_dev, ps[k].n, cudaMemcpyDefault, s));
    }
    cudaEvent_t ev;
    int rc = new_event(h, &ev);
    if (rc) {
      if (tb) ev_destroy(tb);
      return rc;
    }
    CU(cudaEventRecord(ev, s));
    for (size_t k = i; k < j; ++k) ready[ps[k].tensor] = ev;
    const uint64_t bi = h->n_batches++;
    if (tb) {
      uint64_t bytes = 0;
      for (size_t k = i; k < j; ++k) bytes += ps[k].n;
      trace_push(h, {WT_TRACE_INGEST, bi, bytes, tb, ev, false, ev});
    }
  }
  return WT_OK;
}

int ring_setup(Ring &R) {
  if (R.ready) return WT_OK;
  for (int k = 0; k < Ring::kSlots; ++k) {
    if (!R.slot[k]) CU(pinned_alloc(reinterpret_cast<void **>(&R.slot[k]), Ring::kSlotBytes));
    if (!R.done[k]) CU(ev_create(&R.done[k], cudaEventDisableTiming));
  }
  if (!R.stream) CU(cudaStreamCreateWithFlags(&R.stream, cudaStreamNonBlocking));
  R.ready = true;
  return WT_OK;
}

// Opens a WT_OPEN_NOMAP file again for a staged adopt and checks it is the file wt_open
// parsed (same device, inode, size and modification time).  Returns the fd or -1.
int reopen_checked(const File &f) {
  if (wt::fault_injected("open")) {
    set_err(WT_EIO, "%s: open: injected fault", f.path.c_str());
    return -1;
  }
  const int fd = open(f.path.c_str(), O_RDONLY | O_CLOEXEC);
  if (fd < 0) {
    set_err(WT_EIO, "%s: open: %s", f.path.c_str(), strerror(errno));
    return -1;
  }
  struct stat st;
  if (fstat(fd, &st) != 0 || (uint64_t)st.st_dev != f.st_dev || (uint64_t)st.st_ino != f.st_ino ||
      (size_t)st.st_size != f.size ||
      (int64_t)st.st_mtim.tv_sec * 1000000000ll + st.st_mtim.tv_nsec != f.mtime_ns) {
    close(fd);
    set_err(WT_EIO, "%s: the file changed since wt_open", f.path.c_str());
    return -1;
  }
  return fd;
}

// The staged half of a mixed adopt runs on the ring's own stream, after `after` (an event
// recorded on the caller's stream).
struct StagedJoin {
  cudaEvent_t after = nullptr;
};

// Staged: page cache -> pinned slot (host threads: memcpy from the mapping, or pread for a
// WT_OPEN_NOMAP file, which then needs no mapping at all) -> HBM (the gather kernel reading
// the pinned slot over the host link: one launch per up to kMaxGather pieces, so a slot of many
// small tensors costs one or two launches instead of one copy call per tensor).
int adopt_staged(wt_handle *h, const std::vector<Range> &rs, cudaStream_t s, void **ready,
                 StagedJoin *join = nullptr) {
  Ring &R = g_ring[h->device];
  std::lock_guard<std::mutex> ring_lock(R.mu);
  int rc = ring_setup(R);
  if (rc) return rc;
  if (join) {
    s = R.stream;
    CU(cudaStreamWaitEvent(s, join->after, 0));
  }
  // descriptors of the unmapped files this call reads, opened in parallel and closed on return
  std::vector<int> fds(h->files.size(), -1);
  std::vector<uint32_t> need;
  {
    std::vector<char> seen(h->files.size(), 0);
    for (const Range &r : rs)
      if (!r.src_host && r.n && !seen[r.file]) {
        seen[r.file] = 1;
        need.push_back(r.file);
      }
  }
  struct Closer {
    std::vector<int> &fds;
    ~Closer() {
      for (int fd : fds)
        if (fd >= 0) close(fd);
    }
  } closer{fds};
  Pool &pool = host_pool();
  if (!need.empty()) {
    std::vector<std::string> errs(need.size());
    std::atomic<bool> bad{false};
    pool.parallel_for(need.size(), [&](size_t k) {
      fds[need[k]] = reopen_checked(h->files[need[k]]);
      if (fds[need[k]] < 0) {
        errs[k] = t_err;
        bad = true;
      }
    });
    if (bad)
      for (const std::string &e : errs)
        if (!e.empty()) return set_err(WT_EIO, "wt_adopt: %s", e.c_str());
  }
  struct PieceCopy {
    const Range *r;
    uint64_t roff;  // offset in the range
    size_t off;     // in slot (16-byte aligned)
    size_t n;
  };
  size_t r = 0;
  uint64_t roff = 0;
  while (r < rs.size()) {
    const int slot = R.next;
    R.next = (R.next + 1) % Ring::kSlots;
    if (R.used[slot]) CU(cudaEventSynchronize(R.done[slot]));
    uint8_t *buf = R.slot[slot];
    std::vector<PieceCopy> pcs;
    std::vector<size_t> finished;  // tensors whose last byte is in this slot
    size_t fill = 0;
    while (r < rs.size() && fill < Ring::kSlotBytes) {
      const uint64_t take = std::min<uint64_t>(rs[r].n - roff, Ring::kSlotBytes - fill);
      if (take) pcs.push_back({&rs[r], roff, fill, (size_t)take});
      fill = (fill + take + 63) & ~(size_t)63;  // next piece 64-byte aligned in the slot
      roff += take;
      if (roff == rs[r].n) {
        finished.push_back(rs[r].tensor);
        ++r;
        roff = 0;
      }
    }
    // host copy in pieces of at most 4 MiB across the pool
    std::vector<std::pair<size_t, size_t>> work;  // (piece, sub-offset)
    constexpr size_t kSub = 4u << 20;
    for (size_t p = 0; p < pcs.size(); ++p)
      for (size_t o = 0; o < pcs[p].n; o += kSub) work.push_back({p, o});
    std::atomic<int> io_err{0};
    std::vector<std::string> io_msg(1);
    std::mutex io_mu;
    pool.parallel_for(work.size(), [&](size_t w) {
      const PieceCopy &pc = pcs[work[w].first];
      const size_t o = work[w].second, len = std::min(kSub, pc.n - o);
      uint8_t *dst = buf + pc.off + o;
      if (pc.r->src_host) {
        memcpy(dst, pc.r->src_host + pc.roff + o, len);
        return;
      }
      const int fd = fds[pc.r->file];
      size_t got = 0;
      const bool injected = wt::fault_injected("pread");
      while (!injected && got < len) {
        const ssize_t k = pread(fd, dst + got, len - got, (off_t)(pc.r->foff + pc.roff + o + got));
        if (k <= 0) {
          if (k < 0 && errno == EINTR) continue;
          break;
        }
        got += (size_t)k;
      }
      if (got != len && io_err.exchange(1) == 0) {
        std::lock_guard<std::mutex> g(io_mu);
        io_msg[0] = h->files[pc.r->file].path + (injected ? ": pread: injected fault" : ": pread: short read");
      }
    });
    if (io_err) return set_err(WT_EIO, "wt_adopt: %s", io_msg[0].c_str());
    cudaEvent_t tb = nullptr;
    if (h->timeline) {
      rc = trace_mark(s, &tb);
      if (rc) return rc;
    }
    for (size_t i = 0; i < pcs.size();) {
      wt::GatherBatch gb;
      memset(&gb, 0, sizeof gb);
      uint64_t chunks = 0;
      for (; i < pcs.size() && gb.n < (uint32_t)wt::kMaxGather; ++i) {
        const uint32_t q = gb.n++;
        gb.chunk_prefix[q] = chunks;
        gb.src[q] = buf + pcs[i].off;
        gb.dst[q] = pcs[i].r->dst + pcs[i].roff;
        gb.nbytes[q] = pcs[i].n;
        chunks += (pcs[i].n + (1ull << wt::kGatherChunkLog2) - 1) >> wt::kGatherChunkLog2;
      }
      gb.chunk_prefix[gb.n] = chunks;
      if (chunks) {
        CU(wt::launch_gather(gb, (int)std::min<uint64_t>(chunks, (uint64_t)wt::num_sms()), s));
        h->kernel_launches++;
      }
    }
    CU(cudaEventRecord(R.done[slot], s));
    R.used[slot] = true;
    cudaEvent_t ev = nullptr;
    if (!finished.empty()) {
      rc = new_event(h, &ev);
      if (rc) {
        if (tb) ev_destroy(tb);
        return rc;
      }
      CU(cudaEventRecord(ev, s));
      for (size_t t : finished) ready[t] = ev;
    }
    if (tb) {
      cudaEvent_t te = nullptr;
      rc = trace_mark(s, &te);
      if (rc) {
        ev_destroy(tb);
        return rc;
      }
      uint64_t bytes = 0;
      for (const PieceCopy &pc : pcs) bytes += pc.n;
      trace_push(h, {WT_TRACE_INGEST, h->n_batches++, bytes, tb, te, true, ev});
    } else {
      h->n_batches++;
    }
  }
  return WT_OK;
}

// A GATHER or CE adopt over a WT_OPEN_MAP_LARGE handle whose call holds both mapped files
// (`dv`, through the device route) and small unmapped ones (`st`, through the pinned ring):
// the staged half runs on a helper thread and the ring's stream, ordered after the caller's
// earlier work on `s`, while this thread enqueues the mapped half on `s`; `s` then waits
// for whatever the staged half enqueued, on success and on failure alike, so the call keeps
// its stream semantics (later work on `s` never overlaps a copy of this call).
int adopt_mixed(wt_handle *h, const std::vector<Range> &dv, const std::vector<Range> &st, unsigned mode,
                cudaStream_t s, void **ready) {
  StagedJoin join;
  int rc = new_event(h, &join.after);
  if (rc) return rc;
  CU(cudaEventRecord(join.after, s));
  int rc_st = WT_OK;
  std::string err_st;
  struct Joiner {
    std::thread t;
    ~Joiner() {
      if (t.joinable()) t.join();
    }
  } helper;
  helper.t = std::thread([&] {
    const cudaError_t e = cudaSetDevice(h->device);
    rc_st = e == cudaSuccess ? adopt_staged(h, st, s, ready, &join) : cuda_err(e, "cudaSetDevice");
    if (rc_st) err_st = t_err;
  });
  rc = adopt_device(h, dv, mode, s, ready);
  helper.t.join();
  // The ring's stream is created once and never replaced, so it can be read here without
  // the ring's lock; an event on it now follows every copy the staged half enqueued (and
  // possibly later ones of other calls, which only adds order).
  if (const cudaStream_t rs = g_ring[h->device].stream) {
    cudaEvent_t done = nullptr;
    int rc_j = new_event(h, &done);
    if (rc_j == WT_OK) {
      cudaError_t e = cudaEventRecord(done, rs);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(s, done, 0);
      if (e != cudaSuccess) rc_j = cuda_err(e, "wt_adopt: joining the staged half");
    }
    if (rc_j && !rc && !rc_st) return rc_j;
  }
  if (rc) return rc;
  if (rc_st) return set_err(rc_st, "%s", err_st.c_str());
  return WT_OK;
}

// ------------------------------------------------------------------ GEMV planning
uint32_t pow2ceil(uint32_t v) {
  uint32_t p = 1;
  while (p < v) p <<= 1;
  return p;
}

wt::MatDesc make_mat(const wt_gemv_desc &d) {
  wt::MatDesc m;
  memset(&m, 0, sizeof m);
  const int es = elem_bytes(d.dtype);
  m.W = static_cast<const uint8_t *>(d.W);
  m.x = static_cast<const uint8_t *>(d.x);
  m.y = d.y;
  m.s = static_cast<const uint8_t *>(d.scale);
  m.M = (uint32_t)d.M;
  m.V = (uint32_t)(d.K * es / 16);
  m.rs = m.V;
  const uint32_t rowb = m.V * 16;
  // a consumer thread keeps at most 8 (bf16/f16/f32) or 2 (int8: 16 f16 activations per
  // weight vector, two CTAs per SM) x vectors in registers; the mode limits follow from that
  const uint32_t xj = d.dtype == WT_I8 ? 2 : 8;
  if (m.V <= 32 * xj) {
    m.mode = wt::kModeWarpRows;
    m.G = (uint16_t)(m.V <= 32 ? pow2ceil(m.V) : 32);
    m.rt = wt::kStageBytes / rowb;
    m.vc = m.V;
  } else if (rowb <= (uint32_t)wt::kStageBytes && m.V <= 256 * xj) {
    m.mode = wt::kModeBlockRows;
    m.rt = std::min<uint32_t>(wt::kRowBlock, wt::kStageBytes / rowb);
    m.vc = m.V;
  } else {
    // the plain-load kernels read such rows directly; the TMA kernel gets them only as
    // column segments of at most seg_vectors vectors (make_seg_mat)
    m.mode = wt::kModeLongRows;
    m.rt = 1;
    m.vc = m.V;
  }
  return m;
}

// Multi-column kernel: chunks of at most kColVecMax vectors per row, evened out over the row
// and rounded up to 4 (mod 8): 448 vectors -> 5 chunks of 92 (the last box zero-filled past
// the row's end).
wt::MatDesc make_cols_mat(const wt_gemv_desc &d) {
  wt::MatDesc m;
  memset(&m, 0, sizeof m);
  m.W = static_cast<const uint8_t *>(d.W);
  m.x = static_cast<const uint8_t *>(d.x);
  m.y = d.y;
  m.s = static_cast<const uint8_t *>(d.scale);
  m.M = (uint32_t)d.M;
  m.V = (uint32_t)(d.K * elem_bytes(d.dtype) / 16);
  m.rs = m.V;
  m.mode = wt::kModeCols;
  m.G = (uint16_t)d.cols;
  m.rt = 16;
  const uint32_t nchunk = (m.V + wt::kColVecMax - 1) / wt::kColVecMax;
  m.vc = ((m.V + nchunk - 1) / nchunk + 3) / 8 * 8 + 4;
  return m;
}

// Segment length for rows of V vectors: ceil(V / seg_vectors) segments of nearly equal
// length (a multiple of 8 vectors), so no segment is a sliver.  Depends on (V, dtype) only.
uint32_t seg_length(uint32_t V, int dtype) {
  const uint32_t S = wt::seg_vectors(dtype);
  const uint32_t nseg = (V + S - 1) / S;
  return ((V + nseg - 1) / nseg + 7) / 8 * 8;
}

// Column segment k of a matrix whose rows exceed seg_vectors(dtype): vectors
// [k S, min((k + 1) S, V)) of every row, S = seg_length (row pitch: the full row), x
// advanced to match, no scale, tile mode chosen by the segment's own length, y left for the
// workspace patch.
wt::MatDesc make_seg_mat(const wt_gemv_desc &d, uint32_t k) {
  const int es = elem_bytes(d.dtype);
  const uint32_t V = (uint32_t)(d.K * es / 16);
  const uint32_t S = seg_length(V, d.dtype);
  const uint64_t xvb = d.dtype == WT_I8 ? 32 : 16;  // x bytes per 16-byte weight vector
  const uint32_t v0 = k * S;
  wt_gemv_desc sd = d;
  sd.W = static_cast<const uint8_t *>(d.W) + (uint64_t)v0 * 16;
  sd.x = static_cast<const uint8_t *>(d.x) + (uint64_t)v0 * xvb;
  sd.K = (uint64_t)std::min(S, V - v0) * 16 / es;
  sd.scale = nullptr;
  wt::MatDesc m = make_mat(sd);
  m.s = nullptr;
  m.rs = V;
  return m;
}

// cuTensorMapEncodeTiled, looked up once through the runtime (no link against libcuda).
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// The tensor map of a multi-column matrix: W as [M rows, 2V] 8-byte elements (row pitch
// V * 16 bytes), box {2 vc, kColTileRows}, no swizzle, zero fill outside the matrix.
int encode_cols_map(const wt::MatDesc &m, uint8_t *out) {
  static_assert(sizeof(CUtensorMap) == wt::kTensorMapBytes, "tensor map size");
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return set_err(WT_ECUDA, "wt_pass: cuTensorMapEncodeTiled is not available from the driver");
  const cuuint64_t dims[2] = {(cuuint64_t)m.V * 2, (cuuint64_t)m.M};
  const cuuint64_t strides[1] = {(cuuint64_t)m.V * 16};
  const cuuint32_t box[2] = {m.vc * 2, (cuuint32_t)wt::kColTileRows};
  const cuuint32_t estr[2] = {1, 1};
  CUtensorMap map;
  const CUresult r = fn(&map, CU_TENSOR_MAP_DATA_TYPE_UINT64, 2, const_cast<uint8_t *>(m.W), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return set_err(WT_ECUDA, "wt_pass: cuTensorMapEncodeTiled failed (%d) for a %u x %u-vector matrix", (int)r, m.M, m.V);
  memcpy(out, &map, sizeof map);
  return WT_OK;
}

// Interleaved slices per CTA for the one-column kernels.  Byte-equal contiguous ranges leave
// CTAs with different mixes of shapes, and shapes stream at different rates (a decoder's
// k/v rows at ~92 % of the copy peak, its down rows above it): the slowest CTA sets the pass.
// Sixteen slices spread over the whole set even that out (large decoder 6342 -> 6864 GB/s).
// int8 weights keep one range per CTA: they are bound by instructions, and each extra piece
// costs an exposed reload of x.
int one_col_slices(int dtype) { return dtype == WT_I8 ? 1 : 16; }

// Which multi-column kernel runs a matrix: tcgen05 (wt_umma.cu) for 2-byte weights with more
// than 8 columns, where its T-independent tensor time wins (bf16 protocol, T = 16: 6529
// against 6370 GB/s); the warp-level MMA kernel (wt_cols.cu) otherwise (T = 1: 6958 against
// 6580; int8 decodes in registers there).  WT_COLS_KERNEL=mma or =umma forces one kernel
// (umma still only for 2-byte weights).
bool cols_on_umma(int dtype, int cols) {
  const char *e = getenv("WT_COLS_KERNEL");
  const int force = e && strcmp(e, "umma") == 0 ? 1 : e && strcmp(e, "mma") == 0 ? 2 : 0;
  if (dtype != WT_BF16 && dtype != WT_F16) return false;
  return force == 1 || (force == 0 && cols > 8);
}

// int8 weights on the tensor cores (T columns, and one column with rows up to K = 8192) run
// the row-owner kernel (wt_q8rows.cu) when its 128-row blocks fill the GPU (at least two per
// CTA slot over the launch): its warps keep no activation registers and meet in no reduction.
// The matched protocol: T = 1 / 8 / 16 at 6663 / 6581 / 6502 GB/s against 6565 / 6250 / 5004
// on the warp-MMA kernel.  Launches of fewer rows keep the warp-MMA kernel's 16-row tiles,
// which spread over 8 times as many CTAs.  WT_COLS_KERNEL=mma or =q8rows forces one kernel
// for every int8 matrix (the parity tests run each routing).
bool i8_on_q8rows(uint64_t blocks) {
  const char *e = getenv("WT_COLS_KERNEL");
  if (e && strcmp(e, "mma") == 0) return false;
  if (e && strcmp(e, "q8rows") == 0) return true;
  return blocks >= 2ull * wt::num_sms();
}

// The two tensor maps of a row-owner int8 matrix (see wt::launch_gemm_q8_rows).
int encode_q8rows_maps(const wt::MatDesc &m, uint8_t *out) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return set_err(WT_ECUDA, "wt_pass: cuTensorMapEncodeTiled is not available from the driver");
  const uint64_t K = (uint64_t)m.V * 16;
  CUtensorMap mw, mx;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)m.M};
    const cuuint64_t strides[1] = {(cuuint64_t)K};
    const cuuint32_t box[2] = {192, (cuuint32_t)wt::kQ8RowsBlock};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(&mw, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(m.W), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_err(WT_ECUDA, "wt_pass: tensor map of int8 W failed (%d)", (int)r);
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)m.G};
    const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    const cuuint32_t box[2] = {64, 16};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(&mx, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<uint8_t *>(m.x), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_err(WT_ECUDA, "wt_pass: tensor map of fp16 X failed (%d)", (int)r);
  }
  memcpy(out, &mw, sizeof mw);
  memcpy(out + wt::kTensorMapBytes, &mx, sizeof mx);
  return WT_OK;
}

// int8 weights with one activation column go to the tensor-core kernels at T = 1: the CUDA-core
// kernel is issue-bound (ncu: 66.5 % issue active, not_selected on top), while the MMA paths
// decode a 16-byte vector straight into an MMA operand with 1.6x fewer instructions (matched
// protocol: 6386 GB/s on CUDA cores, 6565 on the warp-MMA kernel, 6663 on the row-owner
// kernel).  They take rows up to seg_vectors(int8) vectors (K <= 8192); longer rows keep the
// CUDA-core kernel's cross-CTA split-K, since the MMA kernels give a whole row to one CTA.
// WT_I8_ONECOL=cuda keeps every int8 one-column matrix on the CUDA-core kernel (its parity
// tests run both ways).
bool i8_onecol_on_mma(uint32_t V) {
  const char *e = getenv("WT_I8_ONECOL");
  if (e && strcmp(e, "cuda") == 0) return false;
  return V <= wt::seg_vectors(WT_I8);
}

// The two tensor maps of a tcgen05 multi-column matrix (2-byte weights; see wt::UmmaLaunch).
int encode_umma_maps(const wt::MatDesc &m, uint8_t *out) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return set_err(WT_ECUDA, "wt_pass: cuTensorMapEncodeTiled is not available from the driver");
  const uint64_t K = (uint64_t)m.V * 8;
  CUtensorMap mw, mx;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)m.M};
    const cuuint64_t strides[1] = {(cuuint64_t)m.V * 16};
    const cuuint32_t box[2] = {64, 128};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(&mw, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<uint8_t *>(m.W), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_err(WT_ECUDA, "wt_pass: tensor map of W failed (%d)", (int)r);
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)m.G};
    const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    const cuuint32_t box[2] = {64, 16};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(&mx, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<uint8_t *>(m.x), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_err(WT_ECUDA, "wt_pass: tensor map of X failed (%d)", (int)r);
  }
  memcpy(out, &mw, sizeof mw);
  memcpy(out + wt::kTensorMapBytes, &mx, sizeof mx);
  return WT_OK;
}

// Split the rows of `mats` (in order) into grid * slices contiguous slices of nearly
// equal bytes, cut at row boundaries; slice j goes to CTA j % grid, so every CTA streams
// `slices` slices spread over the whole set and gets a similar mix of shapes.  The grid is
// at most ctas_per_sm CTAs per SM (all resident at once: the launch is persistent).
void partition(const std::vector<wt::MatDesc> &mats, int &grid, std::vector<wt::Piece> &pieces,
               std::vector<uint32_t> &begin, uint32_t row_align = 1, int slices = 1, int ctas_per_sm = 1) {
  uint64_t B = 0;
  std::vector<uint64_t> start(mats.size() + 1, 0);
  for (size_t i = 0; i < mats.size(); ++i) {
    start[i] = B;
    B += (uint64_t)mats[i].M * mats[i].V * 16;
  }
  start[mats.size()] = B;
  constexpr uint64_t kMinCtaBytes = 64 << 10;
  grid = (int)std::max<uint64_t>(
      1, std::min<uint64_t>((uint64_t)wt::num_sms() * ctas_per_sm, (B + kMinCtaBytes - 1) / kMinCtaBytes));
  // slices of at least 2 MiB: a slice costs the consumers a reload of x, and a slice shorter
  // than a tile makes its stages partial.  WT_MIN_SLICE_BYTES (>= 4096) lowers the floor so
  // that tests reach the many-slices-per-CTA partition on sets far smaller than a decoder.
  uint64_t min_slice = 2ull << 20;
  if (const char *e = getenv("WT_MIN_SLICE_BYTES")) {
    const uint64_t v = strtoull(e, nullptr, 10);
    if (v >= 4096) min_slice = v;
  }
  slices = (int)std::max<uint64_t>(1, std::min<uint64_t>((uint64_t)slices, B / ((uint64_t)grid * min_slice)));
  const int nslice = grid * slices;
  // cut c (1..nslice-1) at the row boundary nearest byte B*c/nslice
  std::vector<std::pair<uint32_t, uint32_t>> cuts;  // (mat, row)
  cuts.push_back({0, 0});
  size_t m = 0;
  for (int c = 1; c < nslice; ++c) {
    const uint64_t T = (uint64_t)((unsigned __int128)B * c / nslice);
    while (m + 1 < mats.size() && start[m + 1] <= T) ++m;
    const uint64_t rb = (uint64_t)mats[m].V * 16;
    uint64_t row = (T - start[m] + rb / 2) / rb;
    row = (row + row_align / 2) / row_align * row_align;  // whole tiles per slice
    std::pair<uint32_t, uint32_t> cut = {(uint32_t)m, (uint32_t)std::min<uint64_t>(row, mats[m].M)};
    if (cut.second == mats[m].M && m + 1 < mats.size()) cut = {(uint32_t)m + 1, 0};
    if (cut < cuts.back()) cut = cuts.back();
    cuts.push_back(cut);
  }
  cuts.push_back({(uint32_t)mats.size(), 0});
  begin.assign(1, 0);
  for (int c = 0; c < grid; ++c) {
    for (int j = c; j < nslice; j += grid) {
      auto a = cuts[j], b = cuts[j + 1];
      while (a < b) {
        const uint32_t rend = a.first == b.first ? b.second : mats[a.first].M;
        if (rend > a.second) pieces.push_back({a.first, a.second, rend, 0});
        if (a.first == b.first) break;
        a = {a.first + 1, 0};
      }
    }
    begin.push_back((uint32_t)pieces.size());
  }
}

size_t align16(size_t v) { return (v + 15) & ~(size_t)15; }

template <class T>
size_t append(std::vector<uint8_t> &tab, const std::vector<T> &v) {
  const size_t off = align16(tab.size());
  tab.resize(off + v.size() * sizeof(T));
  if (!v.empty()) memcpy(tab.data() + off, v.data(), v.size() * sizeof(T));
  return off;
}

int validate_desc(const wt_gemv_desc &d, size_t i) {
  if (d.dtype != WT_F32 && d.dtype != WT_BF16 && d.dtype != WT_F16 && d.dtype != WT_I8)
    return set_err(d.dtype == WT_U8 ? WT_ENOTSUP : WT_EINVAL, "desc %zu: dtype %d has no GEMV", i, d.dtype);
  if (d.dtype == WT_I8 && d.M > 0 && d.K > 0 && d.scale == nullptr)
    return set_err(WT_EINVAL, "desc %zu: int8 weights need fp16 row scales", i);
  if (d.dtype != WT_I8 && d.scale != nullptr) return set_err(WT_EINVAL, "desc %zu: scale is for int8 weights only", i);
  if (d.cols < 0 || d.cols > 16) return set_err(WT_EINVAL, "desc %zu: cols %d outside 0..16", i, (int)d.cols);
  if (d.cols > 0 && d.dtype == WT_F32)
    return set_err(WT_ENOTSUP, "desc %zu: the multi-column kernel takes bf16, f16 or int8 weights", i);
  if (d.M > 0x7fffffffull || d.K > 0x7fffffffull) return set_err(WT_EINVAL, "desc %zu: M or K above 2^31-1", i);
  if (d.M > 0 && d.y == nullptr) return set_err(WT_EINVAL, "desc %zu: null y", i);
  if (d.M > 0 && d.K > 0 && (d.W == nullptr || d.x == nullptr)) return set_err(WT_EINVAL, "desc %zu: null W or x", i);
  return WT_OK;
}

// Bounds of device buffers, checked on the host before anything is enqueued: a range that
// starts in a device allocation must end inside it (cuMemGetAddressRange, looked up once
// through the runtime).  The last allocation seen is cached, so a slab of many tensors costs
// one query.  Host memory (mappings, pinned buffers) cannot be asked and passes; mappings
// have their own checks.
struct RangeCache {
  uintptr_t lo = 0, hi = 0;
};

using AddrRangeFn = CUresult (*)(CUdeviceptr *, size_t *, CUdeviceptr);

AddrRangeFn addr_range_fn() {
  static AddrRangeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<AddrRangeFn>(p);
  });
  return fn;
}

// false only when [p, p + n) starts inside a device allocation and runs past its end
bool device_range_ok(const void *p, uint64_t n, RangeCache &c) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  if (n == 0 || (a >= c.lo && a + n <= c.hi && a + n >= a)) return true;
  AddrRangeFn fn = addr_range_fn();
  CUdeviceptr base = 0;
  size_t size = 0;
  if (!fn || fn(&base, &size, (CUdeviceptr)a) != CUDA_SUCCESS) return true;
  c.lo = (uintptr_t)base;
  c.hi = (uintptr_t)base + size;
  return a + n <= c.hi && a + n >= a;
}

// Where W lives: 0 = device memory (cudaMalloc, a memory pool, managed): the TMA kernels
// stream from there; 1 = host memory the device can load from (pinned or registered, or
// pageable where the device reads through the host page tables); -1 = neither.
int memory_class(const void *p, int device) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return 0;
  if (a.type == cudaMemoryTypeHost) return 1;
  int ats = 0;
  cudaDeviceGetAttribute(&ats, cudaDevAttrPageableMemoryAccessUsesHostPageTables, device);
  return ats ? 1 : -1;
}

// The mapping holding [p, p + n) (whole range inside one file mapping), or nullptr.
const File *mapping_of(const wt_handle *h, const void *p, uint64_t n) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  auto it = std::upper_bound(h->by_base.begin(), h->by_base.end(), std::make_pair(a, UINT32_MAX));
  if (it == h->by_base.begin()) return nullptr;
  const File &f = h->files[std::prev(it)->second];
  const uintptr_t s = reinterpret_cast<uintptr_t>(f.base);
  return (a >= s && a + n <= s + f.size && a + n >= a) ? &f : nullptr;
}

int build_plan(wt_handle *h, const wt_gemv_desc *d, size_t n, Plan *P) {
  // One group per distinct wait_event (no event is a class of its own), in order of first
  // appearance: each GEMV depends on its own event only, so descriptors of batches that
  // interleave (two ingest streams, say) still make one wait and one launch per batch.
  std::vector<std::vector<size_t>> members;
  {
    std::vector<std::pair<uintptr_t, size_t>> seen;  // (event, group), sorted by event
    for (size_t k = 0; k < n; ++k) {
      const uintptr_t e = reinterpret_cast<uintptr_t>(d[k].wait_event);
      auto it = std::lower_bound(seen.begin(), seen.end(), std::make_pair(e, (size_t)0));
      if (it == seen.end() || it->first != e) {
        it = seen.insert(it, {e, members.size()});
        members.emplace_back();
      }
      members[it->second].push_back(k);
    }
  }
  for (const std::vector<size_t> &mem : members) {
    Plan::Group g;
    g.first = mem.front();
    // cols_dt: warp-MMA multi-column with T <= 8, colsw_dt: with 8 < T <= 16
    std::vector<wt::MatDesc> by_dt[4], mapped_dt[4], cols_dt[4], umma_dt[4], mcols_dt[4], colsw_dt[4], q8r_dt[4],
        q8r1_dt[4];  // row-owner int8 launches with two 8-column tiles (T > 8) and with one
    std::vector<wt::MatDesc> i8c[2];  // int8 on the tensor cores, T <= 8 and T > 8: kernel chosen below
    uint64_t i8_blocks = 0;           // their 128-row blocks
    std::vector<int64_t> seg_ws[4];  // per by_dt entry: workspace float offset of its partials, or -1
    std::vector<wt::SegReduce> reds;
    std::vector<size_t> red_ws;      // per reds entry: workspace float offset
    RangeCache rcw, rcx, rcy, rcs;
    for (const size_t k : mem) {
      const wt_gemv_desc &q = d[k];
      if (q.M == 0) continue;
      const int es = elem_bytes(q.dtype);
      {
        // every operand that starts in a device allocation must end inside it
        const uint64_t T = q.cols > 0 ? (uint64_t)q.cols : 1;
        const uint64_t xes = q.dtype == WT_I8 ? 2 : (uint64_t)es;
        if (!device_range_ok(q.y, q.M * T * 4, rcy) || !device_range_ok(q.W, q.M * q.K * es, rcw) ||
            !device_range_ok(q.x, q.K * T * xes, rcx) || (q.scale && !device_range_ok(q.scale, q.M * 2, rcs)))
          return set_err(WT_EINVAL, "wt_pass: an operand of desc %zu runs past the end of its device allocation", k);
      }
      const uint32_t ncol = q.cols > 0 ? (uint32_t)q.cols : 1;
      g.wbytes += q.M * q.K * (uint64_t)es;
      if (q.K == 0) {
        g.zero.push_back({q.y, q.M * ncol});
        continue;
      }
      const bool fast = ((reinterpret_cast<uintptr_t>(q.W) | reinterpret_cast<uintptr_t>(q.x)) & 15) == 0 &&
                        (q.K * es) % 16 == 0;
      const File *f = mapping_of(h, q.W, q.M * q.K * es);
      if (!f && inside_mapping(h, q.W, q.M * q.K * es))
        return set_err(WT_EINVAL, "wt_pass: W of desc %zu straddles the end of a mapping", k);
      if (f) {
        // map endpoint: the kernel reads the mapped rows in place over the host link
        if (f->route == WT_ROUTE_NONE || !f->dev)
          return set_err(WT_ENOTSUP, "wt_pass: W of desc %zu lies in %s, which has no device route", k, f->path.c_str());
        const uint64_t off = reinterpret_cast<const uint8_t *>(q.W) - f->base;
        if (!h->prefaulted && !f->populated) prefault(f->base + off, q.M * q.K * es);
        wt_gemv_desc qd = q;
        qd.W = f->dev + off;
        if (fast && q.cols == 0) {
          mapped_dt[q.dtype].push_back(make_mat(qd));
        } else if (fast && q.dtype != WT_F32) {
          wt::MatDesc m = make_mat(qd);
          m.cols = (uint32_t)q.cols;
          mcols_dt[q.dtype].push_back(m);
        } else {
          g.generic.push_back({q.dtype, static_cast<const uint8_t *>(qd.W), static_cast<const uint8_t *>(q.x), q.y, q.M, q.K,
                               static_cast<const uint8_t *>(q.scale), ncol});
        }
      } else if (const int mc = memory_class(q.W, h->device); mc != 0) {
        if (mc < 0) return set_err(WT_ENOTSUP, "wt_pass: W of desc %zu is host memory this device cannot read", k);
        // host memory outside this handle (another mapping, a file-backed DLPack tensor, a
        // pinned buffer): plain loads only, as for the map endpoint; TMA streams device memory
        if (fast && q.cols == 0) {
          mapped_dt[q.dtype].push_back(make_mat(q));
        } else if (fast && q.dtype != WT_F32) {
          wt::MatDesc m = make_mat(q);
          m.cols = (uint32_t)q.cols;
          mcols_dt[q.dtype].push_back(m);
        } else {
          g.generic.push_back({q.dtype, static_cast<const uint8_t *>(q.W), static_cast<const uint8_t *>(q.x), q.y, q.M, q.K,
                               static_cast<const uint8_t *>(q.scale), ncol});
        }
      } else if (fast && q.cols > 0 && q.dtype == WT_I8) {
        i8c[q.cols > 8 ? 1 : 0].push_back(make_cols_mat(q));
        i8_blocks += (q.M + wt::kQ8RowsBlock - 1) / wt::kQ8RowsBlock;
      } else if (fast && q.cols > 0) {
        (cols_on_umma(q.dtype, q.cols) ? umma_dt : q.cols > 8 ? colsw_dt : cols_dt)[q.dtype].push_back(make_cols_mat(q));
      } else if (fast && q.dtype == WT_I8 && i8_onecol_on_mma((uint32_t)(q.K / 16))) {
        // y[M] is Y[1, M] and x[K] is X[1, K]: the one-column GEMV as a T = 1 tensor-core GEMV
        wt_gemv_desc q1 = q;
        q1.cols = 1;
        i8c[0].push_back(make_cols_mat(q1));
        i8_blocks += (q.M + wt::kQ8RowsBlock - 1) / wt::kQ8RowsBlock;
      } else if (fast && q.K * es / 16 > wt::seg_vectors(q.dtype)) {
        // long rows: column segments spread over CTAs, summed by the second pass
        const uint32_t V = (uint32_t)(q.K * es / 16);
        const uint32_t S = seg_length(V, q.dtype);
        const uint32_t nseg = (V + S - 1) / S;
        const size_t off = P->ws_floats;
        P->ws_floats += (size_t)nseg * q.M;
        for (uint32_t k = 0; k < nseg; ++k) {
          by_dt[q.dtype].push_back(make_seg_mat(q, k));
          seg_ws[q.dtype].push_back((int64_t)(off + (size_t)k * q.M));
        }
        wt::SegReduce r;
        memset(&r, 0, sizeof r);
        r.y = q.y;
        r.s = static_cast<const uint8_t *>(q.scale);
        r.M = (uint32_t)q.M;
        r.nseg = nseg;
        reds.push_back(r);
        red_ws.push_back(off);
        g.reduce_rows = std::max(g.reduce_rows, (uint32_t)q.M);
      } else if (fast) {
        by_dt[q.dtype].push_back(make_mat(q));
        seg_ws[q.dtype].push_back(-1);
      } else {
        g.generic.push_back({q.dtype, static_cast<const uint8_t *>(q.W), static_cast<const uint8_t *>(q.x), q.y, q.M, q.K,
                             static_cast<const uint8_t *>(q.scale), ncol});
      }
    }
    if (!i8c[0].empty() || !i8c[1].empty()) {
      const bool rows = i8_on_q8rows(i8_blocks);
      auto &lo = rows ? q8r1_dt[WT_I8] : cols_dt[WT_I8];
      auto &hi = rows ? q8r_dt[WT_I8] : colsw_dt[WT_I8];
      lo.insert(lo.end(), i8c[0].begin(), i8c[0].end());
      hi.insert(hi.end(), i8c[1].begin(), i8c[1].end());
    }
    for (int pass = 0; pass < 8; ++pass) {
      for (int dt = 0; dt < 4; ++dt) {
        std::vector<wt::MatDesc> &ms = pass == 0   ? by_dt[dt]
                                       : pass == 1 ? mapped_dt[dt]
                                       : pass == 2 ? cols_dt[dt]
                                       : pass == 3 ? umma_dt[dt]
                                       : pass == 4 ? mcols_dt[dt]
                                       : pass == 5 ? colsw_dt[dt]
                                       : pass == 6 ? q8r_dt[dt]
                                                   : q8r1_dt[dt];
        const bool warp_mma = pass == 2 || pass == 5;
        if (ms.empty()) continue;
        Plan::Launch L;
        L.dtype = dt;
        std::vector<wt::Piece> pieces;
        std::vector<uint32_t> begin;
        if (pass == 3) {
          // tcgen05 launch: 128-row tiles, dealt round-robin; two tensor maps per matrix
          L.umma = true;
          uint32_t first = 0;
          for (size_t k = 0; k < ms.size(); ++k) {
            const uint32_t tiles = (ms[k].M + 127) / 128;
            pieces.push_back({(uint32_t)k, first, tiles, 0});
            first += tiles;
          }
          L.nmat = (uint32_t)ms.size();
          L.ntiles = first;
          L.grid = (int)std::max<uint32_t>(1, std::min<uint32_t>((uint32_t)wt::num_sms(), first));
          L.mats = append(P->table, ms);
          L.pieces = append(P->table, pieces);
          L.begin = L.pieces;
          L.maps = (P->table.size() + 127) & ~(size_t)127;
          P->table.resize(L.maps + ms.size() * 2 * wt::kTensorMapBytes);
          for (size_t k = 0; k < ms.size(); ++k) {
            int rc = encode_umma_maps(ms[k], P->table.data() + L.maps + k * 2 * wt::kTensorMapBytes);
            if (rc) return rc;
          }
          g.cols.push_back(L);
          continue;
        }
        if (pass >= 6) {
          // row-owner int8 launch: pieces cut at 128-row blocks, two tensor maps per matrix
          L.q8rows = true;
          L.nt = pass == 6 ? 2 : 1;
          partition(ms, L.grid, pieces, begin, (uint32_t)wt::kQ8RowsBlock, 1, 2);
          L.mats = append(P->table, ms);
          L.pieces = append(P->table, pieces);
          L.begin = append(P->table, begin);
          L.maps = (P->table.size() + 127) & ~(size_t)127;
          P->table.resize(L.maps + ms.size() * 2 * wt::kTensorMapBytes);
          for (size_t k = 0; k < ms.size(); ++k) {
            int rc = encode_q8rows_maps(ms[k], P->table.data() + L.maps + k * 2 * wt::kTensorMapBytes);
            if (rc) return rc;
          }
          g.cols.push_back(L);
          continue;
        }
        if (pass == 0)
          for (const wt::MatDesc &m : ms)
            if (m.mode != wt::kModeWarpRows && m.mode != wt::kModeBlockRows)
              return set_err(WT_ENOTSUP, "wt_pass: internal: a %u-vector row reached the TMA kernel unsegmented", m.V);
        L.nt = pass == 2 ? 1 : pass == 5 ? 2 : 0;
        partition(ms, L.grid, pieces, begin, warp_mma ? (uint32_t)wt::kColTileRows : 1u,
                  pass == 0 ? one_col_slices(dt) : 1,
                  pass == 0 ? wt::gemv_ctas_per_sm(dt) : warp_mma ? wt::gemm_cols_ctas_per_sm(dt, L.nt) : 1);
        L.mapped_cols = pass == 4;
        L.mats = append(P->table, ms);
        if (pass == 0)
          for (size_t k = 0; k < ms.size(); ++k)
            if (seg_ws[dt][k] >= 0)
              P->ws_patches.push_back({L.mats + k * sizeof(wt::MatDesc) + offsetof(wt::MatDesc, y), (size_t)seg_ws[dt][k]});
        L.pieces = append(P->table, pieces);
        L.begin = append(P->table, begin);
        if (warp_mma) {
          L.maps = (P->table.size() + 127) & ~(size_t)127;
          P->table.resize(L.maps + ms.size() * wt::kTensorMapBytes);
          for (size_t k = 0; k < ms.size(); ++k) {
            int rc = encode_cols_map(ms[k], P->table.data() + L.maps + k * wt::kTensorMapBytes);
            if (rc) return rc;
          }
        }
        (pass == 0 ? g.launches : pass == 1 || pass == 4 ? g.mapped : g.cols).push_back(L);
      }
    }
    if (!reds.empty()) {
      g.reduce = append(P->table, reds);
      g.n_reduce = (int)reds.size();
      for (size_t k = 0; k < reds.size(); ++k)
        P->ws_patches.push_back({g.reduce + k * sizeof(wt::SegReduce) + offsetof(wt::SegReduce, ws), red_ws[k]});
    }
    P->groups.push_back(std::move(g));
  }
  if (P->ws_floats) {
    CU(cached_alloc(false, P->device, reinterpret_cast<void **>(&P->ws), P->ws_floats * sizeof(float)));
    for (const auto &pt : P->ws_patches) {
      const float *p = P->ws + pt.second;
      memcpy(P->table.data() + pt.first, &p, sizeof p);
    }
  }
  const size_t bytes = std::max<size_t>(16, align16(P->table.size()));
  CU(cached_alloc(true, P->device, reinterpret_cast<void **>(&P->host), bytes));
  P->table_bytes = bytes;
  memcpy(P->host, P->table.data(), P->table.size());
  if (wt::fault_injected("alloc")) return set_err(WT_ENOMEM, "wt_pass: plan tables: injected allocation fault");
  CU(cached_alloc(false, P->device, reinterpret_cast<void **>(&P->dev), bytes));
  CU(ev_create(&P->uploaded, cudaEventDisableTiming));
  return WT_OK;
}

void destroy_plan(Plan *P) {
  for (const auto &sl : P->last) cudaEventSynchronize(sl.second);
  // a plan a captured graph refers to may still be read by a replay the caller did not wait
  // for: its blocks go back to the cache only once the device is idle
  if (P->pinned) cudaDeviceSynchronize();
  cached_free(false, P->device, P->dev, P->table_bytes);
  cached_free(false, P->device, P->ws, P->ws_floats * sizeof(float));
  cached_free(true, P->device, P->host, P->table_bytes);
  ev_destroy(P->uploaded);
  for (const auto &sl : P->last) ev_destroy(sl.second);
  delete P;
  g_live_plans--;
}

// True if the tables of P are in device memory: the stream-ordered upload of its first use
// has completed.  Queried in relaxed capture mode, so it is legal while a graph is captured.
bool plan_resident(const Plan *P) {
  if (!P->sent) return false;
  cudaStreamCaptureMode m = cudaStreamCaptureModeRelaxed;
  cudaThreadExchangeStreamCaptureMode(&m);
  const cudaError_t q = cudaEventQuery(P->uploaded);
  cudaThreadExchangeStreamCaptureMode(&m);
  if (q != cudaSuccess && q != cudaErrorNotReady) cudaGetLastError();
  return q == cudaSuccess;
}

int run_plan(wt_handle *h, Plan *P, const wt_gemv_desc *d, cudaStream_t s, bool capturing = false) {
  if (capturing) {
    // Inside a stream capture the graph replays later, on its own schedule: the tables must
    // already be resident, and nothing here may depend on events outside the capture.
    if (!plan_resident(P))
      return set_err(WT_EINVAL,
                     "wt_pass: capturing a pass needs the same descriptors run once outside the capture, "
                     "with that stream synchronised, before the capture begins");
    P->pinned = true;
  } else if (!P->sent) {
    CU(cudaMemcpyAsync(P->dev, P->host, std::max<size_t>(16, align16(P->table.size())), cudaMemcpyHostToDevice, s));
    CU(cudaEventRecord(P->uploaded, s));
    P->sent = true;
    P->sent_on = s;
  } else if (s != P->sent_on) {
    CU(cudaStreamWaitEvent(s, P->uploaded, 0));
  }
  for (const Plan::Group &g : P->groups) {
    cudaEvent_t wait = static_cast<cudaEvent_t>(d[g.first].wait_event);
    if (wait) CU(cudaStreamWaitEvent(s, wait, 0));
    cudaEvent_t tb = nullptr;
    if (h->timeline && !capturing) {
      int rc = trace_mark(s, &tb);
      if (rc) return rc;
    }
    struct TraceEnd {  // closes the group's timeline record on every path out of this scope
      wt_handle *h;
      cudaStream_t s;
      cudaEvent_t tb;
      uint64_t bytes;
      cudaEvent_t wait;
      ~TraceEnd() {
        if (!tb) return;
        cudaEvent_t te = nullptr;
        if (trace_mark(s, &te) == WT_OK) trace_push(h, {WT_TRACE_GEMV, h->n_groups, bytes, tb, te, true, wait});
        else ev_destroy(tb);
      }
    } trace_end{h, s, tb, g.wbytes, wait};
    if (!capturing) h->n_groups++;
    for (const Plan::Zero &z : g.zero) CU(cudaMemsetAsync(z.y, 0, z.M * sizeof(float), s));
    for (const Plan::Launch &L : g.launches) {
      wt::GemvLaunch gl;
      gl.dtype = L.dtype;
      gl.grid = L.grid;
      gl.mats = reinterpret_cast<const wt::MatDesc *>(P->dev + L.mats);
      gl.pieces = reinterpret_cast<const wt::Piece *>(P->dev + L.pieces);
      gl.begin = reinterpret_cast<const uint32_t *>(P->dev + L.begin);
      gl.status = h->status;
      gl.stall = wt::fault_injected("stall") ? 1 : 0;
      // Inside a captured graph of consecutive passes, each pass may start its launch and
      // prologue while the previous one finishes (a programmatic edge); a group gated on an
      // event, and every pass issued from the host, keep the plain stream order (measured:
      // programmatic launches issued one by one from the host made small passes slower).
      gl.pdl = capturing && !wait ? 1 : 0;
      if (h->stamping) {
        if ((size_t)L.grid > h->stamp_cap) {
          if (capturing)
            return set_err(WT_EINVAL, "wt_pass: a stamped pass needs the same descriptors run once outside the capture");
          const size_t cap = std::max<size_t>((size_t)L.grid, 2u * (size_t)wt::num_sms());
          uint64_t *buf = nullptr;
          CU(dev_alloc(reinterpret_cast<void **>(&buf), cap * wt::kStampFields * sizeof(uint64_t)));
          if (h->stamp_dev) {
            cudaDeviceSynchronize();  // earlier stamped launches may still write the old buffer
            dev_free(h->stamp_dev, h->stamp_cap * wt::kStampFields * sizeof(uint64_t));
          }
          h->stamp_dev = buf;
          h->stamp_cap = cap;
        }
        gl.stamps = h->stamp_dev;
        h->stamp_ctas = L.grid;
      }
      CU(wt::launch_gemv(gl, s));
      h->kernel_launches++;
    }
    if (g.n_reduce) {
      CU(wt::launch_seg_reduce(reinterpret_cast<const wt::SegReduce *>(P->dev + g.reduce), g.n_reduce, g.reduce_rows, s));
      h->kernel_launches++;
    }
    for (const Plan::Launch &L : g.mapped) {
      wt::GemvLaunch gl;
      gl.dtype = L.dtype;
      gl.grid = L.grid;
      gl.mats = reinterpret_cast<const wt::MatDesc *>(P->dev + L.mats);
      gl.pieces = reinterpret_cast<const wt::Piece *>(P->dev + L.pieces);
      gl.begin = reinterpret_cast<const uint32_t *>(P->dev + L.begin);
      gl.status = h->status;
      CU(L.mapped_cols ? wt::launch_gemv_mapped_cols(gl, s) : wt::launch_gemv_mapped(gl, s));
      h->kernel_launches++;
    }
    for (const Plan::Launch &L : g.cols) {
      wt::GemvLaunch gl;
      gl.dtype = L.dtype;
      gl.grid = L.grid;
      gl.mats = reinterpret_cast<const wt::MatDesc *>(P->dev + L.mats);
      gl.pieces = reinterpret_cast<const wt::Piece *>(P->dev + L.pieces);
      gl.begin = reinterpret_cast<const uint32_t *>(P->dev + L.begin);
      gl.status = h->status;
      gl.maps = P->dev + L.maps;
      gl.nt = L.nt;
      if (L.q8rows) {
        CU(wt::launch_gemm_q8_rows(gl, s));
      } else if (L.umma) {
        wt::UmmaLaunch ul;
        ul.dtype = L.dtype;
        ul.grid = L.grid;
        ul.mats = gl.mats;
        ul.pieces = gl.pieces;
        ul.nmat = L.nmat;
        ul.ntiles = L.ntiles;
        ul.status = h->status;
        ul.maps = gl.maps;
        CU(wt::launch_gemm_cols_umma(ul, s));
      } else {
        CU(wt::launch_gemm_cols(gl, s));
      }
      h->kernel_launches++;
    }
    for (const Plan::Generic &q : g.generic) {
      CU(wt::launch_gemv_generic(q.dtype, q.W, q.x, q.y, q.M, q.K, q.scale, q.cols, s));
      h->kernel_launches++;
    }
  }
  if (!capturing) {
    // one completion event per stream the plan has run on: the plan's blocks are reused only
    // after its latest run on every one of them.  Past kPlanStreams streams, the oldest entry
    // is waited for and taken over, so a caller that cycles through streams holds few events.
    constexpr size_t kPlanStreams = 8;
    cudaEvent_t done = nullptr;
    for (const auto &sl : P->last)
      if (sl.first == s) done = sl.second;
    if (!done && P->last.size() >= kPlanStreams) {
      done = P->last.front().second;
      CU(cudaEventSynchronize(done));
      P->last.erase(P->last.begin());
      P->last.push_back({s, done});
    } else if (!done) {
      CU(ev_create(&done, cudaEventDisableTiming));
      P->last.push_back({s, done});
    }
    CU(cudaEventRecord(done, s));
  }
  return WT_OK;
}

int close_impl(wt_handle *h) {
  int rc = WT_OK;
  if (!h->host_only && h->device >= 0) {
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != h->device) cudaSetDevice(h->device);
    for (cudaEvent_t e : h->events) cudaEventSynchronize(e);
    for (auto &t : h->trace) {
      ev_destroy(t.begin);
      if (t.own_end && t.end) {
        cudaEventSynchronize(t.end);
        ev_destroy(t.end);
      }
    }
    h->trace.clear();
    for (Plan *P : h->plans) destroy_plan(P);
    h->plans.clear();
    for (cudaEvent_t e : h->events) ev_destroy(e);
    h->events.clear();
    status_give(h->device, h->status);
    h->status = nullptr;
    if (h->stamp_dev) {
      dev_free(h->stamp_dev, h->stamp_cap * wt::kStampFields * sizeof(uint64_t));
      h->stamp_dev = nullptr;
    }
    for (File &f : h->files) unmap_file(f);
    if (cur >= 0 && cur != h->device) cudaSetDevice(cur);
  } else {
    for (File &f : h->files) unmap_file(f);
  }
  delete h;
  g_live_handles--;
  return rc;
}

}  // namespace

int wt::set_error(int code, const char *msg) { return set_err(code, "%s", msg); }

bool wt::fault_injected(const char *site) {
  const char *e = getenv("WT_FAULT");
  if (!e || !*e) return false;
  static std::mutex mu;
  static std::string last;
  static int count = 0;
  std::lock_guard<std::mutex> g(mu);
  if (last != e) {
    last = e;
    count = 0;
  }
  const char *colon = strchr(e, ':');
  const size_t len = colon ? (size_t)(colon - e) : strlen(e);
  if (len != strlen(site) || strncmp(e, site, len) != 0) return false;
  const int n = colon ? atoi(colon + 1) : 1;
  return ++count == n;
}

// ====================================================================== C ABI
#pragma GCC visibility push(default)
extern "C" {

const char *wt_last_error(void) { return t_err.c_str(); }

int wt_abi_version(void) { return 4; }

int wt_open(const char *const *paths, int n_paths, unsigned flags, wt_handle **out) {
  if (!out) return set_err(WT_EINVAL, "wt_open: out is NULL");
  *out = nullptr;
  if (n_paths < 0 || (n_paths > 0 && !paths)) return set_err(WT_EINVAL, "wt_open: bad path list");
  const unsigned route_req = flags & WT_ROUTE_MASK;
  if (flags & ~(WT_ROUTE_MASK | WT_OPEN_HOST_ONLY | WT_OPEN_PREFAULT | WT_OPEN_TIMELINE | WT_OPEN_NOMAP |
                WT_OPEN_STAMPS | WT_OPEN_MAP_LARGE))
    return set_err(WT_EINVAL, "wt_open: unknown flag bits 0x%x", flags);
  const bool nomap = (flags & WT_OPEN_NOMAP) != 0;
  if (nomap && (flags & WT_OPEN_MAP_LARGE))
    return set_err(WT_EINVAL, "wt_open: WT_OPEN_NOMAP maps nothing: no WT_OPEN_MAP_LARGE");
  uint64_t map_min = 0;
  if (flags & WT_OPEN_MAP_LARGE) {
    map_min = WT_MAP_MIN_BYTES;
    if (const char *e = getenv("WT_MAP_MIN_BYTES")) {
      char *end = nullptr;
      const unsigned long long v = strtoull(e, &end, 10);
      if (!end || end == e || *end) return set_err(WT_EINVAL, "wt_open: WT_MAP_MIN_BYTES=%s is not a byte count", e);
      map_min = v;
    }
  }
  if (nomap && (route_req == WT_ROUTE_REGISTER || route_req == WT_ROUTE_DIRECT || (flags & WT_OPEN_PREFAULT)))
    return set_err(WT_EINVAL, "wt_open: WT_OPEN_NOMAP maps nothing: no REGISTER or DIRECT route, no PREFAULT");
  wt_handle *h = nullptr;
  try {
    h = new wt_handle();
    g_live_handles++;
    h->host_only = (flags & WT_OPEN_HOST_ONLY) != 0;
    h->timeline = (flags & WT_OPEN_TIMELINE) != 0 && !h->host_only;
    h->stamping = (flags & WT_OPEN_STAMPS) != 0 && !h->host_only;
    h->files.resize(n_paths);
    for (int i = 0; i < n_paths; ++i) {
      if (!paths[i]) {
        delete h;
        g_live_handles--;
        return set_err(WT_EINVAL, "wt_open: path %d is NULL", i);
      }
      h->files[i].path = paths[i];
    }
    // parse + map in parallel; keep the first failure in file order
    std::vector<int> rcs(n_paths, WT_OK);
    std::vector<std::string> errs(n_paths);
    int64_t t0 = now_ns();
    host_pool().parallel_for((size_t)n_paths, [&](size_t i) {
      rcs[i] = open_one(h->files[i], nomap, map_min);
      if (rcs[i]) errs[i] = t_err;
    });
    h->open_times.index_ms = (now_ns() - t0) * 1e-6;
    for (const File &f : h->files) {
      h->open_times.index_cpu_ms += f.index_ns * 1e-6;
      h->open_times.map_cpu_ms += f.map_ns * 1e-6;
      h->open_times.files_mapped += f.base ? 1 : 0;
    }
    for (int i = 0; i < n_paths; ++i) {
      if (rcs[i]) {
        std::string msg = errs[i];
        close_impl(h);
        return set_err(rcs[i], "%s", msg.c_str());
      }
    }
    for (int f = 0; f < n_paths; ++f)
      for (uint32_t e = 0; e < h->files[f].tensors.size(); ++e) h->order.push_back({(uint32_t)f, e});
    for (int f = 0; f < n_paths; ++f)
      if (h->files[f].base) h->by_base.push_back({reinterpret_cast<uintptr_t>(h->files[f].base), (uint32_t)f});
    std::sort(h->by_base.begin(), h->by_base.end());
    if (flags & WT_OPEN_PREFAULT) {
      t0 = now_ns();
      host_pool().parallel_for((size_t)n_paths, [&](size_t i) {
        if (h->files[i].base) prefault(h->files[i].base, h->files[i].size);
      });
      h->prefaulted = true;
      h->open_times.prefault_ms = (now_ns() - t0) * 1e-6;
    }
    if (h->host_only) {
      for (File &f : h->files) f.route = WT_ROUTE_NONE;
      *out = h;
      return WT_OK;
    }
    cudaError_t ce = cudaGetDevice(&h->device);
    if (ce != cudaSuccess) {
      close_impl(h);
      return cuda_err(ce, "cudaGetDevice");
    }
    int rc = prepare_device(h->device);
    if (rc) {
      close_impl(h);
      return rc;
    }
    int ats = 0;
    t0 = now_ns();
    cudaDeviceGetAttribute(&ats, cudaDevAttrPageableMemoryAccessUsesHostPageTables, h->device);
    for (File &f : h->files) {
      unsigned want = f.base ? route_req : WT_ROUTE_NONE;
      if (want == WT_ROUTE_AUTO) want = ats ? WT_ROUTE_DIRECT : WT_ROUTE_REGISTER;
      if (want == WT_ROUTE_DIRECT) {
        if (!ats) {
          close_impl(h);
          return set_err(WT_ENOTSUP, "%s: device does not read pageable memory through host page tables", f.path.c_str());
        }
        f.route = WT_ROUTE_DIRECT;
        f.dev = f.base;
      } else if (want == WT_ROUTE_REGISTER) {
        // Read-only registration first (the mapping is PROT_READ); a driver that refuses the
        // flag for file-backed pages gets a plain mapped registration, and wt_file_registration
        // reports which one the file holds.
        const bool injected = wt::fault_injected("register");
        unsigned rf = cudaHostRegisterMapped | cudaHostRegisterReadOnly;
        cudaError_t e = injected ? cudaErrorMemoryAllocation : cudaHostRegister(f.base, f.size, rf);
        if (e != cudaSuccess && !injected) {
          cudaGetLastError();
          rf = cudaHostRegisterMapped;
          e = cudaHostRegister(f.base, f.size, rf);
        }
        if (e == cudaSuccess) {
          f.registered = true;
          f.reg_flags = rf;
          f.populated = true;  // registration pins (and so maps) every page
          void *dp = nullptr;
          e = cudaHostGetDevicePointer(&dp, f.base, 0);
          if (e != cudaSuccess) {
            close_impl(h);
            return cuda_err(e, "cudaHostGetDevicePointer");
          }
          f.route = WT_ROUTE_REGISTER;
          f.dev = static_cast<const uint8_t *>(dp);
        } else if (route_req == WT_ROUTE_AUTO) {
          cudaGetLastError();
          f.route = WT_ROUTE_NONE;
        } else {
          close_impl(h);
          return cuda_err(e, "cudaHostRegister");
        }
      } else {
        f.route = WT_ROUTE_NONE;
      }
    }
    h->open_times.route_ms = (now_ns() - t0) * 1e-6;
    for (const File &f : h->files) h->open_times.files_registered += f.registered ? 1 : 0;
    ce = status_take(h->device, &h->status);
    if (ce != cudaSuccess) {
      close_impl(h);
      return cuda_err(ce, "status word");
    }
    *out = h;
    return WT_OK;
  } catch (const std::bad_alloc &) {
    if (h) close_impl(h);
    return set_err(WT_ENOMEM, "wt_open: out of host memory");
  } catch (...) {
    if (h) close_impl(h);
    return set_err(WT_EINVAL, "wt_open: unexpected failure");
  }
}

int wt_num_tensors(const wt_handle *h, size_t *n) {
  if (!h || !n) return set_err(WT_EINVAL, "wt_num_tensors: NULL argument");
  *n = h->order.size();
  return WT_OK;
}

int wt_dlpack_tensor(const wt_handle *h, size_t i, unsigned flags, DLManagedTensorVersioned **out) {
  if (!out) return set_err(WT_EINVAL, "wt_dlpack_tensor: out is NULL");
  *out = nullptr;
  if (!h) return set_err(WT_EINVAL, "wt_dlpack_tensor: NULL handle");
  if (i >= h->order.size()) return set_err(WT_EINVAL, "wt_dlpack_tensor: tensor %zu out of range", i);
  if (h->host_only && !(flags & WT_DLPACK_HOST))
    return set_err(WT_EINVAL, "wt_dlpack_tensor: host-only handle: ask for WT_DLPACK_HOST");
  const Tensor &t = h->tensor(i);
  const File &f = h->files[h->order[i].first];
  return wt::dlpack_map(f.path.c_str(), t.offset, t.nbytes, t.dtype, t.ndim, t.shape, flags, out);
}

int wt_num_files(const wt_handle *h, size_t *n) {
  if (!h || !n) return set_err(WT_EINVAL, "wt_num_files: NULL argument");
  *n = h->files.size();
  return WT_OK;
}

int wt_tensor_info(const wt_handle *h, size_t i, wt_tensor_meta *out) {
  if (!h || !out) return set_err(WT_EINVAL, "wt_tensor_info: NULL argument");
  if (i >= h->order.size()) return set_err(WT_EINVAL, "wt_tensor_info: index %zu out of range", i);
  const Tensor &t = h->tensor(i);
  out->name = t.name.c_str();
  out->dtype = t.dtype;
  out->ndim = t.ndim;
  for (int d = 0; d < 4; ++d) out->shape[d] = t.shape[d];
  out->nbytes = t.nbytes;
  out->file = h->order[i].first;
  out->offset = t.offset;
  out->host_ptr = h->files[out->file].base ? h->files[out->file].base + t.offset : nullptr;
  return WT_OK;
}

int wt_tensor_table(const wt_handle *h, size_t first, size_t n, wt_tensor_meta *out) {
  if (!h || (n && !out)) return set_err(WT_EINVAL, "wt_tensor_table: NULL argument");
  if (first > h->order.size() || n > h->order.size() - first)
    return set_err(WT_EINVAL, "wt_tensor_table: tensors [%zu, %zu) out of range", first, first + n);
  for (size_t k = 0; k < n; ++k) wt_tensor_info(h, first + k, out + k);
  return WT_OK;
}

int wt_tensor_names(const wt_handle *h, char *buf, size_t cap, size_t *needed) {
  if (!h || !needed || (cap && !buf)) return set_err(WT_EINVAL, "wt_tensor_names: NULL argument");
  size_t total = 0;
  for (size_t i = 0; i < h->order.size(); ++i) total += h->tensor(i).name.size() + 1;
  *needed = total;
  if (cap < total) return cap ? set_err(WT_EINVAL, "wt_tensor_names: buffer of %zu bytes, %zu needed", cap, total) : WT_OK;
  size_t pos = 0;
  for (size_t i = 0; i < h->order.size(); ++i) {
    const std::string &nm = h->tensor(i).name;
    memcpy(buf + pos, nm.c_str(), nm.size() + 1);
    pos += nm.size() + 1;
  }
  return WT_OK;
}

int wt_tensor_groups(const wt_handle *h, uint32_t *group, int32_t *block, size_t *n_groups) {
  if (!h || !n_groups || (!h->order.empty() && (!group || !block)))
    return set_err(WT_EINVAL, "wt_tensor_groups: NULL argument");
  // base name -> group, for the row blocks; every other tensor is a group of its own
  std::unordered_map<std::string_view, uint32_t> by_base;  // views of the handle's own names
  by_base.reserve(h->order.size());
  uint32_t n = 0;
  for (size_t i = 0; i < h->order.size(); ++i) {
    const std::string &nm = h->tensor(i).name;
    const size_t at = nm.rfind("#r");
    int64_t k = -1;
    if (at != std::string::npos) {
      const size_t nd = nm.size() - at - 2;
      if (nd >= 1 && nd <= 9) {
        k = 0;
        for (size_t c = at + 2; c < nm.size() && k >= 0; ++c)
          k = (nm[c] >= '0' && nm[c] <= '9') ? k * 10 + (nm[c] - '0') : -1;
      }
    }
    if (k < 0) {
      group[i] = n++;
      block[i] = -1;
      continue;
    }
    auto ins = by_base.emplace(std::string_view(nm.data(), at), n);
    if (ins.second) ++n;
    group[i] = ins.first->second;
    block[i] = (int32_t)k;
  }
  *n_groups = n;
  return WT_OK;
}

int wt_find(const wt_handle *h, const char *name, size_t *i) {
  if (!h || !name || !i) return set_err(WT_EINVAL, "wt_find: NULL argument");
  for (size_t k = 0; k < h->order.size(); ++k)
    if (h->tensor(k).name == name) {
      *i = k;
      return WT_OK;
    }
  return set_err(WT_EINVAL, "wt_find: no tensor named '%s'", name);
}

int wt_file_route(const wt_handle *h, size_t f, unsigned *route) {
  if (!h || !route) return set_err(WT_EINVAL, "wt_file_route: NULL argument");
  if (f >= h->files.size()) return set_err(WT_EINVAL, "wt_file_route: file %zu out of range", f);
  *route = h->files[f].route;
  return WT_OK;
}

int wt_file_registration(const wt_handle *h, size_t f, unsigned *flags) {
  if (!h || !flags) return set_err(WT_EINVAL, "wt_file_registration: NULL argument");
  if (f >= h->files.size()) return set_err(WT_EINVAL, "wt_file_registration: file %zu out of range", f);
  *flags = h->files[f].registered ? h->files[f].reg_flags : 0u;
  return WT_OK;
}

int wt_open_times(const wt_handle *h, wt_open_phases *out) {
  if (!h || !out) return set_err(WT_EINVAL, "wt_open_times: NULL argument");
  *out = h->open_times;
  return WT_OK;
}

int wt_adopt(wt_handle *h, const size_t *idx, void *const *dst, size_t n, unsigned mode, void *stream,
             void **ready) {
  if (!h) return set_err(WT_EINVAL, "wt_adopt: NULL handle");
  if (h->host_only) return set_err(WT_ENOTSUP, "wt_adopt: handle was opened host-only");
  if (n == 0) return WT_OK;
  if (!idx || !dst || !ready) return set_err(WT_EINVAL, "wt_adopt: NULL array");
  if (mode > WT_ADOPT_STAGED) return set_err(WT_EINVAL, "wt_adopt: unknown mode %u", mode);
  std::lock_guard<std::mutex> g(h->mu);
  try {
    std::vector<Range> rs, st;  // st: small unmapped files of a MAP_LARGE handle (GATHER / CE)
    rs.reserve(n);
    RangeCache rc_dst;
    for (size_t k = 0; k < n; ++k) {
      if (idx[k] >= h->order.size()) return set_err(WT_EINVAL, "wt_adopt: tensor index %zu out of range", idx[k]);
      const File &f = h->files[h->order[idx[k]].first];
      const Tensor &t = h->tensor(idx[k]);
      if (t.nbytes && !dst[k]) return set_err(WT_EINVAL, "wt_adopt: dst[%zu] is NULL", k);
      if (t.nbytes && inside_mapping(h, dst[k], t.nbytes))
        return set_err(WT_EINVAL, "wt_adopt: dst[%zu] lies inside a read-only mapping", k);
      if (!device_range_ok(dst[k], t.nbytes, rc_dst))
        return set_err(WT_EINVAL, "wt_adopt: dst[%zu] (%llu bytes) runs past the end of its device allocation", k,
                       (unsigned long long)t.nbytes);
      if (mode != WT_ADOPT_STAGED && f.route == WT_ROUTE_NONE && !f.small)
        return set_err(WT_ENOTSUP, "wt_adopt: %s has no device route; use WT_ADOPT_STAGED", f.path.c_str());
      ready[k] = nullptr;
      const Range r{k, h->order[idx[k]].first, t.offset, f.base ? f.base + t.offset : nullptr,
                    f.dev ? f.dev + t.offset : nullptr, static_cast<uint8_t *>(dst[k]), t.nbytes,
                    f.populated || h->prefaulted};
      if (mode != WT_ADOPT_STAGED && f.small) {
        st.push_back(r);
      } else {
        rs.push_back(r);
      }
    }
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (mode == WT_ADOPT_STAGED) return adopt_staged(h, rs, s, ready);
    if (st.empty()) return adopt_device(h, rs, mode, s, ready);
    if (rs.empty()) return adopt_staged(h, st, s, ready);
    return adopt_mixed(h, rs, st, mode, s, ready);
  } catch (const std::bad_alloc &) {
    return set_err(WT_ENOMEM, "wt_adopt: out of host memory");
  }
}

int wt_pass(wt_handle *h, const wt_gemv_desc *d, size_t n, void *stream) {
  if (!h) return set_err(WT_EINVAL, "wt_pass: NULL handle");
  if (h->host_only) return set_err(WT_ENOTSUP, "wt_pass: handle was opened host-only");
  if (n == 0) return WT_OK;
  if (!d) return set_err(WT_EINVAL, "wt_pass: NULL descriptors");
  for (size_t i = 0; i < n; ++i) {
    int rc = validate_desc(d[i], i);
    if (rc) return rc;
    if (d[i].M && inside_mapping(h, d[i].y, d[i].M * std::max<int32_t>(1, d[i].cols) * sizeof(float)))
      return set_err(WT_EINVAL, "wt_pass: y of desc %zu lies inside a read-only mapping", i);
  }
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(static_cast<cudaStream_t>(stream), &cs) != cudaSuccess) {
    cudaGetLastError();
    cs = cudaStreamCaptureStatusNone;
  }
  const bool capturing = cs == cudaStreamCaptureStatusActive;
  std::lock_guard<std::mutex> g(h->mu);
  try {
    // Plans are keyed by the descriptors with each wait_event replaced by the ordinal of its
    // first appearance: calls that differ only in which events they wait on share one plan.
    std::vector<wt_gemv_desc> kd(d, d + n);
    {
      std::vector<std::pair<uintptr_t, uintptr_t>> seen;  // (event, ordinal), sorted by event
      for (size_t i = 0; i < n; ++i) {
        const uintptr_t e = reinterpret_cast<uintptr_t>(d[i].wait_event);
        if (!e) continue;
        auto it = std::lower_bound(seen.begin(), seen.end(), std::make_pair(e, (uintptr_t)0));
        if (it == seen.end() || it->first != e) it = seen.insert(it, {e, seen.size() + 1});
        kd[i].wait_event = reinterpret_cast<void *>(it->second);
      }
    }
    const uint8_t *kb = reinterpret_cast<const uint8_t *>(kd.data());
    std::vector<uint8_t> key(kb, kb + n * sizeof(wt_gemv_desc));
    Plan *P = nullptr;
    for (auto it = h->plans.begin(); it != h->plans.end(); ++it)
      if ((*it)->key == key) {
        P = *it;
        h->plans.erase(it);
        h->plans.push_front(P);
        break;
      }
    if (!P && capturing)  // building a plan allocates: not allowed inside a capture
      return set_err(WT_EINVAL,
                     "wt_pass: capturing a pass needs the same descriptors run once outside the capture, "
                     "with that stream synchronised, before the capture begins");
    if (!P) {
      P = new Plan();
      g_live_plans++;
      P->device = h->device;
      P->key = std::move(key);
      int rc = build_plan(h, d, n, P);
      if (rc) {
        destroy_plan(P);
        return rc;
      }
      h->plans.push_front(P);
      // least recently used plans beyond 32 go, except those a captured graph refers to
      size_t live = h->plans.size();
      for (auto it = std::prev(h->plans.end()); live > 32 && it != h->plans.begin();) {
        auto cur = it--;
        if ((*cur)->pinned) continue;
        destroy_plan(*cur);
        h->plans.erase(cur);
        --live;
      }
    }
    return run_plan(h, P, d, static_cast<cudaStream_t>(stream), capturing);
  } catch (const std::bad_alloc &) {
    return set_err(WT_ENOMEM, "wt_pass: out of host memory");
  }
}

static int checksum_impl(wt_handle *h, const void *const *ptr, const uint64_t *nbytes, size_t n,
                         uint64_t *out_dev, void *stream, bool plain) {
  if (!h) return set_err(WT_EINVAL, "wt_checksum: NULL handle");
  if (h->host_only) return set_err(WT_ENOTSUP, "wt_checksum: handle was opened host-only");
  if (n == 0) return WT_OK;
  if (!ptr || !nbytes || !out_dev) return set_err(WT_EINVAL, "wt_checksum: NULL array");
  for (size_t i = 0; i < n; ++i) {
    if (nbytes[i] && !ptr[i]) return set_err(WT_EINVAL, "wt_checksum: ptr[%zu] is NULL", i);
    if (nbytes[i] > wt::kMaxFnvBufferBytes)
      return set_err(WT_EINVAL, "wt_checksum: buffer %zu: %llu bytes is not a device buffer size", i,
                     (unsigned long long)nbytes[i]);
    if (plain && nbytes[i] > (256ull << 20)) return set_err(WT_EINVAL, "wt_checksum_plain: buffer %zu above 256 MiB", i);
  }
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  std::lock_guard<std::mutex> g(h->mu);
  std::vector<uint64_t *> outs(n);
  for (size_t i = 0; i < n; ++i) outs[i] = out_dev + i;
  for (size_t i0 = 0; i0 < n; i0 += wt::kMaxFnv) {
    const size_t m = std::min<size_t>(wt::kMaxFnv, n - i0);
    std::unique_ptr<wt::FnvBatch> b(new wt::FnvBatch);
    const size_t scratch = wt::fnv_fill_batch(*b, ptr + i0, nbytes + i0, outs.data() + i0, m);
    if (plain) {
      CU(wt::launch_fnv_plain(*b, s));
      h->kernel_launches++;
    } else {
      void *sc = nullptr;
      CU(cudaMallocAsync(&sc, scratch, s));
      const cudaError_t e = wt::launch_fnv_tree(*b, sc, s);
      cudaFreeAsync(sc, s);
      CU(e);
      h->kernel_launches += wt::fnv_tree_launches(*b);
    }
  }
  return WT_OK;
}

int wt_checksum(wt_handle *h, const void *const *ptr, const uint64_t *nbytes, size_t n, uint64_t *out_dev,
                void *stream) {
  return checksum_impl(h, ptr, nbytes, n, out_dev, stream, false);
}

int wt_checksum_plain(wt_handle *h, const void *const *ptr, const uint64_t *nbytes, size_t n,
                      uint64_t *out_dev, void *stream) {
  return checksum_impl(h, ptr, nbytes, n, out_dev, stream, true);
}

int wt_device_status(wt_handle *h, int *status) {
  if (!h || !status) return set_err(WT_EINVAL, "wt_device_status: NULL argument");
  if (h->host_only) {
    *status = 0;
    return WT_OK;
  }
  CU(cudaMemcpy(status, h->status, sizeof(int), cudaMemcpyDeviceToHost));
  return WT_OK;
}

int wt_residency(const wt_handle *h, uint64_t *resident, uint64_t *total) {
  if (!h || !resident || !total) return set_err(WT_EINVAL, "wt_residency: NULL argument");
  const size_t pg = (size_t)sysconf(_SC_PAGESIZE);
  uint64_t res = 0, tot = 0;
  std::vector<unsigned char> vec;
  for (const File &f : h->files) {
    if (!f.base) return set_err(WT_ENOTSUP, "wt_residency: %s is not mapped (WT_OPEN_NOMAP or MAP_LARGE)", f.path.c_str());
    const size_t pages = (f.size + pg - 1) / pg;
    vec.assign(pages, 0);
    if (pages && mincore(f.base, f.size, vec.data()) != 0)
      return set_err(WT_EIO, "wt_residency: mincore(%s): %s", f.path.c_str(), strerror(errno));
    for (size_t i = 0; i < pages; ++i)
      if (vec[i] & 1) res += std::min<uint64_t>(pg, f.size - i * pg);
    tot += f.size;
  }
  *resident = res;
  *total = tot;
  return WT_OK;
}

int wt_kernel_launches(const wt_handle *h, uint64_t *n) {
  if (!h || !n) return set_err(WT_EINVAL, "wt_kernel_launches: NULL argument");
  *n = h->kernel_launches;
  return WT_OK;
}

int wt_trace(wt_handle *h, void *origin, wt_trace_rec *out, size_t cap, size_t *n) {
  if (!h || !n || (cap && !out)) return set_err(WT_EINVAL, "wt_trace: NULL argument");
  if (!h->timeline) return set_err(WT_EINVAL, "wt_trace: the handle was not opened with WT_OPEN_TIMELINE");
  if (!origin) return set_err(WT_EINVAL, "wt_trace: NULL origin event");
  std::lock_guard<std::mutex> g(h->mu);
  const cudaEvent_t o = static_cast<cudaEvent_t>(origin);
  CU(cudaEventSynchronize(o));
  *n = h->trace.size();
  for (size_t k = 0; k < h->trace.size() && k < cap; ++k) {
    const auto &t = h->trace[k];
    CU(cudaEventSynchronize(t.end));
    float b = 0.f, e = 0.f;
    CU(cudaEventElapsedTime(&b, o, t.begin));
    CU(cudaEventElapsedTime(&e, o, t.end));
    out[k].kind = t.kind;
    out[k].pad = 0;
    out[k].index = t.index;
    out[k].bytes = t.bytes;
    out[k].event = t.event;
    out[k].begin_ms = b;
    out[k].end_ms = e;
  }
  for (auto &t : h->trace) {
    ev_destroy(t.begin);
    if (t.own_end) ev_destroy(t.end);
  }
  h->trace.clear();
  return WT_OK;
}

static_assert(WT_STAMP_ENTRY == wt::kStEntry && WT_STAMP_PROLOGUE == wt::kStPrologue &&
                  WT_STAMP_OPERANDS == wt::kStOperands && WT_STAMP_FIRST_COPY == wt::kStFirstCopy &&
                  WT_STAMP_FIRST_FULL == wt::kStFirstFull && WT_STAMP_LAST_FULL == wt::kStLastFull &&
                  WT_STAMP_EXIT == wt::kStExit && WT_STAMP_SM == wt::kStSm && WT_STAMP_FIELDS == wt::kStampFields,
              "the stamp record of include/wt.h is the kernel's");

int wt_pass_stamps(wt_handle *h, uint64_t *out, size_t cap, size_t *n) {
  if (!h || !n || (cap && !out)) return set_err(WT_EINVAL, "wt_pass_stamps: NULL argument");
  if (!h->stamping) return set_err(WT_EINVAL, "wt_pass_stamps: the handle was not opened with WT_OPEN_STAMPS");
  std::lock_guard<std::mutex> g(h->mu);
  *n = (size_t)h->stamp_ctas;
  if (!h->stamp_ctas) return WT_OK;
  // the handle's device, whichever device is current: every stamped launch has finished first
  int cur = -1;
  CU(cudaGetDevice(&cur));
  if (cur != h->device) CU(cudaSetDevice(h->device));
  cudaError_t e = cudaDeviceSynchronize();
  const size_t k = std::min(cap, (size_t)h->stamp_ctas);
  if (e == cudaSuccess && k) e = cudaMemcpy(out, h->stamp_dev, k * wt::kStampFields * sizeof(uint64_t), cudaMemcpyDeviceToHost);
  if (cur != h->device) cudaSetDevice(cur);
  if (e != cudaSuccess) return cuda_err(e, "wt_pass_stamps");
  return WT_OK;
}

int wt_live(wt_live_counts *out) {
  if (!out) return set_err(WT_EINVAL, "wt_live: NULL argument");
  out->handles = g_live_handles.load();
  out->plans = g_live_plans.load();
  out->events = g_live_events.load();
  out->device_bytes = g_dev_bytes.load();
  out->pinned_bytes = g_pinned_bytes.load();
  out->cached_device_bytes = g_dev_cached.load();
  out->cached_pinned_bytes = g_pinned_cached.load();
  return WT_OK;
}

int wt_close(wt_handle *h) {
  if (!h) return WT_OK;
  return close_impl(h);
}

}  // extern "C"
#pragma GCC visibility pop
