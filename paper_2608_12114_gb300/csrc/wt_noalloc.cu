// wt_checksum_noalloc: the leaf-tree digest of wt_checksum for callers that must
// not allocate device memory.
//
// Some callers cannot call cudaMalloc at the moment they want a digest: code
// running inside an allocator hook (it would re-enter the allocator it is
// serving), programs that have handed all device memory to their own pool up
// front (a serving engine's weight/KV arena), and loops that cannot afford the
// device-wide synchronisation cudaFree implies.  wt_checksum needs a temporary
// array of leaf digests and takes it from cudaMallocAsync; this entry point
// uses a fixed array compiled into the library instead.
//
// The array below is a file-scope __device__ object: every GPU that loads this
// library holds its ~9 MiB until the process exits.  Host code cannot use its
// name as a device address, so the first call on each device (with that device
// current) asks the runtime for the address with cudaGetSymbolAddress and
// caches it together with the CUDA context that was current; that first call
// should come before any stream capture.  A call made under another context
// (after cudaDeviceReset, or under a context the caller created with the
// driver API) looks the address up again, since the module, and with it the
// array, is loaded afresh in each context.  All calls
// share the array, and nothing in it needs to start at zero: each call writes
// every leaf slot it later reads.  Two calls whose kernels overlap on the GPU
// (different streams, no ordering between them) race on the array.
#include <cstring>
#include <mutex>

#include <cuda.h>  // CUcontext and cuCtxGetCurrent's signature (resolved through the runtime)

#include "../../include/wt.h"
#include "wt_fnv.h"
#include "wt_kernels.h"

namespace {

constexpr uint64_t kNoAllocMaxLeaves = 1ull << 20;  // 4096-byte leaves: 4 GiB of input per call
// leaf digests plus the chunk tables of the parallel second level (at most one chunk per
// kChunkWords leaves and one partial chunk per buffer of a batch)
constexpr uint64_t kNoAllocWords =
    kNoAllocMaxLeaves +
    ((kNoAllocMaxLeaves / wt::kChunkWords + wt::kMaxFnv) * wt::kChunkScratchBytes + wt::kMaxFnv * 8 + 2048) / 8;
__device__ __align__(256) uint64_t g_noalloc_leaves[kNoAllocWords];

std::mutex g_mu;
uint64_t *g_leaves_addr[64] = {nullptr};
CUcontext g_leaves_ctx[64] = {nullptr};  // the context g_leaves_addr[dev] belongs to

using CtxGetCurrentFn = CUresult (*)(CUcontext *);

// cuCtxGetCurrent, looked up once through the runtime (no link against libcuda).
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  return fn;
}

int fail(int code, const char *msg) { return wt::set_error(code, msg); }  // readable via wt_last_error

}  // namespace

extern "C" __attribute__((visibility("default"))) int wt_checksum_noalloc(
    const void *const *ptr, const uint64_t *nbytes, size_t n, uint64_t *out_dev, void *stream) {
  if (n == 0) return WT_OK;
  if (!ptr || !nbytes || !out_dev) return fail(WT_EINVAL, "wt_checksum_noalloc: NULL array");
  // Each buffer is bounded before it is counted, so the sum below cannot wrap.
  uint64_t leaves = 0;
  for (size_t i = 0; i < n; ++i) {
    if (nbytes[i] && !ptr[i]) return fail(WT_EINVAL, "wt_checksum_noalloc: NULL buffer");
    if (nbytes[i] > kNoAllocMaxLeaves * wt::kLeafBytes) {
      leaves = kNoAllocMaxLeaves + 1;
      break;
    }
    leaves += (nbytes[i] + wt::kLeafBytes - 1) / wt::kLeafBytes;
    if (leaves > kNoAllocMaxLeaves) break;
  }
  if (leaves > kNoAllocMaxLeaves)
    return fail(WT_EINVAL,
                "wt_checksum_noalloc: input needs more than 1048576 leaves of 4096 bytes (4 GiB per call); "
                "split the call or use wt_checksum");
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) return fail(WT_ECUDA, "wt_checksum_noalloc: cudaGetDevice failed");
  // The context current now (null before the runtime's first call on this device: the
  // symbol lookup below then creates the primary context, and it is read again after).
  CtxGetCurrentFn get_ctx = ctx_get_current();
  if (!get_ctx) return fail(WT_ECUDA, "wt_checksum_noalloc: cuCtxGetCurrent is not available");
  CUcontext ctx = nullptr;
  if (get_ctx(&ctx) != CUDA_SUCCESS) ctx = nullptr;
  uint64_t *scratch;
  {
    std::lock_guard<std::mutex> g(g_mu);
    if (!ctx || !g_leaves_addr[dev] || g_leaves_ctx[dev] != ctx) {
      void *p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_leaves);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        return fail(WT_ECUDA, "wt_checksum_noalloc: cudaGetSymbolAddress of the leaf array failed");
      }
      if (!ctx && (get_ctx(&ctx) != CUDA_SUCCESS || !ctx))
        return fail(WT_ECUDA, "wt_checksum_noalloc: no CUDA context on the current device");
      g_leaves_addr[dev] = static_cast<uint64_t *>(p);
      g_leaves_ctx[dev] = ctx;
    }
    scratch = g_leaves_addr[dev];
  }
  // Batches run in order on one stream, so each reuses the array from slot 0.
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  static thread_local wt::FnvBatch b;  // 18 KB: kept off the stack
  uint64_t *outs[wt::kMaxFnv];
  for (size_t i0 = 0; i0 < n; i0 += wt::kMaxFnv) {
    const size_t m = n - i0 < (size_t)wt::kMaxFnv ? n - i0 : (size_t)wt::kMaxFnv;
    for (size_t k = 0; k < m; ++k) outs[k] = out_dev + i0 + k;
    const size_t need = wt::fnv_fill_batch(b, ptr + i0, nbytes + i0, outs, m);
    if (need > sizeof(g_noalloc_leaves)) return fail(WT_EINVAL, "wt_checksum_noalloc: batch scratch exceeds the fixed array");
    e = wt::launch_fnv_tree(b, scratch, s);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(WT_ECUDA, "wt_checksum_noalloc: kernel launch failed");
    }
  }
  return WT_OK;
}
