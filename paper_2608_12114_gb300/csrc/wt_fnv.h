// Internal interface of the FNV-1a-64 digest kernels (wt_fnv.cu) for the host library
// (wt_host.cpp, wt_noalloc.cu).  Not part of the public C ABI (include/wt.h).
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace wt {

// ---------------------------------------------------------------- FNV-1a-64
constexpr int kMaxFnv = 512;  // buffers per launch: the batch is an 18 KB kernel parameter
constexpr uint64_t kLeafBytes = 4096;
// Largest buffer a digest call accepts (1 TiB, above any device's memory): bounds the leaf and
// chunk counts so that no size the caller passes can wrap them.
constexpr uint64_t kMaxFnvBufferBytes = 1ull << 40;

// The tree digest's second level is a serial FNV chain over 8 bytes per leaf.  Buffers of
// more than kParallelLeaves leaves split that chain into chunks of kChunkWords leaf digests
// and combine the chunks in parallel (exact; see the kernels), others run it in one thread.
constexpr uint64_t kParallelLeaves = 4096;
constexpr uint32_t kChunkWords = 512;

struct FnvBatch {
  uint32_t n;
  uint32_t pad;
  uint64_t leaf_prefix[kMaxFnv + 1];   // first global leaf of buffer i; [n] = total leaves
  uint32_t chunk_prefix[kMaxFnv + 1];  // first global chunk of buffer i; [n] = total chunks
  const uint8_t *ptr[kMaxFnv];
  uint64_t nbytes[kMaxFnv];
  uint64_t *out[kMaxFnv];  // device address of the digest of buffer i
};

// Fills n, ptr, nbytes, out and both prefixes from the buffers; returns the device scratch
// bytes launch_fnv_tree needs for the batch (leaf digests, then the chunk tables).
size_t fnv_fill_batch(FnvBatch &b, const void *const *ptr, const uint64_t *nbytes, uint64_t *const *out, size_t n);

// Device scratch per chunk of the parallel second level: a 256-entry low-byte table and four
// 32-bit words (starting low byte, B, starting lo, H).
constexpr size_t kChunkScratchBytes = 256 + 4 * 4;

// Kernel launches of launch_fnv_tree for the batch: leaves, combine, and five chunk passes.
int fnv_tree_launches(const FnvBatch &b);

cudaError_t launch_fnv_tree(const FnvBatch &b, void *scratch, cudaStream_t s);
cudaError_t launch_fnv_plain(const FnvBatch &b, cudaStream_t s);

}  // namespace wt
