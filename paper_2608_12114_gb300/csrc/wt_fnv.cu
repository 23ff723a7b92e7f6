// sm_103a kernels of the per-buffer FNV-1a-64 digests that prove ingested bytes equal the
// file's: the literal serial digest, and the tree digest (FNV-1a-64 of each 4 KiB leaf,
// then FNV-1a-64 over the buffer's length and its leaf digests).  The second level of the
// tree runs in parallel chunks for large buffers, with the exact result of the serial chain.
#include <cstring>

#include "wt_device.cuh"
#include "wt_fnv.h"
#include "wt_kernels.h"

namespace wt {

namespace {

// ------------------------------------------------------------------ FNV-1a-64
// The 64-bit state is held as two 32-bit words.  With p = 2^40 + 0x1b3 and x = lo ^ b,
//   (hi 2^32 + x) p mod 2^64 = (hi 0x1b3 + (x << 8) + high32(x 0x1b3)) 2^32 + low32(x 0x1b3),
// since hi 2^72 vanishes and x 2^40 keeps only (x << 8) in the high word.  The serial chain
// through a byte is then an xor and one 32 x 32 multiply on the low word; the high word is a
// multiply-add beside it.  The constants are FNV-1a-64's offset basis and prime.
constexpr uint32_t kFnvOffLo = 0x84222325u, kFnvOffHi = 0xcbf29ce4u;
constexpr uint32_t kFnvP = 0x1b3u;

struct Fnv {
  uint32_t lo = kFnvOffLo, hi = kFnvOffHi;
  __device__ __forceinline__ void byte(uint32_t b) {
    const uint32_t x = lo ^ b;
    const uint64_t w = (uint64_t)x * kFnvP;
    lo = (uint32_t)w;
    hi = hi * kFnvP + ((uint32_t)(w >> 32) + (x << 8));
  }
  // A word's four bytes, little-endian: the low word's chain first (the byte xored into the
  // low byte, one 32 x 32 -> 64 multiply), then the high word's four multiply-adds in one
  // Horner run, since hi' = hi p + t with t from the low word's step alone.  The masked xor
  // is one lop3 (a ^ (b & c), truth table 0x78) on the shifted word.  Measured on GB300 over
  // 1 GiB of leaves: 3.89 TB/s byte at a time, 4.28 TB/s this way, 4.40 TB/s with the
  // 64-byte slices of 8-warp blocks below.
  __device__ __forceinline__ void word(uint32_t v) {
    uint32_t t[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      uint32_t x;
      asm("lop3.b32 %0, %1, %2, 0xff, 0x78;" : "=r"(x) : "r"(lo), "r"(v >> (8 * k)));
      const uint64_t w = (uint64_t)x * kFnvP;
      lo = (uint32_t)w;
      t[k] = (uint32_t)(w >> 32) + (x << 8);
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) hi = hi * kFnvP + t[k];
  }
  __device__ __forceinline__ void vec(const uint4 &v) {
    word(v.x);
    word(v.y);
    word(v.z);
    word(v.w);
  }
  __device__ __forceinline__ void le64(uint64_t v) {
    word((uint32_t)v);
    word((uint32_t)(v >> 32));
  }
  __device__ __forceinline__ uint64_t value() const { return ((uint64_t)hi << 32) | lo; }
};

__device__ __forceinline__ uint32_t find_buf(const FnvBatch &b, uint64_t leaf) {
  uint32_t lo = 0, hi = b.n - 1;
  while (lo < hi) {
    uint32_t mid = (lo + hi + 1) >> 1;
    if (b.leaf_prefix[mid] <= leaf) lo = mid; else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// One thread per 4 KiB leaf.  A warp stages 64-byte slices of its 32 leaves in shared
// memory with coalesced asynchronous 16-byte copies (four lanes per leaf slice, eight
// leaves per warp instruction), double-buffered: slice s + 1 is in flight while each lane
// hashes its own row of slice s.  Rows are padded to 80 bytes, so the lanes that read at
// once use distinct banks.  A warp whose 32 leaves are whole, 16-byte aligned and from one
// buffer (every warp inside a large tensor) computes the copy addresses directly; other
// warps fetch each leaf's pointer and length from its lane.  Blocks of 8 warps hold 40 KB of
// staging; 64-byte slices in 8-warp blocks measured 4.40 TB/s against 4.28 with 128-byte
// slices in 4-warp blocks and 4.00 with 256-byte slices (1 GiB of leaves, GB300).
constexpr int kFnvWarps = 8;
constexpr int kSlice = 64;
constexpr int kSliceStride = kSlice + 16;
constexpr int kLanesPerLeaf = kSlice / 16;
constexpr int kLeavesPerRound = 32 / kLanesPerLeaf;

__device__ __forceinline__ void fnv_stage_fast(uint8_t (*dst)[kSliceStride], const uint8_t *wbase, uint32_t s0,
                                               int lane) {
  const int sub = lane / kLanesPerLeaf, q = lane % kLanesPerLeaf;
  const uint8_t *src = wbase + (size_t)sub * kLeafBytes + s0 + q * 16;
#pragma unroll
  for (int r = 0; r < 32; r += kLeavesPerRound)
    cp_async16(smem_u32(&dst[r + sub][q * 16]), src + (size_t)r * kLeafBytes);
  cp_async_commit();
}

__device__ __forceinline__ void fnv_stage(uint8_t (*dst)[kSliceStride], const uint8_t *lp, uint32_t llen,
                                          uint32_t s0, int lane) {
  const int sub = lane / kLanesPerLeaf, q = lane % kLanesPerLeaf;
#pragma unroll 2
  for (int r = 0; r < 32; r += kLeavesPerRound) {
    const int src = r + sub;
    const uint8_t *p = reinterpret_cast<const uint8_t *>(__shfl_sync(0xffffffffu, (unsigned long long)lp, src));
    const uint32_t n = __shfl_sync(0xffffffffu, llen, src);
    const uint32_t o = s0 + q * 16;
    uint8_t *d = &dst[src][q * 16];
    if (p != nullptr && o < n) {
      if (o + 16 <= n && ((reinterpret_cast<uintptr_t>(p) + o) & 15) == 0) {
        cp_async16(smem_u32(d), p + o);
      } else {
        for (uint32_t k = 0; k < 16 && o + k < n; ++k) d[k] = p[o + k];
      }
    }
  }
  cp_async_commit();
}

__global__ void __launch_bounds__(kFnvWarps * 32) fnv_leaf_kernel(const __grid_constant__ FnvBatch b,
                                                                   uint64_t *leaves) {
  __shared__ __align__(16) uint8_t buf[kFnvWarps][2][32][kSliceStride];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t total = b.leaf_prefix[b.n];
  const uint64_t nwarps = (uint64_t)gridDim.x * kFnvWarps;
  for (uint64_t base = ((uint64_t)blockIdx.x * kFnvWarps + warp) * 32; base < total; base += nwarps * 32) {
    const uint64_t leaf = base + lane;
    const bool mine = leaf < total;
    const uint8_t *lp = nullptr;
    uint32_t llen = 0, t = 0xffffffffu;
    if (mine) {
      t = find_buf(b, leaf);
      const uint64_t off = (leaf - b.leaf_prefix[t]) * kLeafBytes;
      lp = b.ptr[t] + off;
      llen = (uint32_t)min(kLeafBytes, b.nbytes[t] - off);
    }
    const uint32_t t0 = __shfl_sync(0xffffffffu, t, 0);
    const bool fast = __all_sync(0xffffffffu, mine && t == t0 && llen == kLeafBytes &&
                                                   (reinterpret_cast<uintptr_t>(lp) & 15) == 0);
    const uint8_t *wbase = reinterpret_cast<const uint8_t *>(__shfl_sync(0xffffffffu, (unsigned long long)lp, 0));
    // slices the longest leaf of the warp needs (warp-uniform)
    const uint32_t nsl = (__reduce_max_sync(0xffffffffu, llen) + kSlice - 1) / kSlice;
    Fnv h;
    if (nsl) {
      if (fast) fnv_stage_fast(buf[warp][0], wbase, 0, lane);
      else fnv_stage(buf[warp][0], lp, llen, 0, lane);
    }
    for (uint32_t si = 0; si < nsl; ++si) {
      if (si + 1 < nsl) {
        if (fast) fnv_stage_fast(buf[warp][(si + 1) & 1], wbase, (si + 1) * kSlice, lane);
        else fnv_stage(buf[warp][(si + 1) & 1], lp, llen, (si + 1) * kSlice, lane);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      __syncwarp();
      const uint32_t s0 = si * kSlice;
      if (mine && s0 < llen) {
        const uint32_t m = min((uint32_t)kSlice, llen - s0);
        const uint8_t *row = buf[warp][si & 1][lane];
        uint32_t k = 0;
        for (; k + 16 <= m; k += 16) h.vec(*reinterpret_cast<const uint4 *>(row + k));
        for (; k < m; ++k) h.byte(row[k]);
      }
      __syncwarp();  // every lane is done with this buffer before it is refilled
    }
    if (mine) leaves[leaf] = h.value();
  }
}

// ---- second level: FNV-1a over LE64(nbytes), then the LE64 of each leaf digest
//
// The chain costs one dependent xor and 32 x 32 multiply per byte.  For a buffer of L
// leaves that is 8 L bytes in one thread (a 1 GB tensor: 2 MB of chain).  Larger buffers
// split the leaf stream into chunks of kChunkWords digests and combine them exactly in
// parallel, from three facts about one FNV step (all arithmetic mod 2^32):
//  1. the low byte of lo evolves on its own: l' = ((l ^ b) p) & 0xff;
//  2. lo ^ b = lo + d with d = (l ^ b) - l, so lo' = (lo + d) p, and over a chunk of m bytes
//     lo_end = p^m lo_start + B, where B depends only on the chunk's bytes and the low
//     byte of lo_start (so the chain run from lo = that low byte alone gives B);
//  3. hi' = hi p + t with t a function of lo and b alone, so hi_end = p^m hi_start + H,
//     where H is the chunk's hi run from 0 along the true lo sequence.
// Passes: (1) l_end for all 256 starting low bytes of every chunk; (2) per buffer, walk the
// chunks' low bytes through those tables; (3) per chunk, B from its starting low byte;
// (4) per buffer, lo at every chunk start (lo' = p^m lo + B); (5) per chunk, H from the true
// lo start; (6) per buffer, fold the H values into hi.  The result equals the serial chain
// bit for bit.

// p^e mod 2^32 by square and multiply
__device__ __forceinline__ uint32_t fnv_pow(uint32_t e) {
  uint32_t r = 1, q = kFnvP;
  for (; e; e >>= 1, q *= q)
    if (e & 1) r *= q;
  return r;
}

struct FnvScratch {
  uint64_t *leaves;   // [total leaves]
  uint8_t *ltab;      // [chunks][256]: low byte at the chunk's end per starting low byte
  uint32_t *lstart;   // [chunks]: low byte of lo at the chunk's start
  uint32_t *bpart;    // [chunks]: B
  uint32_t *lo_start; // [chunks]
  uint32_t *hpart;    // [chunks]: H
  uint64_t *head;     // [n]: hi << 32 | lo after LE64(nbytes); lo replaced by the final lo
};

__device__ __forceinline__ uint32_t find_chunk_buf(const FnvBatch &b, uint32_t c) {
  uint32_t lo = 0, hi = b.n - 1;
  while (lo < hi) {
    uint32_t mid = (lo + hi + 1) >> 1;
    if (b.chunk_prefix[mid] <= c) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Leaf digests [first, last) of chunk c.
__device__ __forceinline__ void chunk_range(const FnvBatch &b, uint32_t c, uint64_t &first, uint64_t &last) {
  const uint32_t t = find_chunk_buf(b, c);
  first = b.leaf_prefix[t] + (uint64_t)(c - b.chunk_prefix[t]) * kChunkWords;
  last = min(first + kChunkWords, b.leaf_prefix[t + 1]);
}

// Pass 1: one block of 64 threads per chunk, four starting low bytes per thread, two per
// register in 16-bit lanes: (u 0xb3) < 2^16 for u < 256 and 0xb3 = p mod 256, so one
// multiply advances two starts and the lanes never carry into each other.  The mask of one
// byte step merges with the xor of the next (one three-input logic op).  The chunk's
// digests are staged in shared memory and read as broadcasts.
__global__ void __launch_bounds__(64) fnv_table_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  __shared__ uint64_t words[kChunkWords];
  const uint32_t c = blockIdx.x, tid = threadIdx.x;
  uint64_t first, last;
  chunk_range(b, c, first, last);
  const uint32_t w = (uint32_t)(last - first);
  for (uint32_t i = tid; i < w; i += blockDim.x) words[i] = sc.leaves[first + i];
  __syncthreads();
  constexpr uint32_t kMask = 0x00ff00ffu;
  uint32_t r0 = tid | (tid + 64) << 16, r1 = (tid + 128) | (tid + 192) << 16;
  for (uint32_t i = 0; i < w; ++i) {
    const uint64_t v = words[i];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const uint32_t half = k < 4 ? (uint32_t)v : (uint32_t)(v >> 32);
      const uint32_t bb = __byte_perm(half, 0, 0x4040u | (k & 3) | (k & 3) << 8);  // b in both lanes
      r0 = ((r0 & kMask) ^ bb) * 0xb3u;
      r1 = ((r1 & kMask) ^ bb) * 0xb3u;
    }
  }
  uint8_t *lt = sc.ltab + (size_t)c * 256;
  lt[tid] = (uint8_t)r0;
  lt[tid + 64] = (uint8_t)(r0 >> 16);
  lt[tid + 128] = (uint8_t)r1;
  lt[tid + 192] = (uint8_t)(r1 >> 16);
}

// Serial chain over leaves [l0, l1) from state h; kCombineAhead digests are loaded ahead.
constexpr int kCombineAhead = 16;
template <class H>
__device__ __forceinline__ void fnv_leaf_run(H &h, const uint64_t *leaves, uint64_t l0, uint64_t l1) {
  uint64_t r[kCombineAhead];
#pragma unroll
  for (int j = 0; j < kCombineAhead; ++j) r[j] = l0 + j < l1 ? leaves[l0 + j] : 0;
  for (uint64_t l = l0; l < l1; l += kCombineAhead) {
#pragma unroll
    for (int j = 0; j < kCombineAhead; ++j) {
      if (l + j < l1) {
        const uint64_t v = r[j];
        const uint64_t ln = l + j + kCombineAhead;
        if (ln < l1) r[j] = leaves[ln];
        h.le64(v);
      }
    }
  }
}

// The low word alone (fact 2): what pass 3 needs.
struct FnvLo {
  uint32_t lo;
  __device__ __forceinline__ void le64(uint64_t v) {
#pragma unroll
    for (int k = 0; k < 8; ++k) lo = (lo ^ (uint32_t)((v >> (8 * k)) & 0xffu)) * kFnvP;
  }
};

// One warp per buffer.  Small buffers: lane 0 runs the whole chain.  Chunked buffers: pass 2,
// the low-byte walk, in lane 0, over table rows the warp copies into a shared-memory ring
// kWalkAhead chunks ahead (one lookup per chunk instead of one L2 round trip).
constexpr int kWalkAhead = 8;

__global__ void __launch_bounds__(32) fnv_combine_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  __shared__ __align__(16) uint8_t rows[kWalkAhead][256];
  const uint32_t t = blockIdx.x;
  const int lane = threadIdx.x;
  const uint64_t l0 = b.leaf_prefix[t], l1 = b.leaf_prefix[t + 1];
  const uint32_t c0 = b.chunk_prefix[t], c1 = b.chunk_prefix[t + 1];
  Fnv h;
  h.le64(b.nbytes[t]);
  if (c0 == c1) {
    if (lane == 0) {
      fnv_leaf_run(h, sc.leaves, l0, l1);
      *b.out[t] = h.value();
    }
    return;
  }
  const uint32_t nc = c1 - c0;
  // row of chunk c0 + j into slot j % kWalkAhead; one commit group per call, empty past the end
  auto fetch = [&](uint32_t j) {
    if (j < nc && lane < 16)
      cp_async16(smem_u32(rows[j % kWalkAhead] + lane * 16), sc.ltab + (size_t)(c0 + j) * 256 + lane * 16);
    cp_async_commit();
  };
  for (uint32_t j = 0; j < (uint32_t)kWalkAhead; ++j) fetch(j);
  uint32_t l = h.lo & 0xffu;
  for (uint32_t j = 0; j < nc; ++j) {
    cp_async_wait<kWalkAhead - 1>();  // this lane's copy of row j has landed
    __syncwarp();                     // and every lane's
    if (lane == 0) {
      sc.lstart[c0 + j] = l;
      l = rows[j % kWalkAhead][l];
    }
    __syncwarp();  // lane 0 is done with slot j % kWalkAhead before it is refilled
    fetch(j + kWalkAhead);
  }
  cp_async_wait<0>();
  if (lane == 0) sc.head[t] = h.value();
}

// Pass 3: one thread per chunk, the low word from its starting low byte: B = lo_end - p^m l.
__global__ void fnv_bpart_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  const uint32_t c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= b.chunk_prefix[b.n]) return;
  uint64_t first, last;
  chunk_range(b, c, first, last);
  const uint32_t l = sc.lstart[c];
  FnvLo h{l};
  fnv_leaf_run(h, sc.leaves, first, last);
  sc.bpart[c] = h.lo - fnv_pow(8 * (uint32_t)(last - first)) * l;
}

// Pass 4: one thread per chunked buffer, lo at every chunk start.
__global__ void fnv_scan_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= b.n) return;
  const uint32_t c0 = b.chunk_prefix[t], c1 = b.chunk_prefix[t + 1];
  if (c0 == c1) return;
  const uint64_t l0 = b.leaf_prefix[t], l1 = b.leaf_prefix[t + 1];
  const uint32_t pfull = fnv_pow(8 * kChunkWords);
  const uint64_t head = sc.head[t];
  uint32_t lo = (uint32_t)head;
  for (uint32_t c = c0; c < c1; ++c) {
    sc.lo_start[c] = lo;
    const uint64_t first = l0 + (uint64_t)(c - c0) * kChunkWords;
    const uint32_t w = (uint32_t)min((uint64_t)kChunkWords, l1 - first);
    lo = (w == kChunkWords ? pfull : fnv_pow(8 * w)) * lo + sc.bpart[c];
  }
  sc.head[t] = (head & 0xffffffff00000000ull) | lo;
}

// Pass 5: one thread per chunk, the exact chain from (lo_start, 0).
__global__ void fnv_exact_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  const uint32_t c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= b.chunk_prefix[b.n]) return;
  uint64_t first, last;
  chunk_range(b, c, first, last);
  Fnv h;
  h.lo = sc.lo_start[c];
  h.hi = 0;
  fnv_leaf_run(h, sc.leaves, first, last);
  sc.hpart[c] = h.hi;
}

// Pass 6: one thread per chunked buffer, hi folded over its chunks.
__global__ void fnv_finish_kernel(const __grid_constant__ FnvBatch b, FnvScratch sc) {
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= b.n) return;
  const uint32_t c0 = b.chunk_prefix[t], c1 = b.chunk_prefix[t + 1];
  if (c0 == c1) return;
  const uint64_t l0 = b.leaf_prefix[t], l1 = b.leaf_prefix[t + 1];
  const uint32_t pfull = fnv_pow(8 * kChunkWords);
  const uint64_t head = sc.head[t];
  uint32_t hi = (uint32_t)(head >> 32);
  for (uint32_t c = c0; c < c1; ++c) {
    const uint64_t first = l0 + (uint64_t)(c - c0) * kChunkWords;
    const uint32_t w = (uint32_t)min((uint64_t)kChunkWords, l1 - first);
    hi = (w == kChunkWords ? pfull : fnv_pow(8 * w)) * hi + sc.hpart[c];
  }
  *b.out[t] = ((uint64_t)hi << 32) | (uint32_t)head;
}

// One thread per buffer: the literal serial FNV-1a-64.
__global__ void fnv_plain_kernel(const __grid_constant__ FnvBatch b) {
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= b.n) return;
  const uint8_t *p = b.ptr[t];
  const uint64_t n = b.nbytes[t];
  Fnv h;
  uint64_t i = 0;
  // bytes up to the first 16-byte boundary, then vectors, then the tail
  while (i < n && ((reinterpret_cast<uintptr_t>(p) + i) & 15) != 0) h.byte(p[i++]);
  const uint4 *v = reinterpret_cast<const uint4 *>(p + i);
  const uint64_t nv = (n - i) >> 4;
  for (uint64_t k = 0; k < nv; ++k) h.vec(v[k]);
  for (i += nv << 4; i < n; ++i) h.byte(p[i]);
  *b.out[t] = h.value();
}

}  // namespace

static size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Scratch layout of one batch: leaves, ltab, lstart, bpart, lo_start, hpart, head
// (256-byte aligned).
static FnvScratch fnv_layout(const FnvBatch &b, void *base, size_t *bytes) {
  const uint64_t L = b.leaf_prefix[b.n];
  const uint64_t C = b.chunk_prefix[b.n];
  constexpr int kParts = 7;
  const size_t len[kParts] = {L * 8, C * 256, C * 4, C * 4, C * 4, C * 4, (size_t)b.n * 8};
  size_t off[kParts];
  size_t o = 0;
  for (int i = 0; i < kParts; ++i) {
    off[i] = o;
    o = align256(o + len[i]);
  }
  if (bytes) *bytes = o;
  FnvScratch sc;
  const uintptr_t p = reinterpret_cast<uintptr_t>(base);
  sc.leaves = reinterpret_cast<uint64_t *>(p + off[0]);
  sc.ltab = reinterpret_cast<uint8_t *>(p + off[1]);
  sc.lstart = reinterpret_cast<uint32_t *>(p + off[2]);
  sc.bpart = reinterpret_cast<uint32_t *>(p + off[3]);
  sc.lo_start = reinterpret_cast<uint32_t *>(p + off[4]);
  sc.hpart = reinterpret_cast<uint32_t *>(p + off[5]);
  sc.head = reinterpret_cast<uint64_t *>(p + off[6]);
  return sc;
}

size_t fnv_fill_batch(FnvBatch &b, const void *const *ptr, const uint64_t *nbytes, uint64_t *const *out, size_t n) {
  memset(&b, 0, sizeof b);
  b.n = (uint32_t)n;
  uint64_t leaves = 0;
  uint32_t chunks = 0;
  for (size_t k = 0; k < n; ++k) {
    b.leaf_prefix[k] = leaves;
    b.chunk_prefix[k] = chunks;
    b.ptr[k] = static_cast<const uint8_t *>(ptr[k]);
    b.nbytes[k] = nbytes[k];
    b.out[k] = out[k];
    const uint64_t l = (nbytes[k] + kLeafBytes - 1) / kLeafBytes;
    leaves += l;
    if (l > kParallelLeaves) chunks += (uint32_t)((l + kChunkWords - 1) / kChunkWords);
  }
  b.leaf_prefix[n] = leaves;
  b.chunk_prefix[n] = chunks;
  size_t bytes = 0;
  fnv_layout(b, nullptr, &bytes);
  return bytes;
}

int fnv_tree_launches(const FnvBatch &b) {
  if (b.n == 0) return 0;
  return (b.leaf_prefix[b.n] ? 1 : 0) + 1 + (b.chunk_prefix[b.n] ? 5 : 0);
}

cudaError_t launch_fnv_tree(const FnvBatch &b, void *scratch, cudaStream_t s) {
  if (b.n == 0) return cudaSuccess;
  const FnvScratch sc = fnv_layout(b, scratch, nullptr);
  const uint64_t total = b.leaf_prefix[b.n];
  const uint32_t chunks = b.chunk_prefix[b.n];
  cudaError_t e;
  if (total > 0) {
    const uint64_t warps = (total + 31) / 32;
    const uint64_t blocks = (warps + kFnvWarps - 1) / kFnvWarps;
    const uint64_t cap = (uint64_t)num_sms() * 24;
    fnv_leaf_kernel<<<(int)(blocks < cap ? blocks : cap), kFnvWarps * 32, 0, s>>>(b, sc.leaves);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (chunks) {
    fnv_table_kernel<<<chunks, 64, 0, s>>>(b, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  fnv_combine_kernel<<<b.n, 32, 0, s>>>(b, sc);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (chunks) {
    fnv_bpart_kernel<<<(chunks + 127) / 128, 128, 0, s>>>(b, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    fnv_scan_kernel<<<(b.n + 127) / 128, 128, 0, s>>>(b, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    fnv_exact_kernel<<<(chunks + 127) / 128, 128, 0, s>>>(b, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    fnv_finish_kernel<<<(b.n + 127) / 128, 128, 0, s>>>(b, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_fnv_plain(const FnvBatch &b, cudaStream_t s) {
  if (b.n == 0) return cudaSuccess;
  fnv_plain_kernel<<<(b.n + 63) / 64, 64, 0, s>>>(b);
  return cudaGetLastError();
}

}  // namespace wt
