// Multi-column GEMV on the 5th-generation tensor cores (tcgen05) for 2-byte weights:
// Y[t] = W X[t], t < T <= 16, the operation of gemm_cols_kernel (wt_cols.cu) with the
// accumulator in tensor memory and the MMA issued by one thread.
//
// A CTA owns row tiles of 128 rows (one UMMA M) and walks K in chunks of 64 elements:
//
//   producer warp   per stage, two TMA 2-D boxes on one mbarrier: the W tile (128 x 64,
//                   written in the 128-byte-swizzled K-major layout the MMA reads) and the X
//                   tile (16 x 64, same layout, columns past T zero-filled); ten stages keep
//                   160 KB of W in flight per SM
//   MMA thread      four tcgen05.mma kind::f16 (M 128, N 16, K 16) per stage into one of two
//                   TMEM accumulators; tcgen05.commit frees the stage and, after the last
//                   chunk, hands the accumulator to the epilogue
//   epilogue warps  tcgen05.ld (32 lanes x 16 columns per warp) and the stores of Y
//
// The tensor-core time does not grow with T (N = 16 always), so this kernel serves T > 8,
// where the warp-level MMA kernel slows down.  int8 weights stay on that kernel: their
// decode runs in registers there, while here it would have to pass through shared memory
// before every MMA (measured: 3.1 TB/s against 5.8-6.0 TB/s).
//
// Every mbarrier wait is bounded; a timeout records WT_ETIMEDOUT and every role stops.  The
// allocating warp frees the tensor memory after the whole CTA has synchronised.
#include "wt_device.cuh"
#include "wt_kernels.h"

namespace wt {

namespace {

constexpr int kUBM = 128;       // rows per tile (UMMA M)
constexpr int kUBK = 64;        // K elements per stage (128 bytes per row)
constexpr int kUBN = 16;        // X columns (UMMA N)
constexpr uint32_t kUATile = kUBM * kUBK * 2;   // 16 KB
constexpr uint32_t kUXTile = kUBN * kUBK * 2;   // 2 KB
constexpr uint32_t kUStage = kUATile + kUXTile;  // 18 KB
constexpr int kUStages = 10;
constexpr int kUThreads = 256;  // 8 warps: 0 producer, 1 MMA + TMEM, 4-7 epilogue
constexpr uint32_t kUTmemCols = 32;  // two accumulators of 16 fp32 columns
constexpr size_t kUBarOff = (size_t)kUStages * kUStage;
constexpr int kUBars = 2 * kUStages + 4;  // full, empty per stage; acc_full, acc_empty x 2
constexpr size_t kUSmem = kUBarOff + kUBars * 8 + 16 + 1024;  // + 1024 for alignment
static_assert(kUStage % 1024 == 0, "stages keep the 1024-byte alignment of the 128-byte swizzle");
static_assert(kUSmem <= 232448, "shared memory of one CTA");

__device__ __forceinline__ void tma_2d(uint32_t dst, const void *tmap, int32_t x, int32_t y, uint32_t bar,
                                       uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(tmap), "r"(x), "r"(y), "r"(bar), "l"(pol)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile in the 128-byte swizzled layout: rows of
// 128 bytes, 8-row groups 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sdesc(uint32_t addr) {
  return (uint64_t)((addr & 0x3FFFF) >> 4)      // start address
         | ((uint64_t)1 << 16)                  // leading byte offset (unused when swizzled)
         | ((uint64_t)(1024 >> 4) << 32)        // stride byte offset
         | ((uint64_t)1 << 46)                  // version
         | ((uint64_t)2 << 61);                 // 128-byte swizzle
}

// Instruction descriptor, kind::f16: fp32 accumulate, A and B of type ab (0 f16, 1 bf16),
// both K-major, N = 16, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t ab) {
  return (1u << 4) | (ab << 7) | (ab << 10) | ((uint32_t)(kUBN >> 3) << 17) | ((uint32_t)(kUBM >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

// 32 lanes x 16 consecutive fp32 columns of tensor memory: one row per thread of the warp.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
      "%14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

struct UTile {
  uint32_t mat, row0;
};

// Tile i of the launch (row tiles of all matrices in order): binary search over the prefix
// of tile counts kept in Piece.r0 of each matrix's piece (pieces[m] = {m, first tile, tiles}).
__device__ __forceinline__ UTile tile_of(const Piece *pieces, uint32_t nmat, uint32_t i) {
  uint32_t lo = 0, hi = nmat;
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) / 2;
    if (pieces[mid].r0 <= i) lo = mid;
    else hi = mid;
  }
  return {lo, (i - pieces[lo].r0) * (uint32_t)kUBM};
}

template <int DT>
__global__ void __launch_bounds__(kUThreads, 1)
    gemm_cols_umma_kernel(const MatDesc *__restrict__ mats, const Piece *__restrict__ pieces, uint32_t nmat,
                          uint32_t ntiles, int *status, const uint8_t *__restrict__ maps) {
  static_assert(DT == 1 || DT == 2, "2-byte weights only");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t *gbase = smem_raw + (base - smem_u32(smem_raw));
  const uint32_t full0 = base + (uint32_t)kUBarOff;
  const uint32_t empty0 = full0 + kUStages * 8;
  const uint32_t accf0 = empty0 + kUStages * 8;
  const uint32_t acce0 = accf0 + 2 * 8;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(gbase + kUBarOff + kUBars * 8);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kUStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf0 + 8 * b, 1);
      mbar_init(acce0 + 8 * b, 128);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kUTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- producer
    if (lane == 0) {
      const uint64_t pol = l2_evict_first_policy();
      uint32_t it = 0;
      bool live = true;
      for (uint32_t i = blockIdx.x; i < ntiles && live; i += gridDim.x) {
        const UTile t = tile_of(pieces, nmat, i);
        const MatDesc md = mats[t.mat];
        const uint8_t *wmap = maps + (size_t)t.mat * 2 * kTensorMapBytes;
        const uint8_t *xmap = wmap + kTensorMapBytes;
        const uint32_t nk = (md.V * 8 + kUBK - 1) / kUBK;
        for (uint32_t kc = 0; kc < nk; ++kc, ++it) {
          const uint32_t s = it % kUStages;
          if (it >= kUStages && !bounded_wait(empty0 + 8 * s, ((it / kUStages) - 1) & 1, abort_flag, status)) {
            live = false;
            break;
          }
          const uint32_t st = base + s * kUStage;
          const uint32_t bar = full0 + 8 * s;
          mbar_expect_tx(bar, kUStage);
          tma_2d(st, wmap, (int32_t)(kc * kUBK), (int32_t)t.row0, bar, pol);
          tma_2d(st + kUATile, xmap, (int32_t)(kc * kUBK), 0, bar, pol);
        }
      }
      if (*abort_flag) {
        // drain: copies of the last stages may still be landing
        const uint32_t first = it > (uint32_t)kUStages ? it - kUStages : 0;
        for (uint32_t j = first; j < it; ++j) {
          const long long t0 = clock64();
          while (!mbar_try_wait(full0 + 8 * (j % kUStages), (j / kUStages) & 1) && clock64() - t0 < kWaitCycles) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t kI = idesc_f16(DT == 1 ? 1u : 0u);
      uint32_t it = 0, tl = 0;
      bool live = true;
      for (uint32_t i = blockIdx.x; i < ntiles && live; i += gridDim.x, ++tl) {
        const UTile t = tile_of(pieces, nmat, i);
        const MatDesc md = mats[t.mat];
        const uint32_t nk = (md.V * 8 + kUBK - 1) / kUBK;
        const uint32_t buf = tl & 1;
        if (tl >= 2 && !bounded_wait(acce0 + 8 * buf, ((tl >> 1) - 1) & 1, abort_flag, status)) break;
        tc_fence_after();
        const uint32_t dacc = tmem + buf * kUBN;
        for (uint32_t kc = 0; kc < nk; ++kc, ++it) {
          const uint32_t s = it % kUStages;
          if (!bounded_wait(full0 + 8 * s, (it / kUStages) & 1, abort_flag, status)) {
            live = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = base + s * kUStage;
#pragma unroll
          for (int k = 0; k < kUBK / 16; ++k)
            umma(dacc, sdesc(st + k * 32), sdesc(st + kUATile + k * 32), kI, (kc | k) != 0);
          umma_commit(empty0 + 8 * s);  // the stage is free once these MMAs have read it
        }
        if (live) umma_commit(accf0 + 8 * buf);  // the accumulator is complete
      }
      // wait (bounded) for the last MMAs before the tensor memory can be released
      if (it > 0) {
        const uint32_t j = it - 1;
        const long long t0 = clock64();
        while (!mbar_try_wait(empty0 + 8 * (j % kUStages), (j / kUStages) & 1) && clock64() - t0 < kWaitCycles) {
        }
      }
    }
  } else if (warp >= 4) {
    // ---------------- epilogue: warp w reads lanes 32 (w % 4) .. +31 (rows of the tile)
    const uint32_t q = warp & 3;
    uint32_t tl = 0;
    for (uint32_t i = blockIdx.x; i < ntiles; i += gridDim.x, ++tl) {
      const uint32_t buf = tl & 1;
      if (!bounded_wait(accf0 + 8 * buf, (tl >> 1) & 1, abort_flag, status)) break;
      tc_fence_after();
      float v[16];
      tmem_ld16(tmem + ((q * 32u) << 16) + buf * kUBN, v);
      tc_fence_before();
      mbar_arrive(acce0 + 8 * buf);
      const UTile t = tile_of(pieces, nmat, i);
      const MatDesc md = mats[t.mat];
      const uint32_t row = t.row0 + q * 32 + lane;
      if (row < md.M) {
#pragma unroll
        for (int c = 0; c < kUBN; ++c)
          if ((uint32_t)c < md.G) md.y[(uint64_t)c * md.M + row] = v[c];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kUTmemCols) : "memory");
  }
}

}  // namespace

cudaError_t gemm_cols_umma_prepare() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(gemm_cols_umma_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kUSmem)) !=
      cudaSuccess)
    return e;
  return cudaFuncSetAttribute(gemm_cols_umma_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kUSmem);
}

cudaError_t launch_gemm_cols_umma(const UmmaLaunch &L, cudaStream_t s) {
  if (L.ntiles == 0) return cudaSuccess;
  if (L.maps == nullptr) return cudaErrorInvalidValue;
  switch (L.dtype) {
    case 1: gemm_cols_umma_kernel<1><<<L.grid, kUThreads, kUSmem, s>>>(L.mats, L.pieces, L.nmat, L.ntiles, L.status, L.maps); break;
    case 2: gemm_cols_umma_kernel<2><<<L.grid, kUThreads, kUSmem, s>>>(L.mats, L.pieces, L.nmat, L.ntiles, L.status, L.maps); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace wt
