// Multi-column GEMV for int8 weights with fp16 row scales and T > 8 activation columns,
// Y[t] = diag(s) W X[t] (the paper's multi-column packed-int8 kernel at the top of its
// T-sweep, Sec. 4.3), with every warp owning whole rows.
//
// The warp-MMA kernel (wt_cols.cu) splits K across its warps: each warp keeps the
// activations of its share of a K chunk in registers for every column, and the warps' partial
// tiles meet in shared memory at the end of each super block.  With 16 columns of fp16
// activations that register block is as large as the weights it multiplies, and the kernel
// runs latency-bound on reloading it (ncu at T = 16: 63 % DRAM, stalls on the X loads and on
// fixed-latency dependencies).  Here the roles turn around:
//
//   producer warp   per stage, one TMA 2-D box of W (128 rows x 192 int8: the row pitch of
//                   192 bytes puts the rows g and g + 1 a quarter-warp reads 64 bytes apart in
//                   the banks) and three boxes of X (16 columns x 64 fp16 each, 128-byte
//                   swizzle, columns past T zero-filled) on one mbarrier
//   8 MMA warps     warp w owns rows 16w .. 16w + 15 of the 128-row block for the whole of K:
//                   it decodes its two rows' int8 straight into f16 MMA operands, takes the B
//                   operand from the staged X, accumulates m16n8k16 MMAs in registers, and
//                   stores its 16 x T outputs itself after the last chunk
//
// so there is no X register block and no cross-warp reduction; the activations of a stage
// are read from shared memory by all eight warps.  As in wt_cols.cu, the four k values a
// thread holds in one MMA are four consecutive weights of one 16-byte vector and the same
// four activations of its column, since the sum over k does not depend on the order of k.
//
// Every mbarrier wait is bounded; a timeout records WT_ETIMEDOUT and every role stops.
#include <cuda_fp16.h>

#include "wt_device.cuh"
#include "wt_kernels.h"
#include "wt_q8rows.h"

namespace wt {

namespace {

constexpr int kQWarps = 8;                       // MMA warps
constexpr int kQThreads = (kQWarps + 1) * 32;    // + one producer warp
constexpr int kQRows = 16 * kQWarps;             // rows per block
constexpr int kQKc = 192;                        // int8 weights per row per stage
constexpr int kQSub = kQKc / 64;                 // X boxes per stage (64 fp16 = 128 bytes each)
constexpr uint32_t kQWBytes = kQRows * kQKc;     // 24 KB
constexpr uint32_t kQXBytes = kQSub * 16 * 128;  // 6 KB
constexpr uint32_t kQStage = kQWBytes + kQXBytes;
constexpr int kQStages = 3;
constexpr size_t kQBarOff = (size_t)kQStages * kQStage;
constexpr size_t kQFlagOff = kQBarOff + 2 * kQStages * sizeof(uint64_t);
constexpr size_t kQSmem = kQFlagOff + 16 + 1024;  // + 1024: the swizzled boxes sit 1024-aligned
static_assert(kQWBytes % 1024 == 0 && kQStage % 1024 == 0, "X boxes stay 1024-byte aligned");
static_assert(2 * (kQSmem + 1024) <= 233472, "two CTAs per SM");
static_assert(kQKc % 64 == 0 && (kQKc % 128) == 64, "row pitch 64 bytes past a multiple of 128");

__device__ __forceinline__ void tma_box(uint32_t dst, const void *tmap, int32_t x, int32_t y, uint32_t bar,
                                        uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(tmap), "r"(x), "r"(y), "r"(bar), "l"(pol)
      : "memory");
}

// L2 policy for the activations: every 128-row block of a matrix reads the same X again, so
// X stays in L2 while the weights stream past it with evict_first.
__device__ __forceinline__ uint64_t l2_evict_last_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ void mma_f16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                        uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// One stage for warp `warp`: rows 16 warp + g and + g + 8 of the W tile against the staged X.
// Thread (g, t) takes bytes [64q + 16t, 64q + 16t + 16) of each row for q < kQSub (four MMAs
// of four k each), and of X column c = g + 8n the same 16 activations: 32 bytes of row c of
// X box q, whose 16-byte chunks 2t and 2t + 1 the 128-byte swizzle has moved to chunk ^ (c & 7).
template <int NT>
__device__ __forceinline__ void q8rows_stage(uint32_t stage, int warp, uint32_t g, uint32_t t,
                                             float (&acc)[2][NT][4]) {
  const uint32_t wrow = stage + (uint32_t)(16 * warp + g) * kQKc;
  const uint32_t xs = stage + kQWBytes;
#pragma unroll
  for (int q = 0; q < kQSub; ++q) {
    const uint4 w0 = lds128(wrow + q * 64 + t * 16);
    const uint4 w1 = lds128(wrow + 8 * kQKc + q * 64 + t * 16);
    uint32_t xr[NT][8];
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      const uint32_t c = g + 8 * n;  // c & 7 == g
      const uint32_t rowb = xs + q * 2048 + c * 128;
      const uint4 x0 = lds128(rowb + (((2 * t) ^ g) << 4));
      const uint4 x1 = lds128(rowb + (((2 * t + 1) ^ g) << 4));
      xr[n][0] = x0.x, xr[n][1] = x0.y, xr[n][2] = x0.z, xr[n][3] = x0.w;
      xr[n][4] = x1.x, xr[n][5] = x1.y, xr[n][6] = x1.z, xr[n][7] = x1.w;
    }
    const uint32_t ra[4] = {w0.x, w0.y, w0.z, w0.w};
    const uint32_t rb[4] = {w1.x, w1.y, w1.z, w1.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      // word j = weights k 4j..4j+3 of the thread's 16; their activations are X words 2j, 2j+1
      const uint32_t u0 = ra[j] ^ 0x80808080u, u1 = rb[j] ^ 0x80808080u;
      const uint32_t a0 = i8x2_to_f16x2(u0, 0x4140u), a2 = i8x2_to_f16x2(u0, 0x4342u);
      const uint32_t a1 = i8x2_to_f16x2(u1, 0x4140u), a3 = i8x2_to_f16x2(u1, 0x4342u);
#pragma unroll
      for (int n = 0; n < NT; ++n) mma_f16(acc[j & 1][n], a0, a1, a2, a3, xr[n][2 * j], xr[n][2 * j + 1]);
    }
  }
}

template <int NT>
__global__ void __launch_bounds__(kQThreads, 2)
    gemm_q8_rows_kernel(const MatDesc *__restrict__ mats, const Piece *__restrict__ pieces,
                        const uint32_t *__restrict__ begin, int *status, const uint8_t *__restrict__ maps) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t *gbase = smem_raw + (base - smem_u32(smem_raw));
  const uint32_t full0 = base + (uint32_t)kQBarOff;
  const uint32_t empty0 = full0 + kQStages * 8;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(gbase + kQFlagOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t p0 = begin[blockIdx.x];
  const uint32_t p1 = begin[blockIdx.x + 1];

  if (threadIdx.x == 0) {
    for (int s = 0; s < kQStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kQWarps);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();

  if (warp == kQWarps) {
    // ---------------- producer: one thread issues every tensor copy of the CTA
    if (lane == 0) {
      const uint64_t pol = l2_evict_first_policy(), xpol = l2_evict_last_policy();
      uint32_t it = 0;
      bool live = true;
      for (uint32_t pi = p0; pi < p1 && live; ++pi) {
        const Piece pc = pieces[pi];
        const MatDesc md = mats[pc.mat];
        const uint8_t *tw = maps + (size_t)pc.mat * 2 * kTensorMapBytes;
        const uint8_t *tx = tw + kTensorMapBytes;
        const uint32_t K = md.V * 16;
        for (uint32_t rb = pc.r0; rb < pc.r1 && live; rb += kQRows) {
          for (uint32_t k0 = 0; k0 < K; k0 += kQKc) {
            const uint32_t s = it % kQStages;
            if (it >= kQStages && !bounded_wait(empty0 + 8 * s, ((it / kQStages) - 1) & 1, abort_flag, status)) {
              live = false;
              break;
            }
            const uint32_t bar = full0 + 8 * s;
            const uint32_t dst = base + s * kQStage;
            mbar_expect_tx(bar, kQStage);  // whole boxes, zero fill included
            tma_box(dst, tw, (int32_t)k0, (int32_t)rb, bar, pol);
#pragma unroll
            for (int q = 0; q < kQSub; ++q) tma_box(dst + kQWBytes + q * 2048, tx, (int32_t)(k0 + 64 * q), 0, bar, xpol);
            ++it;
          }
        }
      }
      if (!live || *abort_flag) {
        // drain: the copies of the last (up to kQStages) issued stages may still be in flight
        const uint32_t first = it > (uint32_t)kQStages ? it - kQStages : 0;
        for (uint32_t j = first; j < it; ++j) {
          const long long t0 = clock64();
          while (!mbar_try_wait(full0 + 8 * (j % kQStages), (j / kQStages) & 1) && clock64() - t0 < kWaitCycles) {
          }
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- MMA warps: warp owns 16 rows of every 128-row block
    const uint32_t g = lane >> 2, t = lane & 3;
    uint32_t it = 0;
    for (uint32_t pi = p0; pi < p1; ++pi) {
      const Piece pc = pieces[pi];
      const MatDesc md = mats[pc.mat];
      const uint32_t K = md.V * 16, T = md.G;
      for (uint32_t rb = pc.r0; rb < pc.r1; rb += kQRows) {
        float acc[2][NT][4];
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int n = 0; n < NT; ++n) acc[h][n][0] = acc[h][n][1] = acc[h][n][2] = acc[h][n][3] = 0.f;
        for (uint32_t k0 = 0; k0 < K; k0 += kQKc) {
          const uint32_t s = it % kQStages;
          bounded_wait(full0 + 8 * s, (it / kQStages) & 1, abort_flag, status);
          q8rows_stage<NT>(base + s * kQStage, warp, g, t, acc);
          __syncwarp();
          if (lane == 0) mbar_arrive(empty0 + 8 * s);
          ++it;
        }
        // C fragment: (g, 2t), (g, 2t + 1), (g + 8, 2t), (g + 8, 2t + 1) of each 8-column tile
        const uint32_t r0 = rb + 16 * warp + g, r1 = r0 + 8;
        const float s0 = r0 < md.M ? __half2float(reinterpret_cast<const __half *>(md.s)[r0]) : 0.f;
        const float s1 = r1 < md.M ? __half2float(reinterpret_cast<const __half *>(md.s)[r1]) : 0.f;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          const uint32_t c0 = 2 * t + 8 * n;
          if (r0 < md.M) {
            if (c0 < T) md.y[(uint64_t)c0 * md.M + r0] = (acc[0][n][0] + acc[1][n][0]) * s0;
            if (c0 + 1 < T) md.y[(uint64_t)(c0 + 1) * md.M + r0] = (acc[0][n][1] + acc[1][n][1]) * s0;
          }
          if (r1 < md.M) {
            if (c0 < T) md.y[(uint64_t)c0 * md.M + r1] = (acc[0][n][2] + acc[1][n][2]) * s1;
            if (c0 + 1 < T) md.y[(uint64_t)(c0 + 1) * md.M + r1] = (acc[0][n][3] + acc[1][n][3]) * s1;
          }
        }
      }
    }
  }
  __syncthreads();
}

template <int NT>
cudaError_t q8rows_attr() {
  return cudaFuncSetAttribute(gemm_q8_rows_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kQSmem);
}

}  // namespace

cudaError_t gemm_q8_rows_prepare() {
  cudaError_t e = q8rows_attr<1>();
  return e != cudaSuccess ? e : q8rows_attr<2>();
}

cudaError_t launch_gemm_q8_rows(const GemvLaunch &L, cudaStream_t s) {
  if (L.grid <= 0) return cudaSuccess;
  if (L.maps == nullptr) return cudaErrorInvalidValue;
  switch (L.nt) {
    case 1: gemm_q8_rows_kernel<1><<<L.grid, kQThreads, kQSmem, s>>>(L.mats, L.pieces, L.begin, L.status, L.maps); break;
    case 2: gemm_q8_rows_kernel<2><<<L.grid, kQThreads, kQSmem, s>>>(L.mats, L.pieces, L.begin, L.status, L.maps); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace wt
