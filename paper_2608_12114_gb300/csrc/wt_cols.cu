// Multi-column GEMV: Y[t, :] = diag(s) W X[t, :] for t < T <= 16 activation columns, every
// weight read once per pass and reused by all T columns (the paper's multi-column packed-int8
// kernel and its T-sweep, Sec. 4.3 / Sec. 6; speculative batches reuse each weight read).
//
// W streams HBM -> shared memory on an mbarrier ring of 2-D TMA tensor copies: one copy per
// stage brings a tile of 16 rows x vc 16-byte vectors (a box of the matrix seen as
// [M, 2V] 8-byte elements; rows and vectors past the end arrive as zeros).  Per-row 1-D
// copies of 1.5 KB were issue-bound near 3.4 TB/s; one box per 16 rows is not.  The row
// pitch vc * 16 is 64 bytes past a multiple of 128, so the two rows a quarter-warp reads
// fall in different banks.  Eight consumer warps split each tile
// along K and multiply on the tensor cores with warp-level m16n8k16 MMAs (fp32 accumulate):
//
//   A (16 x 16)  16 weight rows, decoded in registers (int8 -> exact f16; bf16/f16 as is)
//   B (16 x 8)   8 activation columns (two MMAs per A for T > 8)
//
// The sum over k does not depend on the order of k, so each thread's four k values of one
// MMA are four consecutive elements of one 16-byte weight vector, and its B values are the
// same four k of X: A and B fragments come straight from whole vector loads, and an int8
// word decodes into exactly the two f16x2 registers a fragment needs.
//
// Four 16-row tiles (two for int8 with T > 8) form a super block whose X registers are loaded
// once per K chunk.  At
// the end of a super block the warps' partial tiles meet in shared memory and are summed in
// warp order (deterministic; rows never depend on the partition across CTAs).
//
// Why warp-level MMAs and not tcgen05: the A operand is decoded from int8 in registers and
// goes to the MMA from there; tcgen05 takes A only from shared or tensor memory, which would
// add a store and a fence per decoded tile, and for T <= 16 the tensor rate is far from the
// bound either way (2 * 16 flops per weight byte at most).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "wt_device.cuh"
#include "wt_kernels.h"

namespace wt {

namespace {

constexpr int kColWarps = 8;  // consumer warps
constexpr int kColConsumers = kColWarps * 32;
constexpr int kColThreads = kColConsumers + 32;  // + one producer warp
constexpr int kColRows = kColTileRows;           // rows of one stage (one MMA tile)
constexpr int kColGroups = (kColVecMax / 4 + kColWarps - 1) / kColWarps;  // 4-vector groups per warp
constexpr uint32_t kColStageBytes = kColRows * kColVecMax * 16;
static_assert(kColVecMax % 8 == 4, "row pitch 64 bytes past a multiple of 128");
static_assert(kColStageBytes % 128 == 0, "stages stay 128-byte aligned for the tensor copies");

// Per-launch geometry: NT = 8-column MMA tiles (T <= 8: 1, else 2).  int8 weights run two
// CTAs per SM with half the ring each (the same bytes in flight per SM, twice the warps; the
// int8 path is latency-bound on its decode).  The cross-warp partials of one 16-row tile take
// 16 x 8 NT floats per warp, in two alternating halves.
template <int DT, int NT>
struct ColGeo {
  static constexpr int kCtasPerSm = DT == 3 ? 2 : 1;
  static constexpr int kStages = kCtasPerSm == 2 ? 3 : 6;
  // 16-row tiles per super block (X registers are loaded once per super block and chunk):
  // four, or two for int8 with 16 columns, which then fits two CTAs per SM (registers and
  // partial buffers halve; X is reloaded every 32 rows instead of 64)
  static constexpr int kBlocks = DT == 3 && NT == 2 ? 2 : 4;
  // accumulator sets per tile (even / odd k16 steps: shorter MMA chains); int8 with 16
  // columns keeps one, its two column tiles already give two independent chains per A
  static constexpr int kAcc = DT == 3 && NT == 2 ? 1 : 2;
  static constexpr int kSuper = kColRows * kBlocks;
  static constexpr uint32_t kRedStride = 128 * NT;  // floats per (tile, warp)
  static constexpr size_t kRedFloats = (size_t)kBlocks * kColWarps * kRedStride;  // one half
  static constexpr size_t kRedOff = (size_t)kStages * kColStageBytes;
  static constexpr size_t kBarOff = kRedOff + 2 * kRedFloats * sizeof(float);
  static constexpr size_t kFlagOff = kBarOff + 2 * kStages * sizeof(uint64_t);
  static constexpr size_t kSmem = kFlagOff + 16;
};
static_assert(ColGeo<1, 2>::kSmem <= 232448 && 2 * (ColGeo<3, 1>::kSmem + 1024) <= 233472 &&
                  2 * (ColGeo<3, 2>::kSmem + 1024) <= 233472,
              "multi-column shared memory");

// 32-bit words of X per weight vector: 16 fp16 activations for an int8 vector, else 8.
template <int DT>
struct ColX {
  static constexpr int W = DT == 3 ? 8 : 4;
};

template <int DT>
__device__ __forceinline__ float col_scale(const uint8_t *s, uint64_t row) {
  if constexpr (DT == 3) return __half2float(reinterpret_cast<const __half *>(s)[row]);
  return 1.f;
}

// d += A B on one 16x8x16 tile; bf16 operands for DT 1, f16 otherwise.
template <int DT>
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  if constexpr (DT == 1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  } else {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
}

// The activations of weight vector `vec` (global vector index col * V + v) of one column.
template <int DT>
__device__ __forceinline__ void load_xvec(const uint8_t *X, uint64_t vec, bool ok, uint32_t (&xr)[ColX<DT>::W]) {
  const uint4 *p = reinterpret_cast<const uint4 *>(X) + (DT == 3 ? 2 * vec : vec);
  const uint4 a = ok ? __ldg(p) : make_uint4(0, 0, 0, 0);
  xr[0] = a.x;
  xr[1] = a.y;
  xr[2] = a.z;
  xr[3] = a.w;
  if constexpr (DT == 3) {
    const uint4 b = ok ? __ldg(p + 1) : make_uint4(0, 0, 0, 0);
    xr[4] = b.x;
    xr[5] = b.y;
    xr[6] = b.z;
    xr[7] = b.w;
  }
}

// 2-D tensor copy of one box into this CTA's shared memory, completion counted on `bar`.
// x (in 8-byte elements) is always a multiple of 2: 16-byte aligned.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void *tmap, int32_t x, int32_t y, uint32_t bar,
                                            uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(tmap), "r"(x), "r"(y), "r"(bar), "l"(pol)
      : "memory");
}

// One stage: rows g and g + 8 of the tile against this warp's vectors of the chunk.
// Thread (g, t) takes vector (q * warps + warp) * 4 + t of group q.
// The box holds vc vectors per row at pitch vc * 16; rows and vectors past the matrix are
// zeros, so only whole groups past vc are skipped.
template <int DT, int NT, int H>
__device__ __forceinline__ void cols_stage(uint32_t tile, uint32_t vc, int warp, uint32_t g, uint32_t t,
                                           const uint32_t (&xr)[kColGroups][NT][ColX<DT>::W], float (&acc)[H][NT][4]) {
  const uint32_t pitch = vc * 16;
#pragma unroll
  for (int q = 0; q < kColGroups; ++q) {
    const uint32_t v0 = (uint32_t)(q * kColWarps + warp) * 4;
    if (v0 >= vc) continue;  // warp-uniform: the box ends before this group
    const uint32_t v = v0 + t;
    const uint4 w0 = lds128(tile + g * pitch + v * 16);
    const uint4 w1 = lds128(tile + (g + 8) * pitch + v * 16);
    const uint32_t ra[4] = {w0.x, w0.y, w0.z, w0.w};
    const uint32_t rb[4] = {w1.x, w1.y, w1.z, w1.w};
    if constexpr (DT == 3) {
      // word j = weights k 4j..4j+3 of the vector; its activations are x words 2j, 2j+1
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t u0 = ra[j] ^ 0x80808080u, u1 = rb[j] ^ 0x80808080u;
        const uint32_t a0 = i8x2_to_f16x2(u0, 0x4140u), a2 = i8x2_to_f16x2(u0, 0x4342u);
        const uint32_t a1 = i8x2_to_f16x2(u1, 0x4140u), a3 = i8x2_to_f16x2(u1, 0x4342u);
#pragma unroll
        for (int n = 0; n < NT; ++n)
          mma16816<2>(acc[(j & 1) % H][n], a0, a1, a2, a3, xr[q][n][2 * j], xr[q][n][2 * j + 1]);
      }
    } else {
      // words 2s, 2s+1 = elements 4s..4s+3 of the vector
#pragma unroll
      for (int s = 0; s < 2; ++s) {
#pragma unroll
        for (int n = 0; n < NT; ++n)
          mma16816<DT>(acc[s % H][n], ra[2 * s], rb[2 * s], ra[2 * s + 1], rb[2 * s + 1], xr[q][n][2 * s],
                       xr[q][n][2 * s + 1]);
      }
    }
  }
}

struct Ring {
  uint32_t stage0, full0, empty0;
  volatile int *abort_flag;
  int *status;
};

// Consumer side of one piece (rows [r0, r1) of one matrix), NT = 8-column MMA tiles.
template <int DT, int NT>
__device__ __forceinline__ void cols_piece(const MatDesc &md, const Piece &pc, const Ring &R, float *red_base,
                                           uint32_t &it, uint32_t &par, int warp, int lane) {
  const uint32_t V = md.V, vc = md.vc, T = md.G;
  const uint32_t nchunk = (V + vc - 1) / vc;
  const uint32_t g = lane >> 2, t = lane & 3;
  const int ct = threadIdx.x;
  constexpr int kColBlocks = ColGeo<DT, NT>::kBlocks;
  constexpr int kColSuper = ColGeo<DT, NT>::kSuper;
  for (uint32_t sb = pc.r0; sb < pc.r1; sb += kColSuper) {
    const uint32_t rows = min((uint32_t)kColSuper, pc.r1 - sb);
    const uint32_t nrb = (rows + kColRows - 1) / kColRows;
    constexpr int H = ColGeo<DT, NT>::kAcc;
    float acc[kColBlocks][H][NT][4];
#pragma unroll
    for (int b = 0; b < kColBlocks; ++b)
#pragma unroll
      for (int h = 0; h < H; ++h)
#pragma unroll
        for (int n = 0; n < NT; ++n) acc[b][h][n][0] = acc[b][h][n][1] = acc[b][h][n][2] = acc[b][h][n][3] = 0.f;
    for (uint32_t c = 0; c < nchunk; ++c) {
      const uint32_t nv = min(vc, V - c * vc);
      uint32_t xr[kColGroups][NT][ColX<DT>::W];
#pragma unroll
      for (int q = 0; q < kColGroups; ++q) {
        const uint32_t v = (uint32_t)(q * kColWarps + warp) * 4 + t;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          const uint32_t col = g + 8 * n;
          load_xvec<DT>(md.x, (uint64_t)col * V + (uint64_t)c * vc + v, v < nv && col < T, xr[q][n]);
        }
      }
#pragma unroll
      for (int b = 0; b < kColBlocks; ++b) {
        if ((uint32_t)b < nrb) {
          const uint32_t s = it % ColGeo<DT, NT>::kStages;
          bounded_wait(R.full0 + 8 * s, (it / ColGeo<DT, NT>::kStages) & 1, R.abort_flag, R.status);
          cols_stage<DT, NT, H>(R.stage0 + s * kColStageBytes, vc, warp, g, t, xr, acc[b]);
          __syncwarp();
          if (lane == 0) mbar_arrive(R.empty0 + 8 * s);
          ++it;
        }
      }
    }
    // warp partials -> red[b][warp][col][row]; C fragment: (g, 2t), (g, 2t+1), (g+8, 2t), (g+8, 2t+1).
    // Two halves alternate, so one barrier per super block suffices: a half is rewritten
    // only after every thread has passed the next super block's barrier.
    constexpr uint32_t kStride = ColGeo<DT, NT>::kRedStride;
    float *red = red_base + par * ColGeo<DT, NT>::kRedFloats;
    par ^= 1;
#pragma unroll
    for (int b = 0; b < kColBlocks; ++b) {
      if ((uint32_t)b < nrb) {
        float *r = red + (b * kColWarps + warp) * kStride;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          const uint32_t c0 = 2 * t + 8 * n;
          r[c0 * 16 + g] = acc[b][0][n][0] + (H == 2 ? acc[b][H - 1][n][0] : 0.f);
          r[(c0 + 1) * 16 + g] = acc[b][0][n][1] + (H == 2 ? acc[b][H - 1][n][1] : 0.f);
          r[c0 * 16 + g + 8] = acc[b][0][n][2] + (H == 2 ? acc[b][H - 1][n][2] : 0.f);
          r[(c0 + 1) * 16 + g + 8] = acc[b][0][n][3] + (H == 2 ? acc[b][H - 1][n][3] : 0.f);
        }
      }
    }
    named_bar(1, kColConsumers);
    for (uint32_t o = ct; o < nrb * kStride; o += kColConsumers) {
      const uint32_t b = o / kStride, e = o % kStride, col = e >> 4, row = b * kColRows + (e & 15);
      if (col < T && row < rows) {
        const float *r = red + b * kColWarps * kStride + e;
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kColWarps; ++w) sum += r[w * kStride];
        md.y[(uint64_t)col * md.M + sb + row] = sum * col_scale<DT>(md.s, sb + row);
      }
    }
  }
}

template <int DT, int NT>
__global__ void __launch_bounds__(kColThreads, (ColGeo<DT, NT>::kCtasPerSm))
    gemm_cols_kernel(const MatDesc *__restrict__ mats, const Piece *__restrict__ pieces,
                     const uint32_t *__restrict__ begin, int *status, const uint8_t *__restrict__ maps) {
  using Geo = ColGeo<DT, NT>;
  constexpr int kColStages = Geo::kStages;
  extern __shared__ __align__(128) uint8_t smem[];
  Ring R;
  R.stage0 = smem_u32(smem);
  R.full0 = smem_u32(smem + Geo::kBarOff);
  R.empty0 = R.full0 + kColStages * 8;
  R.abort_flag = reinterpret_cast<volatile int *>(smem + Geo::kFlagOff);
  R.status = status;
  float *red = reinterpret_cast<float *>(smem + Geo::kRedOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t p0 = begin[blockIdx.x];
  const uint32_t p1 = begin[blockIdx.x + 1];

  if (threadIdx.x == 0) {
    for (int s = 0; s < kColStages; ++s) {
      mbar_init(R.full0 + 8 * s, 1);
      mbar_init(R.empty0 + 8 * s, kColWarps);
    }
    *R.abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();

  if (warp == kColWarps) {
    // ---------------- producer: one thread issues every bulk copy of the CTA
    if (lane == 0) {
      const uint64_t pol = l2_evict_first_policy();
      uint32_t it = 0;
      bool live = true;
      for (uint32_t pi = p0; pi < p1 && live; ++pi) {
        const Piece pc = pieces[pi];
        const MatDesc md = mats[pc.mat];
        const uint8_t *tmap = maps + (size_t)pc.mat * kTensorMapBytes;
        const uint32_t nchunk = (md.V + md.vc - 1) / md.vc;
        for (uint32_t sb = pc.r0; sb < pc.r1 && live; sb += Geo::kSuper) {
          const uint32_t rows = min((uint32_t)Geo::kSuper, pc.r1 - sb);
          const uint32_t nrb = (rows + kColRows - 1) / kColRows;
          for (uint32_t c = 0; c < nchunk && live; ++c) {
            for (uint32_t b = 0; b < nrb; ++b) {
              const uint32_t s = it % kColStages;
              if (it >= kColStages &&
                  !bounded_wait(R.empty0 + 8 * s, ((it / kColStages) - 1) & 1, R.abort_flag, status)) {
                live = false;
                break;
              }
              const uint32_t bar = R.full0 + 8 * s;
              mbar_expect_tx(bar, kColRows * md.vc * 16);  // the whole box, zero fill included
              tma_load_2d(R.stage0 + s * kColStageBytes, tmap, (int32_t)(2 * c * md.vc),
                          (int32_t)(sb + b * kColRows), bar, pol);
              ++it;
            }
          }
        }
      }
      if (!live || *R.abort_flag) {
        // drain: the copies of the last (up to kColStages) issued stages may still be in flight
        const uint32_t first = it > (uint32_t)kColStages ? it - kColStages : 0;
        for (uint32_t j = first; j < it; ++j) {
          const long long t0 = clock64();
          while (!mbar_try_wait(R.full0 + 8 * (j % kColStages), (j / kColStages) & 1) &&
                 clock64() - t0 < kWaitCycles) {
          }
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- consumers: 8 warps (every matrix of the launch has T <= 8 NT)
    uint32_t it = 0, par = 0;
    for (uint32_t pi = p0; pi < p1; ++pi) {
      const Piece pc = pieces[pi];
      const MatDesc md = mats[pc.mat];
      cols_piece<DT, NT>(md, pc, R, red, it, par, warp, lane);
    }
  }
  __syncthreads();
}

}  // namespace

int gemm_cols_ctas_per_sm(int dtype, int nt) { return dtype == 3 ? 2 : 1; }

template <int DT, int NT>
static cudaError_t cols_attr() {
  return cudaFuncSetAttribute(gemm_cols_kernel<DT, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)ColGeo<DT, NT>::kSmem);
}

cudaError_t gemm_cols_prepare() {
  cudaError_t e;
  if ((e = cols_attr<1, 1>()) != cudaSuccess || (e = cols_attr<1, 2>()) != cudaSuccess ||
      (e = cols_attr<2, 1>()) != cudaSuccess || (e = cols_attr<2, 2>()) != cudaSuccess ||
      (e = cols_attr<3, 1>()) != cudaSuccess)
    return e;
  return cols_attr<3, 2>();
}

template <int DT, int NT>
static void cols_launch(const GemvLaunch &L, cudaStream_t s) {
  gemm_cols_kernel<DT, NT><<<L.grid, kColThreads, ColGeo<DT, NT>::kSmem, s>>>(L.mats, L.pieces, L.begin, L.status,
                                                                             L.maps);
}

cudaError_t launch_gemm_cols(const GemvLaunch &L, cudaStream_t s) {
  if (L.maps == nullptr || (L.nt != 1 && L.nt != 2)) return cudaErrorInvalidValue;
  switch (L.dtype * 4 + L.nt) {
    case 1 * 4 + 1: cols_launch<1, 1>(L, s); break;
    case 1 * 4 + 2: cols_launch<1, 2>(L, s); break;
    case 2 * 4 + 1: cols_launch<2, 1>(L, s); break;
    case 2 * 4 + 2: cols_launch<2, 2>(L, s); break;
    case 3 * 4 + 1: cols_launch<3, 1>(L, s); break;
    case 3 * 4 + 2: cols_launch<3, 2>(L, s); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace wt
