// sm_103a kernels of the file-backed weight path.
//
//   gather_kernel      host-mapped file bytes -> HBM, 16-byte vector loads and
//                      stores (the ingest step: the copy the paper calls the
//                      ingestion tax, Sec. 1 and Sec. 2.2, done once at the
//                      host-link rate)
//   gemv_tma_kernel    y = W x per matrix, fp32 accumulate: the bandwidth-bound
//                      consumer pass (Sec. 3.1: one single-token GEMV per
//                      matrix).  W streams HBM -> shared memory through 1-D TMA
//                      bulk copies on an mbarrier ring; warps reduce with
//                      shuffles.  No tensor cores: ~1 flop per weight byte.
//
// The FNV-1a-64 digest kernels are in wt_fnv.cu.
//
// Every wait on an mbarrier is bounded (clock64 budget); a wait that runs out
// records WT_ETIMEDOUT in the caller's status word, makes every later wait of
// the CTA return at once, and the producer drains its own copies in flight
// before the CTA exits.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "wt_device.cuh"
#include "wt_kernels.h"

namespace wt {

namespace {

int g_num_sms[64] = {0};

// ------------------------------------------------------------------ element math
template <int DT>
struct Elem;
template <>
struct Elem<0> {  // f32
  static constexpr int kEPV = 4;
  __device__ static __forceinline__ void unpack(const uint4 &v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
  }
  __device__ static __forceinline__ float scalar(const uint8_t *p, uint64_t i) {
    uint32_t u = (uint32_t)p[4 * i] | ((uint32_t)p[4 * i + 1] << 8) | ((uint32_t)p[4 * i + 2] << 16) |
                 ((uint32_t)p[4 * i + 3] << 24);
    return __uint_as_float(u);
  }
};
template <>
struct Elem<1> {  // bf16: the high half of an IEEE single
  static constexpr int kEPV = 8;
  __device__ static __forceinline__ void unpack(const uint4 &v, float (&f)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
  __device__ static __forceinline__ float scalar(const uint8_t *p, uint64_t i) {
    uint32_t u = (uint32_t)p[2 * i] | ((uint32_t)p[2 * i + 1] << 8);
    return __uint_as_float(u << 16);
  }
};
template <>
struct Elem<2> {  // f16
  static constexpr int kEPV = 8;
  __device__ static __forceinline__ void unpack(const uint4 &v, float (&f)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __half2 h = *reinterpret_cast<const __half2 *>(&w[i]);
      float2 t = __half22float2(h);
      f[2 * i] = t.x;
      f[2 * i + 1] = t.y;
    }
  }
  __device__ static __forceinline__ float scalar(const uint8_t *p, uint64_t i) {
    uint16_t u = (uint16_t)(p[2 * i] | (p[2 * i + 1] << 8));
    return __half2float(__ushort_as_half(u));
  }
};

template <>
struct Elem<3> {  // int8 weights (their activations are f16, their rows carry f16 scales)
  static constexpr int kEPV = 16;
  __device__ static __forceinline__ float scalar(const uint8_t *p, uint64_t i) { return (float)(int8_t)p[i]; }
};

// Element type of x for weights of type DT: int8 weights take f16 activations.
template <int DT>
struct XElem {
  static constexpr int value = DT == 3 ? 2 : DT;
};

// x vectors a consumer thread keeps in registers (16-byte weight vectors it covers).  An
// int8 vector needs 32 bytes of f16 x, and the int8 kernel runs two CTAs per SM under a
// 96-register cap, so it keeps two (rows of up to 512 vectors; longer ones are segmented).
template <int DT>
struct XJ {
  static constexpr int value = DT == 3 ? 2 : 8;
};

// Vector counts above XJ never reach a kernel of that type (the planner keeps them out);
// clamping keeps every template instantiation inside the register array.
#define WT_NJC(n) ((n) <= XJ<DT>::value ? (n) : XJ<DT>::value)

// Row scale applied at the store: f16 per row for int8 weights, 1 otherwise.
template <int DT>
__device__ __forceinline__ float row_scale(const uint8_t *s, uint64_t row) {
  if constexpr (DT == 3) return s ? __half2float(reinterpret_cast<const __half *>(s)[row]) : 1.f;
  return 1.f;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ------------------------------------------------------------------ gather
__global__ void __launch_bounds__(256) gather_kernel(const __grid_constant__ GatherBatch b) {
  const uint64_t total = b.chunk_prefix[b.n];
  for (uint64_t c = blockIdx.x; c < total; c += gridDim.x) {
    // range holding chunk c (binary search over the prefix in parameter space)
    uint32_t lo = 0, hi = b.n - 1;
    while (lo < hi) {
      uint32_t mid = (lo + hi + 1) >> 1;
      if (b.chunk_prefix[mid] <= c) lo = mid; else hi = mid - 1;
    }
    const uint64_t off = (c - b.chunk_prefix[lo]) << kGatherChunkLog2;
    const uint64_t n = b.nbytes[lo];
    const uint64_t len = min((uint64_t)1 << kGatherChunkLog2, n - off);
    const uint8_t *src = b.src[lo] + off;
    uint8_t *dst = b.dst[lo] + off;
    if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0) {
      const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
      uint4 *d4 = reinterpret_cast<uint4 *>(dst);
      const uint32_t n16 = (uint32_t)(len >> 4);
      uint32_t i = threadIdx.x;
      const uint32_t st = blockDim.x;
      for (; i + 3 * st < n16; i += 4 * st) {
        uint4 a0 = s4[i], a1 = s4[i + st], a2 = s4[i + 2 * st], a3 = s4[i + 3 * st];
        d4[i] = a0;
        d4[i + st] = a1;
        d4[i + 2 * st] = a2;
        d4[i + 3 * st] = a3;
      }
      for (; i < n16; i += st) d4[i] = s4[i];
      for (uint32_t t = (n16 << 4) + threadIdx.x; t < len; t += st) dst[t] = src[t];
    } else {
      for (uint32_t t = threadIdx.x; t < len; t += blockDim.x) dst[t] = src[t];
    }
  }
}

// ------------------------------------------------------------------ GEMV
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kGemvThreads = kConsumers + 32;
constexpr int kRedRows = 64;  // rows whose warp partials are gathered before one cross-warp sum

// Shared-memory layout of one CTA: the stage ring, its full/empty barriers, the cross-warp
// partials and the abort flag.  int8 weights run two CTAs per SM with half the ring each
// (the same bytes in flight per SM, twice the warps: that path is latency-bound on its
// decode, not on HBM).
template <int DT>
struct GemvGeo {
  static constexpr int kCtasPerSm = DT == 3 ? 2 : 1;
  static constexpr int kStages = DT == 3 ? 3 : 6;
  static constexpr size_t kBarOff = (size_t)kStages * kStageBytes;
  static constexpr size_t kRedOff = kBarOff + 2 * kStages * sizeof(uint64_t);
  static constexpr size_t kFlagOff = kRedOff + 2 * kConsumerWarps * kRedRows * sizeof(float);
  static constexpr size_t kSmem = kFlagOff + 16;
};
static_assert(GemvGeo<1>::kSmem <= 232448 && 2 * (GemvGeo<3>::kSmem + 1024) <= 233472, "GEMV shared memory");

// Two fp32 values in one 64-bit register; fma.rn.f32x2 performs two independent
// round-to-nearest FMAs (the same arithmetic as two fmaf calls) in one instruction.
__device__ __forceinline__ uint64_t pack2(uint32_t lo, uint32_t hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ float sum2(uint64_t v) {
  uint32_t lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=r"(lo), "=r"(hi) : "l"(v));
  return __uint_as_float(lo) + __uint_as_float(hi);
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// A 16-byte vector as fp32 pairs (element 2i in the low half, 2i+1 in the high half).
// For int8 weights (DT 3) the unit is a quad instead: x is held as four f16 per 64-bit
// register, matching one 32-bit word of four weights (see dot16).
template <int DT>
struct Pairs {
  static constexpr int N = DT == 3 ? 4 : Elem<DT>::kEPV / 2;
  __device__ static __forceinline__ uint64_t get(const uint4 &v, int i) {
    const uint32_t w = i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
    if (DT == 1) return pack2(w << 16, w & 0xffff0000u);  // bf16
    if (DT == 2) {                                          // f16
      const float2 t = __half22float2(*reinterpret_cast<const __half2 *>(&w));
      return pack2(__float_as_uint(t.x), __float_as_uint(t.y));
    }
    return i == 0 ? pack2(v.x, v.y) : pack2(v.z, v.w);  // f32
  }
};

// c + a.lo * b.lo + a.hi * b.hi: fp16 operands, fp32 products and sums (fma.rn.f32.f16:
// the product of two f16 values is exact in fp32, one rounding per FMA).
__device__ __forceinline__ float fma_h2(uint32_t a, uint32_t b, float c) {
  float d;
  asm("{\n\t.reg .f16 al, ah, bl, bh;\n\t"
      "mov.b32 {al, ah}, %1;\n\t"
      "mov.b32 {bl, bh}, %2;\n\t"
      "fma.rn.f32.f16 %0, al, bl, %3;\n\t"
      "fma.rn.f32.f16 %0, ah, bh, %0;\n\t}"
      : "=f"(d)
      : "r"(a), "r"(b), "f"(c));
  return d;
}

// Four running fp32 partial sums of one row (two f32x2 registers).
struct Acc4 {
  uint64_t a = 0, b = 0;
  __device__ __forceinline__ float total() const { return sum2(a) + sum2(b); }
};

template <int DT>
__device__ __forceinline__ void dot16(const uint4 &w, const uint64_t (&xp)[Pairs<DT>::N], Acc4 &acc) {
  if constexpr (DT == 3) {
    // one word = four int8 weights -> two exact f16x2 words -> four mixed-precision FMAs
    uint32_t f[4];
    asm("mov.b64 {%0, %1}, %2;" : "=r"(f[0]), "=r"(f[1]) : "l"(acc.a));
    asm("mov.b64 {%0, %1}, %2;" : "=r"(f[2]), "=r"(f[3]) : "l"(acc.b));
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t u = ws[i] ^ 0x80808080u;
      const uint32_t h01 = i8x2_to_f16x2(u, 0x4140u);
      const uint32_t h23 = i8x2_to_f16x2(u, 0x4342u);
      float c = __uint_as_float(f[i]);
      c = fma_h2(h01, (uint32_t)xp[i], c);
      c = fma_h2(h23, (uint32_t)(xp[i] >> 32), c);
      f[i] = __float_as_uint(c);
    }
    acc.a = pack2(f[0], f[1]);
    acc.b = pack2(f[2], f[3]);
  } else {
#pragma unroll
    for (int i = 0; i < Pairs<DT>::N; ++i) {
      if (i & 1) acc.b = fma2(Pairs<DT>::get(w, i), xp[i], acc.b);
      else acc.a = fma2(Pairs<DT>::get(w, i), xp[i], acc.a);
    }
  }
}

template <int DT>
__device__ __forceinline__ void load_xpairs(const uint8_t *x, uint32_t v, bool ok, uint64_t (&xp)[Pairs<DT>::N]) {
  if constexpr (DT == 3) {
    // the 16 f16 activations of weight vector v: 32 bytes
    const uint4 a = ok ? __ldg(reinterpret_cast<const uint4 *>(x) + 2 * v) : make_uint4(0, 0, 0, 0);
    const uint4 b = ok ? __ldg(reinterpret_cast<const uint4 *>(x) + 2 * v + 1) : make_uint4(0, 0, 0, 0);
    xp[0] = pack2(a.x, a.y);
    xp[1] = pack2(a.z, a.w);
    xp[2] = pack2(b.x, b.y);
    xp[3] = pack2(b.z, b.w);
  } else {
    const uint4 t = ok ? __ldg(reinterpret_cast<const uint4 *>(x) + v) : make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int i = 0; i < Pairs<DT>::N; ++i) xp[i] = Pairs<DT>::get(t, i);
  }
}

// Sums N per-lane values (N a power of two) over the 32 lanes with N/2 + N/4 + ... + 1
// halving exchanges, then plain exchanges for the remaining offsets.  Afterwards every
// lane holds the full sum of value index lane >> (5 - log2 N).  Fixed data flow, so the
// result is deterministic.
template <int N>
__device__ __forceinline__ float transpose_reduce(float (&v)[N], int lane) {
  int o = 16;
#pragma unroll
  for (int n = N; n > 1; n >>= 1, o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int k = 0; k < n / 2; ++k) {
      const float send = up ? v[k] : v[k + n / 2];
      const float keep = up ? v[k + n / 2] : v[k];
      v[k] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  float t = v[0];
  for (; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  return t;
}

template <int N>
struct Log2 {
  static constexpr int value = N <= 1 ? 0 : 1 + Log2<(N > 1 ? N / 2 : 1)>::value;
};
template <>
struct Log2<1> {
  static constexpr int value = 0;
};

// Warp-rows tile: each warp owns whole rows, G lanes per row, NJ 16-byte vectors per
// lane per row.  U rows are loaded before any is used (latency of shared loads overlaps).
template <int DT, int NJ>
__device__ __forceinline__ void tile_warp_rows(uint32_t tile, uint32_t V, uint32_t nr, uint32_t G,
                                               uint32_t gl, uint32_t sub, uint32_t rpw, int warp, int lane,
                                               const uint64_t (&xp)[XJ<DT>::value][Pairs<DT>::N], float *y,
                                               const uint8_t *sr) {
  constexpr int U = NJ == 1 ? 8 : NJ == 2 ? 4 : (NJ <= 4 ? 2 : 1);
  const uint32_t step = kConsumerWarps * rpw;
  for (uint32_t base = warp * rpw; base < nr; base += U * step) {
    uint4 w[U][NJ];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t row = base + u * step + sub;
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        const uint32_t v = gl + j * G;
        w[u][j] = lds_or_zero(tile + (row * V + v) * 16, row < nr && v < V);
      }
    }
    float t[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      Acc4 acc;
#pragma unroll
      for (int j = 0; j < NJ; ++j) dot16<DT>(w[u][j], xp[j], acc);
      t[u] = acc.total();
    }
    if (G == 32) {
      const float sum = transpose_reduce<U>(t, lane);
      constexpr int L = Log2<U>::value;
      const uint32_t row = base + (uint32_t)(lane >> (5 - L)) * step;
      if ((lane & ((32 >> L) - 1)) == 0 && row < nr) y[row] = sum * row_scale<DT>(sr, row);
    } else {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        for (uint32_t o = G >> 1; o > 0; o >>= 1) t[u] += __shfl_xor_sync(0xffffffffu, t[u], o);
        const uint32_t row = base + u * step + sub;
        if (gl == 0 && row < nr) y[row] = t[u] * row_scale<DT>(sr, row);
      }
    }
  }
}

// Short-row tile (V <= 16 vectors): G = pow2ceil(V) lanes per row, one vector per lane,
// 32 / G rows per warp per sweep.  Eight sweeps are loaded before use and their
// reductions over the G lanes are unrolled, so the eight shuffle chains interleave.
template <int DT, int G>
__device__ __forceinline__ void tile_small_rows(uint32_t tile, uint32_t V, uint32_t nr, int warp, int lane,
                                                const uint64_t (&xp)[Pairs<DT>::N], float *y, const uint8_t *sr) {
  constexpr int RPW = 32 / G;
  constexpr int U = 8;
  const uint32_t gl = lane & (G - 1);
  const uint32_t sub = lane / G;
  const uint32_t step = kConsumerWarps * RPW;
  for (uint32_t base = warp * RPW; base < nr; base += U * step) {
    uint4 w[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t row = base + u * step + sub;
      w[u] = lds_or_zero(tile + (row * V + gl) * 16, row < nr && gl < V);
    }
    float t[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      Acc4 acc;
      dot16<DT>(w[u], xp, acc);
      t[u] = acc.total();
    }
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) {
#pragma unroll
      for (int u = 0; u < U; ++u) t[u] += __shfl_xor_sync(0xffffffffu, t[u], o);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t row = base + u * step + sub;
      if (gl == 0 && row < nr) y[row] = t[u] * row_scale<DT>(sr, row);
    }
  }
}

// Block-rows tile of exactly NR rows: all consumer threads share each row; thread ct
// holds vectors ct + 256 j.  Warp partials land in rb[q * warps + warp].
template <int DT, int NJ, int NR>
__device__ __forceinline__ void tile_block_rows(uint32_t tile, uint32_t V, int ct, int warp, int lane,
                                                const uint64_t (&xp)[XJ<DT>::value][Pairs<DT>::N], float *rb) {
  constexpr int NP = NR <= 1 ? 1 : NR <= 2 ? 2 : NR <= 4 ? 4 : 8;
  uint4 w[NR][NJ];
#pragma unroll
  for (int q = 0; q < NR; ++q) {
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
      const uint32_t v = ct + j * kConsumers;
      w[q][j] = lds_or_zero(tile + (q * V + v) * 16, j + 1 < NJ || v < V);
    }
  }
  float t[NP];
#pragma unroll
  for (int q = 0; q < NP; ++q) {
    t[q] = 0.f;
    if (q < NR) {
      Acc4 acc;
#pragma unroll
      for (int j = 0; j < NJ; ++j) dot16<DT>(w[q < NR ? q : 0][j], xp[j], acc);
      t[q] = acc.total();
    }
  }
  const float sum = transpose_reduce<NP>(t, lane);
  constexpr int L = Log2<NP>::value;
  const int q = lane >> (5 - L);
  if ((lane & ((32 >> L) - 1)) == 0 && q < NR) rb[q * kConsumerWarps + warp] = sum;
}

// Sum of the consumer warps' partials of one row, in warp order (deterministic).
__device__ __forceinline__ float sum_warps(const float *p) {
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) t += p[w];
  return t;
}

template <int DT>
__device__ __forceinline__ bool block_rows_dispatch(uint32_t nj, uint32_t nr, uint32_t tile, uint32_t V, int ct,
                                                    int warp, int lane, const uint64_t (&xp)[XJ<DT>::value][Pairs<DT>::N],
                                                    float *rb) {
#define WT_BR(NJ, NR) \
  case NJ * 8 + NR: tile_block_rows<DT, WT_NJC(NJ), NR>(tile, V, ct, warp, lane, xp, rb); return true;
  switch (nj * 8 + nr) {
    WT_BR(1, 1) WT_BR(1, 2) WT_BR(1, 3) WT_BR(1, 4) WT_BR(1, 5) WT_BR(1, 6) WT_BR(1, 7) WT_BR(1, 8)
    WT_BR(2, 1) WT_BR(2, 2) WT_BR(2, 3) WT_BR(2, 4) WT_BR(2, 5) WT_BR(2, 6) WT_BR(2, 7)
    WT_BR(3, 1) WT_BR(3, 2) WT_BR(3, 3)
    WT_BR(4, 1) WT_BR(4, 2)
    WT_BR(5, 1) WT_BR(6, 1) WT_BR(7, 1) WT_BR(8, 1)
    default: return false;
  }
#undef WT_BR
}

// Consumer warp 0 records when it saw its first and its latest stage land.
__device__ __forceinline__ void stamp_full(uint64_t *st, uint32_t it, int warp, int lane) {
  if (warp == 0 && lane == 0) {
    const uint64_t t = globaltimer_ns();
    if (it == 0) st[kStFirstFull] = t;
    st[kStLastFull] = t;
  }
}

// ST: the stamping instantiation, which also writes the per-CTA times of StampField to
// stamps[blockIdx.x * kStampFields ...]; otherwise identical.
template <int DT, bool ST>
__global__ void __launch_bounds__(kGemvThreads, GemvGeo<DT>::kCtasPerSm)
    gemv_tma_kernel(const MatDesc *__restrict__ mats, const Piece *__restrict__ pieces,
                    const uint32_t *__restrict__ begin, int *status, int stall, uint64_t *stamps) {
  constexpr int NP = Pairs<DT>::N;
  constexpr int kStages = GemvGeo<DT>::kStages;
  uint64_t *const st = ST ? stamps + (uint64_t)blockIdx.x * kStampFields : nullptr;
  if (ST && threadIdx.x == 0) {
    st[kStEntry] = globaltimer_ns();
    st[kStFirstCopy] = st[kStFirstFull] = st[kStLastFull] = 0;
  }
  extern __shared__ __align__(128) uint8_t smem[];
  const uint32_t stage0 = smem_u32(smem);
  const uint32_t full0 = smem_u32(smem + GemvGeo<DT>::kBarOff);
  const uint32_t empty0 = full0 + kStages * 8;
  float *red = reinterpret_cast<float *>(smem + GemvGeo<DT>::kRedOff);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + GemvGeo<DT>::kFlagOff);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t p0 = begin[blockIdx.x];
  const uint32_t p1 = begin[blockIdx.x + 1];

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kConsumerWarps);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();
  if (ST && threadIdx.x == 0) st[kStPrologue] = globaltimer_ns();
  // Up to here only the plan tables (written once, by the upload before the first launch) and
  // shared memory are touched, so under a programmatic launch this prologue may overlap the
  // previous kernel of the stream; W, x, y and the scales are read or written only after that
  // kernel has completed.  The next pass may then be launched at once: its CTAs take an SM
  // only as this grid leaves it.  Without a programmatic launch both are no-ops.
  griddep_wait();
  griddep_launch();
  if (ST && threadIdx.x == 0) st[kStOperands] = globaltimer_ns();

  if (warp == kConsumerWarps) {
    // ---------------- producer: one thread issues every bulk copy of the CTA
    if (lane == 0 && !stall) {
      const uint64_t pol = l2_evict_first_policy();
      uint32_t it = 0;
      bool live = true;
      for (uint32_t pi = p0; pi < p1 && live; ++pi) {
        const Piece pc = pieces[pi];
        const MatDesc md = mats[pc.mat];
        const uint64_t rowb = (uint64_t)md.rs * 16;  // row pitch (the full row for a column segment)
        const uint32_t vb = md.V * 16;                // tile rows sit at V * 16 pitch in shared memory
        for (uint32_t r = pc.r0; r < pc.r1 && live; r += md.rt) {
          const uint32_t nr = min(md.rt, pc.r1 - r);
          const uint32_t s = it % kStages;
          if (it >= kStages && !bounded_wait(empty0 + 8 * s, ((it / kStages) - 1) & 1, abort_flag, status)) {
            live = false;
            break;
          }
          const uint32_t dst = stage0 + s * kStageBytes;
          const uint32_t bar = full0 + 8 * s;
          if (ST && it == 0) st[kStFirstCopy] = globaltimer_ns();
          mbar_expect_tx(bar, nr * vb);
          if (md.rs == md.V) {
            bulk_g2s(dst, md.W + (uint64_t)r * rowb, nr * vb, bar, pol);  // contiguous rows: one copy
          } else {
            for (uint32_t q = 0; q < nr; ++q) bulk_g2s(dst + q * vb, md.W + (uint64_t)(r + q) * rowb, vb, bar, pol);
          }
          ++it;
        }
      }
      if (!live || *abort_flag) {
        // drain: the copies of the last (up to kStages) issued stages may still be in flight
        const uint32_t first = it > (uint32_t)kStages ? it - kStages : 0;
        for (uint32_t j = first; j < it; ++j) {
          const long long t0 = clock64();
          while (!mbar_try_wait(full0 + 8 * (j % kStages), (j / kStages) & 1) &&
                 clock64() - t0 < kWaitCycles) {
          }
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- consumers: 8 warps
    const int ct = threadIdx.x;  // 0..255
    uint32_t it = 0;
    int par = 0;
    uint64_t xp[XJ<DT>::value][NP];
    for (uint32_t pi = p0; pi < p1; ++pi) {
      const Piece pc = pieces[pi];
      const MatDesc md = mats[pc.mat];
      const uint32_t V = md.V;
      if (md.mode == kModeWarpRows) {
        const uint32_t G = md.G;
        const uint32_t gl = lane & (G - 1);
        const uint32_t sub = lane / G;
        const uint32_t rpw = 32 / G;
        const uint32_t nj = (V + G - 1) / G;
#pragma unroll
        for (int j = 0; j < XJ<DT>::value; ++j) {
          const uint32_t v = gl + j * G;
          load_xpairs<DT>(md.x, v, j < (int)nj && v < V, xp[j]);
        }
        for (uint32_t r = pc.r0; r < pc.r1; r += md.rt) {
          const uint32_t nr = min(md.rt, pc.r1 - r);
          const uint32_t s = it % kStages;
          bounded_wait(full0 + 8 * s, (it / kStages) & 1, abort_flag, status);
          if (ST) stamp_full(st, it, warp, lane);
          const uint32_t tile = stage0 + s * kStageBytes;
          float *y = md.y + r;
          const uint8_t *sr = md.s ? md.s + 2ull * r : nullptr;  // f16 row scales (int8 weights)
          if (G < 32) {
            switch (G) {
              case 1: tile_small_rows<DT, 1>(tile, V, nr, warp, lane, xp[0], y, sr); break;
              case 2: tile_small_rows<DT, 2>(tile, V, nr, warp, lane, xp[0], y, sr); break;
              case 4: tile_small_rows<DT, 4>(tile, V, nr, warp, lane, xp[0], y, sr); break;
              case 8: tile_small_rows<DT, 8>(tile, V, nr, warp, lane, xp[0], y, sr); break;
              default: tile_small_rows<DT, 16>(tile, V, nr, warp, lane, xp[0], y, sr); break;
            }
          } else switch (nj) {
            case 1: tile_warp_rows<DT, WT_NJC(1)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 2: tile_warp_rows<DT, WT_NJC(2)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 3: tile_warp_rows<DT, WT_NJC(3)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 4: tile_warp_rows<DT, WT_NJC(4)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 5: tile_warp_rows<DT, WT_NJC(5)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 6: tile_warp_rows<DT, WT_NJC(6)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            case 7: tile_warp_rows<DT, WT_NJC(7)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
            default: tile_warp_rows<DT, WT_NJC(8)>(tile, V, nr, G, gl, sub, rpw, warp, lane, xp, y, sr); break;
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(empty0 + 8 * s);
          ++it;
        }
      } else if (md.mode == kModeBlockRows) {
        // whole consumer group shares each row; one tile = up to kRowBlock full rows
        const uint32_t nj = (V + kConsumers - 1) / kConsumers;
#pragma unroll
        for (int j = 0; j < XJ<DT>::value; ++j) {
          const uint32_t v = ct + j * kConsumers;
          load_xpairs<DT>(md.x, v, j < (int)nj && v < V, xp[j]);
        }
        // Warp partials of up to kRedRows rows collect in one half of `red`; the consumer
        // group then synchronises once and sums them (one barrier per kRedRows rows).
        uint32_t g0 = pc.r0, gn = 0;
        for (uint32_t r = pc.r0; r < pc.r1; r += md.rt) {
          const uint32_t nr = min(md.rt, pc.r1 - r);
          const uint32_t s = it % kStages;
          bounded_wait(full0 + 8 * s, (it / kStages) & 1, abort_flag, status);
          if (ST) stamp_full(st, it, warp, lane);
          const uint32_t tile = stage0 + s * kStageBytes;
          float *rb = red + par * (kConsumerWarps * kRedRows) + gn * kConsumerWarps;
          if (!block_rows_dispatch<DT>(nj, nr, tile, V, ct, warp, lane, xp, rb) && ct == 0)
            atomicCAS(status, 0, -1);  // unreachable by construction of the plan
          __syncwarp();
          if (lane == 0) mbar_arrive(empty0 + 8 * s);
          ++it;
          gn += nr;
          if (r + nr >= pc.r1 || gn + md.rt > (uint32_t)kRedRows) {
            named_bar(1, kConsumers);
            const float *gb = red + par * (kConsumerWarps * kRedRows);
            for (uint32_t q = ct; q < gn; q += kConsumers) md.y[g0 + q] = sum_warps(gb + q * kConsumerWarps) * row_scale<DT>(md.s, g0 + q);
            par ^= 1;
            g0 += gn;
            gn = 0;
          }
        }
      }
    }
  }
  __syncthreads();
  if (ST && threadIdx.x == 0) {
    st[kStExit] = globaltimer_ns();
    st[kStSm] = sm_id();
  }
}

// Map endpoint: one lane group per row (G = pow2ceil(V) lanes for rows shorter than 32
// vectors, the whole warp otherwise); each lane keeps four 16-byte loads of the mapped rows
// in flight; x comes from L1/L2.  Link-bound by design (the weights never enter HBM).
template <int DT>
__global__ void __launch_bounds__(256) gemv_mapped_kernel(const MatDesc *__restrict__ mats,
                                                          const Piece *__restrict__ pieces,
                                                          const uint32_t *__restrict__ begin) {
  constexpr int NP = Pairs<DT>::N;
  constexpr int kWarps = 8;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (uint32_t pi = begin[blockIdx.x]; pi < begin[blockIdx.x + 1]; ++pi) {
    const Piece pc = pieces[pi];
    const MatDesc md = mats[pc.mat];
    const uint32_t V = md.V;
    const uint32_t G = V >= 32 ? 32u : (V <= 1 ? 1u : 1u << (32 - __clz(V - 1)));
    const uint32_t gl = lane & (G - 1), sub = lane / G, rpw = 32 / G;
    for (uint32_t base = pc.r0 + warp * rpw; base < pc.r1; base += kWarps * rpw) {
      const uint32_t row = base + sub;
      const bool valid = row < pc.r1;
      const uint4 *w4 = reinterpret_cast<const uint4 *>(md.W + (uint64_t)(valid ? row : pc.r0) * V * 16);
      Acc4 acc;
      for (uint32_t v = gl; v < V; v += 4 * G) {
        uint4 w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t vv = v + u * G;
          w[u] = (valid && vv < V) ? w4[vv] : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t vv = v + u * G;
          uint64_t xp[NP];
          load_xpairs<DT>(md.x, vv, vv < V, xp);
          dot16<DT>(w[u], xp, acc);
        }
      }
      float t = acc.total();
      for (uint32_t o = G >> 1; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
      if (valid && gl == 0) md.y[row] = t * row_scale<DT>(md.s, row);
    }
  }
}

// Map endpoint with T activation columns: the one-column mapped kernel's loads of W, each
// vector multiplied against every column's x (from L1/L2) into its own accumulators; the
// link-bound W stream is read once for all T columns.
template <int DT>
__global__ void __launch_bounds__(256, 1) gemv_mapped_cols_kernel(const MatDesc *__restrict__ mats,
                                                               const Piece *__restrict__ pieces,
                                                               const uint32_t *__restrict__ begin) {
  constexpr int NP = Pairs<DT>::N;
  constexpr int kWarps = 8;
  constexpr int kMaxT = 16;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (uint32_t pi = begin[blockIdx.x]; pi < begin[blockIdx.x + 1]; ++pi) {
    const Piece pc = pieces[pi];
    const MatDesc md = mats[pc.mat];
    const uint32_t V = md.V, T = md.cols;
    const uint64_t xstride = (uint64_t)V * (DT == 3 ? 32 : 16);  // bytes of one x column
    const uint32_t G = V >= 32 ? 32u : (V <= 1 ? 1u : 1u << (32 - __clz(V - 1)));
    const uint32_t gl = lane & (G - 1), sub = lane / G, rpw = 32 / G;
    for (uint32_t base = pc.r0 + warp * rpw; base < pc.r1; base += kWarps * rpw) {
      const uint32_t row = base + sub;
      const bool valid = row < pc.r1;
      const uint4 *w4 = reinterpret_cast<const uint4 *>(md.W + (uint64_t)(valid ? row : pc.r0) * V * 16);
      Acc4 acc[kMaxT];
      for (uint32_t v = gl; v < V; v += 4 * G) {
        uint4 w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t vv = v + u * G;
          w[u] = (valid && vv < V) ? w4[vv] : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t vv = v + u * G;
          // decode the vector once (int8: exact f16x2 words; else fp32 pairs), use it T times
          uint32_t dh[8];
          uint64_t dp[NP];
          if constexpr (DT == 3) {
            const uint32_t ws[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const uint32_t q = ws[i] ^ 0x80808080u;
              dh[2 * i] = i8x2_to_f16x2(q, 0x4140u);
              dh[2 * i + 1] = i8x2_to_f16x2(q, 0x4342u);
            }
          } else {
#pragma unroll
            for (int i = 0; i < NP; ++i) dp[i] = Pairs<DT>::get(w[u], i);
          }
#pragma unroll
          for (int t = 0; t < kMaxT; ++t) {
            if ((uint32_t)t < T) {
              uint64_t xp[NP];
              load_xpairs<DT>(md.x + t * xstride, vv, vv < V, xp);
              if constexpr (DT == 3) {
                uint32_t f[4];
                asm("mov.b64 {%0, %1}, %2;" : "=r"(f[0]), "=r"(f[1]) : "l"(acc[t].a));
                asm("mov.b64 {%0, %1}, %2;" : "=r"(f[2]), "=r"(f[3]) : "l"(acc[t].b));
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  float c = __uint_as_float(f[i]);
                  c = fma_h2(dh[2 * i], (uint32_t)xp[i], c);
                  c = fma_h2(dh[2 * i + 1], (uint32_t)(xp[i] >> 32), c);
                  f[i] = __float_as_uint(c);
                }
                acc[t].a = pack2(f[0], f[1]);
                acc[t].b = pack2(f[2], f[3]);
              } else {
#pragma unroll
                for (int i = 0; i < NP; ++i) {
                  if (i & 1) acc[t].b = fma2(dp[i], xp[i], acc[t].b);
                  else acc[t].a = fma2(dp[i], xp[i], acc[t].a);
                }
              }
            }
          }
        }
      }
      const float sc = valid ? row_scale<DT>(md.s, row) : 0.f;
#pragma unroll
      for (int t = 0; t < kMaxT; ++t) {
        if ((uint32_t)t < T) {
          float r = acc[t].total();
          for (uint32_t o = G >> 1; o > 0; o >>= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
          if (valid && gl == 0) md.y[(uint64_t)t * md.M + row] = r * sc;
        }
      }
    }
  }
}

// Fallback: one warp per row, byte-assembled scalar loads (any alignment).  Column c of a
// multi-column call reads x + c * K elements and writes y + c * M.
template <int DT>
__global__ void gemv_generic_kernel(const uint8_t *W, const uint8_t *x, float *y, uint64_t M,
                                    uint64_t K, const uint8_t *s, uint32_t cols) {
  const uint64_t warps = (uint64_t)gridDim.x * (blockDim.x >> 5);
  const int lane = threadIdx.x & 31;
  constexpr int kXes = 16 / Elem<XElem<DT>::value>::kEPV;
  for (uint64_t row = (uint64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < M;
       row += warps) {
    const uint8_t *wr = W + row * K * (uint64_t)(16 / Elem<DT>::kEPV);
    for (uint32_t c = 0; c < cols; ++c) {
      const uint8_t *xc = x + (uint64_t)c * K * kXes;
      float acc = 0.f;
      for (uint64_t k = lane; k < K; k += 32)
        acc = fmaf(Elem<DT>::scalar(wr, k), Elem<XElem<DT>::value>::scalar(xc, k), acc);
      acc = warp_sum(acc);
      if (lane == 0) y[(uint64_t)c * M + row] = acc * row_scale<DT>(s, row);
    }
  }
}

// Second pass of cross-CTA split-K: one thread per output row, segments summed in order.
__global__ void seg_reduce_kernel(const SegReduce *__restrict__ tab) {
  const SegReduce r = tab[blockIdx.y];
  const uint32_t row = blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= r.M) return;
  float sum = 0.f;
  for (uint32_t k = 0; k < r.nseg; ++k) sum += r.ws[(uint64_t)k * r.M + row];
  r.y[row] = r.s ? sum * __half2float(reinterpret_cast<const __half *>(r.s)[row]) : sum;
}

}  // namespace

// ------------------------------------------------------------------ launchers
int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (g_num_sms[dev] == 0) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    g_num_sms[dev] = n > 0 ? n : 1;
  }
  return g_num_sms[dev];
}

cudaError_t launch_gather(const GatherBatch &b, int grid, cudaStream_t s) {
  if (b.n == 0 || b.chunk_prefix[b.n] == 0) return cudaSuccess;
  gather_kernel<<<grid, 256, 0, s>>>(b);
  return cudaGetLastError();
}

size_t gemv_smem_bytes(int dtype) { return dtype == 3 ? GemvGeo<3>::kSmem : GemvGeo<1>::kSmem; }
int gemv_ctas_per_sm(int dtype) { return dtype == 3 ? GemvGeo<3>::kCtasPerSm : GemvGeo<1>::kCtasPerSm; }

template <int DT>
static cudaError_t gemv_attr() {
  const cudaError_t e =
      cudaFuncSetAttribute(gemv_tma_kernel<DT, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)GemvGeo<DT>::kSmem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemv_tma_kernel<DT, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)GemvGeo<DT>::kSmem);
}

cudaError_t gemv_prepare() {
  cudaError_t e;
  if ((e = gemv_attr<0>()) != cudaSuccess || (e = gemv_attr<1>()) != cudaSuccess || (e = gemv_attr<2>()) != cudaSuccess)
    return e;
  return gemv_attr<3>();
}

// With L.pdl the launch carries programmatic stream serialization: inside a captured graph of
// consecutive passes, the next pass's launch and prologue overlap the tail of the one before;
// the kernel waits for that one's completion before it touches any operand.
template <int DT>
static cudaError_t gemv_launch(const GemvLaunch &L, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)L.grid);
  cfg.blockDim = dim3(kGemvThreads);
  cfg.dynamicSmemBytes = GemvGeo<DT>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = L.pdl ? 1 : 0;
  if (L.stamps)
    return cudaLaunchKernelEx(&cfg, gemv_tma_kernel<DT, true>, L.mats, L.pieces, L.begin, L.status, L.stall, L.stamps);
  return cudaLaunchKernelEx(&cfg, gemv_tma_kernel<DT, false>, L.mats, L.pieces, L.begin, L.status, L.stall,
                            (uint64_t *)nullptr);
}

cudaError_t launch_gemv(const GemvLaunch &L, cudaStream_t s) {
  if (L.grid <= 0) return cudaSuccess;
  switch (L.dtype) {
    case 0: return gemv_launch<0>(L, s);
    case 1: return gemv_launch<1>(L, s);
    case 2: return gemv_launch<2>(L, s);
    case 3: return gemv_launch<3>(L, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemv_mapped(const GemvLaunch &L, cudaStream_t s) {
  if (L.grid <= 0) return cudaSuccess;
  switch (L.dtype) {
    case 0: gemv_mapped_kernel<0><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    case 1: gemv_mapped_kernel<1><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    case 2: gemv_mapped_kernel<2><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    case 3: gemv_mapped_kernel<3><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_gemv_mapped_cols(const GemvLaunch &L, cudaStream_t s) {
  if (L.grid <= 0) return cudaSuccess;
  switch (L.dtype) {
    case 1: gemv_mapped_cols_kernel<1><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    case 2: gemv_mapped_cols_kernel<2><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    case 3: gemv_mapped_cols_kernel<3><<<L.grid, 256, 0, s>>>(L.mats, L.pieces, L.begin); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_gemv_generic(int dtype, const uint8_t *W, const uint8_t *x, float *y, uint64_t M,
                                uint64_t K, const uint8_t *sc, uint32_t cols, cudaStream_t s) {
  if (M == 0) return cudaSuccess;
  if (cols == 0) cols = 1;
  const uint64_t blocks64 = (M + 7) / 8;
  const int grid = (int)(blocks64 < (uint64_t)num_sms() * 8 ? blocks64 : (uint64_t)num_sms() * 8);
  switch (dtype) {
    case 0: gemv_generic_kernel<0><<<grid, 256, 0, s>>>(W, x, y, M, K, sc, cols); break;
    case 1: gemv_generic_kernel<1><<<grid, 256, 0, s>>>(W, x, y, M, K, sc, cols); break;
    case 2: gemv_generic_kernel<2><<<grid, 256, 0, s>>>(W, x, y, M, K, sc, cols); break;
    case 3: gemv_generic_kernel<3><<<grid, 256, 0, s>>>(W, x, y, M, K, sc, cols); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_seg_reduce(const SegReduce *tab, int n, uint32_t max_rows, cudaStream_t s) {
  if (n == 0 || max_rows == 0) return cudaSuccess;
  const dim3 grid((max_rows + 255) / 256, (unsigned)n);
  seg_reduce_kernel<<<grid, 256, 0, s>>>(tab);
  return cudaGetLastError();
}

}  // namespace wt
