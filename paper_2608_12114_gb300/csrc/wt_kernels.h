// Internal interface between the host library (wt_host.cpp) and the sm_103a
// kernels (wt_kernels.cu).  Not part of the public C ABI (include/wt.h).
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace wt {

// ---------------------------------------------------------------- ingest gather
// One launch copies up to kMaxGather (src, dst, nbytes) ranges; the whole
// descriptor set travels in the kernel's parameter space (no device table).
constexpr int kMaxGather = 128;
constexpr int kGatherChunkLog2 = 16;  // 64 KiB of one range per CTA iteration

struct GatherBatch {
  uint32_t n;
  uint32_t pad;
  uint64_t chunk_prefix[kMaxGather + 1];  // first chunk index of range i; [n] = total
  const uint8_t *src[kMaxGather];
  uint8_t *dst[kMaxGather];
  uint64_t nbytes[kMaxGather];
};

cudaError_t launch_gather(const GatherBatch &b, int grid, cudaStream_t s);

// ---------------------------------------------------------------- GEMV
// Tile geometry.  A stage is one TMA bulk transfer target in shared memory.
constexpr int kStageBytes = 32768;
constexpr int kConsumerWarps = 8;
constexpr int kRowBlock = 8;  // rows of a block-mode tile

enum GemvMode : uint16_t {
  kModeWarpRows = 0,   // rows of <= 256 vectors: each warp owns whole rows
  kModeBlockRows = 1,  // 256 < vectors <= kStageBytes/16: whole CTA per row, full-row tiles
  kModeLongRows = 2,   // rows longer than one stage: split into column segments before any TMA launch
  kModeCols = 3,       // multi-column kernel (G = T columns): 16-row tiles x vc-vector chunks
};

// Multi-column kernel: at most kColVecMax 16-byte vectors of a row per stage, and a chunk
// length vc = 4 (mod 8) so that the stage's row pitch vc * 16 is 64 bytes past a multiple
// of 128 (the two rows a quarter-warp reads fall in different banks).
constexpr int kColVecMax = 92;
constexpr int kColTileRows = 16;
constexpr int kTensorMapBytes = 128;  // one CUtensorMap

struct alignas(16) MatDesc {
  const uint8_t *W;
  const uint8_t *x;
  float *y;
  const uint8_t *s;  // f16 row scales (int8 weights), else null
  uint32_t M;     // rows
  uint32_t V;     // 16-byte vectors per row (K * sizeof(elem) / 16)
  uint32_t rt;    // rows per tile (modes 0/1) or per row block (mode 2)
  uint32_t vc;    // vectors per column chunk (mode 2); V otherwise
  uint16_t mode;  // GemvMode
  uint16_t G;     // mode 0: lanes per row (power of two <= 32); kModeCols: columns T
  uint32_t rs;    // row pitch in 16-byte vectors: V, or the full row of a column segment
                  // (segments are split-K only); s == nullptr then means "no scale yet"
  uint32_t cols;  // map endpoint with T activation columns: T (X [T, K], Y [T, M]); else 0
  uint32_t pad;
};
static_assert(sizeof(MatDesc) == 64, "MatDesc is one 64-byte record");

// Cross-CTA split-K: rows longer than seg_vectors(dtype) are cut into column segments of
// that many vectors (the last one shorter).  Each segment is a matrix of its own (row pitch
// the full row; tile mode by its own length: a full segment is one 32 KB or 16 KB row per
// stage, whole-CTA "block rows") writing partial sums to a workspace; a second pass sums the
// segments of each row in segment order and applies the row scale.  Segment boundaries
// depend only on the matrix, so a row's result never depends on how rows and segments were
// spread over CTAs.
constexpr uint32_t kSegVec = 2048;  // bf16 / f16 / f32: 32 KB per segment row
constexpr uint32_t seg_vectors(int dtype) { return dtype == 3 ? kSegVec / 4 : kSegVec; }  // int8: 8 KB

struct alignas(16) SegReduce {
  const float *ws;   // nseg x M partial sums (segment-major)
  float *y;          // M outputs
  const uint8_t *s;  // f16 row scales (int8 weights) or null
  uint32_t M;
  uint32_t nseg;
};

// y[row] = (sum over segments of ws[seg * M + row], in segment order) * scale[row], for
// every SegReduce of the table.
cudaError_t launch_seg_reduce(const SegReduce *tab, int n, uint32_t max_rows, cudaStream_t s);

struct alignas(16) Piece {
  uint32_t mat;  // index into the launch's MatDesc table
  uint32_t r0;   // first row
  uint32_t r1;   // one past the last row
  uint32_t pad;
};

struct GemvLaunch {
  int dtype;               // WT_F32 / WT_BF16 / WT_F16 / WT_I8 (x f16, f16 row scales)
  int grid;                // CTAs; CTA b owns pieces [begin[b], begin[b+1])
  const MatDesc *mats;     // device
  const Piece *pieces;     // device
  const uint32_t *begin;   // device, grid + 1 entries
  int *status;             // device status word (bounded-wait failures)
  const uint8_t *maps = nullptr;  // multi-column kernel: one TMA tensor map per MatDesc
                                  // (kTensorMapBytes each, 128-byte aligned, device)
  int stall = 0;  // failure test (host fault site "stall"): the producer issues no copy, so
                  // every consumer wait runs out, reports WT_ETIMEDOUT and the CTA exits
  int nt = 0;     // multi-column kernel: 8-column MMA tiles of every matrix (T <= 8 nt)
  int pdl = 0;    // one-column kernel: launch with programmatic stream serialization (the
                  // launch and prologue may overlap the previous kernel of the stream)
  uint64_t *stamps = nullptr;  // one-column kernel: non-null runs the stamping instantiation,
                               // kStampFields words per CTA (grid x kStampFields, device)
};

// Per-CTA stamps of the one-column kernel (%globaltimer nanoseconds, but kStSm): the record
// layout of wt_pass_stamps.  A time the CTA never reached (no rows: no copy, no stage) is 0.
enum StampField : int {
  kStEntry = 0,      // CTA entry
  kStPrologue = 1,   // barriers initialised (shared-memory set-up done)
  kStOperands = 2,   // past the wait for the previous grid: operands may be read
  kStFirstCopy = 3,  // first bulk copy issued (after the plan-table reads)
  kStFirstFull = 4,  // first stage landed, as consumer warp 0 saw it
  kStLastFull = 5,   // last stage landed, as consumer warp 0 saw it
  kStExit = 6,       // every warp done
  kStSm = 7,         // %smid of the CTA (not a time)
  kStampFields = 8
};

cudaError_t gemv_prepare();  // one-time function attributes
cudaError_t launch_gemv(const GemvLaunch &L, cudaStream_t s);
size_t gemv_smem_bytes(int dtype);
int gemv_ctas_per_sm(int dtype);  // resident CTAs per SM the one-column launch is sized for

// Map endpoint (the paper's adoption, contract C1): W is read in place from a file mapping
// the device reaches over the host link, with 16-byte loads and no TMA; same tables as
// launch_gemv (MatDesc.W holds the device-readable address of the mapped rows).
cudaError_t launch_gemv_mapped(const GemvLaunch &L, cudaStream_t s);
// The map endpoint with T <= 16 activation columns (MatDesc.cols = T): each mapped weight
// vector is loaded once over the host link and used for every column.
cudaError_t launch_gemv_mapped_cols(const GemvLaunch &L, cudaStream_t s);

// Multi-column GEMV Y[t] = diag(s) W X[t] (t < T <= 16; X [T, K] and Y [T, M] row-major) on the
// tensor cores (wt_cols.cu); dtype WT_BF16 / WT_F16 / WT_I8, tables as for launch_gemv with
// MatDesc.mode = kModeCols, MatDesc.G = T and MatDesc.vc = vectors per chunk (<= kColVecMax,
// vc = 4 mod 8), plus GemvLaunch.maps: per matrix a 2-D tensor map of W viewed as
// [M, 2V] 8-byte elements with box {2 vc, kColTileRows} (rows and columns past the end
// arrive as zeros).
// One launch holds matrices of one dtype and one nt (GemvLaunch.nt: 1 for T <= 8, 2 for
// 8 < T <= 16); int8 with nt = 1 runs two CTAs per SM (gemm_cols_ctas_per_sm).
cudaError_t gemm_cols_prepare();
cudaError_t launch_gemm_cols(const GemvLaunch &L, cudaStream_t s);
int gemm_cols_ctas_per_sm(int dtype, int nt);

// The same multi-column GEMV on tcgen05 for 2-byte weights (wt_umma.cu): row tiles of 128
// rows, K in chunks of 64 elements, accumulators in tensor memory.  pieces[m] = {m, first
// tile of matrix m, its tiles, 0}; CTA b takes tiles b, b + grid, ...  maps holds two tensor
// maps per matrix: W ([M, K] 2-byte elements, box {64, 128}, 128-byte swizzle) and X ([T, K]
// 2-byte elements, box {64, 16}, 128-byte swizzle).
struct UmmaLaunch {
  int dtype;
  int grid;
  const MatDesc *mats;
  const Piece *pieces;
  uint32_t nmat;
  uint32_t ntiles;
  int *status;
  const uint8_t *maps;
};
cudaError_t gemm_cols_umma_prepare();
cudaError_t launch_gemm_cols_umma(const UmmaLaunch &L, cudaStream_t s);

// Fallback for operands the tiled kernels cannot take (unaligned W/x, rows whose byte length
// is not a multiple of 16, or multi-column W read in place from a mapping): one warp per
// row, scalar loads.  cols = 0 or 1: y = W x; cols = T > 1: Y [T, M] from X [T, K].
cudaError_t launch_gemv_generic(int dtype, const uint8_t *W, const uint8_t *x, float *y,
                                uint64_t M, uint64_t K, const uint8_t *scale, uint32_t cols,
                                cudaStream_t s);

int num_sms();  // of the current device (cached per device)

// Records `msg` as this thread's wt_last_error() text and returns `code`.
int set_error(int code, const char *msg);

// Host-side fault injection (tests): true when WT_FAULT="<site>[:<n>]" names this site and
// this is its n-th call (n = 1 by default) since the variable last changed.  Sites: open,
// pread, mmap, register, alloc (the call fails as if the system or CUDA call had), and stall
// (a resident GEMV launch whose producer issues nothing: its bounded waits run out).
bool fault_injected(const char *site);

}  // namespace wt

struct DLManagedTensorVersioned;

namespace wt {

// The producer's core (wt_dlpack.cpp): maps bytes [off, off + nbytes) of `path` read-only and
// shared (whole pages), exposes them per WT_DLPACK_* flags and returns a capsule of shape
// shape[0..ndim) with compact strides.
int dlpack_map(const char *path, uint64_t off, uint64_t nbytes, int32_t dtype, int ndim, const uint64_t *shape,
               unsigned flags, DLManagedTensorVersioned **out);

}  // namespace wt
