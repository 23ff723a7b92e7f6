// Internal interface of the row-owner int8 multi-column kernel (wt_q8rows.cu) for the host
// library (wt_host.cpp).  Not part of the public C ABI (include/wt.h).
#pragma once

#include "wt_kernels.h"

namespace wt {

// int8 weights with T activation columns, every warp owning 16 rows of a 128-row block for the
// whole of K.  Tables as for launch_gemm_cols, with pieces cut at multiples of kQ8RowsBlock
// rows, GemvLaunch.nt = 8-column MMA tiles (1 or 2), and GemvLaunch.maps holding two tensor
// maps per matrix: W ([M, K] uint8, box {192, 128}, no swizzle) and X ([T, K] fp16, box
// {64, 16}, 128-byte swizzle; columns past T zero-filled).  Two CTAs per SM.
constexpr int kQ8RowsBlock = 128;
cudaError_t gemm_q8_rows_prepare();
cudaError_t launch_gemm_q8_rows(const GemvLaunch &L, cudaStream_t s);

}  // namespace wt
