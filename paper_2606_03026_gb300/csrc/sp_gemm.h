// sp_gemm.h -- host interface of the tensor-core (tcgen05) dense path.
#pragma once

#include <cuda.h>

#include "sp_internal.h"

namespace sp {

// TMA descriptors of the two bf16 operands: A = spike rows [rows][Kp],
// B = weights [N][Kp], both K-major.
struct GemmMaps {
  CUtensorMap a;
  CUtensorMap b;
};

int gemm_k_pad(int K);                  // K rounded up to the 64-column K block
cudaError_t gemm_make_maps(const __nv_bfloat16* Xb, int rows_alloc, const __nv_bfloat16* Wb,
                           int N, int Kp, GemmMaps* out);
cudaError_t launch_w_to_bf16(const int8_t* W, int64_t ldw, int N, int K, __nv_bfloat16* Wb,
                             cudaStream_t s);
// TMA descriptor of u8 spike rows X [T][ldx] (nonzero = spike) read in
// 64-column x 128-row boxes, zero past K and T.  X 16-byte aligned,
// ldx % 16 == 0.
cudaError_t gemm_make_x8_map(const void* X, int64_t ldx, int T, int K, CUtensorMap* out);
// fp32 elements of one split-K partial (one 128 x 256 output tile).
constexpr int kGemmPartialElems = 128 * 256;
// K splits the launch will use for a T x N output (1 = no split): as many as
// leave no SM idle while every cluster of splits stays resident at once.
int gemm_splits(bool fused_x, int T, int N, int Kp, int part_units);
// ACC = X W^T on the tensor cores with the acc / y epilogue, K split S ways
// (gemm_splits) over a thread-block cluster; the partials meet in p.part (at
// least one per SM: p.part_units >= SM count).  mapA is the bf16 staging copy
// of X (gemm_make_maps), or with fused_x (requires S >= 2) the u8 spike rows
// themselves (gemm_make_x8_map), converted to bf16 inside the kernel.
cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, bool fused_x, int S,
                        int T, int N, int Kp, const GemmParams& p, cudaStream_t s);

}  // namespace sp
