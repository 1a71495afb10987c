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
// fp32 elements of one split-K partial (one 128 x 256 output tile).
constexpr int kGemmPartialElems = 128 * 256;
// ACC = X W^T on the tensor cores with the acc / y epilogue.  Splits K over
// a thread-block cluster when the output has fewer tiles than SMs; the
// partials meet in p.part (at least one per SM: p.part_units >= SM count).
cudaError_t launch_gemm(const GemmMaps& maps, int T, int N, int Kp, const GemmParams& p,
                        cudaStream_t s);

}  // namespace sp
