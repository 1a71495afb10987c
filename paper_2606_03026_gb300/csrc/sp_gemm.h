// sp_gemm.h -- host interface of the tensor-core (tcgen05) dense path.
#pragma once

#include <cuda.h>

#include "sp_internal.h"

namespace sp {

// TMA descriptors of the two e4m3 operands, both K-major: A = 0/1 spike bytes
// [rows][Kp], B = the weight planes [N][2 Kp] (per 64-column K block, 64
// bytes of e4m3(16 h) then 64 bytes of e4m3(l), w = 16 h + l).
struct GemmMaps {
  CUtensorMap a;
  CUtensorMap b;
};

int gemm_k_pad(int K);                  // K rounded up to the 64-column K block
cudaError_t gemm_make_maps(const uint8_t* Xs, int rows_alloc, const uint8_t* Wq, int N, int Kp,
                           GemmMaps* out);
// The weight planes from W (column-major INT8 [K][ldw]) into Wq [N][2 Kp].
cudaError_t launch_w_to_e4m3(const int8_t* W, int64_t ldw, int N, int K, uint8_t* Wq,
                             cudaStream_t s);
// TMA descriptor of caller-owned 0/1 spike rows X [T][ldx] (SP_SPIKES_BOOL8),
// read in place in 64-column x 128-row boxes, zero past K and T.  X 16-byte
// aligned, ldx % 16 == 0.
cudaError_t gemm_make_rows_map(const void* X, int64_t ldx, int T, int K, CUtensorMap* out);
// fp32 elements of one split-K partial (one 128 x 256 output tile).
constexpr int kGemmPartialElems = 128 * 256;
// K splits the launch will use for a T x N output (1 = no split): as many as
// leave no SM idle while every cluster of splits stays resident at once.
int gemm_splits(int T, int N, int Kp, int part_units);
// ACC = X W^T on the tensor cores with the acc / y epilogue, K split S ways
// (gemm_splits) over a thread-block cluster; the partials meet in p.part (at
// least one per SM: p.part_units >= SM count).  mapA is the 0/1 staging copy
// of X (gemm_make_maps) or the caller's 0/1 rows (gemm_make_rows_map).
cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, int S, int T, int N,
                        int Kp, const GemmParams& p, cudaStream_t s);

// Grouped form: the output tiles of up to kGemmMaxMembers independent
// contractions (one per plan of a group, each with its own operands, sizes
// and outputs) in ONE persistent launch, every tile over its whole K.
constexpr int kGemmMaxMembers = SPIKE_PROJ_MAX_GROUP;
struct GemmMember {
  CUtensorMap a;          // 0/1 spike rows [>= T][Kp] (staging copy or caller's bool8 rows)
  CUtensorMap b;          // weight planes [N][2 Kp]
  GemmParams p;           // scale, acc, y, T, N, K of this member (part unused)
  int32_t tiles_n;        // ceil(N / 256)
  int32_t nkb;            // Kp / 64 K blocks
  int32_t unit_begin;     // first output tile of this member in the launch
  int32_t unit_end;       // one past its last
};
// Kernel parameters of one grouped launch, passed by value (__grid_constant__;
// about 24 KB at 64 members, inside the 32 KB kernel-parameter limit).
struct GemmGroupArgs {
  GemmMember m[kGemmMaxMembers];
  int32_t count;          // members
  int32_t units;          // output tiles of all members
  int* err;               // device error word
};
cudaError_t launch_gemm_group(const GemmGroupArgs& a, cudaStream_t s);

}  // namespace sp
