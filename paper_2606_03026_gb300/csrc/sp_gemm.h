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
  CUtensorMap b;          // 256-row boxes (one output tile's channels)
  CUtensorMap b128;       // the same operand in 128-row boxes (half a tile)
  CUtensorMap p64;        // one plane of one K block: 128 rows x 64 bytes, 64-byte swizzle
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

// Small-T form (sp_gemm_small.cu): T <= kGemmSmallMaxT spike rows in any
// input format, read directly (no staging copy), the product computed
// transposed (128 output channels per CTA as the MMA's M, the tokens as its
// N) with K split over a cluster of S in {1, 2, 4, 8} CTAs that reduces
// through distributed shared memory.  Each CTA holds the 0 / 1 bytes of its K
// range of all T rows, at most kGemmSmallMaxKB K blocks of 64 columns.
constexpr int kGemmSmallMaxT = 64;
constexpr int kGemmSmallMaxS = 8;
constexpr int kGemmSmallMaxKB = 16;
struct GemmSmallArgs {
  const void* spikes;     // row t at spikes + t * ld elements (sp_fmt)
  int32_t fmt;
  int64_t ld;
  const float* scale;
  int32_t* acc;           // [T][N] or null
  float* y;               // [T][N] or null
  int32_t T, TN;          // rows, and the MMA's N (T rounded up to 16)
  int32_t N, K;
  int32_t S;              // K ranges = cluster size
  int32_t nkb;            // Kp / 64
  int* err;
  int32_t fault;          // Fault armed for this launch
};
// K splits of the small-T form for this shape, 0 when it does not apply
// (T > kGemmSmallMaxT, or K too long for the per-CTA spike slice).
int gemm_small_splits(int T, int N, int Kp);
// mapW: the weight planes, one plane of one K block per box (GemmMaps::p64).
cudaError_t launch_gemm_small(const CUtensorMap& mapW, const GemmSmallArgs& a, cudaStream_t s);

// Grouped form: the output tiles of up to kGemmMaxMembers independent
// contractions (one per plan of a group, each with its own operands, sizes
// and outputs) in ONE persistent launch, every tile over its whole K.
constexpr int kGemmMaxMembers = SPIKE_PROJ_MAX_GROUP;
struct GemmMember {
  CUtensorMap a;          // 0/1 spike rows [>= T][Kp] (staging copy or caller's bool8 rows)
  CUtensorMap b;          // weight planes [N][2 Kp] in boxes of 256 / CL rows (GemmMaps)
  GemmParams p;           // scale, acc, y, T, N, K of this member (part unused)
  int32_t tiles_n;        // ceil(N / 256)
  int32_t nkb;            // Kp / 64 K blocks
  int32_t unit_begin;     // first output tile of this member in the launch
  int32_t unit_end;       // one past its last
};
// Kernel parameters of one grouped launch, passed by value (__grid_constant__;
// about 24 KB at 64 members, inside the 32 KB kernel-parameter limit).  A
// unit is CL row tiles of one member with the same 256 channels; with CL = 2
// a CTA pair computes it with the 2-SM MMA (M = 256), each CTA loading its
// own 128 spike rows and half of the 256 weight rows.
//
// Tail split: when the units do not fill the last round of the persistent
// grid, each of the last r units is cut into S ranges of its K blocks (S =
// min(clusters / r, 4)), so the last round runs r S sub-units on as many
// clusters.  Sub-unit 0 of a split unit owns the output; each other sub-unit
// writes its fp32 partial (per CTA one 128 x 256 tile) to part and raises a
// per-warp flag, which the owner's warp waits for (bounded), adds and
// clears.  The launcher fills whole / tail_s / total.
struct GemmGroupArgs {
  GemmMember m[kGemmMaxMembers];
  int32_t count;          // members
  int32_t units;          // units of all members
  int32_t cl;             // CTAs per unit (1, or 2 for the CTA-pair MMA)
  int* err;               // device error word
  float* part;            // tail-split partials, kGemmGroupSlots x 128 x 256 fp32 (or null)
  uint32_t* flags;        // kGemmGroupSlots x 8 words, zero between launches
  int32_t whole;          // units run over their whole K (the first ones)
  int32_t tail_s;         // K ranges per tail unit (1: no split)
  int32_t total;          // whole + (units - whole) * tail_s
};
// Partial tiles (128 x 256 fp32, one per CTA of a helper sub-unit) that the
// tail split may need: at most one per SM.
constexpr int kGemmGroupSlots = 160;
// CTAs per unit for a grouped launch whose members have these tile counts:
// 2 unless pairing row tiles adds more than 1/8 of idle (row-padding) tiles.
int gemm_group_cluster(const int* tiles_m, const int* tiles_n, int count);
cudaError_t launch_gemm_group(const GemmGroupArgs& a, cudaStream_t s);

}  // namespace sp
