// sp_dense.cu -- continuous-input projections (Section 2.3: for continuous
// inputs the INT8 weights are converted to FP32, multiplied with the FP32
// activations and accumulated, and the row scale is applied after; Section
// 2.2: these projections keep row-major weights, one contiguous dot product
// per output):
//
//   y[b][m] = s_m * sum_k float(W[m * ldw + k]) * x[b][k]
//
// for B <= 4 activation rows and up to 128 problems per launch (e.g. the
// query/key/value, attention-output and FFN up projections of every block of a
// decode step).  The weights stream from HBM once per call, so the kernel is
// HBM-bound: algorithmic bytes = sum over problems of N * K.
//
// A unit is 4 consecutive rows of one problem, owned by one warp.  Lane l
// covers the 16-column chunks l, l + 32, l + 64, ... of the row (16-byte
// weight loads, 512 contiguous bytes per warp instruction), issuing the loads
// of one chunk of all 4 rows before any arithmetic.  A weight byte
// becomes a float exactly through its bias (w + 128 in the low byte of 2^23's
// mantissa, minus 2^23 + 128).  Each lane accumulates with fmaf in ascending
// k, the 32 lane sums meet in a 5-level butterfly, and one FP32 multiply by s_m
// gives y.  Every output is therefore an FP32 sum of K products of depth at
// most 16 * ceil(K / 512) + 5, whatever the grid, so the error bound and the
// result are the same on every run.
#include "sp_ptx.cuh"
#include "sp_rows.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int kDenseRows = 4;        // rows per unit (one warp)
constexpr int kDenseThreads = 256;
// Per activation count B: 16-column chunks per lane loaded per round, and
// CTAs per SM the registers must allow.  One chunk of 4 rows per round: the
// converted weights stay in registers for the B activation rows, and more
// warps with less in flight each stream faster than fewer warps with three
// chunks (measured on the 22-block step: B = 1 at 32 warps per SM 5.1 TB/s
// against 3.6 with three chunks; B = 2 / 3 / 4 at 16 warps per SM 2.9 / 2.3 /
// 1.7 TB/s against 2.5 / 1.6 / 1.3).
template <int B> struct DenseShape { static constexpr int batch = 1, min_ctas = 2; };
template <> struct DenseShape<1> { static constexpr int batch = 1, min_ctas = 4; };

struct DenseParams {
  int32_t count, B;
  int32_t units;                       // total over problems
  DenseProblem prob[kDenseMaxProblems];
  int32_t unit_end[kDenseMaxProblems]; // prefix sums of each problem's units
};

template <int B>
__global__ void __launch_bounds__(kDenseThreads, DenseShape<B>::min_ctas)
dense_kernel(const __grid_constant__ DenseParams p) {
  constexpr int kDenseBatch = DenseShape<B>::batch;
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int nwarps = gridDim.x * (kDenseThreads / 32);
  int j = 0;                                   // problem of the current unit (units ascend)
  for (int u = blockIdx.x * (kDenseThreads / 32) + (threadIdx.x >> 5); u < p.units; u += nwarps) {
    while (u >= p.unit_end[j]) ++j;
    const DenseProblem& P = p.prob[j];
    const int row0 = (u - (j ? p.unit_end[j - 1] : 0)) * kDenseRows;
    const int nrows = min(kDenseRows, P.N - row0);
    const int nch = (P.K + 511) / 512;        // chunk rounds of the whole warp
    float acc[kDenseRows][B];
#pragma unroll
    for (int r = 0; r < kDenseRows; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b) acc[r][b] = 0.f;

    for (int i0 = 0; i0 < nch; i0 += kDenseBatch) {
      // weights: up to 3 chunks x 4 rows of 16 bytes in flight
      uint4 w[kDenseRows][kDenseBatch];
#pragma unroll
      for (int c = 0; c < kDenseBatch; ++c) {
        const int k = 16 * (lane + 32 * (i0 + c));
#pragma unroll
        for (int r = 0; r < kDenseRows; ++r) {
          w[r][c] = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);   // biased zeros
          if (k < P.K && r < nrows) {
            // the row is ldw >= K bytes with ldw % 16 == 0: the 16 bytes at k
            // lie inside it; bytes at or past K meet a zero activation
            const uint4 v = ld_weights16(P.W + (int64_t)(row0 + r) * P.ldw + k);
            w[r][c] = make_uint4(v.x ^ 0x80808080u, v.y ^ 0x80808080u, v.z ^ 0x80808080u,
                                 v.w ^ 0x80808080u);
          }
        }
      }
#pragma unroll
      for (int c = 0; c < kDenseBatch; ++c) {
        const int k = 16 * (lane + 32 * (i0 + c));
        if (k >= P.K) continue;
#pragma unroll
        for (int b = 0; b < B; ++b) {
          float xv[16];
          load_x16(P.x + (int64_t)b * P.ldx, k, P.K, xv);
#pragma unroll
          for (int r = 0; r < kDenseRows; ++r) {
            const uint32_t ww[4] = {w[r][c].x, w[r][c].y, w[r][c].z, w[r][c].w};
#pragma unroll
            for (int e = 0; e < 16; ++e)
              acc[r][b] = fmaf(byte_to_float(ww[e >> 2], (uint32_t)(e & 3)), xv[e], acc[r][b]);
          }
        }
      }
    }
    // butterfly over the 32 lanes; every lane ends with the full sums
#pragma unroll
    for (int r = 0; r < kDenseRows; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b)
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) acc[r][b] += __shfl_xor_sync(0xffffffffu, acc[r][b], d);
#pragma unroll
    for (int r = 0; r < kDenseRows; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b)
        if (lane == r * B + b && r < nrows)
          P.y[(int64_t)b * P.ldy + row0 + r] = __fmul_rn(__ldg(P.scale + row0 + r), acc[r][b]);
  }
}

int g_dense_sms = 0;

// Resident CTAs of dense_kernel<B> per SM (0 before the first query).
template <int B>
int dense_ctas_per_sm() {
  static int n = 0;
  if (n == 0 && cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, dense_kernel<B>, kDenseThreads, 0) !=
                    cudaSuccess) {
    (void)cudaGetLastError();
    n = 1;
  }
  return n > 0 ? n : 1;
}

template <int B>
cudaError_t launch_dense_t(const DenseParams& p, cudaStream_t s) {
  // one wave of resident CTAs (never more than the units need): every unit a
  // warp takes from the grid-stride sequence starts without waiting for a CTA
  const int warps_per_cta = kDenseThreads / 32;
  int grid = g_dense_sms * dense_ctas_per_sm<B>();
  const int need = (p.units + warps_per_cta - 1) / warps_per_cta;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  return launch_pdl(dense_kernel<B>, dim3(grid), dim3(kDenseThreads), 0, s, p);
}

}  // namespace

cudaError_t launch_dense(const DenseProblem* probs, int count, int B, cudaStream_t s) {
  if (g_dense_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_dense_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  DenseParams p;
  p.count = count;
  p.B = B;
  int units = 0;
  for (int j = 0; j < count; ++j) {
    p.prob[j] = probs[j];
    units += (probs[j].N + kDenseRows - 1) / kDenseRows;
    p.unit_end[j] = units;
  }
  for (int j = count; j < kDenseMaxProblems; ++j) p.unit_end[j] = units;
  p.units = units;
  switch (B) {
    case 1: return launch_dense_t<1>(p, s);
    case 2: return launch_dense_t<2>(p, s);
    case 3: return launch_dense_t<3>(p, s);
    default: return launch_dense_t<4>(p, s);
  }
}

}  // namespace sp
