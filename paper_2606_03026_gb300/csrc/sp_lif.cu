// sp_lif.cu -- spike producer: one leaky integrate-and-fire step written
// straight into the packed spike rows (SP_SPIKES_BITS32) that the gather,
// union and GEMM paths read.  The paper names LIF dynamics (Section 1)
// without giving the update; the library uses this reading:
//
//   v <- fmaf(beta, v, I)      one FP32 fused multiply-add
//   x  = (v >= theta)          the spike
//   v <- v - theta where x     soft reset, one FP32 subtract
//
// Every operation is IEEE FP32 with round-to-nearest (the library is built
// without fast-math, so subnormals are kept), so v and the bits are the same
// as the definition's on every run.  One warp per 32-neuron word: lane l
// updates neuron 32 w + l (coalesced 128-byte reads and writes of v and I)
// and the warp's ballot is spike word w; bits at or past K are 0.  Rows
// whose elements are 16-byte aligned (v, I 16-byte aligned, ld % 4 == 0) take
// a vector form when the state is large (at least 2^22 neurons): lane l
// holds neurons 4l .. 4l + 3 of a 128-neuron group (one
// 16-byte load of v and of I, two groups in flight per lane), and the group's
// 4 spike words are assembled from 4 ballots (bit j of ballot c, for lane
// 8w + j, is neuron 32w + 4j + c).  The state
// may be read from one buffer and written to another (vin == vout updates it
// in place), and each row may have its own neuron count (the rows of a group
// of projections with different K).
#include "sp_internal.h"
#include "sp_ptx.cuh"

namespace sp {
namespace {

constexpr int kLifThreads = 256;

struct LifParams {
  const float* vin;       // row r at vin + r * ld
  float* vout;            // idem; may equal vin
  const float* I;         // idem
  int64_t ld;
  float beta, theta;
  uint32_t* bits;         // row r at bits + r * ld_bits words
  int64_t ld_bits;
  int32_t rows;
  int32_t K;              // neurons per row (the largest when per_row)
  int32_t per_row;        // 1: row r has Krow[r] neurons (rows <= kMaxProblems)
  int32_t Krow[kMaxProblems];
};

__global__ void __launch_bounds__(kLifThreads)
lif_kernel(const __grid_constant__ LifParams p) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int words = (p.K + 31) / 32;
  const int64_t total = (int64_t)p.rows * words;
  const int64_t nwarps = (int64_t)gridDim.x * (kLifThreads / 32);
  for (int64_t wi = (int64_t)blockIdx.x * (kLifThreads / 32) + (threadIdx.x >> 5); wi < total;
       wi += nwarps) {
    const int64_t r = wi / words;
    const int w = (int)(wi - r * words);
    const int K = p.per_row ? p.Krow[r] : p.K;
    if (32 * w >= K) continue;               // warp-uniform: past this row's last word
    const int k = 32 * w + lane;
    bool fire = false;
    if (k < K) {
      float u = fmaf(p.beta, p.vin[r * p.ld + k], p.I[r * p.ld + k]);
      fire = u >= p.theta;
      if (fire) u = __fsub_rn(u, p.theta);
      p.vout[r * p.ld + k] = u;
    }
    const uint32_t word = __ballot_sync(0xffffffffu, fire);
    if (lane == 0) p.bits[r * p.ld_bits + w] = word;
  }
}

// Bit j of the low byte of x moved to bit 4j (j < 8).
__device__ __forceinline__ uint32_t spread4(uint32_t x) {
  x &= 0xffu;
  x = (x | (x << 12)) & 0x000f000fu;
  x = (x | (x << 6)) & 0x03030303u;
  x = (x | (x << 3)) & 0x11111111u;
  return x;
}

// One LIF step of the 4 neurons at k .. k + 3 of a row (those < K).
__device__ __forceinline__ void lif4(const LifParams& p, const float* vr, float* vw, const float* ir,
                                     int k, int K, bool (&fire)[4]) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f), cur = v;
  if (k + 4 <= K) {
    v = *reinterpret_cast<const float4*>(vr + k);
    cur = __ldg(reinterpret_cast<const float4*>(ir + k));
  } else {
    float* pv = &v.x;
    float* pc = &cur.x;
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (k + e < K) {
        pv[e] = vr[k + e];
        pc[e] = ir[k + e];
      }
  }
  float u[4] = {fmaf(p.beta, v.x, cur.x), fmaf(p.beta, v.y, cur.y), fmaf(p.beta, v.z, cur.z),
                fmaf(p.beta, v.w, cur.w)};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    fire[e] = k + e < K && u[e] >= p.theta;
    if (fire[e]) u[e] = __fsub_rn(u[e], p.theta);
  }
  if (k + 4 <= K) {
    *reinterpret_cast<float4*>(vw + k) = make_float4(u[0], u[1], u[2], u[3]);
  } else {
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (k + e < K) vw[k + e] = u[e];
  }
}

__global__ void __launch_bounds__(kLifThreads)
lif_kernel_v4(const __grid_constant__ LifParams p) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int K = p.K;
  const int groups = (K + 127) / 128;            // 128-neuron groups per row
  const int words = (K + 31) / 32;
  const int64_t total = (int64_t)p.rows * groups;
  const int64_t nwarps = (int64_t)gridDim.x * (kLifThreads / 32);
  for (int64_t gi = (int64_t)blockIdx.x * (kLifThreads / 32) + (threadIdx.x >> 5); gi < total;
       gi += 2 * nwarps) {
    bool fire[2][4];
    int64_t row[2];
    int g[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {                // two groups' loads in flight
      const int64_t item = gi + q * nwarps;
      row[q] = item / groups;
      g[q] = (int)(item - row[q] * groups);
      if (item < total) {
        const int64_t off = row[q] * p.ld;
        lif4(p, p.vin + off, p.vout + off, p.I + off, 128 * g[q] + 4 * lane, K, fire[q]);
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) fire[q][e] = false;
      }
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      uint32_t bal[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) bal[e] = __ballot_sync(0xffffffffu, fire[q][e]);
      const int w = 4 * g[q] + lane;             // lanes 0..3 write the group's words
      if (lane < 4 && gi + q * nwarps < total && w < words) {
        uint32_t word = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) word |= spread4(bal[e] >> (8 * lane)) << e;
        p.bits[row[q] * p.ld_bits + w] = word;
      }
    }
  }
}

int g_lif_sms = 0;

cudaError_t launch_lif_params(const LifParams& p, cudaStream_t s) {
  if (g_lif_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_lif_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  // the vector form for large states only: at decode sizes (a few hundred
  // thousand neurons) its small grid made the following decode launch start
  // later (producer + decode step 16.2 against 14.7 us with the scalar form)
  const bool vec = !p.per_row && (int64_t)p.rows * p.K >= ((int64_t)1 << 22) && p.ld % 4 == 0 &&
                   ((uintptr_t)p.vin & 15) == 0 && ((uintptr_t)p.vout & 15) == 0 &&
                   ((uintptr_t)p.I & 15) == 0;
  const int64_t total_warps =
      vec ? ((int64_t)p.rows * ((p.K + 127) / 128) + 1) / 2 : (int64_t)p.rows * ((p.K + 31) / 32);
  const int64_t need = (total_warps + kLifThreads / 32 - 1) / (kLifThreads / 32);
  int64_t grid = (int64_t)g_lif_sms * 8;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  if (vec) return launch_pdl(lif_kernel_v4, dim3((unsigned)grid), dim3(kLifThreads), 0, s, p);
  return launch_pdl(lif_kernel, dim3((unsigned)grid), dim3(kLifThreads), 0, s, p);
}

}  // namespace

cudaError_t launch_lif(float* v, const float* I, int K, int rows, int64_t ld, float beta,
                       float theta, uint32_t* bits, int64_t ld_bits, cudaStream_t s) {
  LifParams p = {};
  p.vin = v;
  p.vout = v;
  p.I = I;
  p.ld = ld;
  p.beta = beta;
  p.theta = theta;
  p.bits = bits;
  p.ld_bits = ld_bits;
  p.rows = rows;
  p.K = K;
  return launch_lif_params(p, s);
}

cudaError_t launch_lif_rows(const float* vin, float* vout, const float* I, const int32_t* Ks,
                            int rows, int64_t ld, float beta, float theta, uint32_t* bits,
                            int64_t ld_bits, cudaStream_t s) {
  if (rows < 1 || rows > kMaxProblems) return cudaErrorInvalidValue;
  LifParams p = {};
  p.vin = vin;
  p.vout = vout;
  p.I = I;
  p.ld = ld;
  p.beta = beta;
  p.theta = theta;
  p.bits = bits;
  p.ld_bits = ld_bits;
  p.rows = rows;
  p.per_row = 1;
  for (int r = 0; r < rows; ++r) {
    p.Krow[r] = Ks[r];
    if (Ks[r] > p.K) p.K = Ks[r];
  }
  return launch_lif_params(p, s);
}

}  // namespace sp
