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
// and the warp's ballot is spike word w; bits at or past K are 0.  The state
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

int g_lif_sms = 0;

cudaError_t launch_lif_params(const LifParams& p, cudaStream_t s) {
  if (g_lif_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_lif_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const int64_t total_warps = (int64_t)p.rows * ((p.K + 31) / 32);
  const int64_t need = (total_warps + kLifThreads / 32 - 1) / (kLifThreads / 32);
  int64_t grid = (int64_t)g_lif_sms * 8;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
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
