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
// and the warp's ballot is spike word w; bits at or past K are 0.
#include "sp_internal.h"
#include "sp_ptx.cuh"

namespace sp {
namespace {

constexpr int kLifThreads = 256;

__global__ void __launch_bounds__(kLifThreads)
lif_kernel(float* __restrict__ v, const float* __restrict__ I, int K, int rows, int64_t ld,
           float beta, float theta, uint32_t* __restrict__ bits, int64_t ld_bits) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int words = (K + 31) / 32;
  const int64_t total = (int64_t)rows * words;
  const int64_t nwarps = (int64_t)gridDim.x * (kLifThreads / 32);
  for (int64_t wi = (int64_t)blockIdx.x * (kLifThreads / 32) + (threadIdx.x >> 5); wi < total;
       wi += nwarps) {
    const int64_t r = wi / words;
    const int w = (int)(wi - r * words);
    const int k = 32 * w + lane;
    bool fire = false;
    if (k < K) {
      float u = fmaf(beta, v[r * ld + k], I[r * ld + k]);
      fire = u >= theta;
      if (fire) u = __fsub_rn(u, theta);
      v[r * ld + k] = u;
    }
    const uint32_t word = __ballot_sync(0xffffffffu, fire);
    if (lane == 0) bits[r * ld_bits + w] = word;
  }
}

int g_lif_sms = 0;

}  // namespace

cudaError_t launch_lif(float* v, const float* I, int K, int rows, int64_t ld, float beta,
                       float theta, uint32_t* bits, int64_t ld_bits, cudaStream_t s) {
  if (g_lif_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_lif_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const int64_t total_warps = (int64_t)rows * ((K + 31) / 32);
  const int64_t need = (total_warps + kLifThreads / 32 - 1) / (kLifThreads / 32);
  int64_t grid = (int64_t)g_lif_sms * 8;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  return launch_pdl(lif_kernel, dim3((unsigned)grid), dim3(kLifThreads), 0, s, v, I, K, rows, ld,
                    beta, theta, bits, ld_bits);
}

}  // namespace sp
