// sp_probe.cu -- measurement aid: the practical bandwidth ceiling of a gather
// access pattern.  Not part of the method.
//
// A decode step reads |A_j| * N bytes of active columns; the gather kernel
// reads every active column as 512-byte tile segments (one 16-byte vector per
// lane of a warp) after loading and compacting the spike words and before a
// cluster reduction.  This kernel reads exactly a given list of pieces (512,
// 1024 or 1536 contiguous bytes: tile segments, or whole columns of a 1536-
// channel projection) with none of that work: the pieces are precomputed on
// the host, dealt out round-robin over every warp of the grid (so each warp
// holds at most one more piece than any other), and each lane issues all of
// its loads in one round before folding them.  Launched with the same grid shape (4 CTAs of
// 256 threads per SM) and the same programmatic dependent launch as the
// gather, its time per launch in a CUDA graph is the floor for that access
// pattern on this GPU: the launch, the dependency wait, DRAM latency and the
// random-access DRAM rate, without the method's own prologue and epilogue.
// With no pieces it measures the launch and dependency floor alone.
//
// The XOR of every 32-bit word read is folded into *sink (one atomicXor per
// warp), so a test can check that exactly the listed bytes were read.
#include "sp_internal.h"
#include "sp_ptx.cuh"

namespace sp {
namespace {

constexpr int kProbeThreads = 256;
constexpr int kProbeVecs = 15;           // 16-byte loads per lane in flight (one round)

__device__ __forceinline__ uint4 ld_stream16(const uint8_t* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Piece i (PV x 512 contiguous bytes at base + 16 * offsets16[i]) is read by
// warp i % warps, lane l reading bytes 16 l + 512 v of it (v < PV).
template <int PV>
__global__ void __launch_bounds__(kProbeThreads, 4)
probe_gather_kernel(const uint8_t* __restrict__ base, const uint32_t* __restrict__ offsets16,
                    int count, uint32_t* sink) {
  constexpr int kPieces = kProbeVecs / PV;
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warps = (int)(gridDim.x * blockDim.x) >> 5;
  const int gw = (int)(blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  uint32_t x = 0u;
  for (int i0 = gw; i0 < count; i0 += warps * kPieces) {
    uint4 v[kPieces * PV];
#pragma unroll
    for (int b = 0; b < kPieces; ++b) {
      const int i = i0 + b * warps;
      const uint8_t* p =
          i < count ? base + (size_t)__ldg(offsets16 + i) * 16u + lane * 16 : nullptr;
#pragma unroll
      for (int q = 0; q < PV; ++q)
        v[b * PV + q] = p ? ld_stream16(p + q * 512) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int b = 0; b < kPieces * PV; ++b) x ^= v[b].x ^ v[b].y ^ v[b].z ^ v[b].w;
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) x ^= __shfl_xor_sync(0xffffffffu, x, d);
  if (lane == 0 && x != 0u) atomicXor(sink, x);
}

}  // namespace

cudaError_t launch_probe_gather(const uint8_t* base, const uint32_t* offsets16, int count,
                                int piece_bytes, uint32_t* sink, cudaStream_t s) {
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)(4 * sms)), block(kProbeThreads);
  switch (piece_bytes) {
    case 512: return launch_pdl(probe_gather_kernel<1>, grid, block, 0, s, base, offsets16, count, sink);
    case 1024: return launch_pdl(probe_gather_kernel<2>, grid, block, 0, s, base, offsets16, count, sink);
    case 1536: return launch_pdl(probe_gather_kernel<3>, grid, block, 0, s, base, offsets16, count, sink);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace sp
