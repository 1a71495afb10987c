// sp_union.cu -- batched decode with shared column fetches, and the density
// probe used by the dispatcher.
//
// Union kernel: B spike rows share one weight matrix.  Eq. (sparse) holds per
// row; a column that fires in several rows need only be fetched once.  A
// work unit is (output tile of 256 channels, chunk of 256 columns):
//   1. load the chunk's spike word of every row (8 words per row) and OR them
//      into the union U of the chunk,
//   2. copy the union columns' 256-byte tile segments into shared memory with
//      cp.async (each column of U read once, inactive columns never),
//   3. each warp takes whole rows; for every active column of its row it adds
//      the shared-memory segment into biased 16-bit lanes (lane = 8 channels;
//      at most 256 columns per chunk, so the lanes cannot overflow),
//   4. single-chunk problems write acc / y directly; otherwise the row sums go
//      into the workspace as fp32 with 16-byte red.add (exact: integers below
//      2^24), and the CTA that completes an output tile (atomic ticket) reads
//      the tile back in 16-byte groups, 16 loads per thread in flight, writes
//      acc and y = s * float(acc) for every row, and re-zeroes the workspace.
//      Nothing waits on another CTA.
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int kUnionWordsPerChunk = kUnionCK / 32;              // 8
constexpr size_t kUnionSmemTile = (size_t)kUnionCK * kUnionNT;   // 64 KB
constexpr size_t kUnionSmemMask = (size_t)kUnionMaxRows * kUnionWordsPerChunk * 4;  // 8 KB
constexpr size_t kUnionSmem = kUnionSmemTile + kUnionSmemMask;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void red_add_v4(float* addr, float a, float b, float c, float d) {
  asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(addr), "f"(a),
               "f"(b), "f"(c), "f"(d)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

__global__ void __launch_bounds__(kUnionThreads)
union_kernel(const __grid_constant__ UnionParams p) {
  extern __shared__ __align__(16) uint8_t smem[];
  uint8_t* s_tile = smem;                                                  // [CK][NT]
  uint32_t* s_mask = reinterpret_cast<uint32_t*>(smem + kUnionSmemTile);   // [B][8]
  __shared__ uint32_t s_union[kUnionWordsPerChunk];
  __shared__ int s_uidx[kUnionCK];
  __shared__ int s_ucount;
  __shared__ int s_last;

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int ntile = ceil_div(p.N, kUnionNT);
  const int kch = ceil_div(p.K, kUnionCK);
  const int units = ntile * kch;

  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const int nt = u / kch;
    const int kc = u - nt * kch;
    const int n0 = nt * kUnionNT;
    const int k0 = kc * kUnionCK;

    // ---- 1. spike words of every row, and their union ------------------------
    if (threadIdx.x < kUnionWordsPerChunk) s_union[threadIdx.x] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < p.B * kUnionWordsPerChunk; i += kUnionThreads) {
      const int t = i / kUnionWordsPerChunk;
      const int w = i - t * kUnionWordsPerChunk;
      const uint32_t word =
          spike_word(spike_row(p.spikes, p.fmt, t, p.ld_spikes), p.fmt, p.K, k0 + 32 * w);
      s_mask[i] = word;
      if (word) atomicOr(&s_union[w], word);
    }
    __syncthreads();
    if (warp == 0) {
      const int n = compact_words(s_union, kUnionWordsPerChunk, 0, s_uidx);
      if (lane == 0) s_ucount = n;
    }
    __syncthreads();
    const int ucount = s_ucount;

    // ---- 2. fetch each union column's tile segment once ----------------------
    {
      const int seg = threadIdx.x & 15;                    // 16-byte segment
      const int ch = n0 + seg * 16;
      if (ch < p.N) {
        for (int i = threadIdx.x >> 4; i < ucount; i += kUnionThreads / 16) {
          const int kofs = s_uidx[i];
          cp_async16(s_tile + (size_t)kofs * kUnionNT + seg * 16,
                     p.W + (int64_t)(k0 + kofs) * p.ldw + ch);
        }
      }
      cp_async_wait_all();
    }
    __syncthreads();

    // ---- 3. per-row sums from shared memory ----------------------------------
    const int ch = n0 + lane * 8;
    for (int t = warp; t < p.B; t += kUnionWarps) {
      uint32_t ev0 = 0u, od0 = 0u, ev1 = 0u, od1 = 0u;
      int n = 0;
#pragma unroll 1
      for (int w = 0; w < kUnionWordsPerChunk; ++w) {
        uint32_t bits = s_mask[t * kUnionWordsPerChunk + w];
        while (bits) {
          const int kofs = w * 32 + __ffs(bits) - 1;
          bits &= bits - 1u;
          const uint2 v = *reinterpret_cast<const uint2*>(s_tile + (size_t)kofs * kUnionNT + lane * 8);
          acc_bytes(v.x, ev0, od0);
          acc_bytes(v.y, ev1, od1);
          ++n;
        }
      }
      int o[8];
      unbias16(ev0, od0, n, o);
      unbias16(ev1, od1, n, o + 4);
      if (ch < p.N && p.fault == kFaultAbort && kch == 1) {
        if (lane == 0) atomicExch(p.err, kErrInjected);   // test fault: output unwritten
      } else if (ch < p.N) {
        if (kch == 1) {
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            if (p.acc) p.acc[(int64_t)t * p.N + ch + q] = o[q];
            if (p.y) p.y[(int64_t)t * p.N + ch + q] = scale_out(__ldg(p.scale + ch + q), o[q]);
          }
        } else {
          // integer partials below 2^24 added as fp32 (exact), 16 bytes at a time
          float* ws = reinterpret_cast<float*>(p.ws) + (int64_t)t * p.N + ch;
          if (o[0] | o[1] | o[2] | o[3])
            red_add_v4(ws, (float)o[0], (float)o[1], (float)o[2], (float)o[3]);
          if (o[4] | o[5] | o[6] | o[7])
            red_add_v4(ws + 4, (float)o[4], (float)o[5], (float)o[6], (float)o[7]);
        }
      }
    }

    // ---- 4. completion ticket per output tile ----------------------------------
    if (kch > 1) {
      __threadfence();
      __syncthreads();
      if (threadIdx.x == 0) {
        const uint32_t prev = atomicAdd(p.tickets + nt, 1u);
        int last = prev == (uint32_t)(kch - 1);
        if (last && p.fault == kFaultAbort) {   // test fault: workspace and ticket left dirty
          atomicExch(p.err, kErrInjected);
          last = 0;
        }
        if (last) atomicExch(p.tickets + nt, 0u);
        s_last = last;
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        // every (row, 4-channel group) of the tile: N % 16 == 0, so groups
        // never straddle N; 16 loads of each thread in flight before any store
        const int groups = min(kUnionNT, p.N - n0) / 4;
        const int total = p.B * groups;
        constexpr int kBatch = 16;
        // acc / y may be only 4-byte aligned (rows are 64-byte multiples apart)
        const bool vec_out = ((reinterpret_cast<uintptr_t>(p.acc) | reinterpret_cast<uintptr_t>(p.y)) & 15u) == 0;
        for (int i0 = threadIdx.x; i0 < total; i0 += kUnionThreads * kBatch) {
          float4 v[kBatch];
#pragma unroll
          for (int j = 0; j < kBatch; ++j) {
            const int i = i0 + j * kUnionThreads;
            if (i < total) {
              const int t = i / groups;
              const int n = n0 + 4 * (i - t * groups);
              v[j] = __ldcg(reinterpret_cast<const float4*>(reinterpret_cast<float*>(p.ws) +
                                                              (int64_t)t * p.N + n));
            }
          }
#pragma unroll
          for (int j = 0; j < kBatch; ++j) {
            const int i = i0 + j * kUnionThreads;
            if (i < total) {
              const int t = i / groups;
              const int n = n0 + 4 * (i - t * groups);
              __stcg(reinterpret_cast<float4*>(reinterpret_cast<float*>(p.ws) + (int64_t)t * p.N + n),
                     make_float4(0.f, 0.f, 0.f, 0.f));
              const int o[4] = {__float2int_rn(v[j].x), __float2int_rn(v[j].y), __float2int_rn(v[j].z),
                                __float2int_rn(v[j].w)};
              int32_t* acc_row = p.acc ? p.acc + (int64_t)t * p.N : nullptr;
              float* y_row = p.y ? p.y + (int64_t)t * p.N : nullptr;
              if (vec_out) {
                if (acc_row) *reinterpret_cast<int4*>(acc_row + n) = make_int4(o[0], o[1], o[2], o[3]);
                if (y_row)
                  *reinterpret_cast<float4*>(y_row + n) =
                      make_float4(scale_out(__ldg(p.scale + n), o[0]), scale_out(__ldg(p.scale + n + 1), o[1]),
                                  scale_out(__ldg(p.scale + n + 2), o[2]), scale_out(__ldg(p.scale + n + 3), o[3]));
              } else {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                  if (acc_row) acc_row[n + q] = o[q];
                  if (y_row) y_row[n + q] = scale_out(__ldg(p.scale + n + q), o[q]);
                }
              }
            }
          }
        }
      }
    }
    __syncthreads();
  }
}

// Density probe: out[0] += sum over rows of |A_t| (out zeroed by the caller).
// One thread per (row, 32-column word), grid-stride; warp sums, one atomic
// per warp.
__global__ void density_kernel(const void* spikes, int fmt, int64_t ld, int B, int K,
                               int32_t* out) {
  const int nw = ceil_div(K, 32);
  const int64_t total_words = (int64_t)nw * B;
  int total = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total_words;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / nw);
    const int w = (int)(i - (int64_t)t * nw);
    total += __popc(spike_word(spike_row(spikes, fmt, t, ld), fmt, K, 32 * w));
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) total += __shfl_xor_sync(0xffffffffu, total, d);
  if ((threadIdx.x & 31) == 0 && total) atomicAdd(out, total);
}

int g_union_grid = 0;

}  // namespace

cudaError_t launch_union(const UnionParams& p, cudaStream_t s) {
  if (p.B <= 0) return cudaSuccess;
  if (p.B > kUnionMaxRows) return cudaErrorInvalidValue;
  if (g_union_grid == 0) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(union_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kUnionSmem);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, union_kernel, kUnionThreads,
                                                      kUnionSmem);
    if (e != cudaSuccess) return e;
    g_union_grid = sms * (per_sm > 0 ? per_sm : 1);
  }
  const int units = ceil_div(p.N, kUnionNT) * ceil_div(p.K, kUnionCK);
  const int grid = units < g_union_grid ? units : g_union_grid;
  union_kernel<<<grid, kUnionThreads, kUnionSmem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_density(const void* spikes, int fmt, int64_t ld, int B, int K, int32_t* out,
                           cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(out, 0, 2 * sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  const int64_t words = (int64_t)ceil_div(K, 32) * B;
  const int threads = 256;
  int64_t grid = (words + threads - 1) / threads;
  if (grid > 2048) grid = 2048;
  if (grid < 1) grid = 1;
  density_kernel<<<(int)grid, threads, 0, s>>>(spikes, fmt, ld, B, K, out);
  return cudaGetLastError();
}

}  // namespace sp
