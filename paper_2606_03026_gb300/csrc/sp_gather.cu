// sp_gather.cu -- active-column gather-sum (Section 2.2, Eq. (sparse)):
//
//   acc_m = sum_{k in A} Q[k*ldw + m],   y_m = s_m * float(acc_m)
//
// for one or many (projection, token) problems in a single launch.
//
// Decomposition: a work unit is (problem j, token t, output tile of 512
// channels, chunk of 512 input columns).  Per unit the CTA
//   1. reads the chunk's 16 spike words and compacts them into the ascending
//      list of active columns (warp popcount + shuffle scan),
//   2. lets each of its 8 warps stream every 8th listed column: one 16-byte
//      load per lane covers 512 contiguous bytes of the column, accumulated
//      as biased 16-bit lanes (at most 64 columns per warp, never overflows),
//   3. sums the 8 warps through shared memory and
//      - writes acc / y directly when the problem has a single K chunk, or
//      - adds into the INT32 workspace with red.add, then takes a ticket:
//        the CTA that completes the tile (ticket == chunks - 1) reads the
//        workspace back, writes acc and y = s * float(acc), and re-zeroes the
//        workspace and the ticket for the next call.  No CTA ever waits on
//        another.
// Inactive columns are never read.  Integer sums are order-free, so the
// result is bit-identical to the definition whatever the CTA schedule.
#include "sp_spikes.cuh"

namespace sp {
namespace {

template <int NP>
__device__ __forceinline__ int find_problem(const GatherParamsT<NP>& p, int u) {
  int lo = 0, hi = p.nprob - 1;            // largest j with unit_begin_j * B <= u
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.prob[mid].unit_begin * p.B <= u) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <int NP>
__global__ void __launch_bounds__(kGatherThreads)
gather_kernel(const __grid_constant__ GatherParamsT<NP> p) {
  __shared__ uint32_t s_words[kGatherCK / 32];
  __shared__ int s_idx[kGatherCK];
  __shared__ __align__(16) int s_red[kGatherWarps][kGatherNT];
  __shared__ int s_count;
  __shared__ int s_last;

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;

  for (int u = blockIdx.x; u < p.units_total; u += gridDim.x) {
    // ---- decode the unit ---------------------------------------------------
    const int j = find_problem(p, u);
    const GatherProblem& P = p.prob[j];
    const int upt = gather_units(P.N, P.K);
    const int ul = u - P.unit_begin * p.B;
    const int t = ul / upt;
    const int r = ul - t * upt;
    const int kch = gather_kchunks(P.K);
    const int ntile = gather_ntiles(P.N);
    const int nt = r / kch;
    const int kc = r - nt * kch;
    if (t >= p.B || nt >= ntile) {           // cannot happen for a valid table
      if (threadIdx.x == 0) atomicExch(p.err, kErrBadUnit);
      return;
    }
    const int n0 = nt * kGatherNT;
    const int k0 = kc * kGatherCK;
    const int64_t row = (int64_t)j * p.B + t;

    // ---- 1. spike words of the chunk -> active list -------------------------
    const void* srow = spike_row(p.spikes, p.fmt, row, p.ld_spikes);
    if (threadIdx.x < kGatherCK / 32)
      s_words[threadIdx.x] = spike_word(srow, p.fmt, P.K, k0 + threadIdx.x * 32);
    __syncthreads();
    if (warp == 0) {
      const int n = compact_words(s_words, kGatherCK / 32, k0, s_idx);
      if (lane == 0) s_count = n;
    }
    __syncthreads();
    const int cnt = s_count;

    // ---- 2. stream the active columns of this output tile -------------------
    const int ch = n0 + lane * 16;          // first channel of this lane
    const bool lane_on = ch < P.N;
    const int8_t* wcol = P.W + ch;
    const int64_t ldw = P.ldw;
    uint32_t ev[4] = {0u, 0u, 0u, 0u}, od[4] = {0u, 0u, 0u, 0u};
    int mine = 0;
    int i = warp;
    for (; i + 3 * kGatherWarps < cnt; i += 4 * kGatherWarps) {
      const int c0 = s_idx[i], c1 = s_idx[i + kGatherWarps];
      const int c2 = s_idx[i + 2 * kGatherWarps], c3 = s_idx[i + 3 * kGatherWarps];
      uint4 v0 = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
      uint4 v1 = v0, v2 = v0, v3 = v0;
      if (lane_on) {
        v0 = ld_weights16(wcol + c0 * ldw);
        v1 = ld_weights16(wcol + c1 * ldw);
        v2 = ld_weights16(wcol + c2 * ldw);
        v3 = ld_weights16(wcol + c3 * ldw);
      }
      acc_bytes(v0.x, ev[0], od[0]); acc_bytes(v0.y, ev[1], od[1]);
      acc_bytes(v0.z, ev[2], od[2]); acc_bytes(v0.w, ev[3], od[3]);
      acc_bytes(v1.x, ev[0], od[0]); acc_bytes(v1.y, ev[1], od[1]);
      acc_bytes(v1.z, ev[2], od[2]); acc_bytes(v1.w, ev[3], od[3]);
      acc_bytes(v2.x, ev[0], od[0]); acc_bytes(v2.y, ev[1], od[1]);
      acc_bytes(v2.z, ev[2], od[2]); acc_bytes(v2.w, ev[3], od[3]);
      acc_bytes(v3.x, ev[0], od[0]); acc_bytes(v3.y, ev[1], od[1]);
      acc_bytes(v3.z, ev[2], od[2]); acc_bytes(v3.w, ev[3], od[3]);
      mine += 4;
    }
    for (; i < cnt; i += kGatherWarps) {
      uint4 v = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
      if (lane_on) v = ld_weights16(wcol + s_idx[i] * ldw);
      acc_bytes(v.x, ev[0], od[0]); acc_bytes(v.y, ev[1], od[1]);
      acc_bytes(v.z, ev[2], od[2]); acc_bytes(v.w, ev[3], od[3]);
      ++mine;
    }

    // ---- 3. reduce the warps -------------------------------------------------
    {
      int o[16];
      unbias16(ev[0], od[0], mine, o + 0);
      unbias16(ev[1], od[1], mine, o + 4);
      unbias16(ev[2], od[2], mine, o + 8);
      unbias16(ev[3], od[3], mine, o + 12);
      int4* dst = reinterpret_cast<int4*>(&s_red[warp][lane * 16]);
      dst[0] = make_int4(o[0], o[1], o[2], o[3]);
      dst[1] = make_int4(o[4], o[5], o[6], o[7]);
      dst[2] = make_int4(o[8], o[9], o[10], o[11]);
      dst[3] = make_int4(o[12], o[13], o[14], o[15]);
    }
    __syncthreads();

    int32_t* acc_row = p.acc ? p.acc + row * p.ld_out : nullptr;
    float* y_row = p.y ? p.y + row * p.ld_out : nullptr;
    if (kch == 1) {
      for (int o = threadIdx.x; o < kGatherNT; o += kGatherThreads) {
        const int n = n0 + o;
        if (n >= P.N) break;
        int v = 0;
#pragma unroll
        for (int w = 0; w < kGatherWarps; ++w) v += s_red[w][o];
        if (acc_row) acc_row[n] = v;
        if (y_row) y_row[n] = scale_out(__ldg(P.scale + n), v);
      }
    } else {
      int32_t* ws = p.ws + (int64_t)P.ws_begin * p.B + (int64_t)t * P.N;
      for (int o = threadIdx.x; o < kGatherNT; o += kGatherThreads) {
        const int n = n0 + o;
        if (n >= P.N) break;
        int v = 0;
#pragma unroll
        for (int w = 0; w < kGatherWarps; ++w) v += s_red[w][o];
        if (v) atomicAdd(ws + n, v);
      }
      __threadfence();
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t* tk = p.tickets + (int64_t)P.ticket_begin * p.B + (int64_t)t * ntile + nt;
        const uint32_t prev = atomicAdd(tk, 1u);
        const int last = prev == (uint32_t)(kch - 1);
        if (last) atomicExch(tk, 0u);       // every chunk has arrived: reset
        s_last = last;
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        for (int o = threadIdx.x; o < kGatherNT; o += kGatherThreads) {
          const int n = n0 + o;
          if (n >= P.N) break;
          const int v = __ldcg(ws + n);
          __stcg(ws + n, 0);
          if (acc_row) acc_row[n] = v;
          if (y_row) y_row[n] = scale_out(__ldg(P.scale + n), v);
        }
      }
    }
    __syncthreads();   // shared buffers are reused by the next unit
  }
}

template <int NP>
cudaError_t launch_gather_t(const GatherParamsT<NP>& p, cudaStream_t s) {
  static int grid_cap = 0;                  // SMs x resident CTAs per SM
  if (p.units_total <= 0) return cudaSuccess;
  if (grid_cap == 0) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_kernel<NP>,
                                                      kGatherThreads, 0);
    if (e != cudaSuccess) return e;
    grid_cap = sms * (per_sm > 0 ? per_sm : 1);
  }
  const int grid = p.units_total < grid_cap ? p.units_total : grid_cap;
  gather_kernel<NP><<<grid, kGatherThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gather(const GatherParams1& p, cudaStream_t s) { return launch_gather_t(p, s); }
cudaError_t launch_gather(const GatherParamsG& p, cudaStream_t s) { return launch_gather_t(p, s); }

}  // namespace sp
