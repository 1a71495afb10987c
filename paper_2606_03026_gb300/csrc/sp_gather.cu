// sp_gather.cu -- active-column gather-sum (Section 2.2, Eq. (sparse)):
//
//   acc_m = sum_{k in A} Q[k*ldw + m],   y_m = s_m * float(acc_m)
//
// for one or many (projection, token) problems in a single launch: batch-1
// decode, a group of independent projections (a whole decode step), and the
// per-token strategy of the batched call.
//
// Decomposition: a work unit is (problem j, token t, output tile of 512
// channels, chunk of 512 input columns), and one 128-thread CTA does one
// unit.  Units are small (about 26 KB of active columns at 10% spikes) and
// many CTAs fit on an SM, so all units of a decode step are resident at once
// and the memory system sees the whole step's column reads together.  Per
// unit, with no CTA-wide barrier before the data loads:
//   1. every warp reads the chunk's 16 spike words and compacts them (warp
//      popcount and shuffle scan); warp w keeps the active columns whose rank
//      is w modulo 4,
//   2. each lane issues its warp's column loads, up to 19 at once (16 bytes
//      of the 512-byte tile row per column: 11 into registers with
//      ld.global.nc, not allocated in L1, and 8 into shared memory with
//      cp.async) and adds them into biased 16-bit lanes (at most 128 columns
//      per warp, so the lanes cannot overflow),
//   3. the 4 warps are summed through shared memory and
//      - acc / y are written directly when the problem has a single chunk, or
//      - the partial is added into the workspace with 16-byte fp32 vector
//        reductions (exact: integer values below 2^24); the CTA that
//        completes the tile (atomic ticket == chunks - 1) reads the workspace
//        back, writes acc and y = s * float(acc), and re-zeroes the workspace
//        and the ticket.  No CTA ever waits on another.
// Inactive columns are never read.  Integer sums are order-free, so the
// result is bit-identical to the definition whatever the CTA schedule.
#include <atomic>

#include "sp_ptx.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int kWarps = kGatherWarps;               // 4
constexpr int kWords = kGatherCK / 32;             // spike words per chunk (16)
constexpr int kPerWarp = kGatherCK / kWarps;       // column-list capacity per warp
constexpr int kLoadBatch = 11;                     // column loads per lane into registers (72 registers)
constexpr int kSmemSlots = 8;                      // further column loads per lane into shared memory
static_assert(kGatherNT == 4 * kGatherThreads, "one 4-channel vector per thread in the flush");

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

__device__ __forceinline__ void red_add_v4(float* addr, float a, float b, float c, float d) {
  asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(addr), "f"(a),
               "f"(b), "f"(c), "f"(d)
               : "memory");
}

// CTA x of the first grid row prefetches rows x, x + gridDim.x, ... of the
// (problem, token) spike rows into L2, one 128-byte line per thread.
template <int NP>
__device__ __forceinline__ void prefetch_spike_rows(const GatherParamsT<NP>& p) {
  const int rows = p.nprob * p.B;
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const int j = r / p.B;
    const int K = p.prob[j].K;
    const int64_t bytes = p.fmt == SP_SPIKES_BITS32 ? ((int64_t)K + 31) / 32 * 4 : (int64_t)K;
    const char* row = static_cast<const char*>(spike_row(p.spikes, p.fmt, r, p.ld_spikes));
    for (int64_t off = (int64_t)threadIdx.x * 128; off < bytes; off += (int64_t)kGatherThreads * 128)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(row + off));
  }
}

template <int NP>
__global__ void __launch_bounds__(kGatherThreads, 7)
gather_kernel(const __grid_constant__ GatherParamsT<NP> p) {
  __shared__ int s_cols[kWarps][kPerWarp];
  // Per warp: the landing slots of its shared-memory column loads, reused for
  // its 512 partial sums once its loads are consumed (each warp touches only
  // its own region until the barrier before the cross-warp sum).
  union WarpArea {
    uint4 stage[kSmemSlots][32];
    int red[kGatherNT];
  };
  __shared__ __align__(16) WarpArea s_area[kWarps];
  __shared__ int s_last;

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  // the next launch may take free SM slots now; this grid's own memory work
  // starts once the previous kernel has finished
  pdl_launch_dependents();
  pdl_wait();
  // The first grid row starts first: it pulls every spike row of the launch
  // into L2 before the column-load burst fills the DRAM queues, so that units
  // that start late do not wait behind that burst for their spike words.
  if (blockIdx.y == 0) prefetch_spike_rows(p);

  // grid = (tokens x units of the largest problem, problems): token t, unit x
  // of problem blockIdx.y; the output tile is the fastest index so that the
  // tiles of one column chunk run side by side
  {
    const int j = blockIdx.y;
    const int t = (int)(blockIdx.x / (unsigned)p.max_units);
    const int x = (int)blockIdx.x - t * p.max_units;
    const GatherProblem& P = p.prob[j];
    const int kch = gather_kchunks(P.K);
    const int ntile = gather_ntiles(P.N);
    if (x >= ntile * kch) return;           // this problem has fewer units
    const int kc = x / ntile;
    const int nt = x - kc * ntile;
    const int n0 = nt * kGatherNT;
    const int k0 = kc * kGatherCK;
    const int64_t row = (int64_t)j * p.B + t;

    // ---- 1. this warp's share of the chunk's active columns -------------------
    const void* srow = spike_row(p.spikes, p.fmt, row, p.ld_spikes);
    const uint32_t word = lane < kWords ? spike_word(srow, p.fmt, P.K, k0 + 32 * lane) : 0u;
    const int c = __popc(word);
    int incl = c;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += v;
    }
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    {
      uint32_t w = word;
      int rank = incl - c;
      while (w) {
        const int b = __ffs(w) - 1;
        w &= w - 1u;
        if ((rank & (kWarps - 1)) == warp) s_cols[warp][rank >> 2] = k0 + 32 * lane + b;
        ++rank;
      }
    }
    __syncwarp();
    const int mine = (total - warp + kWarps - 1) / kWarps;   // ranks warp, warp+4, ...

    // ---- 2. stream the columns of this output tile -------------------------------
    const int ch = n0 + lane * 16;          // first channel of this lane
    const bool lane_on = ch < P.N;
    const int8_t* wcol = P.W + ch;
    const int64_t ldw = P.ldw;
    uint32_t ev[4] = {0u, 0u, 0u, 0u}, od[4] = {0u, 0u, 0u, 0u};
    uint4* stage = &s_area[warp].stage[0][lane];     // slot b at stage[32 * b]
    // Rounds of up to kLoadBatch + kSmemSlots columns per warp, all in flight
    // together (one round covers a unit at 10% spikes): the columns past the
    // register batch are copied into shared memory with cp.async first, then
    // the register batch is loaded and added, then the shared-memory columns.
    for (int i0 = 0; i0 < mine; i0 += kLoadBatch + kSmemSlots) {
      const int ns = min(kSmemSlots, mine - i0 - kLoadBatch);   // warp-uniform, may be <= 0
      if (lane_on)
        for (int b = 0; b < ns; ++b)
          cp_async16(stage + 32 * b, wcol + s_cols[warp][i0 + kLoadBatch + b] * ldw);
      cp_async_commit();
      uint4 v[kLoadBatch];
#pragma unroll
      for (int b = 0; b < kLoadBatch; ++b) {
        v[b] = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
        if (lane_on && i0 + b < mine) v[b] = ld_weights16(wcol + s_cols[warp][i0 + b] * ldw);
      }
#pragma unroll
      for (int b = 0; b < kLoadBatch; ++b) {
        acc_bytes(v[b].x, ev[0], od[0]);
        acc_bytes(v[b].y, ev[1], od[1]);
        acc_bytes(v[b].z, ev[2], od[2]);
        acc_bytes(v[b].w, ev[3], od[3]);
      }
      cp_async_wait_all();                  // this lane's copies have landed
      for (int b = 0; b < ns; ++b) {
        const uint4 w = stage[32 * b];
        acc_bytes(w.x, ev[0], od[0]);
        acc_bytes(w.y, ev[1], od[1]);
        acc_bytes(w.z, ev[2], od[2]);
        acc_bytes(w.w, ev[3], od[3]);
      }
    }
    // padding loads (0x80 bytes) add 0 to the biased lanes: only the `mine`
    // real columns carry the +128 bias
    const int nacc = mine;

    // ---- 3. reduce the warps -------------------------------------------------
    {
      int o[16];
      unbias16(ev[0], od[0], nacc, o + 0);
      unbias16(ev[1], od[1], nacc, o + 4);
      unbias16(ev[2], od[2], nacc, o + 8);
      unbias16(ev[3], od[3], nacc, o + 12);
      __syncwarp();                         // every lane is done with the warp's slots
      int4* dst = reinterpret_cast<int4*>(&s_area[warp].red[lane * 16]);
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
        const int v = s_area[0].red[o] + s_area[1].red[o] + s_area[2].red[o] + s_area[3].red[o];
        if (acc_row) acc_row[n] = v;
        if (y_row) y_row[n] = scale_out(__ldg(P.scale + n), v);
      }
    } else {
      // Partials go into the workspace as fp32 16-byte vector reductions (one
      // per thread: channels n0 + 4i .. n0 + 4i + 3).  fp32 is exact here:
      // every partial and every sum is an integer of magnitude <= 128 * K <
      // 2^24, so the result does not depend on the order of the additions.
      float* ws = reinterpret_cast<float*>(p.ws) + (int64_t)P.ws_begin * p.B + (int64_t)t * P.N;
      const int o = threadIdx.x * 4;
      const int n = n0 + o;                 // N % 16 == 0: the 4 channels are all valid or none
      if (n < P.N) {
        const int4 r0 = *reinterpret_cast<const int4*>(&s_area[0].red[o]);
        const int4 r1 = *reinterpret_cast<const int4*>(&s_area[1].red[o]);
        const int4 r2 = *reinterpret_cast<const int4*>(&s_area[2].red[o]);
        const int4 r3 = *reinterpret_cast<const int4*>(&s_area[3].red[o]);
        const int v0 = r0.x + r1.x + r2.x + r3.x, v1 = r0.y + r1.y + r2.y + r3.y;
        const int v2 = r0.z + r1.z + r2.z + r3.z, v3 = r0.w + r1.w + r2.w + r3.w;
        if (v0 | v1 | v2 | v3) red_add_v4(ws + n, (float)v0, (float)v1, (float)v2, (float)v3);
      }
      // Release: the barrier orders the CTA's reductions before thread 0, whose
      // GPU-scope fence makes them visible before its ticket increment.  The
      // thread that completes the tile fences again (acquire) before the CTA
      // reads the workspace back.
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t* tk = p.tickets + (int64_t)P.ticket_begin * p.B + (int64_t)t * ntile + nt;
        __threadfence();
        const uint32_t prev = atomicAdd(tk, 1u);
        const int last = prev == (uint32_t)(kch - 1);
        if (last) {
          atomicExch(tk, 0u);               // every chunk has arrived: reset
          __threadfence();
        }
        s_last = last;
      }
      __syncthreads();
      if (s_last && n < P.N) {
        const float4 f = __ldcg(reinterpret_cast<const float4*>(ws + n));
        __stcg(reinterpret_cast<float4*>(ws + n), make_float4(0.f, 0.f, 0.f, 0.f));
        const int v[4] = {__float2int_rn(f.x), __float2int_rn(f.y), __float2int_rn(f.z),
                          __float2int_rn(f.w)};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (acc_row) acc_row[n + k] = v[k];
          if (y_row) y_row[n + k] = scale_out(__ldg(P.scale + n + k), v[k]);
        }
      }
    }
  }
}

// Asks for the largest shared-memory carveout once per device, so that 7
// CTAs (7 x 18 KB of shared memory) fit on an SM beside their L1.
template <int NP>
cudaError_t set_carveout() {
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_relaxed) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(gather_kernel<NP>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           (int)cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_relaxed);
  return e;
}

template <int NP>
cudaError_t launch_gather_t(const GatherParamsT<NP>& p, cudaStream_t s) {
  if (p.units_total <= 0 || p.B <= 0 || p.max_units <= 0) return cudaSuccess;
  const cudaError_t e = set_carveout<NP>();
  if (e != cudaSuccess) return e;
  if ((int64_t)p.max_units * p.B > 0x7fffffffll) return cudaErrorInvalidConfiguration;
  // one CTA per unit; the hardware keeps every unit of a decode step resident
  // (7 CTAs of 128 threads per SM) and schedules the rest in waves
  const dim3 grid((unsigned)(p.max_units * p.B), (unsigned)p.nprob, 1);
  return launch_pdl(gather_kernel<NP>, grid, dim3(kGatherThreads), 0, s, p);
}

}  // namespace

cudaError_t launch_gather(const GatherParams1& p, cudaStream_t s) { return launch_gather_t(p, s); }
cudaError_t launch_gather(const GatherParamsG& p, cudaStream_t s) { return launch_gather_t(p, s); }

}  // namespace sp
