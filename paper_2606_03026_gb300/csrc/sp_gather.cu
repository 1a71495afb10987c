// sp_gather.cu -- active-column gather-sum (Section 2.2, Eq. (sparse)):
//
//   acc_m = sum_{k in A} Q[k*ldw + m],   y_m = s_m * float(acc_m)
//
// for one or many (projection, token) problems in a single launch: batch-1
// decode, a group of independent projections (a whole decode step), and the
// per-token strategy of the batched call.
//
// Two forms share the per-unit work.  A unit is (problem j, token t, output
// tile of 512 channels, chunk of input columns); per unit, with no CTA-wide
// barrier before the data loads:
//   1. every warp reads the chunk's spike words (one per lane) and compacts
//      them (warp popcount and shuffle scan); warp w of W keeps the active
//      columns whose rank is w modulo W,
//   2. each lane issues its warp's column loads in rounds that keep them all
//      in flight (16 bytes of the 512-byte tile row per column: a batch into
//      registers with ld.global.nc, not allocated in L1, and a batch into
//      shared memory with cp.async) and adds them into biased 16-bit lanes
//      (at most 256 columns per warp, so the lanes cannot overflow),
//   3. the warps' partials meet in shared memory.
// Cluster form (one token per problem, K <= 6 x 1024: batch-1 decode and
// grouped decode steps): 256-thread CTAs, chunks of up to 1024 columns, and
// the chunk CTAs of a tile in one thread-block cluster that reduces its
// partials through distributed shared memory (no workspace, no atomics).
// Ticket form (any batch and K): 128-thread CTAs, 512-column chunks; acc / y
// are written directly when a tile has a single chunk, else the partial is
// added into the workspace with 16-byte fp32 vector reductions (exact:
// integer values below 2^24) and the CTA that completes the tile (atomic
// ticket == chunks - 1) reads the workspace back, writes acc and
// y = s * float(acc), and re-zeroes the workspace and the ticket.  No CTA
// ever waits on another.
// Inactive columns are never read.  Integer sums are order-free, so the
// result is bit-identical to the definition whatever the CTA schedule.
#include <atomic>

#include "sp_ptx.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

static_assert(kGatherNT == 4 * kGatherThreads, "one 4-channel vector per thread in the flush");
static_assert((kGatherWarps & (kGatherWarps - 1)) == 0 && (kGatherClusterWarps & (kGatherClusterWarps - 1)) == 0,
              "warp counts are powers of two (rank residues by mask)");
static_assert(kGatherNT / 4 <= kGatherClusterThreads, "one 4-channel group per thread");

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

// Stores 16 bytes into a peer CTA's shared memory (shared::cluster address
// `remote`) and counts them on the peer's mbarrier `remote_bar` (also a
// shared::cluster address of that CTA); the store is asynchronous.
__device__ __forceinline__ void st_async_v4(uint32_t remote, uint32_t remote_bar, int4 v) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.s32 [%0], {%1, %2, %3, %4}, [%5];"
               ::"r"(remote), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(remote_bar)
               : "memory");
}

// CTA x of the first grid row prefetches rows x, x + gridDim.x, ... of the
// (problem, token) spike rows into L2, one 128-byte line per thread, and the
// scales of problems x, x + gridDim.x, ... (read only at the very end, when a
// DRAM round trip would add to the kernel's tail).
template <int NP>
__device__ __forceinline__ void prefetch_spike_rows(const GatherParamsT<NP>& p) {
  const int rows = p.nprob * p.B;
  if (p.lif_I) {                            // LIF mode: the state and current rows
    for (int r = blockIdx.x; r < rows; r += gridDim.x) {
      const int64_t bytes = (int64_t)p.prob[r].K * 4;
      const char* vr = reinterpret_cast<const char*>(p.lif_vin + (int64_t)r * p.lif_ld);
      const char* ir = reinterpret_cast<const char*>(p.lif_I + (int64_t)r * p.lif_ld);
      for (int64_t off = (int64_t)threadIdx.x * 128; off < bytes; off += (int64_t)blockDim.x * 128) {
        asm volatile("prefetch.global.L2 [%0];" ::"l"(vr + off));
        asm volatile("prefetch.global.L2 [%0];" ::"l"(ir + off));
      }
    }
    return;
  }
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const int j = r / p.B;
    const int K = p.prob[j].K;
    const int64_t bytes = p.fmt == SP_SPIKES_BITS32 ? ((int64_t)K + 31) / 32 * 4 : (int64_t)K;
    const char* row = static_cast<const char*>(spike_row(p.spikes, p.fmt, r, p.ld_spikes));
    for (int64_t off = (int64_t)threadIdx.x * 128; off < bytes; off += (int64_t)blockDim.x * 128)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(row + off));
  }
  if (p.y == nullptr) return;
  for (int j = blockIdx.x; j < p.nprob; j += gridDim.x) {
    const char* sc = reinterpret_cast<const char*>(p.prob[j].scale);
    for (int off = threadIdx.x * 128; off < p.prob[j].N * 4; off += blockDim.x * 128)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(sc + off));
  }
}

// Shared memory of one unit with W warps, chunks of at most MAXCK columns and
// S shared-memory column slots per lane.  Per warp: its column list, and the
// landing slots of its shared-memory column loads, reused for its 512 partial
// sums once its loads are consumed (each warp touches only its own area
// until the barrier before the cross-warp sum).
template <int W, int MAXCK, int S>
struct UnitSmem {
  int cols[W][MAXCK / W];
  union WarpArea {
    uint4 stage[S][32];
    int red[kGatherNT];
  } area[W];
};

// One unit: the active columns of spike-row chunk [k0, k0 + ck) (ck a
// multiple of 32, at most MAXCK <= 1024) summed over output channels
// [n0, n0 + 512) of problem P by W warps.  Each lane keeps up to L column
// loads in registers and S more landing in shared memory in flight.  Leaves
// warp w's partial sums in sm.area[w].red and ends with a CTA barrier.
template <int W, int MAXCK, int L, int S>
__device__ __forceinline__ void unit_partial(UnitSmem<W, MAXCK, S>& sm, const GatherProblem& P,
                                             const void* srow, int fmt, int n0, int k0, int ck,
                                             const uint32_t* s_words = nullptr) {
  static_assert(MAXCK % 32 == 0 && MAXCK / 32 <= 32, "one spike word per lane");
  static_assert(MAXCK / W <= 256, "biased 16-bit lanes hold at most 257 columns");
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;

  // ---- 1. this warp's share of the chunk's active columns ---------------------
  // the chunk's spike words: from the spike row, or already in shared memory
  // (s_words[i] = columns k0 + 32 i .. k0 + 32 i + 31, bits past K clear)
  const uint32_t word = lane < ck / 32
                            ? (s_words ? s_words[lane] : spike_word(srow, fmt, P.K, k0 + 32 * lane))
                            : 0u;
  const int c = __popc(word);
  int incl = c;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += v;
  }
  const int total = __shfl_sync(0xffffffffu, incl, 31);
  {
    // this lane's bits of rank = warp (mod W): local indices i0, i0 + W, ...
    const int r0 = incl - c;                // rank of the lane's first set bit
    const int i0 = (warp - r0) & (W - 1);   // W is a power of two
    for (int i = i0; i < c; i += W)
      sm.cols[warp][(r0 + i) / W] = k0 + 32 * lane + (int)__fns(word, 0u, i + 1);
  }
  __syncwarp();
  const int mine = (total - warp + W - 1) / W;       // ranks warp, warp + W, ...

  // ---- 2. stream the columns of this output tile -------------------------------
  const int ch = n0 + lane * 16;            // first channel of this lane
  const bool lane_on = ch < P.N;
  const int8_t* wcol = P.W + ch;
  const int64_t ldw = P.ldw;
  uint32_t ev[4] = {0u, 0u, 0u, 0u}, od[4] = {0u, 0u, 0u, 0u};
  uint4* stage = &sm.area[warp].stage[0][lane];     // slot b at stage[32 * b]
  // Rounds of up to L + S columns per warp, all in flight together: the
  // columns past the register batch are copied into shared memory with
  // cp.async first, then the register batch is loaded and added, then the
  // shared-memory columns.
  for (int i0 = 0; i0 < mine; i0 += L + S) {
    const int ns = min(S, mine - i0 - L);   // warp-uniform, may be <= 0
    if (lane_on)
      for (int b = 0; b < ns; ++b) cp_async16(stage + 32 * b, wcol + sm.cols[warp][i0 + L + b] * ldw);
    cp_async_commit();
    uint4 v[L];
#pragma unroll
    for (int b = 0; b < L; ++b) {
      v[b] = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
      if (lane_on && i0 + b < mine) v[b] = ld_weights16(wcol + sm.cols[warp][i0 + b] * ldw);
    }
#pragma unroll
    for (int b = 0; b < L; ++b) {
      acc_bytes(v[b].x, ev[0], od[0]);
      acc_bytes(v[b].y, ev[1], od[1]);
      acc_bytes(v[b].z, ev[2], od[2]);
      acc_bytes(v[b].w, ev[3], od[3]);
    }
    cp_async_wait_all();                    // this lane's copies have landed
    for (int b = 0; b < ns; ++b) {
      const uint4 w = stage[32 * b];
      acc_bytes(w.x, ev[0], od[0]);
      acc_bytes(w.y, ev[1], od[1]);
      acc_bytes(w.z, ev[2], od[2]);
      acc_bytes(w.w, ev[3], od[3]);
    }
  }

  // ---- 3. per-warp partials ------------------------------------------------------
  // padding loads (0x80 bytes) add 0 to the biased lanes: only the `mine`
  // real columns carry the +128 bias
  int o[16];
  unbias16(ev[0], od[0], mine, o + 0);
  unbias16(ev[1], od[1], mine, o + 4);
  unbias16(ev[2], od[2], mine, o + 8);
  unbias16(ev[3], od[3], mine, o + 12);
  __syncwarp();                             // every lane is done with the warp's slots
  int4* dst = reinterpret_cast<int4*>(&sm.area[warp].red[lane * 16]);
  dst[0] = make_int4(o[0], o[1], o[2], o[3]);
  dst[1] = make_int4(o[4], o[5], o[6], o[7]);
  dst[2] = make_int4(o[8], o[9], o[10], o[11]);
  dst[3] = make_int4(o[12], o[13], o[14], o[15]);
  __syncthreads();
}

// Sum of the W warps' partials for tile channels o .. o + 3.
template <int W, int MAXCK, int S>
__device__ __forceinline__ int4 unit_sum4(const UnitSmem<W, MAXCK, S>& sm, int o) {
  int4 s = make_int4(0, 0, 0, 0);
#pragma unroll
  for (int w = 0; w < W; ++w) {
    const int4 r = *reinterpret_cast<const int4*>(&sm.area[w].red[o]);
    s.x += r.x;
    s.y += r.y;
    s.z += r.z;
    s.w += r.w;
  }
  return s;
}

// Scales of channels n .. n + 3 (read only where y is written).
__device__ __forceinline__ float4 scale4(const GatherProblem& P, int n) {
  return make_float4(__ldg(P.scale + n), __ldg(P.scale + n + 1), __ldg(P.scale + n + 2),
                     __ldg(P.scale + n + 3));
}

// acc and y = s * float(acc) of channels n .. n + 3, sc = their scales.
__device__ __forceinline__ void write4(int32_t* acc_row, float* y_row, int n, int4 v, float4 sc) {
  // one 16-byte store each where the rows allow it (the output may also be
  // page-locked host memory, where every transaction crosses the link)
  const bool v4 = ((reinterpret_cast<uintptr_t>(acc_row) | reinterpret_cast<uintptr_t>(y_row)) & 15u) == 0;
  if (v4) {
    if (acc_row) *reinterpret_cast<int4*>(acc_row + n) = v;
    if (y_row)
      *reinterpret_cast<float4*>(y_row + n) = make_float4(
          scale_out(sc.x, v.x), scale_out(sc.y, v.y), scale_out(sc.z, v.z), scale_out(sc.w, v.w));
    return;
  }
  if (acc_row) {
    acc_row[n] = v.x;
    acc_row[n + 1] = v.y;
    acc_row[n + 2] = v.z;
    acc_row[n + 3] = v.w;
  }
  if (y_row) {
    y_row[n] = scale_out(sc.x, v.x);
    y_row[n + 1] = scale_out(sc.y, v.y);
    y_row[n + 2] = scale_out(sc.z, v.z);
    y_row[n + 3] = scale_out(sc.w, v.w);
  }
}

// ---------------------------------------------------------------------------
// Ticket form: any number of tokens and chunks.  128-thread CTAs, one per
// (problem, token, 512-channel tile, 512-column chunk) unit.  Grid = (tokens
// x units of the largest problem, problems); the output tile is the fastest
// index so that the tiles of one column chunk run side by side.
constexpr int kTicketWarps = kGatherWarps;         // 4
constexpr int kTicketLoads = 11;                   // column loads per lane in registers (72 registers)
constexpr int kTicketSlots = 8;                    // and in shared memory
using TicketSmem = UnitSmem<kTicketWarps, kGatherCK, kTicketSlots>;

template <int NP>
__global__ void __launch_bounds__(kGatherThreads, 7)
gather_kernel(const __grid_constant__ GatherParamsT<NP> p) {
  __shared__ TicketSmem sm;
  __shared__ int s_last;
  // The next launch may take free SM slots now.  The first grid row starts
  // first: it pulls every spike row of the launch into L2 before the
  // column-load burst fills the DRAM queues, so that units that start late
  // do not wait behind that burst for their spike words.  A prefetch hands
  // no data to the kernel, so it may run before the wait for the previous
  // kernel (if that kernel writes the rows, L2 simply holds its writes);
  // every load and store of this grid comes after the wait.
  pdl_launch_dependents();
  if (blockIdx.y == 0) prefetch_spike_rows(p);
  pdl_wait();

  const int j = blockIdx.y;
  const int t = (int)(blockIdx.x / (unsigned)p.max_units);
  const int x = (int)blockIdx.x - t * p.max_units;
  const GatherProblem& P = p.prob[j];
  const int kch = gather_kchunks(P.K);
  const int ntile = gather_ntiles(P.N);
  if (x >= ntile * kch) return;             // this problem has fewer units
  const int kc = x / ntile;
  const int nt = x - kc * ntile;
  const int n0 = nt * kGatherNT;
  const int64_t row = (int64_t)j * p.B + t;
  unit_partial<kTicketWarps, kGatherCK, kTicketLoads, kTicketSlots>(
      sm, P, spike_row(p.spikes, p.fmt, row, p.ld_spikes), p.fmt, n0, kc * kGatherCK, kGatherCK);

  int32_t* acc_row = p.acc ? p.acc + row * p.ld_out : nullptr;
  float* y_row = p.y ? p.y + row * p.ld_out : nullptr;
  const int o = threadIdx.x * 4;
  const int n = n0 + o;                     // N % 16 == 0: the 4 channels are all valid or none
  if (kch == 1) {
    if (p.fault == kFaultAbort) {           // test fault: the output stays unwritten
      if (threadIdx.x == 0) atomicExch(p.err, kErrInjected);
      return;
    }
    if (n < P.N) write4(acc_row, y_row, n, unit_sum4(sm, o), y_row ? scale4(P, n) : float4{});
    return;
  }
  // Partials go into the workspace as fp32 16-byte vector reductions (one per
  // thread).  fp32 is exact here: every partial and every sum is an integer
  // of magnitude <= 128 * K < 2^24, so the result does not depend on the
  // order of the additions.
  float* ws = reinterpret_cast<float*>(p.ws) + (int64_t)P.ws_begin * p.B + (int64_t)t * P.N;
  if (n < P.N) {
    const int4 v = unit_sum4(sm, o);
    if (v.x | v.y | v.z | v.w) red_add_v4(ws + n, (float)v.x, (float)v.y, (float)v.z, (float)v.w);
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
    int last = prev == (uint32_t)(kch - 1);
    if (last && p.fault == kFaultAbort) {   // test fault: workspace and ticket left dirty
      atomicExch(p.err, kErrInjected);
      last = 0;
    }
    if (last) {
      atomicExch(tk, 0u);                   // every chunk has arrived: reset
      __threadfence();
    }
    s_last = last;
  }
  __syncthreads();
  if (s_last && n < P.N) {
    const float4 f = __ldcg(reinterpret_cast<const float4*>(ws + n));
    __stcg(reinterpret_cast<float4*>(ws + n), make_float4(0.f, 0.f, 0.f, 0.f));
    write4(acc_row, y_row, n,
           make_int4(__float2int_rn(f.x), __float2int_rn(f.y), __float2int_rn(f.z),
                     __float2int_rn(f.w)),
           y_row ? scale4(P, n) : float4{});
  }
}

// ---------------------------------------------------------------------------
// Cluster form: one token per problem, at most CL chunks of at most 1024
// columns per tile.  256-thread CTAs in clusters of CL (6 for a group of
// projections; 12 or 16 for a single projection, which then spreads over more
// SMs); a cluster holds tpc tiles x kch chunks of one problem (rank = tile
// slot * kch + chunk; kch divides CL); the grid lists the clusters one by one
// (or is (clusters of the largest problem x CL, problems)).  The 128
// 4-channel groups of a tile are split into kch contiguous runs, run c owned
// by the CTA of chunk c.  Every CTA stores its partial of each group into the
// owner's shared memory with st.async (distributed shared memory), which
// counts the bytes on the owner's mbarrier; the owner's threads wait on that
// barrier alone, add the kch partials of their groups and write acc / y.  No
// workspace, no atomics, no cluster-wide barrier after the column loads: a
// CTA finishes as soon as its own groups are complete, whatever the other
// tiles of its cluster are doing.  (Ending with a release / acquire cluster
// barrier instead cost 0.5 us per 22-block decode step.)
constexpr int kClusterLoads = 9;                   // column loads per lane in registers (64 registers)
// and in shared memory: 8 for a group (4 CTAs per SM), 16 for a single
// projection's clusters of 12 or 16 (fewer CTAs, each with more columns)
template <int CL> constexpr int cluster_slots() { return CL > 8 ? 16 : 8; }
template <int CL>
using ClusterSmem = UnitSmem<kGatherClusterWarps, kGatherClusterMaxCK, cluster_slots<CL>()>;

// kLif: the fused spike producer (a separate instantiation, so that the plain
// decode carries none of its code)
template <int NP, bool kLif, int CL>
__global__ void __launch_bounds__(kGatherClusterThreads, 4)
gather_cluster_kernel(const __grid_constant__ GatherParamsT<NP> p) {
  extern __shared__ __align__(16) uint8_t dyn_smem[];   // ClusterSmem<CL>, sized at launch
  ClusterSmem<CL>& sm = *reinterpret_cast<ClusterSmem<CL>*>(dyn_smem);
  // [sender chunk][owned group]: kch * ceil(128 / kch) < 128 + kch entries
  __shared__ __align__(16) int4 s_recv[kGatherNT / 4 + CL];
  __shared__ uint32_t s_lif[kLif ? kGatherClusterMaxCK / 32 : 1];   // LIF mode: the chunk's spike words
  __shared__ __align__(8) uint64_t s_bar;   // completes when every partial for s_recv has landed

  // the unit (kernel parameters only: known before the dependency wait)
  const int c = (int)blockIdx.x / CL;
  const int rank = (int)blockIdx.x - c * CL;   // rank in the (CL, 1, 1) cluster
  int j = blockIdx.y, cl = c;
  if (p.ncl_list > 0) {                     // listed clusters: no idle CTAs
    const int e = p.cl_list[c];
    j = e >> 8;
    cl = e & 0xff;
  }
  const GatherProblem& P = p.prob[j];
  const int kch = P.kch;
  const int per = (kGatherNT / 4 + kch - 1) / kch;   // most groups owned by one CTA
  const int ts = rank / kch;
  const int kc = rank - ts * kch;
  const int n0 = (cl * P.tpc + ts) * kGatherNT;
  const bool work = cl < P.ncl && n0 < P.N;  // idle clusters and tile slots past the last tile
  const int owned = min(per, kGatherNT / 4 - kc * per);   // groups this CTA owns
  if (threadIdx.x == 0 && work) {
    // every CTA of the tile stores its partial of each owned group here:
    // kch * owned 16-byte stores, counted in bytes on s_bar
    mbar_init(&s_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    mbar_arrive_expect_tx(&s_bar, (uint32_t)(kch * owned * 16));
  }
  // every CTA of the cluster arrives here and waits (below) before its first
  // store into a peer's shared memory: the peer is then known to be running,
  // with its barrier initialised
  asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory");
  pdl_launch_dependents();
  if (blockIdx.y == 0) prefetch_spike_rows(p);   // before the wait: see gather_kernel
  pdl_wait();
  if (!work) return;                        // nothing is stored into an idle CTA

  // This thread's owned group (a contiguous run of the tile's 4-channel
  // groups), set after the column loads (nothing extra is live across them).
  int n = 0;
  bool owner = false;
  float4 sc = float4{};
  if constexpr (kLif) {
    // fused spike producer: one LIF step of this chunk's neurons (every CTA
    // of the chunk computes the same words from the old state; the CTA of
    // tile slot 0 in cluster 0 writes the new state and the bits)
    const int k0 = kc * P.ck;
    const float* vr = p.lif_vin + (int64_t)j * p.lif_ld;
    const float* ir = p.lif_I + (int64_t)j * p.lif_ld;
    const bool writer = cl == 0 && ts == 0;
    for (int i = threadIdx.x; i < P.ck; i += kGatherClusterThreads) {   // warp-uniform: ck % 32 == 0
      const int k = k0 + i;
      bool fire = false;
      if (k < P.K) {
        float u = fmaf(p.lif_beta, vr[k], ir[k]);
        fire = u >= p.lif_theta;
        if (fire) u = __fsub_rn(u, p.lif_theta);
        if (writer) p.lif_vout[(int64_t)j * p.lif_ld + k] = u;
      }
      const uint32_t w = __ballot_sync(0xffffffffu, fire);
      if ((threadIdx.x & 31) == 0) {
        s_lif[i >> 5] = w;
        if (writer && p.lif_bits && k < P.K) p.lif_bits[(int64_t)j * p.lif_ld_bits + (k >> 5)] = w;
      }
    }
    __syncthreads();
  }
  unit_partial<kGatherClusterWarps, kGatherClusterMaxCK, kClusterLoads, cluster_slots<CL>()>(
      sm, P, kLif ? nullptr : spike_row(p.spikes, p.fmt, j, p.ld_spikes), p.fmt, n0, kc * P.ck,
      P.ck, kLif ? s_lif : nullptr);
  // the owner's scales, read now: their load overlaps the exchange instead
  // of following the owner's wait
  {
    const int g_own = kc * per + (int)threadIdx.x;
    n = n0 + 4 * g_own;
    owner = (int)threadIdx.x < per && g_own < kGatherNT / 4 && n < P.N;
  }
  if (owner && p.y) sc = scale4(P, n);
  asm volatile("barrier.cluster.wait;" ::: "memory");
  const int g = threadIdx.x;              // the 4-channel group of this thread
  // test stall: the first CTA's partials are never stored, so its tile's
  // owners wait until their (shortened) bound runs out
  const bool stall = p.fault == kFaultStall;
  if (g < kGatherNT / 4 && !(stall && blockIdx.x == 0 && blockIdx.y == 0)) {
    const int4 v = unit_sum4(sm, 4 * g);
    const int o = g / per;                // the owning chunk
    const uint32_t dst = (uint32_t)(ts * kch + o);
    st_async_v4(cluster_addr(&s_recv[kc * per + (g - o * per)], dst), cluster_addr(&s_bar, dst), v);
  }
  // the owner's threads wait for the kch partials of their groups (no
  // cluster-wide barrier: a CTA goes on as soon as its own groups are in)
  if ((int)threadIdx.x < per && !mbar_wait(&s_bar, 0, stall ? kStallWaitCycles : kWaitLimitCycles)) {
    if (p.err) atomicExch(p.err, kErrFlagTimeout);   // (the allocation-free call has none)
    return;
  }
  if (p.fault == kFaultAbort) {             // test fault: the output stays unwritten
    if (threadIdx.x == 0) atomicExch(p.err, kErrInjected);
    return;
  }
  if (owner) {
    int4 s = make_int4(0, 0, 0, 0);
    for (int q = 0; q < kch; ++q) {
      const int4 v = s_recv[q * per + threadIdx.x];
      s.x += v.x;
      s.y += v.y;
      s.z += v.z;
      s.w += v.w;
    }
    write4(p.acc ? p.acc + (int64_t)j * p.ld_out : nullptr,
           p.y ? p.y + (int64_t)j * p.ld_out : nullptr, n, s, sc);
  }
}

// Asks for the largest shared-memory carveout once per device and kernel, so
// that every resident CTA's shared memory fits beside L1.
template <typename Kern>
cudaError_t set_carveout(Kern kernel, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_relaxed) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           (int)cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_relaxed);
  return e;
}

// Clusters of the cluster form that can be resident at once (per device).
template <int NP, bool kLif, int CL>
int cluster_capacity() {
  static std::atomic<int> cap[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev >= 64) return 0;
  int n = cap[dev].load(std::memory_order_relaxed);
  if (n != 0) return n;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = CL;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.gridDim = dim3(CL, 1, 1);
  cfg.blockDim = dim3(kGatherClusterThreads, 1, 1);
  cfg.dynamicSmemBytes = sizeof(ClusterSmem<CL>);
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  if (cudaOccupancyMaxActiveClusters(&n, gather_cluster_kernel<NP, kLif, CL>, &cfg) != cudaSuccess ||
      n < 1) {
    (void)cudaGetLastError();
    n = -1;
  }
  cap[dev].store(n, std::memory_order_relaxed);
  return n;
}

// Resident-cluster count of the kernel the launch will use (0 on failure).
template <int NP>
int capacity_for(bool lif, int CL) {
  if (lif) return cluster_capacity<NP, true, 6>();
  switch (CL) {
    case 16: return cluster_capacity<NP, false, 16>();
    case 12: return cluster_capacity<NP, false, 12>();
    default: return cluster_capacity<NP, false, 6>();
  }
}

// Fills the cluster-form fields of q and the cluster size *cl_out; false
// when the launch does not fit the cluster form (several tokens, a chunk
// count above the cluster size, or more clusters than can be resident at
// once).  A group of projections takes clusters of 6 and the fewest chunks
// of at most 1024 columns.  A single projection (which alone would leave
// most SMs idle) takes the cluster size and chunking with the most working
// CTAs among clusters of 16, 12 and 6, chunks of 256 to 1024 columns and at
// most a quarter of the tile slots idle.  Up to kGatherMaxClusterList
// clusters are listed one by one (a 1-D grid of exactly the clusters with
// work, all resident together); more take a (clusters x CL, problems) grid
// in which the problems with fewer clusters leave idle CTAs.
template <int NP>
bool cluster_form(GatherParamsT<NP>& q, int* grid_x, int* grid_y, int* cl_out) {
  if (q.B != 1) return false;
  int CL = 6;
  if (q.nprob == 1 && !q.lif_I) {
    GatherProblem& P = q.prob[0];
    const int ntiles = gather_ntiles(P.N);
    int best = 0;
    for (const int cand : {16, 12, 6}) {
      for (int kch = cand; kch >= 1; --kch) {
        if (cand % kch != 0) continue;
        const int ck = ceil_div(ceil_div(P.K, kch), 32) * 32;
        if (ck > kGatherClusterMaxCK || (ck < 256 && kch > 1)) continue;
        const int tpc = cand / kch;
        const int ncl = ceil_div(ntiles, tpc);
        if (4 * (ncl * tpc - ntiles) > ncl * tpc) continue;   // more than a quarter idle
        const int working = ntiles * kch;
        if (working > best) {
          best = working;
          CL = cand;
          P.kch = kch;
        }
        break;                              // the most chunks this size allows
      }
    }
    if (best == 0) return false;
    P.ck = ceil_div(ceil_div(P.K, P.kch), 32) * 32;
    P.tpc = CL / P.kch;
    P.ncl = ceil_div(ntiles, P.tpc);
  } else {
    for (int j = 0; j < q.nprob; ++j) {
      GatherProblem& P = q.prob[j];
      // the fewest chunks (a divisor of the cluster size) of at most 1024 columns
      int kch = 0;
      for (int d = 1; d <= CL; ++d)
        if (CL % d == 0 && ceil_div(P.K, d) <= kGatherClusterMaxCK) {
          kch = d;
          break;
        }
      if (kch == 0) return false;
      P.kch = kch;
      P.ck = ceil_div(ceil_div(P.K, kch), 32) * 32;
      P.tpc = CL / kch;
      P.ncl = ceil_div(gather_ntiles(P.N), P.tpc);
    }
  }
  int total = 0, widest = 0;
  for (int j = 0; j < q.nprob; ++j) {
    total += q.prob[j].ncl;
    if (q.prob[j].ncl > widest) widest = q.prob[j].ncl;
  }
  if (total > capacity_for<NP>(q.lif_I != nullptr, CL)) return false;
  q.ncl_list = 0;
  if (total <= kGatherMaxClusterList && widest <= 0xff) {
    int c = 0;
    for (int j = 0; j < q.nprob; ++j)
      for (int cl = 0; cl < q.prob[j].ncl; ++cl) q.cl_list[c++] = (uint16_t)((j << 8) | cl);
    q.ncl_list = total;
    *grid_x = total * CL;
    *grid_y = 1;
  } else {
    *grid_x = widest * CL;
    *grid_y = q.nprob;
  }
  *cl_out = CL;
  return true;
}

// Sets the one-time attributes of a cluster-form kernel, once per device: the
// largest shared-memory carveout (the resident-cluster count depends on it),
// for clusters above 8 CTAs the non-portable cluster size, and the dynamic
// shared memory above 48 KB.  (Each is a driver call of about a microsecond:
// set on every launch they made a single decode's host time the bound.)
template <typename Kern>
cudaError_t cluster_attrs(Kern kernel, int CL, size_t smem, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_relaxed) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           (int)cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess && CL > 8)
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess && smem > 48 * 1024)
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_relaxed);
  return e;
}

template <int NP>
cudaError_t launch_gather_t(const GatherParamsT<NP>& p, cudaStream_t s) {
  static std::atomic<uint64_t> carve_t{0}, carve_c{0}, carve_l{0}, carve_12{0}, carve_16{0};
  if (p.units_total <= 0 || p.B <= 0 || p.max_units <= 0) return cudaSuccess;
  // the attributes first: the resident-cluster counts depend on the carveout
  cudaError_t e = p.lif_I
                      ? cluster_attrs(gather_cluster_kernel<NP, true, 6>, 6, sizeof(ClusterSmem<6>), carve_l)
                      : cluster_attrs(gather_cluster_kernel<NP, false, 6>, 6, sizeof(ClusterSmem<6>), carve_c);
  if (e == cudaSuccess && !p.lif_I && p.nprob == 1) {
    e = cluster_attrs(gather_cluster_kernel<NP, false, 12>, 12, sizeof(ClusterSmem<12>), carve_12);
    if (e == cudaSuccess)
      e = cluster_attrs(gather_cluster_kernel<NP, false, 16>, 16, sizeof(ClusterSmem<16>), carve_16);
  }
  if (e != cudaSuccess) return e;
  GatherParamsT<NP> q = p;
  int gx = 0, gy = 0, CL = 6;
  const bool cluster = cluster_form(q, &gx, &gy, &CL);
  if (p.lif_I && !cluster) return cudaErrorNotSupported;   // the fused producer needs the cluster form
  if (cluster) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)gx, (unsigned)gy, 1);
    cfg.blockDim = dim3(kGatherClusterThreads, 1, 1);
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    if (p.lif_I) {
      cfg.dynamicSmemBytes = sizeof(ClusterSmem<6>);
      return cudaLaunchKernelEx(&cfg, gather_cluster_kernel<NP, true, 6>, q);
    }
    switch (CL) {
      case 16:
        cfg.dynamicSmemBytes = sizeof(ClusterSmem<16>);
        return cudaLaunchKernelEx(&cfg, gather_cluster_kernel<NP, false, 16>, q);
      case 12:
        cfg.dynamicSmemBytes = sizeof(ClusterSmem<12>);
        return cudaLaunchKernelEx(&cfg, gather_cluster_kernel<NP, false, 12>, q);
      default:
        cfg.dynamicSmemBytes = sizeof(ClusterSmem<6>);
        return cudaLaunchKernelEx(&cfg, gather_cluster_kernel<NP, false, 6>, q);
    }
  }
  e = set_carveout(gather_kernel<NP>, carve_t);
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
