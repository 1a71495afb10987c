// sp_gemm.cu -- dense tensor-core path for many spike rows at once:
//
//   ACC[t][m] = sum_k X[t][k] * Q[m][k],   Y[t][m] = s_m * float(ACC[t][m])
//
// i.e. Eq. (sparse) for every row of a dense spike matrix (prompt prefill).
//
// The 5th-generation tensor cores of sm_103a have no integer MMA
// (ptxas rejects tcgen05.mma .kind::i8 for this target).  The contraction runs
// as tcgen05.mma .kind::f8f6f4 with both operands e4m3 and fp32 accumulation
// in tensor memory, and it is exact:
//   * spikes are bytes 0 / 1, which e4m3 reads as 0 and 2^-9 (its smallest
//     subnormal), so a 0/1 spike matrix is an MMA operand as it stands;
//   * a weight w in [-128, 127] is split as w = 16 h + l, h = floor(w / 16) in
//     [-8, 7], l in [0, 15].  16 h and l have at most four significant bits
//     and |16 h| <= 128, so both are e4m3 values exactly.  The weight operand
//     holds the two planes side by side along K, and every K step issues one
//     MMA per plane into the same accumulator;
//   * every product is a multiple of 2^-9 and every partial sum n 2^-9 with
//     |n| <= 128 K <= 2^24 (K <= 2^17): an fp32 value, so no addition
//     rounds.  The epilogue scales by 2^9 (exact) and converts to INT32.
// An fp8 MMA runs at twice the bf16 rate, so the two planes take the time of
// one bf16 MMA, while the spike operand is one byte per element and needs no
// conversion pass.
//
// Kernel structure (320 threads):
//   warp 0      TMA producer: per 64-column K block, a 128 x 64 spike box
//               (64-byte swizzle) and a 256 x 128 weight box (both planes,
//               128-byte swizzle) into a 5-stage shared-memory ring
//   warp 1      allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//               and issues tcgen05.mma (M = 128, N = 256, K = 32) from one
//               thread; tcgen05.commit frees ring slots and publishes
//               accumulators
//   warps 2-9   epilogue: warp w reads TMEM lane quarter w % 4 (32 rows);
//               with K whole, warps 2-5 write 32-column chunks; with K split,
//               warps 2-5 and 6-9 take alternate chunks of the partial and
//               the two 16-column halves of every owned chunk
// Whole K (enough output tiles for every SM): one CTA per SM, persistent over
// 128 x 256 tiles; the epilogue of one tile overlaps the next tile's MMAs
// (double-buffered accumulator) and writes acc / y through a shared-memory
// transpose so that every store covers 128 contiguous bytes of a row.
// Split K (few output tiles, e.g. T = 512 rows give 4 x 6 tiles for N =
// 1536): the S CTAs of a thread-block cluster hold one tile for S K ranges.
// Each CTA stores the 32-column chunks it does not own (chunk c belongs to
// cluster rank c % S) into an fp32 workspace that stays in L2, one cluster
// barrier (release / acquire) publishes them, and each owner pulls the S - 1
// partials of each of its chunks into shared memory (bulk copies completing on
// one mbarrier per chunk, so chunk 0 is added while chunk 1 lands), adds them
// to its own accumulator and writes acc / y.
//
// Every mbarrier wait is bounded (2^31 SM cycles, about a second); on
// timeout the kernel sets the error word, stops issuing work, drains what it
// issued and frees its tensor memory before exiting.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "sp_gemm.h"
#include "sp_ptx.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 5;
constexpr int CPT = BN / 32;                  // 32-column chunks per output tile
constexpr int A_BYTES = BM * BK;              // 8 KB: 0/1 spike bytes
constexpr int B_BYTES = BN * BK * 2;          // 32 KB: the 16h and l planes
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 2 * BN;             // double-buffered accumulator
constexpr int kGemmThreads = 320;             // TMA, MMA and 8 epilogue warps
constexpr int TR_STRIDE = 33;                 // padded transpose rows (words)
constexpr size_t SMEM_RING = (size_t)STAGES * STAGE_BYTES;
constexpr int TR16_STRIDE = 17;               // padded 16-column transpose rows
constexpr size_t SMEM_TR = (size_t)8 * 32 * TR16_STRIDE * 4 > (size_t)4 * 32 * TR_STRIDE * 4
                               ? (size_t)8 * 32 * TR16_STRIDE * 4 : (size_t)4 * 32 * TR_STRIDE * 4;
constexpr size_t SMEM_BARS = 256;
constexpr size_t kGemmSmem = 1024 + SMEM_RING + SMEM_TR + SMEM_BARS;
static_assert(kGemmSmem <= 227 * 1024, "shared memory per CTA");
// accumulator units per spike: e4m3 0x01 = 2^-9
constexpr float kUnitsPerSpike = 512.f;

// Instruction descriptor, kind::f8f6f4: D fp32, A and B e4m3 (format 0), both
// K-major, N = 256, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

// Split-K exchange: one partial chunk (32 columns x 128 rows fp32) is 16 KB;
// a rank owns at most kMaxOwned of the CPT chunks of a tile (S >= 2), and the
// S - 1 incoming partials of its chunks fit the idle ring.
constexpr int kPartChunkBytes = 32 * BM * 4;
constexpr int kMaxOwned = (CPT + 1) / 2;
// most peer partials an owner receives: max over S of (S - 1) * ceil(CPT / S)
constexpr int max_incoming_chunks() {
  int m = 0;
  for (int S = 2; S <= 8; ++S) {
    const int n = (S - 1) * ((CPT + S - 1) / S);
    if (n > m) m = n;
  }
  return m;
}
static_assert(max_incoming_chunks() * kPartChunkBytes <= (int)SMEM_RING,
              "split-K partials fit the ring");

struct GemmArgs {
  GemmParams p;
  int tiles_m, tiles_n, splits, kb_per_split, nkb, units;
};

__device__ __forceinline__ void unit_coords(const GemmArgs& a, int u, int& tile, int& mb, int& nb,
                                            int& kb0, int& kb1) {
  tile = u / a.splits;
  const int sp = u - tile * a.splits;
  mb = tile / a.tiles_n;
  nb = tile - mb * a.tiles_n;
  kb0 = sp * a.kb_per_split;
  kb1 = min(a.nkb, kb0 + a.kb_per_split);
}

// Scale of output column n for the calling lane (0 when y is not written).
__device__ __forceinline__ float column_scale(const GemmParams& p, int n) {
  return (p.y && n < p.N) ? __ldg(p.scale + n) : 0.f;
}

// One warp writes a 32-row x 32-column chunk of fp32 sums in accumulator
// units (v[i] = column col0 + i of row row0 + lane): transposed through shared
// memory so that each store instruction covers 32 consecutive columns of one
// row; acc = the exact integer, y = s * float(acc) with sc = the scale of
// column col0 + lane.
__device__ __forceinline__ void store_chunk(const GemmParams& p, uint32_t* tr,
                                            const uint32_t (&v)[32], int row0, int col0,
                                            float sc) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 32; ++i) tr[lane * TR_STRIDE + i] = v[i];
  __syncwarp();
  const int n = col0 + lane;
  const int nrows = p.T - row0 < 32 ? p.T - row0 : 32;
  if (n < p.N) {
    int32_t* acc = p.acc ? p.acc + (int64_t)row0 * p.N + n : nullptr;
    float* y = p.y ? p.y + (int64_t)row0 * p.N + n : nullptr;
    if (nrows == 32) {
      // full chunk: all 32 shared-memory reads into registers before the
      // first global store, so no store orders a later read
      int val[32];
#pragma unroll
      for (int rr = 0; rr < 32; ++rr)
        val[rr] = __float2int_rn(__uint_as_float(tr[rr * TR_STRIDE + lane]) * kUnitsPerSpike);
      if (acc) {
#pragma unroll
        for (int rr = 0; rr < 32; ++rr) acc[(int64_t)rr * p.N] = val[rr];
      }
      if (y) {
#pragma unroll
        for (int rr = 0; rr < 32; ++rr) y[(int64_t)rr * p.N] = scale_out(sc, val[rr]);
      }
    } else {
      for (int rr = 0; rr < nrows; ++rr) {
        const int val = __float2int_rn(__uint_as_float(tr[rr * TR_STRIDE + lane]) * kUnitsPerSpike);
        if (acc) acc[(int64_t)rr * p.N] = val;
        if (y) y[(int64_t)rr * p.N] = scale_out(sc, val);
      }
    }
  }
  __syncwarp();
}

// One warp writes a 32-row x 16-column block of fp32 sums in accumulator
// units (v[i] = column col0 + i of row row0 + lane) through a shared-memory
// transpose: lane l then holds column col0 + (l & 15) of rows 2 rr + (l >> 4),
// so each store instruction covers 64 contiguous bytes of two rows.  sc = the
// scale of column col0 + (lane & 15).
__device__ __forceinline__ void store_block16(const GemmParams& p, uint32_t* tr,
                                              const uint32_t (&v)[16], int row0, int col0,
                                              float sc) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 16; ++i) tr[lane * TR16_STRIDE + i] = v[i];
  __syncwarp();
  const int col = lane & 15, sub = lane >> 4;
  const int n = col0 + col;
  int val[16];
#pragma unroll
  for (int r2 = 0; r2 < 16; ++r2)
    val[r2] = __float2int_rn(__uint_as_float(tr[(2 * r2 + sub) * TR16_STRIDE + col]) * kUnitsPerSpike);
  __syncwarp();
  if (n < p.N) {
    const int nrows = p.T - row0 < 32 ? p.T - row0 : 32;
    if (p.acc) {
      int32_t* acc = p.acc + (int64_t)(row0 + sub) * p.N + n;
#pragma unroll
      for (int r2 = 0; r2 < 16; ++r2)
        if (2 * r2 + sub < nrows) acc[(int64_t)(2 * r2) * p.N] = val[r2];
    }
    if (p.y) {
      float* y = p.y + (int64_t)(row0 + sub) * p.N + n;
#pragma unroll
      for (int r2 = 0; r2 < 16; ++r2)
        if (2 * r2 + sub < nrows) y[(int64_t)(2 * r2) * p.N] = scale_out(sc, val[r2]);
    }
  }
}

__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
            const __grid_constant__ GemmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)STAGES * A_BYTES;
  uint32_t* s_tr = reinterpret_cast<uint32_t*>(smem + SMEM_RING);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SMEM_RING + SMEM_TR);
  uint64_t* full = bars;                 // [STAGES] TMA -> MMA
  uint64_t* empty = bars + STAGES;       // [STAGES] MMA -> TMA
  uint64_t* tfull = bars + 2 * STAGES;   // [2] MMA -> epilogue
  uint64_t* tempty = tfull + 2;          // [2] epilogue -> MMA
  uint64_t* done = tempty + 2;           // all MMAs retired
  uint64_t* pfull = done + 1;            // [kMaxOwned] split K: peers' partials of owned chunk j
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(pfull + kMaxOwned);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // wait bound: a launch with the test stall fault gives up after ~2 ms
  const long long lim = a.p.fault == kFaultStall ? kStallWaitCycles : kWaitLimitCycles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);          // one arrive per epilogue warp
    }
    mbar_init(done, 1);
    for (int j = 0; j < kMaxOwned; ++j) mbar_init(&pfull[j], 1);
    *s_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
  }
  if (warp == 1) tmem_alloc(s_tmem, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  // The set-up above overlaps the previous kernel of the stream (programmatic
  // dependent launch); every global access below comes after it has finished.
  pdl_launch_dependents();
  pdl_wait();

  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int issued = 0;                       // ring slots filled, for the drain
      for (int u = blockIdx.x; u < a.units && !*s_abort; u += gridDim.x) {
        int tile, mb, nb, kb0, kb1;
        unit_coords(a, u, tile, mb, nb, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], ph ^ 1u, lim)) {
            *s_abort = 1;
            atomicExch(a.p.err, kErrMbarTimeout);
            break;
          }
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          // test stall fault: CTA 0's first fill is never issued, so its
          // MMA warp's bounded wait runs out
          if (!(a.p.fault == kFaultStall && blockIdx.x == 0 && issued == 0)) {
            tma_load_2d(sA + (size_t)stage * A_BYTES, &mapA, &full[stage], kb * BK, mb * BM);
            tma_load_2d(sB + (size_t)stage * B_BYTES, &mapB, &full[stage], kb * 2 * BK, nb * BN);
          }
          ++issued;
          if (++stage == STAGES) { stage = 0; ph ^= 1u; }
        }
      }
      // Drain: wait (bounded) until every copy issued into the ring has landed,
      // so no TMA write is in flight when the CTA exits.
      int s = stage;
      uint32_t q = ph;
      for (int i = 0; i < STAGES && i < issued; ++i) {
        if (--s < 0) { s = STAGES - 1; q ^= 1u; }
        mbar_wait(&full[s], q, lim);
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer --------------------------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      for (int u = blockIdx.x; u < a.units && !*s_abort; u += gridDim.x) {
        int tile, mb, nb, kb0, kb1;
        unit_coords(a, u, tile, mb, nb, kb0, kb1);
        if (!mbar_wait(&tempty[ab], aph ^ 1u, lim)) {
          *s_abort = 1;
          atomicExch(a.p.err, kErrMbarTimeout);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(ab * BN);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], ph, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(sA + (size_t)stage * A_BYTES, 512, kSwizzle64);
          const uint64_t bd = smem_desc(sB + (size_t)stage * B_BYTES, 1024, kSwizzle128);
          // descriptor addresses count 16-byte units: +2 = 32 bytes (next 32
          // K elements), +4 = 64 bytes (the l plane of the weight row)
#pragma unroll
          for (int k = 0; k < BK / 32; ++k) {
            mma_e4m3(d, ad + 2u * k, bd + 2u * k, kIdesc, (kb > kb0 || k > 0) ? 1u : 0u);
            mma_e4m3(d, ad + 2u * k, bd + 4u + 2u * k, kIdesc, 1u);
          }
          mma_commit(&empty[stage]);
          if (++stage == STAGES) { stage = 0; ph ^= 1u; }
        }
        if (!ok) {
          *s_abort = 1;
          atomicExch(a.p.err, kErrMbarTimeout);
          break;
        }
        mma_commit(&tfull[ab]);
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
      mma_commit(done);                      // retire every issued MMA
      mbar_wait(done, 0, lim);
    }
  } else if (a.splits == 1) {
    if (warp < 6) {                           // the whole-K epilogue uses warps 2-5
      // ------------------------------ epilogue (whole K) ------------------------
      // Each warp owns one 32-row quarter of the tile (its TMEM lane quarter) and
      // works alone: no barrier joins the epilogue warps, so a warp that gives up
      // on a timed-out wait cannot strand the others.
      const int q = warp & 3;
      uint32_t* tr = s_tr + (size_t)(warp - 2) * 32 * TR_STRIDE;
      int ab = 0;
      uint32_t aph = 0;
      for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
        int tile, mb, nb, kb0, kb1;
        unit_coords(a, u, tile, mb, nb, kb0, kb1);
        if (!mbar_wait(&tfull[ab], aph, lim)) {
          *s_abort = 1;
          if (lane == 0) atomicExch(a.p.err, kErrMbarTimeout);
          break;
        }
        tc_fence_after();
        const int row0 = mb * BM + q * 32;
        for (int c = 0; c < BN; c += 32) {
          uint32_t v[32];
          tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN + c), v);
          if (a.p.fault == kFaultAbort) {    // test fault: the output stays unwritten
            if (lane == 0) atomicExch(a.p.err, kErrInjected);
            continue;
          }
          store_chunk(a.p, tr, v, row0, nb * BN + c, column_scale(a.p, nb * BN + c + lane));
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[ab]);
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
    }
  } else {
    // ---------------- epilogue (split K): reduce-scatter through L2 -----------
    // One unit per CTA.  Wait for this CTA's accumulator.
    if (mbar_wait(&tfull[0], 0, lim)) {
      tc_fence_after();
    } else {
      *s_abort = 1;
      if (lane == 0) atomicExch(a.p.err, kErrMbarTimeout);
    }
  }

  if (a.splits > 1) {
    // Partial of cluster rank r for chunk c, quarter q: 32 columns x 32 rows
    // at part + ((tile * S + r) * CPT + c) * 4096 + q * 1024, column-major with
    // the row fastest, so that a warp writes 128 contiguous bytes (one column
    // of its quarter) per store, and each (r, c) partial is 16 KB contiguous.
    const int S = a.splits;
    const int rank = (int)cluster_ctarank();
    const bool epi = warp >= 2;
    const int q = warp & 3;                  // TMEM lane quarter
    const int half = (warp - 2) >> 2;        // warps 2-5: 0, warps 6-9: 1
    int tile, mb, nb, kb0, kb1;
    unit_coords(a, blockIdx.x, tile, mb, nb, kb0, kb1);
    const float* tile_part = a.p.part + (size_t)tile * S * (BM * BN);
    // scales of this warp's 16 columns of each owned chunk
    float sc[kMaxOwned];
#pragma unroll
    for (int j = 0; j < kMaxOwned; ++j)
      sc[j] = (epi && rank + j * S < BN / 32)
                  ? column_scale(a.p, nb * BN + (rank + j * S) * 32 + half * 16 + (lane & 15))
                  : 0.f;
    if (epi && !*s_abort) {
      // the chunks of this warp's parity, two at a time behind one wait
      float* mine = a.p.part + ((size_t)tile * S + rank) * (BM * BN) + q * 1024 + lane;
      const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16);
      for (int c = half; c < BN / 32; c += 4) {
        uint32_t v0[32], v1[32];
        tmem_ld32_issue(trow + (uint32_t)c * 32u, v0);
        tmem_ld32_issue(trow + (uint32_t)(c + 2) * 32u, v1);
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        reg_pin(v0);
        reg_pin(v1);
        if (c % S != rank) {
          float* dst = mine + (size_t)c * 4096;
#pragma unroll
          for (int i = 0; i < 32; ++i) __stcg(dst + i * 32, __uint_as_float(v0[i]));
        }
        if ((c + 2) % S != rank) {
          float* dst = mine + (size_t)(c + 2) * 4096;
#pragma unroll
          for (int i = 0; i < 32; ++i) __stcg(dst + i * 32, __uint_as_float(v1[i]));
        }
      }
    }
    cluster_sync();                                     // partials published
    // The ring is idle (every MMA of this CTA has completed): one thread pulls
    // the S - 1 peer partials of each owned chunk j into it with bulk copies
    // that complete on pfull[j].
    if (warp == 2 && lane == 0 && !*s_abort) {
      asm volatile("fence.proxy.async.global;" ::: "memory");
      int slot = 0;
      for (int j = 0, c = rank; c < BN / 32; ++j, c += S) {
        mbar_arrive_expect_tx(&pfull[j], (uint32_t)((S - 1) * kPartChunkBytes));
        for (int r = 0; r < S; ++r)
          if (r != rank)
            bulk_load(smem + (size_t)(slot++) * kPartChunkBytes,
                      tile_part + ((size_t)r * CPT + c) * 4096, kPartChunkBytes, &pfull[j]);
      }
    }
    if (epi && !*s_abort) {
      uint32_t* tr = s_tr + (size_t)(warp - 2) * 32 * TR16_STRIDE;
#pragma unroll
      for (int j = 0; j < kMaxOwned; ++j) {
        const int c = rank + j * S;
        if (c >= BN / 32) break;
        if (!mbar_wait(&pfull[j], 0, lim)) {
          *s_abort = 1;
          if (lane == 0) atomicExch(a.p.err, kErrMbarTimeout);
          break;
        }
        uint32_t v[16];
        tmem_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(c * 32 + half * 16), v);
        for (int r = 0; r < S - 1; ++r) {
          const float* src = reinterpret_cast<const float*>(
                                 smem + (size_t)(j * (S - 1) + r) * kPartChunkBytes) +
                             q * 1024 + half * 16 * 32 + lane;
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) + src[i * 32]);
        }
        if (a.p.fault == kFaultAbort) {      // test fault: the output stays unwritten
          if (lane == 0) atomicExch(a.p.err, kErrInjected);
          continue;
        }
        store_block16(a.p, tr, v, mb * BM + q * 32, nb * BN + c * 32 + half * 16, sc[j]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---- grouped persistent launch ------------------------------------------------
//
// The output tiles of every member of a group (e.g. the 22 down projections
// of a 512-token prefill: 22 x 4 x 6 = 528 tiles of 128 x 256) form one list,
// member after member.  A unit is CL row tiles of one member with the same 256
// channels (row tiles CL g + r, r = the CTA's rank in its cluster of CL);
// cluster c of a persistent grid takes units c, c + clusters, ...  Each tile
// runs over its whole K, so no partial leaves the SM, and the epilogue of unit
// i (8 warps: TMEM lane quarter w % 4, 16-column half (w - 2) / 4 of every
// 32-column chunk) overlaps the MMAs of unit i + 1 through the
// double-buffered accumulator.
//
// CL = 2 runs each unit on a CTA pair with the 2-SM MMA (.cta_group::2,
// M = 256): each CTA loads its own 128 spike rows and HALF of the 256
// weight rows of every K block, and one thread of the even CTA issues the
// MMAs, which read both CTAs' shared memory and write each CTA's own 128
// accumulator rows.  Per K block an SM then takes in 24 KB instead of 40 KB
// and its tensor core reads 8 KB instead of 12 KB per MMA, which takes the
// K loop from shared-memory bound to tensor bound; the ring holds 8 stages
// instead of 5.  Both CTAs' copies complete on the even CTA's full barrier
// (which expects the pair's bytes); the even CTA's commits arrive on the
// empty / accumulator barriers of both CTAs; both CTAs' epilogue warps
// release an accumulator on the even CTA's barrier.  A row tile past a
// member's last (T not a multiple of 256) is computed on zero rows (TMA
// fills past T) and writes nothing.

template <int CL>
struct GroupCfg {
  static constexpr int kStages = CL == 2 ? 8 : STAGES;
  static constexpr int kBStage = B_BYTES / CL;      // this CTA's weight rows x 128 B
  static constexpr uint32_t kStageTx = (uint32_t)CL * (A_BYTES + kBStage);
  static constexpr size_t kRing = (size_t)kStages * (A_BYTES + kBStage);
  static constexpr size_t kSmem = 1024 + kRing + SMEM_TR + SMEM_BARS;
  // kind::f8f6f4 instruction descriptor with M = 128 CL
  static constexpr uint32_t kIdesc =
      (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)((BM * CL) >> 4) << 24);
};
static_assert(GroupCfg<1>::kSmem <= 227 * 1024 && GroupCfg<2>::kSmem <= 227 * 1024,
              "shared memory per CTA");
static_assert((2 * GroupCfg<2>::kStages + 5) * 8 + 8 <= (int)SMEM_BARS, "barrier area");

// Member holding unit u (members are few, their unit ranges ascending).
__device__ __forceinline__ int member_of(const GemmGroupArgs& g, int u) {
  int j = 0;
  while (j + 1 < g.count && u >= g.m[j].unit_end) ++j;
  return j;
}

// One unit of a grouped launch as a CTA of rank `rank` sees it.
struct GroupUnit {
  int j;                  // member
  int mb, nb;             // this CTA's row tile and the channel tile
  int kb0, kb1;           // K blocks [kb0, kb1)
  int role;               // 0 whole K, 1 owner of a split unit, 2 helper
  int slot;               // helper: its partial slot; owner: its first helper's
};

template <int CL>
__device__ __forceinline__ GroupUnit group_unit(const GemmGroupArgs& g, int v, int rank) {
  GroupUnit r;
  int u = v, s = 0, S = 1;
  r.role = 0;
  r.slot = 0;
  if (v >= g.whole) {
    S = g.tail_s;
    const int t = (v - g.whole) / S;
    s = v - g.whole - t * S;
    u = g.whole + t;
    r.role = s == 0 ? 1 : 2;
    r.slot = t * (S - 1) + (s == 0 ? 0 : s - 1);
  }
  r.j = member_of(g, u);
  const GemmMember& M = g.m[r.j];
  const int unit = u - M.unit_begin;
  const int mg = unit / M.tiles_n;
  r.nb = unit - mg * M.tiles_n;
  r.mb = mg * CL + rank;
  r.kb0 = s * M.nkb / S;
  r.kb1 = (s + 1) * M.nkb / S;
  return r;
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

template <int CL>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_group_kernel(const __grid_constant__ GemmGroupArgs g) {
  using C = GroupCfg<CL>;
  constexpr int ST = C::kStages;
  constexpr bool kPair = CL == 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)ST * A_BYTES;
  uint32_t* s_tr = reinterpret_cast<uint32_t*>(smem + C::kRing);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kRing + SMEM_TR);
  uint64_t* full = bars;                 // [ST] TMA (both CTAs of a pair) -> MMA
  uint64_t* empty = bars + ST;           // [ST] MMA -> TMA
  uint64_t* tfull = bars + 2 * ST;       // [2] MMA -> epilogue
  uint64_t* tempty = tfull + 2;          // [2] epilogue (both CTAs of a pair) -> MMA
  uint64_t* done = tempty + 2;           // all MMAs retired
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = kPair ? (int)cluster_ctarank() : 0;
  const bool leader = rank == 0;
  const int cluster = (int)blockIdx.x / CL, nclusters = (int)gridDim.x / CL;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 8 * CL);     // one arrive per epilogue warp of the pair
    }
    mbar_init(done, 1);
    *s_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if (kPair) tmem_alloc_pair(s_tmem, TMEM_COLS);
    else tmem_alloc(s_tmem, TMEM_COLS);
  }
  tc_fence_before();
  // both CTAs' barriers exist before either signals the other's
  if (kPair) cluster_sync();
  else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  pdl_launch_dependents();
  pdl_wait();

  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0) {
      const uint32_t full_cl = kPair ? cluster_addr(full, 0) : 0u;   // even CTA's full[0]
      int stage = 0;
      uint32_t ph = 0;
      int issued = 0;
      int last = -1;
      for (int v = cluster; v < g.total && !*s_abort; v += nclusters) {
        const GroupUnit U = group_unit<CL>(g, v, rank);
        const GemmMember& M = g.m[U.j];
        if (U.j != last) {
          tma_prefetch_desc(&M.a);
          tma_prefetch_desc(&M.b);
          last = U.j;
        }
        const int mb = U.mb, nb = U.nb;
        for (int kb = U.kb0; kb < U.kb1; ++kb) {
          if (!mbar_wait(&empty[stage], ph ^ 1u)) {
            *s_abort = 1;
            atomicExch(g.err, kErrMbarTimeout);
            break;
          }
          if (leader) mbar_arrive_expect_tx(&full[stage], C::kStageTx);
          uint8_t* dA = sA + (size_t)stage * A_BYTES;
          uint8_t* dB = sB + (size_t)stage * C::kBStage;
          if (kPair) {
            const uint32_t bar = full_cl + (uint32_t)stage * 8u;
            tma_load_2d_pair(dA, &M.a, bar, kb * BK, mb * BM);
            tma_load_2d_pair(dB, &M.b, bar, kb * 2 * BK, nb * BN + rank * (BN / 2));
          } else {
            tma_load_2d(dA, &M.a, &full[stage], kb * BK, mb * BM);
            tma_load_2d(dB, &M.b, &full[stage], kb * 2 * BK, nb * BN);
          }
          ++issued;
          if (++stage == ST) { stage = 0; ph ^= 1u; }
        }
      }
      // Drain (bounded): the last fills of every slot have landed (the even
      // CTA's full barriers count both CTAs' copies) and been released by
      // the MMA, so nothing is in flight towards either CTA when they exit.
      int s = stage;
      uint32_t q = ph;
      for (int i = 0; i < ST && i < issued; ++i) {
        if (--s < 0) { s = ST - 1; q ^= 1u; }
        if (leader) mbar_wait(&full[s], q);
        mbar_wait(&empty[s], q);
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer --------------------------------
    if (lane == 0 && leader) {
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      for (int v = cluster; v < g.total && !*s_abort; v += nclusters) {
        const GroupUnit U = group_unit<CL>(g, v, rank);
        if (!mbar_wait(&tempty[ab], aph ^ 1u)) {
          *s_abort = 1;
          atomicExch(g.err, kErrMbarTimeout);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(ab * BN);
        bool ok = true;
        for (int kb = U.kb0; kb < U.kb1; ++kb) {
          if (!mbar_wait(&full[stage], ph)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(sA + (size_t)stage * A_BYTES, 512, kSwizzle64);
          const uint64_t bd = smem_desc(sB + (size_t)stage * C::kBStage, 1024, kSwizzle128);
          // +2 = the next 32 K elements, +4 = the l plane of the weight rows
#pragma unroll
          for (int k = 0; k < BK / 32; ++k) {
            const uint32_t acc = (kb > U.kb0 || k > 0) ? 1u : 0u;
            if (kPair) {
              mma_e4m3_pair(d, ad + 2u * k, bd + 2u * k, C::kIdesc, acc);
              mma_e4m3_pair(d, ad + 2u * k, bd + 4u + 2u * k, C::kIdesc, 1u);
            } else {
              mma_e4m3(d, ad + 2u * k, bd + 2u * k, C::kIdesc, acc);
              mma_e4m3(d, ad + 2u * k, bd + 4u + 2u * k, C::kIdesc, 1u);
            }
          }
          if (kPair) mma_commit_pair(&empty[stage], 3);
          else mma_commit(&empty[stage]);
          if (++stage == ST) { stage = 0; ph ^= 1u; }
        }
        if (!ok) {
          *s_abort = 1;
          atomicExch(g.err, kErrMbarTimeout);
          break;
        }
        if (kPair) mma_commit_pair(&tfull[ab], 3);
        else mma_commit(&tfull[ab]);
        if (++ab == 2) { ab = 0; aph ^= 1u; }
      }
      if (kPair) mma_commit_pair(done, 1);
      else mma_commit(done);
      mbar_wait(done, 0);
    }
  } else {
    // ------------------------------ epilogue ----------------------------------
    // Warps work alone (no barrier joins them), so a warp that gives up on a
    // timed-out wait strands no other.
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    uint32_t* tr = s_tr + (size_t)(warp - 2) * 32 * TR16_STRIDE;
    const uint32_t tempty_cl = kPair ? cluster_addr(tempty, 0) : 0u;
    int ab = 0;
    uint32_t aph = 0;
    for (int v = cluster; v < g.total; v += nclusters) {
      const GroupUnit U = group_unit<CL>(g, v, rank);
      const GemmMember& M = g.m[U.j];
      if (!mbar_wait(&tfull[ab], aph)) {
        *s_abort = 1;
        if (lane == 0) atomicExch(g.err, kErrMbarTimeout);
        break;
      }
      tc_fence_after();
      const int row0 = U.mb * BM + q * 32;
      const bool live = row0 < M.p.T;
      const uint32_t trow =
          tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN + half * 16);
      // this warp's 32 x 16 block of chunk c inside a 128 x 256 partial tile
      const size_t pofs = (size_t)(q * 32 + lane) + (size_t)half * 16 * 128;
      if (U.role == 2) {
        // helper: the partial of this CTA's rows to its slot, then this
        // warp's flag (every lane's stores ordered before it)
        float* dst = g.part + (size_t)(U.slot * CL + rank) * (BM * BN) + pofs;
        if (live) {
#pragma unroll 1
          for (int c = 0; c < CPT; ++c) {
            uint32_t v[16];
            tmem_ld16(trow + (uint32_t)(c * 32), v);
#pragma unroll
            for (int i = 0; i < 16; ++i)
              __stcg(dst + (size_t)(c * 32 + i) * 128, __uint_as_float(v[i]));
          }
        }
        __threadfence();
        __syncwarp();
        if (lane == 0) st_release(g.flags + (size_t)(U.slot * CL + rank) * 8 + (warp - 2), 1u);
      } else {
        const int helpers = U.role == 1 ? g.tail_s - 1 : 0;
        bool ok = true;
        for (int h = 0; h < helpers && ok; ++h) {
          // owner: wait (bounded) for the helper's warp that wrote this block
          const uint32_t* f = g.flags + (size_t)((U.slot + h) * CL + rank) * 8 + (warp - 2);
          const long long t0 = clock64();
          while (ld_acquire(f) == 0u) {
            if (clock64() - t0 > kWaitLimitCycles) {
              ok = false;
              break;
            }
          }
        }
        __syncwarp();
        if (!ok) {
          *s_abort = 1;
          if (lane == 0) atomicExch(g.err, kErrFlagTimeout);
        } else if (live) {
#pragma unroll 1
          for (int c = 0; c < CPT; ++c) {
            const int col0 = U.nb * BN + c * 32 + half * 16;
            uint32_t v[16];
            tmem_ld16(trow + (uint32_t)(c * 32), v);
            for (int h = 0; h < helpers; ++h) {
              const float* src = g.part + (size_t)((U.slot + h) * CL + rank) * (BM * BN) + pofs +
                                 (size_t)c * 32 * 128;
#pragma unroll
              for (int i = 0; i < 16; ++i)
                v[i] = __float_as_uint(__uint_as_float(v[i]) + __ldcg(src + (size_t)i * 128));
            }
            if (M.p.fault == kFaultAbort) {   // test fault: the output stays unwritten
              if (lane == 0) atomicExch(g.err, kErrInjected);
              continue;
            }
            store_block16(M.p, tr, v, row0, col0, column_scale(M.p, col0 + (lane & 15)));
          }
        }
        __syncwarp();
        if (lane == 0)
          for (int h = 0; h < helpers; ++h)
            g.flags[(size_t)((U.slot + h) * CL + rank) * 8 + (warp - 2)] = 0u;   // for the next launch
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (kPair) mbar_arrive_cluster(tempty_cl + (uint32_t)ab * 8u);
        else mbar_arrive(&tempty[ab]);
      }
      if (++ab == 2) { ab = 0; aph ^= 1u; }
    }
  }

  tc_fence_before();
  if (kPair) cluster_sync();             // the pair's MMAs, copies and arrivals are over
  else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (kPair) tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---- operand preparation ------------------------------------------------------

// e4m3 encoding (1 sign bit, 4 exponent bits with bias 7, 3 mantissa bits) of
// an integer v with at most four significant bits and |v| <= 448 (exact).
__device__ __forceinline__ uint8_t e4m3_of_small_int(int v) {
  if (v == 0) return 0;
  const uint32_t sign = v < 0 ? 0x80u : 0u;
  const uint32_t m = (uint32_t)(v < 0 ? -v : v);
  const int e = 31 - __clz((int)m);                    // 2^e <= m < 2^(e+1)
  const uint32_t frac = ((m << 3) >> e) & 7u;          // the three bits below the leading one
  return (uint8_t)(sign | (uint32_t)(e + 7) << 3 | frac);
}

// W column-major INT8 [K][ldw] -> the weight operand [N][2 Kp] bytes: for
// every 64-column K block, 64 bytes of e4m3(16 h) then 64 bytes of e4m3(l),
// w = 16 h + l (zero for k >= K).  32 x 32 tiles transposed through shared
// memory.
__global__ void w_to_e4m3_kernel(const int8_t* __restrict__ W, int64_t ldw, int N, int K, int Kp,
                                 uint8_t* __restrict__ Wq) {
  __shared__ int8_t tile[32][33];
  const int k0 = blockIdx.x * 32, m0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;     // 32 x 8
  for (int i = ty; i < 32; i += 8) {
    const int k = k0 + i, m = m0 + tx;
    tile[i][tx] = (k < K && m < N) ? W[(int64_t)k * ldw + m] : (int8_t)0;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += 8) {
    const int m = m0 + i, k = k0 + tx;
    if (m < N && k < Kp) {
      const int w = tile[tx][i];
      const int h = w >> 4;                  // floor(w / 16)
      uint8_t* row = Wq + (int64_t)m * 2 * Kp + (k / BK) * (2 * BK) + (k % BK);
      row[0] = e4m3_of_small_int(16 * h);
      row[BK] = e4m3_of_small_int(w - 16 * h);
    }
  }
}

// Spike rows (any format) -> 0/1 bytes [T][Kp], zero past K.  One thread per
// 16 consecutive columns of a row: one 16-byte store.  kVec: byte rows are
// 16-byte aligned (base and leading dimension), so whole 16-column groups
// load as one vector.
template <bool kVec>
__global__ void spikes_to_01_kernel(const void* __restrict__ spikes, int fmt, int64_t ld, int T,
                                    int K, int Kp, uint8_t* __restrict__ Xs) {
  pdl_launch_dependents();
  pdl_wait();
  const int per_row = Kp / 16;
  const int64_t total = (int64_t)T * per_row;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / per_row);
    const int k = (int)(i - (int64_t)t * per_row) * 16;
    uint4 o = make_uint4(0u, 0u, 0u, 0u);
    if (k < K) {
      const void* row = spike_row(spikes, fmt, t, ld);
      if (fmt != SP_SPIKES_BITS32 && kVec && K - k >= 16) {
        const uint4 w = __ldg(reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(row) + k));
        o = make_uint4(nonzero_bytes_to_01(w.x), nonzero_bytes_to_01(w.y), nonzero_bytes_to_01(w.z),
                       nonzero_bytes_to_01(w.w));
      } else {
        uint32_t bits = 0u;                  // spikes of columns k .. k+15
        if (fmt == SP_SPIKES_BITS32) {
          bits = (__ldg(reinterpret_cast<const uint32_t*>(row) + (k >> 5)) >> (k & 31)) & 0xffffu;
        } else {
          const uint8_t* x = static_cast<const uint8_t*>(row) + k;
          const int n = K - k < 16 ? K - k : 16;
          for (int j = 0; j < n; ++j) bits |= (uint32_t)(__ldg(x + j) != 0) << j;
        }
        if (K - k < 16) bits &= (1u << (K - k)) - 1u;
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t nib = (bits >> (4 * j)) & 0xfu;
          w[j] = (nib & 1u) | (nib & 2u) << 7 | (nib & 4u) << 14 | (nib & 8u) << 21;
        }
        o = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
    *reinterpret_cast<uint4*>(Xs + (int64_t)t * Kp + k) = o;
  }
}

int g_num_sms = 0;
bool g_attr_set = false;

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D byte matrix [outer][inner] with rows `stride` bytes apart, read in
// box_inner x box_outer boxes, zero past the extents.
bool encode_u8_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                  uint64_t stride, uint32_t box_inner, uint32_t box_outer,
                  CUtensorMapSwizzle swizzle) {
  auto enc = get_encode();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {stride};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Largest number of clusters of `size` CTAs that can be resident at once.
int max_active_clusters(int size) {
  static int cache[9] = {0};
  if (cache[size] == 0) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = size;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.gridDim = dim3(size, 1, 1);
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = kGemmSmem;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_kernel, &cfg) != cudaSuccess || n < 1) {
      (void)cudaGetLastError();
      n = -1;
    }
    cache[size] = n;
  }
  return cache[size];
}

cudaError_t set_gemm_attrs() {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kGemmSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 0);
  if (e != cudaSuccess) return e;
  done = true;
  return cudaSuccess;
}

cudaError_t init_sms() {
  if (g_attr_set) return cudaSuccess;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  g_attr_set = true;
  return cudaSuccess;
}

// K splits for a T x N output: split only when the tiles alone leave SMs
// idle, and only as far as every cluster stays resident in a single wave.
int pick_splits(int T, int N, int Kp, int part_units) {
  const int tiles = ceil_div(T, BM) * ceil_div(N, BN);
  const int nkb = Kp / BK;
  int S = 1;
  if (tiles < g_num_sms) {
    S = g_num_sms / tiles;
    if (S > 8) S = 8;
    if (S > nkb / 4) S = nkb / 4;
    if (S < 1) S = 1;
    while (S > 1) {
      const int kbps = ceil_div(nkb, S);
      const int exact = ceil_div(nkb, kbps);            // splits with work
      if (exact == S && max_active_clusters(S) >= tiles && tiles * S <= part_units) break;
      --S;
    }
  }
  return S;
}

}  // namespace

int gemm_k_pad(int K) { return ceil_div(K, BK) * BK; }

cudaError_t gemm_make_maps(const uint8_t* Xs, int rows_alloc, const uint8_t* Wq, int N, int Kp,
                           GemmMaps* out) {
  if (!encode_u8_2d(&out->a, Xs, (uint64_t)Kp, (uint64_t)rows_alloc, (uint64_t)Kp, BK, BM,
                    CU_TENSOR_MAP_SWIZZLE_64B))
    return cudaErrorUnknown;
  if (!encode_u8_2d(&out->b, Wq, (uint64_t)2 * Kp, (uint64_t)N, (uint64_t)2 * Kp, 2 * BK, BN,
                    CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_u8_2d(&out->b128, Wq, (uint64_t)2 * Kp, (uint64_t)N, (uint64_t)2 * Kp, 2 * BK,
                    BN / 2, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_u8_2d(&out->p64, Wq, (uint64_t)2 * Kp, (uint64_t)N, (uint64_t)2 * Kp, BK, BN / 2,
                    CU_TENSOR_MAP_SWIZZLE_64B))
    return cudaErrorUnknown;
  return cudaSuccess;
}

cudaError_t gemm_make_rows_map(const void* X, int64_t ldx, int T, int K, CUtensorMap* out) {
  return encode_u8_2d(out, X, (uint64_t)K, (uint64_t)T, (uint64_t)ldx, BK, BM,
                      CU_TENSOR_MAP_SWIZZLE_64B)
             ? cudaSuccess
             : cudaErrorInvalidValue;
}

cudaError_t launch_w_to_e4m3(const int8_t* W, int64_t ldw, int N, int K, uint8_t* Wq,
                             cudaStream_t s) {
  const int Kp = gemm_k_pad(K);
  dim3 grid(ceil_div(Kp, 32), ceil_div(N, 32)), block(32, 8);
  w_to_e4m3_kernel<<<grid, block, 0, s>>>(W, ldw, N, K, Kp, Wq);
  return cudaGetLastError();
}

cudaError_t launch_spikes_to_01(const void* spikes, int fmt, int64_t ld, int T, int K, int Kp,
                                uint8_t* Xs, cudaStream_t s) {
  const int64_t total = (int64_t)T * (Kp / 16);
  const int threads = 256;
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > 8192) blocks = 8192;
  if (blocks < 1) blocks = 1;
  const bool vec = fmt != SP_SPIKES_BITS32 && (reinterpret_cast<uintptr_t>(spikes) & 15u) == 0 &&
                   ld % 16 == 0;
  if (vec)
    return launch_pdl(spikes_to_01_kernel<true>, dim3((unsigned)blocks), dim3(threads), 0, s, spikes,
                      fmt, ld, T, K, Kp, Xs);
  return launch_pdl(spikes_to_01_kernel<false>, dim3((unsigned)blocks), dim3(threads), 0, s, spikes,
                    fmt, ld, T, K, Kp, Xs);
}

namespace {

// Largest number of clusters of `cl` CTAs of gemm_group_kernel<cl> that can be
// resident at once (-1 when the occupancy query fails).
template <int CL>
int group_active_clusters() {
  static int n = 0;
  if (n == 0) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = CL;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.gridDim = dim3(CL, 1, 1);
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = GroupCfg<CL>::kSmem;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int c = 0;
    if (cudaOccupancyMaxActiveClusters(&c, gemm_group_kernel<CL>, &cfg) != cudaSuccess || c < 1) {
      (void)cudaGetLastError();
      c = -1;
    }
    n = c;
  }
  return n;
}

template <int CL>
cudaError_t launch_group_cl(const GemmGroupArgs& a, cudaStream_t s) {
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_group_kernel<CL>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)GroupCfg<CL>::kSmem);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  int clusters = g_num_sms / CL;
  if (CL > 1) {
    const int resident = group_active_clusters<CL>();
    if (resident < 1) return cudaErrorInvalidConfiguration;
    if (clusters > resident) clusters = resident;
  }
  // Tail split: the r units past the last full round of the grid (all of
  // them when there are fewer units than clusters) are cut into S K ranges
  // so that the last round fills the grid.  Sub-units of the last round land
  // on distinct clusters: the whole units are a multiple of the grid.
  GemmGroupArgs b = a;
  b.whole = a.units;
  b.tail_s = 1;
  const int r = a.units % clusters;
  if (a.part && a.flags && r > 0) {
    int S = clusters / r;
    if (S > 6) S = 6;
    int min_nkb = 1 << 30;
    for (int j = 0; j < a.count; ++j)
      if (a.m[j].unit_end > a.units - r && a.m[j].nkb < min_nkb) min_nkb = a.m[j].nkb;
    while (S > 1 && (min_nkb < 4 * S || r * (S - 1) * CL > kGemmGroupSlots)) --S;
    if (S > 1) {
      b.whole = a.units - r;
      b.tail_s = S;
    }
  }
  b.total = b.whole + (a.units - b.whole) * b.tail_s;
  if (clusters > b.total) clusters = b.total;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = CL;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.gridDim = dim3(clusters * CL, 1, 1);
  cfg.blockDim = dim3(kGemmThreads, 1, 1);
  cfg.dynamicSmemBytes = GroupCfg<CL>::kSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = CL > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, gemm_group_kernel<CL>, b);
}

}  // namespace

int gemm_group_cluster(const int* tiles_m, const int* tiles_n, int count) {
  int64_t tiles = 0, pad2 = 0;
  for (int j = 0; j < count; ++j) {
    tiles += (int64_t)tiles_m[j] * tiles_n[j];
    pad2 += (int64_t)(ceil_div(tiles_m[j], 2) * 2 - tiles_m[j]) * tiles_n[j];
  }
  return pad2 * 8 <= tiles ? 2 : 1;
}

cudaError_t launch_gemm_group(const GemmGroupArgs& a, cudaStream_t s) {
  cudaError_t e = init_sms();
  if (e != cudaSuccess) return e;
  if (a.units < 1) return cudaSuccess;
  switch (a.cl) {
    case 1: return launch_group_cl<1>(a, s);
    case 2: return launch_group_cl<2>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

int gemm_splits(int T, int N, int Kp, int part_units) {
  if (init_sms() != cudaSuccess || set_gemm_attrs() != cudaSuccess) return 1;
  return pick_splits(T, N, Kp, part_units);
}

cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, int S, int T, int N,
                        int Kp, const GemmParams& p, cudaStream_t s) {
  cudaError_t e = init_sms();
  if (e != cudaSuccess) return e;
  e = set_gemm_attrs();
  if (e != cudaSuccess) return e;
  GemmArgs a;
  a.p = p;
  a.tiles_m = ceil_div(T, BM);
  a.tiles_n = ceil_div(N, BN);
  a.nkb = Kp / BK;
  a.kb_per_split = ceil_div(a.nkb, S);
  a.splits = S;
  a.units = a.tiles_m * a.tiles_n * S;
  if (S == 1) {
    const int grid = a.units < g_num_sms ? a.units : g_num_sms;
    return launch_pdl(gemm_kernel, dim3(grid), dim3(kGemmThreads), kGemmSmem, s, mapA, mapB, a);
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(a.units, 1, 1);
  cfg.blockDim = dim3(kGemmThreads, 1, 1);
  cfg.dynamicSmemBytes = kGemmSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, gemm_kernel, mapA, mapB, a);
}

}  // namespace sp
