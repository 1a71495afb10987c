// sp_gemm_small.cu -- tensor-core path for a few spike rows (T <= 64):
//
//   ACC[t][m] = sum_k X[t][k] * Q[m][k],   Y[t][m] = s_m * float(ACC[t][m])
//
// i.e. Eq. (sparse) for each of T tokens (a decode batch), computed
// transposed, D[m][t] = sum_k Q[m][k] X[t][k]: the weights are the MMA's
// 128-row M operand (128 output channels per CTA) and the T spike rows its N
// operand (N = T rounded up to 16), so no MMA row is spent on absent tokens
// as it would be with the tokens in M (a 128-row tile for 64 tokens).
//
// Arithmetic as in the prefill GEMM (sp_gemm.cu): tcgen05.mma kind::f8f6f4,
// both operands e4m3, fp32 accumulation in tensor memory, exact -- spikes are
// bytes 0 / 1 (e4m3 0 and 2^-9), a weight w = 16 h + l is two e4m3 planes
// (the plan's copy, [N][2 Kp]), every partial sum is n 2^-9 with
// |n| <= 128 K < 2^24, and the epilogue scales by 2^9 and converts to INT32.
//
// Decomposition: output tile mt (channels 128 mt ..) x S K ranges, one CTA
// each; the S CTAs of a tile form a thread-block cluster.  Per CTA (320
// threads):
//   warp 0      TMA producer: the two 128 x 64-byte weight boxes (one per
//               plane) of each 64-column K block into an 8-stage ring.  The
//               planes are written once, when the plan is made, so the first
//               ring fills are issued before the dependency wait and overlap
//               the tail of the previous kernel of the stream.
//   warp 1      allocates 64 TMEM columns and issues the MMAs (M = 128,
//               N = TN, K = 32; two per plane per K block) from one thread.
//   warps 2-9   after the dependency wait, expand the CTA's K range of all T
//               spike rows (any input format) into 0 / 1 bytes in the
//               64-byte-swizzled K-major layout the MMA reads (the layout a
//               TMA box with 64-byte swizzle writes), K block by K block.
//   warps 2-5   then read the accumulator (warp w: TMEM lane quarter w % 4,
//               i.e. 32 channels x TN tokens) and reduce it over the
//               cluster: the tokens form groups of 4, group g belongs to
//               cluster rank g % S, every CTA pushes each group's 4 values of
//               its 32 channels into the owner's shared memory with st.async
//               (distributed shared memory), which counts the bytes on the
//               owner's receive mbarrier; the owner waits on that barrier
//               alone, adds the S partials of its groups and writes acc / y
//               (a warp's 32 lanes hold 32 consecutive channels of one
//               token: 128-byte stores).
// No workspace, no atomics, no flags: the inter-CTA waits are one cluster
// barrier (every peer has staged its spike slice, so its receive area is
// free) and the receive mbarriers.  Every mbarrier wait is bounded; on
// timeout the CTA raises the error word, stops issuing, drains its copies and
// frees its tensor memory.
#include <cuda.h>

#include "sp_gemm.h"
#include "sp_ptx.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int kSmM = 128;                     // output channels per tile (MMA M)
constexpr int kSmBK = 64;                     // K columns per K block
constexpr int kSmStages = 8;
constexpr int kSmWBytes = kSmM * 2 * kSmBK;   // 16 KB: 128 channel rows x (64 h + 64 l)
constexpr int kSmXBlock = kGemmSmallMaxT * kSmBK;   // 4 KB: up to 64 token rows x 64 bytes
constexpr int kSmGroups = kGemmSmallMaxT / 4;       // 4-token groups
// (sender, owned group) slots an owner receives: S * ceil(16 / S) = 16 for
// the cluster sizes used (powers of two)
constexpr int kSmRecvSlots = kSmGroups;
constexpr int kSmStageWarps = 8;              // warps 2-9 stage the spike operand
constexpr int kSmThreads = 64 + 32 * kSmStageWarps;
constexpr int kSmTmemCols = kGemmSmallMaxT;
constexpr size_t kSmRing = (size_t)kSmStages * kSmWBytes;
constexpr size_t kSmX = (size_t)kGemmSmallMaxKB * kSmXBlock;
constexpr size_t kSmRecv = (size_t)kSmRecvSlots * kSmM * 16;
constexpr size_t kSmBars = 512;
constexpr size_t kSmSmem = 1024 + kSmRing + kSmX + kSmRecv + kSmBars;
static_assert(kSmSmem <= 227 * 1024, "shared memory per CTA");
static_assert((2 * kSmStages + kGemmSmallMaxKB + 3) * 8 + 8 <= (int)kSmBars, "barrier area");
constexpr float kUnitsPerSpike = 512.f;       // e4m3 0x01 = 2^-9

// Sixteen spikes (bit i = column k0 + i) as sixteen 0 / 1 bytes.
__device__ __forceinline__ uint4 bits16_to_01(uint32_t bits) {
  uint32_t w[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const uint32_t nib = (bits >> (4 * j)) & 0xfu;
    w[j] = (nib & 1u) | (nib & 2u) << 7 | (nib & 4u) << 14 | (nib & 8u) << 21;
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Spikes of row t, columns k0 .. k0 + 15 (k0 % 16 == 0, k0 < K) as 0 / 1 bytes.
__device__ __forceinline__ uint4 spikes16(const GemmSmallArgs& a, int t, int k0) {
  const void* row = spike_row(a.spikes, a.fmt, t, a.ld);
  const int rem = a.K - k0;
  if (a.fmt == SP_SPIKES_BITS32) {
    uint32_t b = (__ldg(static_cast<const uint32_t*>(row) + (k0 >> 5)) >> (k0 & 16)) & 0xffffu;
    if (rem < 16) b &= (1u << rem) - 1u;
    return bits16_to_01(b);
  }
  const uint8_t* x = static_cast<const uint8_t*>(row) + k0;
  if (rem >= 16 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(x));
    return make_uint4(nonzero_bytes_to_01(v.x), nonzero_bytes_to_01(v.y), nonzero_bytes_to_01(v.z),
                      nonzero_bytes_to_01(v.w));
  }
  uint32_t b = 0u;
  const int n = rem < 16 ? rem : 16;
  for (int i = 0; i < n; ++i) b |= (uint32_t)(__ldg(x + i) != 0) << i;
  return bits16_to_01(b);
}

// The two planes of K block kb for output tile mt: the 16 h plane into the
// first 8 KB of dst, the l plane into the second, each 128 channel rows of
// 64 bytes with the 64-byte swizzle.  (With 128-byte rows holding both
// planes, the tensor core took 150 cycles per MMA at any N; with 64-byte
// rows, 48 at N = 64.)
__device__ __forceinline__ void load_planes(uint8_t* dst, const CUtensorMap* map, uint64_t* bar,
                                            int kb, int mt) {
  tma_load_2d(dst, map, bar, kb * 2 * kSmBK, mt * kSmM);
  tma_load_2d(dst + kSmWBytes / 2, map, bar, kb * 2 * kSmBK + kSmBK, mt * kSmM);
}

// The four MMAs of one K block (two 32-column K steps x the two weight
// planes, one accumulator), the commit that frees its ring slot, and a
// non-blocking test of the NEXT block's full barrier issued ahead of them, so
// that its shared-memory latency overlaps the MMA issue.  Returns the test.
__device__ __forceinline__ bool mma_block(uint32_t tmem, uint64_t hd, uint64_t ld, uint64_t xd,
                                          uint32_t idesc, bool accumulate, uint64_t* empty_bar,
                                          uint64_t* next_full, uint32_t next_phase) {
  uint32_t ready;
  asm volatile(
      "{\n\t.reg .pred pn, pa, pt;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 pn, [%1], %2;\n\t"
      "setp.ne.b32 pa, %3, 0;\n\t"
      "setp.eq.b32 pt, 0, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%4], %5, %7, %9, pa;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%4], %6, %7, %9, pt;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%4], %10, %8, %9, pt;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%4], %11, %8, %9, pt;\n\t"
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%12];\n\t"
      "selp.u32 %0, 1, 0, pn;\n\t}"
      : "=r"(ready)
      : "r"(smem_u32(next_full)), "r"(next_phase), "r"((uint32_t)accumulate), "r"(tmem), "l"(hd),
        "l"(ld), "l"(xd), "l"(xd + 2u), "r"(idesc), "l"(hd + 2u), "l"(ld + 2u),
        "r"(smem_u32(empty_bar))
      : "memory");
  return ready != 0;
}

// Stores 16 bytes into CTA `rank`'s shared memory at the address `local`
// has in this CTA (distributed shared memory of the cluster), counted in
// bytes on that CTA's mbarrier at the address `bar` has in this CTA.
__device__ __forceinline__ void st_async_v4(const void* local, const uint64_t* bar, uint32_t rank,
                                            uint4 v) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.u32 [%0], {%1, %2, %3, %4}, [%5];"
               ::"r"(cluster_addr(local, rank)), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w),
               "r"(cluster_addr(bar, rank))
               : "memory");
}

// Token columns 16 c .. 16 c + 15 of this warp's 32 TMEM lanes as floats.
__device__ __forceinline__ void acc_chunk(uint32_t trow, int c, float (&f)[16]) {
  uint32_t v[16];
  tmem_ld16(trow + (uint32_t)(16 * c), v);
#pragma unroll
  for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(v[i]);
}

__global__ void __launch_bounds__(kSmThreads, 1)
gemm_small_kernel(const __grid_constant__ CUtensorMap mapW, const __grid_constant__ GemmSmallArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sW = smem;                                     // [stage] weight boxes
  uint8_t* sX = smem + kSmRing;                           // [K block] TN x 64 spike bytes
  uint4* recv = reinterpret_cast<uint4*>(sX + kSmX);      // [slot][128 channels]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sX + kSmX + kSmRecv);
  uint64_t* full = bars;                 // [stages] TMA -> MMA
  uint64_t* empty = bars + kSmStages;    // [stages] MMA -> TMA
  uint64_t* xready = empty + kSmStages;  // [K block] spike operand staged (one arrival per staging warp)
  uint64_t* tfull = xready + kGemmSmallMaxKB;   // accumulator complete
  uint64_t* done = tfull + 1;            // every MMA retired (MMA thread)
  uint64_t* rbar = done + 1;             // the cluster's partials of this rank's groups landed
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(rbar + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int S = a.S;
  const int rank = S > 1 ? (int)cluster_ctarank() : 0;
  const int mt = (int)blockIdx.x / S;
  const int kb0 = rank * a.nkb / S;
  const int nk = (rank + 1) * a.nkb / S - kb0;            // >= 1 (nkb >= S)
  const int TN = a.TN;
  const long long lim = a.fault == kFaultStall ? kStallWaitCycles : kWaitLimitCycles;
  // test stall fault: CTA 0's first weight box is never issued
  const bool skip_first = a.fault == kFaultStall && blockIdx.x == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kSmStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < kGemmSmallMaxKB; ++b) mbar_init(&xready[b], kSmStageWarps);
    mbar_init(tfull, 1);
    mbar_init(done, 1);
    mbar_init(rbar, 1);
    *s_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (S > 1) {
      // every rank stores its partial of each of this rank's groups (g = rank
      // mod S) for the 128 channels: S x owned x 128 x 16 bytes
      const int G = a.TN / 4;
      const int owned = rank < G ? (G - 1 - rank) / S + 1 : 0;
      mbar_arrive_expect_tx(rbar, (uint32_t)(S * owned * kSmM * 16));
    }
    tma_prefetch_desc(&mapW);
  }
  if (warp == 1) tmem_alloc(s_tmem, kSmTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;

  // First ring fills, before the dependency wait (the planes are plan-owned
  // and immutable after plan creation).
  const int pre = nk < kSmStages ? nk : kSmStages;
  if (warp == 0 && lane == 0) {
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], kSmWBytes);
      if (!(skip_first && i == 0)) load_planes(sW + (size_t)i * kSmWBytes, &mapW, &full[i], kb0 + i, mt);
    }
  }
  pdl_launch_dependents();
  pdl_wait();

  const int q = warp & 3;                  // TMEM lane quarter of an epilogue warp
  const int row = q * 32 + lane;           // channel within the tile
  const int m = mt * kSmM + row;
  const bool epi = warp >= 2 && warp < 6;   // epilogue: TMEM lane quarters 2, 3, 0, 1
  const bool stg = warp >= 2;              // staging warps
  // the scale of this thread's channel, read now so that no load waits in the epilogue
  const float sc = (epi && a.y && m < a.N) ? __ldg(a.scale + m) : 0.f;
  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0) {
      int issued = pre;
      for (int i = pre; i < nk && !*s_abort; ++i) {
        const int stage = i % kSmStages;
        const uint32_t ph = (uint32_t)(i / kSmStages - 1) & 1u;   // phase of the MMA's release
        if (!mbar_wait_sleep(&empty[stage], ph, lim)) {
          *s_abort = 1;
          atomicExch(a.err, kErrMbarTimeout);
          break;
        }
        mbar_arrive_expect_tx(&full[stage], kSmWBytes);
        load_planes(sW + (size_t)stage * kSmWBytes, &mapW, &full[stage], kb0 + i, mt);
        ++issued;
      }
      // Drain (bounded): the last fill of every slot has landed, so no copy
      // is in flight towards this CTA when it exits.
      for (int i = issued - 1; i >= 0 && i >= issued - kSmStages; --i)
        mbar_wait_sleep(&full[i % kSmStages], (uint32_t)(i / kSmStages) & 1u, lim);
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer --------------------------------
    if (lane == 0) {
      const uint32_t idesc =
          (1u << 4) | ((uint32_t)(TN >> 3) << 17) | ((uint32_t)(kSmM >> 4) << 24);
      bool ok = true;
      // The staging warps finish the K blocks in order, so block b staged
      // implies every block before it; `staged` is the last block known done.
      int staged = -1;
      int stage = 0;
      uint32_t fph = 0;
      bool have = false;                   // full[stage] already seen complete
      for (int i = 0; i < nk; ++i) {
        if (i > staged) {
          if (mbar_test(&xready[nk - 1], 0)) staged = nk - 1;
          else if (mbar_test(&xready[i], 0) || mbar_wait_sleep(&xready[i], 0, lim)) staged = i;
          else ok = false;
        }
        if (!ok || (!have && !mbar_wait_sleep(&full[stage], fph, lim))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t hd = smem_desc(sW + (size_t)stage * kSmWBytes, 512, kSwizzle64);
        const uint64_t ld = smem_desc(sW + (size_t)stage * kSmWBytes + kSmWBytes / 2, 512, kSwizzle64);
        const uint64_t xd = smem_desc(sX + (size_t)i * kSmXBlock, 512, kSwizzle64);
        const int nstage = stage + 1 == kSmStages ? 0 : stage + 1;
        const uint32_t nfph = nstage == 0 ? fph ^ 1u : fph;
        have = mma_block(tmem, hd, ld, xd, idesc, i > 0, &empty[stage], &full[nstage], nfph);
        stage = nstage;
        fph = nfph;
      }
      if (!ok) {
        *s_abort = 1;
        atomicExch(a.err, kErrMbarTimeout);
      }
      mma_commit(tfull);
      mma_commit(done);                    // retire every issued MMA
      mbar_wait_sleep(done, 0, lim);
    }
  } else {
    // ------------------ spike operand: rows -> 0 / 1 bytes ----------------------
    // The slice is the CTA's nk K blocks (columns 64 kb0 ..) of the TN rows;
    // K block b of row r goes to byte 64 r + 16 (j ^ ((r >> 1) & 3)) of block
    // b (j = 16-column chunk within the 64-byte row: the 64-byte swizzle).
    // One round of loads: BITS32 words are copied (cp.async) into scratch in
    // the receive area (idle until every CTA of the cluster has staged its
    // slice: see the cluster arrival below) and expanded from there; byte
    // rows are copied straight into their slots (U8 bytes then folded to 0 /
    // 1 in place).  In the expansion a warp covers 8 rows x 4 chunks of one K
    // block: 512 contiguous bytes, no bank conflicts; each warp marks each K
    // block done on its barrier, so the MMAs of block b start while later
    // blocks are still being expanded.
    const int e = warp - 2;                // staging warp 0 .. kSmStageWarps - 1
    const int nw = 2 * nk;                 // words per row of the slice (<= 32)
    constexpr int kScr = 33;               // scratch row stride in words (odd: no bank conflicts)
    uint32_t* scratch = reinterpret_cast<uint32_t*>(recv);   // [row][kScr words]
    if (a.fmt == SP_SPIKES_BITS32) {
#pragma unroll 1
      for (int r = e; r < TN; r += kSmStageWarps) {
        if (lane < nw) {
          const int w = kb0 * 2 + lane;
          uint32_t* dst = scratch + r * kScr + lane;
          if (r < a.T && w * 32 < a.K) {
            const uint32_t* src = static_cast<const uint32_t*>(spike_row(a.spikes, a.fmt, r, a.ld)) + w;
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src)
                         : "memory");
          } else {
            *dst = 0u;
          }
        }
      }
      asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
      __syncwarp();
      // the other staging warps' words too
      asm volatile("bar.sync 1, %0;" ::"n"(32 * kSmStageWarps) : "memory");
      const int rr = lane >> 2, j = lane & 3;
      const int shift = 16 * (j & 1);
#pragma unroll 1
      for (int b = 0; b < nk; ++b) {
        const int k = (kb0 + b) * 64 + 16 * j;
        const int rem = a.K - k;
        const uint32_t mask = rem >= 16 ? 0xffffu : (rem > 0 ? (1u << rem) - 1u : 0u);
        const uint32_t* src = scratch + 2 * b + (j >> 1);
        uint8_t* dst = sX + b * kSmXBlock;
#pragma unroll 2
        for (int r = 8 * e + rr; r < TN; r += 8 * kSmStageWarps) {
          const uint32_t bits = (src[r * kScr] >> shift) & mask;
          uint4 o;
          o.x = ((bits & 0xfu) * 0x204081u) & 0x01010101u;
          o.y = (((bits >> 4) & 0xfu) * 0x204081u) & 0x01010101u;
          o.z = (((bits >> 8) & 0xfu) * 0x204081u) & 0x01010101u;
          o.w = ((bits >> 12) * 0x204081u) & 0x01010101u;
          *reinterpret_cast<uint4*>(dst + r * 64 + ((j ^ ((r >> 1) & 3)) << 4)) = o;
        }
        // generic-proxy stores -> visible to the tensor core (async proxy)
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&xready[b]);
      }
    } else {
      const int rr = lane >> 2, j = lane & 3;
      const int groups = TN / 8;
      bool any_async = false;
#pragma unroll 1
      for (int it = e; it < nk * groups; it += kSmStageWarps) {
        const int b = it / groups;
        const int r = (it - b * groups) * 8 + rr;
        const int k = (kb0 + b) * 64 + 16 * j;
        uint8_t* dst = sX + b * kSmXBlock + r * 64 + ((j ^ ((r >> 1) & 3)) << 4);
        const uint8_t* src = r < a.T && k < a.K
                                 ? static_cast<const uint8_t*>(spike_row(a.spikes, a.fmt, r, a.ld)) + k
                                 : nullptr;
        if (src && a.K - k >= 16 && (reinterpret_cast<uintptr_t>(src) & 15u) == 0) {
          asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src)
                       : "memory");
          any_async = true;
        } else {
          *reinterpret_cast<uint4*>(dst) = src ? spikes16(a, r, k) : make_uint4(0u, 0u, 0u, 0u);
        }
      }
      asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
      if (any_async && a.fmt == SP_SPIKES_U8) {   // any nonzero byte -> 1 (this lane's copies)
#pragma unroll 1
        for (int it = e; it < nk * groups; it += kSmStageWarps) {
          const int b = it / groups;
          const int r = (it - b * groups) * 8 + rr;
          const int k = (kb0 + b) * 64 + 16 * j;
          if (r < a.T && k + 16 <= a.K) {
            uint4* p = reinterpret_cast<uint4*>(sX + b * kSmXBlock + r * 64 +
                                                ((j ^ ((r >> 1) & 3)) << 4));
            const uint4 v = *p;
            *p = make_uint4(nonzero_bytes_to_01(v.x), nonzero_bytes_to_01(v.y),
                            nonzero_bytes_to_01(v.z), nonzero_bytes_to_01(v.w));
          }
        }
      }
    }
    if (a.fmt != SP_SPIKES_BITS32) {
      // generic-proxy stores -> visible to the tensor core (async proxy)
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0)
        for (int b = 0; b < nk; ++b) mbar_arrive(&xready[b]);
    }
  }
  // Every CTA of the cluster arrives once its slice is staged (the receive
  // area held the BITS32 scratch) and waits, below, before its first store
  // into a peer's shared memory.
  if (S > 1) {
    if (stg) asm volatile("bar.sync 1, %0;" ::"n"(32 * kSmStageWarps) : "memory");   // every staging warp is done
    asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory");
  }

  // ---------------- accumulator, reduction over the cluster, output ------------
  // Warp w holds channels 32 (w % 4) .. of the tile (TMEM lanes); the tokens
  // form G = TN / 4 groups of 4 columns, group g owned by cluster rank g % S.
  const int G = TN / 4;
  const int gpo = (G + S - 1) / S;         // most groups one rank owns
  bool ok = true;
  if (epi) {
    // warp-uniform: tcgen05.ld is a .sync.aligned warp instruction
    ok = __all_sync(0xffffffffu, mbar_wait_sleep(tfull, 0, lim) && !*s_abort);
    if (ok) tc_fence_after();
    else if (lane == 0) {
      *s_abort = 1;
      atomicExch(a.err, kErrMbarTimeout);
    }
  }
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
  if (S > 1) {
    asm volatile("barrier.cluster.wait;" ::: "memory");   // every peer has staged its slice
    if (epi && ok) {
#pragma unroll 1
      for (int c = 0; c < TN / 16; ++c) {
        float f[16];
        acc_chunk(trow, c, f);
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const int g = 4 * c + h;
          st_async_v4(&recv[(rank * gpo + g / S) * kSmM + row], rbar, (uint32_t)(g % S),
                      make_uint4(__float_as_uint(f[4 * h]), __float_as_uint(f[4 * h + 1]),
                                 __float_as_uint(f[4 * h + 2]), __float_as_uint(f[4 * h + 3])));
        }
      }
    }
  }
  // every partial of this rank's groups is in its shared memory (no
  // cluster-wide barrier: a CTA writes as soon as its own groups are in)
  bool in = true;
  if (S > 1 && epi) {
    in = mbar_wait(rbar, 0, lim);
    if (!in) {
      *s_abort = 1;
      atomicExch(a.err, kErrFlagTimeout);
    }
  }
  // warp-uniform again (the S = 1 path reads TMEM); only the stores check m < N
  if (epi && __all_sync(0xffffffffu, ok && in && !*s_abort)) {
    if (a.fault == kFaultAbort) {          // test fault: the output stays unwritten
      if (threadIdx.x == 64) atomicExch(a.err, kErrInjected);
    } else {
#pragma unroll 1
      for (int g = rank; g < G; g += S) {
        float f[4] = {0.f, 0.f, 0.f, 0.f};
        if (S > 1) {
#pragma unroll 1
          for (int s = 0; s < S; ++s) {
            const uint4 p = recv[(s * gpo + g / S) * kSmM + row];
            f[0] += __uint_as_float(p.x);
            f[1] += __uint_as_float(p.y);
            f[2] += __uint_as_float(p.z);
            f[3] += __uint_as_float(p.w);
          }
        } else {
          uint32_t v[4];
          tmem_ld4(trow + (uint32_t)(4 * g), v);
#pragma unroll
          for (int i = 0; i < 4; ++i) f[i] = __uint_as_float(v[i]);
        }
        if (m < a.N) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int t = 4 * g + i;
            if (t < a.T) {
              const int val = __float2int_rn(f[i] * kUnitsPerSpike);
              if (a.acc) a.acc[(int64_t)t * a.N + m] = val;
              if (a.y) a.y[(int64_t)t * a.N + m] = scale_out(sc, val);
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kSmTmemCols);
  }
}

int g_sms = 0;

// Largest number of clusters of `size` CTAs of gemm_small_kernel that can be
// resident at once (-1 when the occupancy query fails).
int small_active_clusters(int size) {
  static int cache[kGemmSmallMaxS + 1] = {0};
  if (cache[size] == 0) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = size;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.gridDim = dim3(size, 1, 1);
    cfg.blockDim = dim3(kSmThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmSmem;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_small_kernel, &cfg) != cudaSuccess || n < 1) {
      (void)cudaGetLastError();
      n = -1;
    }
    cache[size] = n;
  }
  return cache[size];
}

cudaError_t small_init() {
  static bool done = false;
  if (done) return cudaSuccess;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemm_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmSmem);
  if (e != cudaSuccess) return e;
  done = true;
  return cudaSuccess;
}

}  // namespace

int gemm_small_splits(int T, int N, int Kp) {
  if (T < 1 || T > kGemmSmallMaxT || small_init() != cudaSuccess) return 0;
  const int tiles = ceil_div(N, kSmM);
  const int nkb = Kp / kSmBK;
  // the most K ranges that keep every CTA's spike slice in shared memory,
  // every cluster resident at once and no SM holding two CTAs
  for (int S = kGemmSmallMaxS; S >= 1; S /= 2) {
    if (S > nkb || ceil_div(nkb, S) > kGemmSmallMaxKB || tiles * S > g_sms) continue;
    if (S > 1 && small_active_clusters(S) < tiles) continue;
    return S;
  }
  return 0;
}

cudaError_t launch_gemm_small(const CUtensorMap& mapW, const GemmSmallArgs& a, cudaStream_t s) {
  cudaError_t e = small_init();
  if (e != cudaSuccess) return e;
  if (a.S < 1 || a.S > kGemmSmallMaxS || (a.S & (a.S - 1)) != 0 || a.T < 1 || a.T > kGemmSmallMaxT || a.TN % 16 != 0 ||
      a.TN < a.T || a.TN > kGemmSmallMaxT || a.nkb < a.S || ceil_div(a.nkb, a.S) > kGemmSmallMaxKB)
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = a.S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)(ceil_div(a.N, kSmM) * a.S), 1, 1);
  cfg.blockDim = dim3(kSmThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, gemm_small_kernel, mapW, a);
}

}  // namespace sp
