// sp_gemm.cu -- dense tensor-core path for many spike rows at once:
//
//   ACC[t][m] = sum_k X[t][k] * Q[m][k],   Y[t][m] = s_m * float(ACC[t][m])
//
// i.e. Eq. (sparse) for every row of a dense spike matrix (prompt prefill).
//
// The 5th-generation tensor cores of sm_103a have no integer MMA
// (ptxas rejects tcgen05.mma .kind::i8 for this target), so the contraction
// runs as tcgen05.mma .kind::f16 with bf16 operands and fp32 accumulation in
// tensor memory.  It is exact: spikes 0/1 and weights in [-128, 127] are bf16
// integers, every product is an integer, and every partial sum is an integer
// of magnitude <= 128 * K < 2^24, so no fp32 addition ever rounds.  The
// epilogue converts the accumulator to INT32 without loss.
//
// Kernel structure (one CTA per SM, persistent over work units):
//   warp 0      TMA producer: 128x64 (X) and 256x64 (W) bf16 boxes, 128-byte
//               swizzle, into a 4-stage shared-memory ring (mbarriers)
//   warp 1      allocates 512 TMEM columns (two 128x256 fp32 accumulators) and
//               issues tcgen05.mma (M=128, N=256, K=16) from one thread;
//               tcgen05.commit frees ring slots and publishes accumulators
//   warps 2-5   epilogue: tcgen05.ld 32 columns at a time, transpose through
//               shared memory so each warp store covers 128 contiguous bytes
//               of one output row, then either write acc / y, or (split K)
//               add the INT32 partial into the workspace; the warp that
//               completes the last split of its 32-row quarter of a tile
//               (atomic ticket per quarter) writes acc / y and re-zeroes the
//               workspace.
// A work unit is (128-row block, 256-column block, K split).  K is split so
// that units ~ number of SMs when the output has few tiles (T = 512 gives only
// 24 tiles of 128x256 for N = 1536).
//
// Every mbarrier wait is bounded (about one second of %globaltimer); on
// timeout the kernel sets the error word, stops issuing work, drains what it
// issued and frees its tensor memory before exiting.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "sp_gemm.h"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;          // 16 KB
constexpr int B_BYTES = BN * BK * 2;          // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 2 * BN;             // double-buffered accumulator
constexpr int kGemmThreads = 192;
constexpr int TR_STRIDE = 33;                 // padded transpose rows (words)
constexpr size_t SMEM_RING = (size_t)STAGES * STAGE_BYTES;
constexpr size_t SMEM_TR = (size_t)4 * 32 * TR_STRIDE * 4;
constexpr size_t SMEM_BARS = 256;
constexpr size_t kGemmSmem = 1024 + SMEM_RING + SMEM_TR + SMEM_BARS;
constexpr uint64_t kWaitLimitNs = 1000000000ull;   // 1 s

// ---- PTX wrappers -------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity; false on timeout.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (;;) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t cols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(cols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(cols)
               : "memory");
}
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on a CTA-local mbarrier once all previously issued MMAs complete.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// 32 lanes x 32 consecutive 32-bit columns: thread i gets row (lane base + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor (tcgen05 format): K-major operand whose rows
// are 128 bytes (64 bf16) laid out by TMA with the 128-byte swizzle; 8-row
// groups are 1024 bytes apart (stride byte offset).  Stage buffers are
// 1024-byte aligned, so the base-offset field is 0.  Advancing K by 16
// elements inside the swizzle atom adds 32 bytes to the start address.
__device__ __forceinline__ uint64_t smem_desc_k128(const void* p) {
  const uint64_t addr = smem_u32(p);
  uint64_t d = (addr >> 4) & 0x3FFFull;    // start address
  d |= (uint64_t)1 << 16;                  // leading byte offset (unused here)
  d |= (uint64_t)(1024 >> 4) << 32;        // stride byte offset
  d |= (uint64_t)1 << 46;                  // descriptor version for tcgen05
  d |= (uint64_t)2 << 61;                  // 128-byte swizzle
  return d;
}
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major,
// N = 256, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);

struct GemmArgs {
  GemmParams p;
  int tiles_m, tiles_n, splits, kb_per_split, nkb, units;
  int32_t* ws;
  uint32_t* tickets;
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
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

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
          if (!mbar_wait(&empty[stage], ph ^ 1u)) {
            *s_abort = 1;
            atomicExch(a.p.err, kErrMbarTimeout);
            break;
          }
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          tma_load_2d(sA + (size_t)stage * A_BYTES, &mapA, &full[stage], kb * BK, mb * BM);
          tma_load_2d(sB + (size_t)stage * B_BYTES, &mapB, &full[stage], kb * BK, nb * BN);
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
        mbar_wait(&full[s], q);
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
        if (!mbar_wait(&tempty[ab], aph ^ 1u)) {
          *s_abort = 1;
          atomicExch(a.p.err, kErrMbarTimeout);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(ab * BN);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], ph)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc_k128(sA + (size_t)stage * A_BYTES);
          const uint64_t bd = smem_desc_k128(sB + (size_t)stage * B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16(d, ad + 2u * k, bd + 2u * k, kIdesc, (kb > kb0 || k > 0) ? 1u : 0u);
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
      mbar_wait(done, 0);
    }
  } else {
    // ------------------------------ epilogue ----------------------------------
    // Each warp owns one 32-row quarter of the tile (its TMEM lane quarter) and
    // works alone: no barrier joins the epilogue warps, so a warp that gives up
    // on a timed-out wait cannot strand the others.
    const int q = warp & 3;
    uint32_t* tr = s_tr + (size_t)(warp - 2) * 32 * TR_STRIDE;
    int ab = 0;
    uint32_t aph = 0;
    const int T = a.p.T, N = a.p.N;
    for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
      int tile, mb, nb, kb0, kb1;
      unit_coords(a, u, tile, mb, nb, kb0, kb1);
      if (!mbar_wait(&tfull[ab], aph)) {
        *s_abort = 1;
        if (lane == 0) atomicExch(a.p.err, kErrMbarTimeout);
        break;
      }
      tc_fence_after();
      const int row0 = mb * BM + q * 32;     // first row of this warp's quarter
      for (int c = 0; c < BN; c += 32) {
        uint32_t v[32];
        tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN + c), v);
        // transpose: lane = row on the way in, lane = column on the way out
#pragma unroll
        for (int i = 0; i < 32; ++i) tr[lane * TR_STRIDE + i] = v[i];
        __syncwarp();
        const int n = nb * BN + c + lane;
        const bool col_ok = n < N;
        const float sc = (col_ok && a.p.y && a.splits == 1) ? __ldg(a.p.scale + n) : 0.f;
        for (int rr = 0; rr < 32; ++rr) {
          const int r = row0 + rr;
          if (r >= T) break;
          const int val = __float2int_rn(__uint_as_float(tr[rr * TR_STRIDE + lane]));
          if (!col_ok) continue;
          const int64_t o = (int64_t)r * N + n;
          if (a.splits == 1) {
            if (a.p.acc) a.p.acc[o] = val;
            if (a.p.y) a.p.y[o] = scale_out(sc, val);
          } else if (val) {
            atomicAdd(a.ws + o, val);
          }
        }
        __syncwarp();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[ab]);
      if (++ab == 2) { ab = 0; aph ^= 1u; }

      if (a.splits > 1) {
        // the warp that completes this quarter's last K split finishes it
        __threadfence();
        __syncwarp();
        int last = 0;
        if (lane == 0) {
          uint32_t* tk = a.tickets + (size_t)tile * 4 + q;
          const uint32_t prev = atomicAdd(tk, 1u);
          last = prev == (uint32_t)(a.splits - 1);
          if (last) atomicExch(tk, 0u);
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          __threadfence();
          const int cols = min(BN, N - nb * BN);
          for (int rr = 0; rr < 32; ++rr) {
            const int r = row0 + rr;
            if (r >= T) break;
            for (int cc = lane; cc < cols; cc += 32) {
              const int n = nb * BN + cc;
              const int64_t o = (int64_t)r * N + n;
              const int val = __ldcg(a.ws + o);
              __stcg(a.ws + o, 0);
              if (a.p.acc) a.p.acc[o] = val;
              if (a.p.y) a.p.y[o] = scale_out(__ldg(a.p.scale + n), val);
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
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---- operand preparation ------------------------------------------------------

// W column-major INT8 [K][ldw] -> bf16 K-major [N][Kp] (zero for k >= K):
// 32x32 tiles transposed through shared memory.
__global__ void w_to_bf16_kernel(const int8_t* __restrict__ W, int64_t ldw, int N, int K, int Kp,
                                 __nv_bfloat16* __restrict__ Wb) {
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
    if (m < N && k < Kp) Wb[(int64_t)m * Kp + k] = __float2bfloat16_rn((float)tile[tx][i]);
  }
}

// Spike rows (either format) -> bf16 0/1 [T][Kp], zero past K.  One thread
// per 8 consecutive columns of a row.
__global__ void spikes_to_bf16_kernel(const void* __restrict__ spikes, int fmt, int64_t ld, int T,
                                      int K, int Kp, __nv_bfloat16* __restrict__ Xb) {
  const int per_row = Kp / 8;
  const int64_t total = (int64_t)T * per_row;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / per_row);
    const int k = (int)(i - (int64_t)t * per_row) * 8;
    uint32_t bits = 0u;                      // spikes of columns k .. k+7
    if (k < K) {
      const void* row = spike_row(spikes, fmt, t, ld);
      if (fmt == SP_SPIKES_BITS32) {
        bits = (__ldg(reinterpret_cast<const uint32_t*>(row) + (k >> 5)) >> (k & 31)) & 0xffu;
      } else {
        const uint8_t* x = reinterpret_cast<const uint8_t*>(row) + k;
        const int n = K - k < 8 ? K - k : 8;
        for (int j = 0; j < n; ++j) bits |= (uint32_t)(__ldg(x + j) != 0) << j;
      }
      if (K - k < 8) bits &= (1u << (K - k)) - 1u;
    }
    // bf16 1.0 = 0x3F80; two columns per 32-bit word
    uint4 o;
    o.x = ((bits >> 0) & 1u ? 0x3F80u : 0u) | ((bits >> 1) & 1u ? 0x3F800000u : 0u);
    o.y = ((bits >> 2) & 1u ? 0x3F80u : 0u) | ((bits >> 3) & 1u ? 0x3F800000u : 0u);
    o.z = ((bits >> 4) & 1u ? 0x3F80u : 0u) | ((bits >> 5) & 1u ? 0x3F800000u : 0u);
    o.w = ((bits >> 6) & 1u ? 0x3F80u : 0u) | ((bits >> 7) & 1u ? 0x3F800000u : 0u);
    *reinterpret_cast<uint4*>(Xb + (int64_t)t * Kp + k) = o;
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

bool encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
               uint32_t box_inner, uint32_t box_outer) {
  auto enc = get_encode();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int gemm_k_pad(int K) { return ceil_div(K, BK) * BK; }
int gemm_ticket_count(int T, int N) { return ceil_div(T, BM) * ceil_div(N, BN) * 4; }

cudaError_t gemm_make_maps(const __nv_bfloat16* Xb, int rows_alloc, const __nv_bfloat16* Wb, int N,
                           int Kp, GemmMaps* out) {
  if (!encode_2d(&out->a, Xb, (uint64_t)Kp, (uint64_t)rows_alloc, BK, BM)) return cudaErrorUnknown;
  if (!encode_2d(&out->b, Wb, (uint64_t)Kp, (uint64_t)N, BK, BN)) return cudaErrorUnknown;
  return cudaSuccess;
}

cudaError_t launch_w_to_bf16(const int8_t* W, int64_t ldw, int N, int K, __nv_bfloat16* Wb,
                             cudaStream_t s) {
  const int Kp = gemm_k_pad(K);
  dim3 grid(ceil_div(Kp, 32), ceil_div(N, 32)), block(32, 8);
  w_to_bf16_kernel<<<grid, block, 0, s>>>(W, ldw, N, K, Kp, Wb);
  return cudaGetLastError();
}

cudaError_t launch_spikes_to_bf16(const void* spikes, int fmt, int64_t ld, int T, int K, int Kp,
                                  __nv_bfloat16* Xb, cudaStream_t s) {
  const int64_t total = (int64_t)T * (Kp / 8);
  const int threads = 256;
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  spikes_to_bf16_kernel<<<(int)blocks, threads, 0, s>>>(spikes, fmt, ld, T, K, Kp, Xb);
  return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmMaps& maps, int T, int N, int Kp, const GemmParams& p,
                        int32_t* ws, uint32_t* tickets, cudaStream_t s) {
  if (!g_attr_set) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kGemmSmem);
    if (e != cudaSuccess) return e;
    g_attr_set = true;
  }
  GemmArgs a;
  a.p = p;
  a.tiles_m = ceil_div(T, BM);
  a.tiles_n = ceil_div(N, BN);
  a.nkb = Kp / BK;
  const int tiles = a.tiles_m * a.tiles_n;
  int splits = g_num_sms / tiles;
  if (splits > a.nkb / 4) splits = a.nkb / 4;
  if (splits < 1) splits = 1;
  a.kb_per_split = ceil_div(a.nkb, splits);
  a.splits = ceil_div(a.nkb, a.kb_per_split);
  a.units = tiles * a.splits;
  a.ws = ws;
  a.tickets = tickets;
  const int grid = a.units < g_num_sms ? a.units : g_num_sms;
  gemm_kernel<<<grid, kGemmThreads, kGemmSmem, s>>>(maps.a, maps.b, a);
  return cudaGetLastError();
}

}  // namespace sp
