// sp_head.cu -- vocabulary head with INT8 activations and candidate-row
// verification (Section 5, trace configuration; Appendix D), one launch per
// call for up to 4 hidden states:
//
//   1. s_x = max(max_k |h_k|, 1e-8) / 127, q_k = clip(rint(h_k / s_x), +-127)
//      (the weight quantiser of Section 2.3 read onto the hidden vector)
//   2. a_m = sum_k Q[m][k] q_k (exact INT32), z_m = s_m * (s_x * float(a_m))
//   3. order by z descending (equal z: lower row first); gap = z_(1) - z_(2)
//   4. gate: verification when gap < tau
//   5. the k_sel first rows are recomputed with the FP32 activations,
//      r_m = s_m * sum_k float(Q[m][k]) h_k (the continuous-input rule)
//   6. token = the candidate with the largest r (equal r: lower row), or,
//      without verification, the first row of the order.
//
// Steps 1-4 reach exactly the definition's values: the codes and the scale
// come from the same IEEE operations, the integer sums are order-free and z
// is two RN multiplies, so z, the gap, the gate and the candidate rows are
// bit-identical to the definition's.  r is an FP32 sum (per lane in ascending
// k, then a 5-level butterfly: depth 16 * ceil(K / 512) + 5), within the
// usual FP32 dot-product bound of the exact value.
//
// Layout of the work.  The weights stream from HBM once (V * K bytes) and
// dominate the traffic, so the kernel is HBM-bound.  Every CTA builds the
// INT8 codes of all hidden states in shared memory.  A warp owns units of 4
// consecutive rows; lane l reads the 16-byte chunks l, l + 32, ... of each
// row and accumulates __dp4a products with the codes.  Each z becomes a
// 64-bit key (z's order-preserving bits, then the complement of the row, so
// that one unsigned comparison orders by z descending and row ascending;
// keys are distinct) and the warp keeps its best 64 keys in a sorted list
// (bitonic sort of 32 new keys, then a bitonic merge with the list).
//
// Every key of the final 64 is in some CTA's list, so the CTA lists are all
// that the selection reads.  Each projection CTA merges its 8 warp lists in
// shared memory (a tree of pairwise bitonic merges), writes one list to the
// workspace, and counts the list's keys in a 4096-bin histogram of their 12
// leading order bits.  A second kernel, one CTA launched as the programmatic
// dependent of the first, takes as a lower bound T the histogram bin that
// holds the 64th best listed key, and in the same round of loads the first
// 4 keys of every list.  The keys >= T (about seventy) are gathered (the
// rest of a list is fetched only when all 4 of its leading keys pass),
// ordered by counting, gated, and the candidates recomputed, 4 rows per warp
// with all their loads in flight.  The projection kernel has little shared
// memory and no clusters: a larger shared-memory carve-out or a cluster
// launch slowed its weight stream.
#include "sp_internal.h"
#include "sp_ptx.cuh"
#include "sp_rows.cuh"
#include "sp_spikes.cuh"

namespace sp {
namespace {

constexpr int kHeadThreads = 256;
constexpr int kHeadWarps = kHeadThreads / 32;
constexpr int kHeadRows = 4;                  // rows per unit (one warp)
constexpr int kHeadList = SPIKE_PROJ_HEAD_MAX_CAND;   // keys per sorted list
constexpr int kSelThreads = 512;              // threads of the selection CTA
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kLead = 4;                      // leading keys of each list read first
constexpr int kHistBits = 12;                 // histogram bins: the keys' leading order bits
constexpr int kHistWords = 1 << kHistBits;    // bins of one hidden state
constexpr int kHeadMaxGrid = 1024;            // projection CTAs (lists) of one call
static_assert(kHeadList == 64, "a list is two keys per lane");
static_assert(SPIKE_PROJ_HEAD_MAX_K % (4 * 256) == 0, "the codes phase covers K in float4 per thread");
static_assert(kSelThreads * 8 == kHistWords, "hist_bound: 8 bins per selection thread");
static_assert(kHeadList == 4 * kSelWarps, "four candidates per selection warp");

typedef unsigned long long hkey;

// Workspace: the CTA lists (projection CTA c's list of hidden state b is
// list b * nlists + c), then per hidden state the histogram of the listed
// keys' 12 leading order bits (4096 bins, an eighth of an octave of z
// each), zero between calls.
constexpr size_t kListBytes = (size_t)SPIKE_PROJ_HEAD_MAX_B * kHeadMaxGrid * kHeadList * 8;
constexpr size_t kHistBytes = (size_t)SPIKE_PROJ_HEAD_MAX_B * kHistWords * 4;

struct HeadParams {
  const int8_t* W;
  int64_t ldw;
  const float* scale;
  int32_t V, K, Kpad, units;
  const float* h;
  int64_t ldh;
  float tau;
  int32_t k_sel;
  int32_t* token;
  int32_t* verified;
  float* gap;
  int32_t* cand;
  float* r;
  float* z;
  int64_t ld_z;
  int32_t B;
  hkey* lists;             // one 64-key list per projection CTA and hidden state
  uint32_t* hist;          // [B][kHistWords]
  int32_t nlists;          // CTAs of the projection kernel
};

// Order-preserving bits of z (both zeros map to the bits of +0).
__device__ __forceinline__ uint32_t order_bits(float z) {
  const uint32_t u = z == 0.0f ? 0u : __float_as_uint(z);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float from_order_bits(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
// Larger key = larger z, or equal z and lower row; 0 is below every key.
__device__ __forceinline__ hkey make_key(float z, int m) {
  return ((hkey)order_bits(z) << 32) | (hkey)(0xffffffffu - (uint32_t)m);
}
__device__ __forceinline__ int key_row(hkey k) { return (int)(0xffffffffu - (uint32_t)k); }
__device__ __forceinline__ float key_z(hkey k) { return from_order_bits((uint32_t)(k >> 32)); }
__device__ __forceinline__ hkey kmax(hkey a, hkey b) { return a > b ? a : b; }
__device__ __forceinline__ hkey kmin(hkey a, hkey b) { return a < b ? a : b; }

// The warp's 32 keys (one per lane) sorted descending: lane l gets the l-th.
__device__ __forceinline__ hkey warp_sort32(hkey v, int lane) {
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1)
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      const hkey o = __shfl_xor_sync(0xffffffffu, v, j);
      const bool lower = (lane & j) == 0;
      const bool desc = (lane & k) == 0;    // k == 32: every lane
      v = (lower == desc) ? kmax(v, o) : kmin(v, o);
    }
  return v;
}

// Sorts a bitonic sequence of 64 keys, element l in a and 32 + l in b of lane
// l, into descending order (half-cleaners of stride 32, 16, ..., 1).
__device__ __forceinline__ void warp_merge64(hkey& a, hkey& b, int lane) {
  const hkey hi = kmax(a, b), lo = kmin(a, b);
  a = hi;
  b = lo;
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const bool lower = (lane & j) == 0;
    const hkey oa = __shfl_xor_sync(0xffffffffu, a, j);
    const hkey ob = __shfl_xor_sync(0xffffffffu, b, j);
    a = lower ? kmax(a, oa) : kmin(a, oa);
    b = lower ? kmax(b, ob) : kmin(b, ob);
  }
}

// List (a, b) <- the best 64 of the list and the 32 keys n (one per lane).
// For descending A and B of equal length, max(A_i, B_{63-i}) holds the best
// 64 of both as a bitonic sequence; n is B with 32 empty keys appended.
__device__ __forceinline__ void list_insert32(hkey& a, hkey& b, hkey n, int lane) {
  n = warp_sort32(n, lane);
  b = kmax(b, __shfl_sync(0xffffffffu, n, 31 - lane));
  warp_merge64(a, b, lane);
}

// Merges the n sorted lists s[0 .. n) (64 keys each, in shared memory) in
// place, pairwise by the CTA's nw warps; the result is s[0].  Every thread
// calls it.
__device__ void tree_merge(hkey* s, int n, int nw) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int stride = 1; stride < n; stride <<= 1) {
    for (int q = warp; q * 2 * stride + stride < n; q += nw) {
      hkey* A = s + (size_t)(q * 2 * stride) * kHeadList;
      const hkey* Bl = A + (size_t)stride * kHeadList;
      hkey a = kmax(A[lane], Bl[63 - lane]);
      hkey b = kmax(A[32 + lane], Bl[31 - lane]);
      warp_merge64(a, b, lane);
      __syncwarp();
      A[lane] = a;
      A[32 + lane] = b;
    }
    __syncthreads();
  }
}

// out[0 .. 64) <- the best min(C, 64) of the C distinct keys buf[0 .. C),
// descending (each placed by counting the larger ones), 0 past C.
__device__ void rank_place(const hkey* buf, int C, hkey* out) {
  const int t = threadIdx.x, nt = blockDim.x;
  for (int i = C + t; i < kHeadList; i += nt) out[i] = 0ull;
  for (int i = t; i < C; i += nt) {
    const hkey ki = buf[i];
    int larger = 0;
    int j = 0;
    for (; j + 8 <= C; j += 8) {                 // 8 loads in flight
      hkey v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = buf[j + e];
#pragma unroll
      for (int e = 0; e < 8; ++e) larger += v[e] > ki;
    }
    for (; j < C; ++j) larger += buf[j] > ki;
    if (larger < kHeadList) out[larger] = ki;
  }
  __syncthreads();
}

// The lower bound of the leading order bits of the histogram bin that holds
// the need-th largest key, from a kHistWords-bin histogram (bin i counts the
// keys whose leading bits are i): thread t of a kSelThreads-thread CTA holds
// bins 8t .. 8t + 7 in c (loaded by the caller, so that the loads can be in
// flight with others), and the suffix sums meet in two barriers.  0 when
// the histogram holds fewer than need keys.  Every thread calls it.
__device__ uint32_t hist_bound(const uint32_t (&c)[8], uint32_t need, uint32_t* s_wtot,
                               uint32_t& s_bin) {
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  uint32_t sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) sum += c[i];
  uint32_t S = sum;                              // keys in the bins of lanes >= this one
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t o = __shfl_down_sync(0xffffffffu, S, d);
    if (lane + d < 32) S += o;
  }
  if (lane == 0) s_wtot[warp] = S;
  if (t == 0) s_bin = 0u;
  __syncthreads();
  for (int w = warp + 1; w < (int)(blockDim.x >> 5); ++w) S += s_wtot[w];
  if (S >= need && S - sum < need) {             // this thread's bins hold the need-th key
    uint32_t cum = S - sum;
#pragma unroll
    for (int i = 7; i >= 0; --i) {
      if (cum + c[i] >= need) {
        s_bin = (uint32_t)(8 * t + i) << (32 - kHistBits);
        break;
      }
      cum += c[i];
    }
  }
  __syncthreads();
  return s_bin;
}

// r of up to 4 candidate rows (rows[j], j < n) for hidden state hb, by one
// warp: per row, lane l sums the 16-byte chunks l, l + 32, ... in ascending k
// with fmaf, then the 5-level butterfly (the continuous-input kernel's
// order); the loads of all the rows and of up to 4 chunks are in flight
// together.
__device__ __forceinline__ void verify_rows4(const HeadParams& p, const float* hb, const int (&rows)[4],
                                             int n, int lane, float (&out)[4]) {
  const int nch = (p.K + 511) / 512;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int c0 = 0; c0 < nch; c0 += 4) {
    uint4 v[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int k = 16 * (lane + 32 * (c0 + t));
        if (j < n && c0 + t < nch && k < p.K) v[j][t] = ld_weights16(p.W + (int64_t)rows[j] * p.ldw + k);
      }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int k = 16 * (lane + 32 * (c0 + t));
      if (c0 + t < nch && k < p.K) {
        float x[16];
        load_x16(hb, k, p.K, x);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (j < n) {
            const uint32_t ww[4] = {v[j][t].x ^ 0x80808080u, v[j][t].y ^ 0x80808080u,
                                    v[j][t].z ^ 0x80808080u, v[j][t].w ^ 0x80808080u};
#pragma unroll
            for (int e = 0; e < 16; ++e)
              acc[j] = fmaf(byte_to_float(ww[e >> 2], (uint32_t)(e & 3)), x[e], acc[j]);
          }
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) {
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) acc[j] += __shfl_xor_sync(0xffffffffu, acc[j], d);
    out[j] = j < n ? __fmul_rn(__ldg(p.scale + rows[j]), acc[j]) : 0.f;
  }
}

// Step 1 for every hidden state: thread t holds h[4t + 1024 i .. +3], i < NV,
// in registers (one read of h); the CTA's maximum |h| meets in one barrier
// and every thread derives s_x; the codes go to shared memory four to a word.
template <int B, int NV>
__device__ __forceinline__ void head_codes(const HeadParams& p, int8_t* s_codes, float* s_red, float* s_sx) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll 1
  for (int b = 0; b < B; ++b) {
    const float* hb = p.h + (int64_t)b * p.ldh;
    float4 hv[NV];
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int k = 4 * (int)threadIdx.x + 4 * kHeadThreads * i;
      hv[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (k + 4 <= p.K) {
        hv[i] = __ldg(reinterpret_cast<const float4*>(hb + k));   // h 16-byte aligned, ldh % 4 == 0
      } else if (k < p.K) {
        hv[i].x = hb[k];
        if (k + 1 < p.K) hv[i].y = hb[k + 1];
        if (k + 2 < p.K) hv[i].z = hb[k + 2];
      }
      mx = fmaxf(mx, fmaxf(fmaxf(fabsf(hv[i].x), fabsf(hv[i].y)), fmaxf(fabsf(hv[i].z), fabsf(hv[i].w))));
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, d));
    if (lane == 0) s_red[warp] = mx;
    __syncthreads();
    float a = s_red[0];
#pragma unroll
    for (int w = 1; w < kHeadWarps; ++w) a = fmaxf(a, s_red[w]);
    const float sx = __fdiv_rn(fmaxf(a, 1e-8f), 127.0f);
    if (threadIdx.x == 0) s_sx[b] = sx;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int k = 4 * (int)threadIdx.x + 4 * kHeadThreads * i;
      if (k < p.Kpad) {
        const float e[4] = {hv[i].x, hv[i].y, hv[i].z, hv[i].w};
        uint32_t packed = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          int c = 0;
          if (k + j < p.K) c = (int)fminf(fmaxf(rintf(__fdiv_rn(e[j], sx)), -127.0f), 127.0f);
          packed |= ((uint32_t)c & 0xffu) << (8 * j);
        }
        *reinterpret_cast<uint32_t*>(s_codes + b * p.Kpad + k) = packed;
      }
    }
    __syncthreads();                             // s_red is rewritten by the next hidden state
  }
}

template <int B> struct HeadShape { static constexpr int min_ctas = 2; };
template <> struct HeadShape<1> { static constexpr int min_ctas = 4; };

// Steps 1-2 and the CTA's lists.
template <int B>
__global__ void __launch_bounds__(kHeadThreads, HeadShape<B>::min_ctas)
head_kernel(const __grid_constant__ HeadParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  hkey* s_all = reinterpret_cast<hkey*>(smem);             // [8][64]
  int8_t* s_codes = reinterpret_cast<int8_t*>(s_all + kHeadWarps * kHeadList);   // [B][Kpad]
  __shared__ float s_red[kHeadWarps];
  __shared__ float s_sx[B];

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = gridDim.x * kHeadWarps;
  const int wg = blockIdx.x * kHeadWarps + warp;
  // The weights are constant (no kernel writes them): the rows of this warp's
  // first unit are prefetched into L2 before the dependency wait.
  if (wg < p.units) {
    for (int r = 0; r < kHeadRows; ++r) {
      const int row = wg * kHeadRows + r;
      if (row >= p.V) break;
      for (int off = lane * 128; off < p.K; off += 32 * 128)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(p.W + (int64_t)row * p.ldw + off));
    }
  }
  pdl_wait();

  // 1. activation scale and INT8 codes of each hidden state (zero past K);
  // a compact form for K <= 2048 (the code runs once per CTA, and its size
  // shows in the start-up)
  if (p.K <= 2 * 4 * kHeadThreads) head_codes<B, 2>(p, s_codes, s_red, s_sx);
  else head_codes<B, SPIKE_PROJ_HEAD_MAX_K / (4 * kHeadThreads)>(p, s_codes, s_red, s_sx);

  // 2. approximate logits; each warp keeps its best 64 keys per hidden state
  hkey la[B], lb[B], pend[B];
#pragma unroll
  for (int b = 0; b < B; ++b) la[b] = lb[b] = pend[b] = 0ull;
  int slot = 0;                                  // units since the last insert
  const int nch = (p.K + 511) / 512;
  for (int u = wg; u < p.units; u += nwarps) {
    const int row0 = u * kHeadRows;
    const int nrows = min(kHeadRows, p.V - row0);
    int acc[kHeadRows][B];
#pragma unroll
    for (int r = 0; r < kHeadRows; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b) acc[r][b] = 0;
    for (int c = 0; c < nch; ++c) {
      const int k = 16 * (lane + 32 * c);
      if (k >= p.K) continue;
      // the row is ldw >= K bytes with ldw % 16 == 0: the 16 bytes at k lie
      // inside it; bytes at or past K meet zero codes
      uint4 w[kHeadRows];
#pragma unroll
      for (int r = 0; r < kHeadRows; ++r)
        w[r] = r < nrows ? ld_weights16(p.W + (int64_t)(row0 + r) * p.ldw + k) : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int b = 0; b < B; ++b) {
        const uint4 q = *reinterpret_cast<const uint4*>(s_codes + b * p.Kpad + k);
#pragma unroll
        for (int r = 0; r < kHeadRows; ++r) {
          int a = acc[r][b];
          a = __dp4a((int)w[r].x, (int)q.x, a);
          a = __dp4a((int)w[r].y, (int)q.y, a);
          a = __dp4a((int)w[r].z, (int)q.z, a);
          a = __dp4a((int)w[r].w, (int)q.w, a);
          acc[r][b] = a;
        }
      }
    }
#pragma unroll
    for (int r = 0; r < kHeadRows; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b)
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) acc[r][b] += __shfl_xor_sync(0xffffffffu, acc[r][b], d);
#pragma unroll
    for (int r = 0; r < kHeadRows; ++r) {
      if (r < nrows) {
        const float s = __ldg(p.scale + row0 + r);
#pragma unroll
        for (int b = 0; b < B; ++b) {
          const float zv = __fmul_rn(s, __fmul_rn(s_sx[b], __int2float_rn(acc[r][b])));
          if (p.z && lane == r * B + b) p.z[(int64_t)b * p.ld_z + row0 + r] = zv;
          if (lane == slot * kHeadRows + r) pend[b] = make_key(zv, row0 + r);
        }
      }
    }
    if (++slot == 32 / kHeadRows) {             // 32 pending keys: insert them
#pragma unroll
      for (int b = 0; b < B; ++b) {
        list_insert32(la[b], lb[b], pend[b], lane);
        pend[b] = 0ull;
      }
      slot = 0;
    }
  }
  if (slot) {
#pragma unroll
    for (int b = 0; b < B; ++b) list_insert32(la[b], lb[b], pend[b], lane);
  }
  // the selection kernel may become resident once every CTA is here (not
  // earlier: its CTAs would take slots from the weight stream)
  pdl_launch_dependents();

  // 3. the CTA's list per hidden state, into the workspace
#pragma unroll
  for (int b = 0; b < B; ++b) {
    s_all[warp * kHeadList + lane] = la[b];
    s_all[warp * kHeadList + 32 + lane] = lb[b];
    __syncthreads();
    tree_merge(s_all, kHeadWarps, kHeadWarps);
    const int64_t slot = (int64_t)b * p.nlists + blockIdx.x;
    if (threadIdx.x < kHeadList) {
      const hkey k = s_all[threadIdx.x];
      __stcg(p.lists + slot * kHeadList + threadIdx.x, k);
      // the listed keys into the histogram (equal bins of a warp summed
      // first): every key of the final selection is a listed key
      const uint32_t real = __ballot_sync(0xffffffffu, k != 0ull);
      if (k != 0ull) {
        const uint32_t bin = (uint32_t)(k >> (64 - kHistBits));
        const uint32_t mb = __match_any_sync(real, bin);
        if (lane == __ffs(mb) - 1) atomicAdd(p.hist + (int64_t)b * kHistWords + bin, (uint32_t)__popc(mb));
      }
    }
    __syncthreads();
  }
}

// Steps 3-6, one CTA of kSelThreads threads, per hidden state: the bound T
// and the leading keys of every list (one round of loads for both), the
// keys >= T, the best 64 of them by counting, the gate, the candidates
// recomputed (warp w: candidates w, w + 16, w + 32, w + 48), the token.  When
// the bound does not narrow the keys to at most kSelThreads (an adversarial
// spread, e.g. equal logits everywhere), or passes fewer than min(V, 64) (a
// histogram left dirty by a call that never reached this kernel), every list
// is merged instead, 15 at a time into a running best 64: slower, and exact
// either way.
__global__ void __launch_bounds__(kSelThreads, 1)
head_select_kernel(const __grid_constant__ HeadParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  hkey* s_lead = reinterpret_cast<hkey*>(smem);            // [nlists][kLead]; 16 lists when merging
  __shared__ hkey s_cand[kSelThreads];
  __shared__ hkey s_best[kHeadList];
  __shared__ float s_r[kHeadList];
  __shared__ int s_long[kSelThreads];
  __shared__ uint32_t s_wtot[kSelWarps];
  __shared__ uint32_t s_bin;
  __shared__ int s_nc, s_nlong;

  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int ks = p.k_sel, nl = p.nlists;
  pdl_launch_dependents();
  pdl_wait();                                    // every CTA list and count is written
  for (int b = 0; b < p.B; ++b) {
    const hkey* lists = p.lists + (int64_t)b * nl * kHeadList;
    // one round of loads: this thread's 8 histogram bins and the leading keys
    // (32 bytes) of lists t and t + kSelThreads
    const uint4* hq = reinterpret_cast<const uint4*>(p.hist + (int64_t)b * kHistWords) + 2 * t;
    const uint4 h0 = __ldcg(hq), h1 = __ldcg(hq + 1);
    ulonglong2 lead[2][2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int l = t + q * kSelThreads;
      if (l < nl) {
        const ulonglong2* src = reinterpret_cast<const ulonglong2*>(lists + (int64_t)l * kHeadList);
        lead[q][0] = __ldcg(src);
        lead[q][1] = __ldcg(src + 1);
      }
    }
    for (int l = t + 2 * kSelThreads; l < nl; l += kSelThreads) {   // more than 1024 lists: never
      const ulonglong2* src = reinterpret_cast<const ulonglong2*>(lists + (int64_t)l * kHeadList);
      const ulonglong2 k01 = __ldcg(src), k23 = __ldcg(src + 1);
      s_lead[l * kLead] = k01.x;
      s_lead[l * kLead + 1] = k01.y;
      s_lead[l * kLead + 2] = k23.x;
      s_lead[l * kLead + 3] = k23.y;
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int l = t + q * kSelThreads;
      if (l < nl) {
        s_lead[l * kLead] = lead[q][0].x;
        s_lead[l * kLead + 1] = lead[q][0].y;
        s_lead[l * kLead + 2] = lead[q][1].x;
        s_lead[l * kLead + 3] = lead[q][1].y;
      }
    }
    if (t == 0) {
      s_nc = 0;
      s_nlong = 0;
    }
    // the bound (its barriers also complete the stores above)
    const uint32_t hc[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
    const uint32_t tb = hist_bound(hc, kHeadList, s_wtot, s_bin);
    const hkey T = tb ? (hkey)tb << 32 : 1ull;   // no bound: every key passes
    for (int l = t; l < nl; l += kSelThreads) {
      int n = 0;
#pragma unroll
      for (int e = 0; e < kLead; ++e) {
        const hkey k = s_lead[l * kLead + e];
        if (k >= T) {
          const int i = atomicAdd(&s_nc, 1);
          if (i < kSelThreads) s_cand[i] = k;
          ++n;
        }
      }
      if (n == kLead) {                          // the list may continue past its leading keys
        const int j = atomicAdd(&s_nlong, 1);
        if (j < kSelThreads) s_long[j] = l;
      }
    }
    __syncthreads();
    const int nlong = s_nlong;
    for (int j = warp; j < min(nlong, kSelThreads); j += kSelWarps) {
      const hkey* L = lists + (int64_t)s_long[j] * kHeadList;
      for (int e = kLead + lane; e < kHeadList; e += 32) {
        const hkey k = __ldcg(L + e);
        if (k >= T) {
          const int i = atomicAdd(&s_nc, 1);
          if (i < kSelThreads) s_cand[i] = k;
        }
      }
    }
    __syncthreads();
    const int C = s_nc;
    if (C <= kSelThreads && nlong <= kSelThreads && C >= min(p.V, kHeadList)) {
      rank_place(s_cand, C, s_best);
    } else {
      hkey* s16 = s_lead;                        // 16 lists: the running best, then 15 more
      for (int i = t; i < kHeadList; i += kSelThreads) s16[i] = 0ull;
      for (int base = 0; base < nl; base += 15) {
        const int cnt = min(15, nl - base);
        for (int e = t; e < 15 * kHeadList; e += kSelThreads)
          s16[kHeadList + e] = e / kHeadList < cnt ? __ldcg(lists + (int64_t)base * kHeadList + e) : 0ull;
        __syncthreads();
        tree_merge(s16, 16, kSelWarps);
      }
      for (int i = t; i < kHeadList; i += kSelThreads) s_best[i] = s16[i];
      __syncthreads();
    }
    const float g = __fsub_rn(key_z(s_best[0]), key_z(s_best[1]));
    const bool open = g < p.tau;
    if (open) {
      const float* hb = p.h + (int64_t)b * p.ldh;
      int rows[4];
      int n = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = warp + kSelWarps * j;
        rows[j] = i < ks ? key_row(s_best[i]) : 0;
        if (i < ks) n = j + 1;
      }
      if (n > 0) {
        float rv[4];
        verify_rows4(p, hb, rows, n, lane, rv);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (j < n && lane == 0) s_r[warp + kSelWarps * j] = rv[j];
      }
      __syncthreads();
    }
    if (warp == 0) {
      int token = key_row(s_best[0]);
      if (open) {
        // largest r, equal r: lower row (starting from candidate 0, so the
        // token is always a candidate)
        float br = s_r[0];
        int bm = token;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const int i = lane + 32 * q;
          if (i < ks) {
            const float rv = s_r[i];
            const int m = key_row(s_best[i]);
            if (rv > br || (rv == br && m < bm)) {
              br = rv;
              bm = m;
            }
            if (p.r) p.r[(int64_t)b * ks + i] = rv;
          }
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) {
          const float orv = __shfl_xor_sync(0xffffffffu, br, d);
          const int om = __shfl_xor_sync(0xffffffffu, bm, d);
          if (orv > br || (orv == br && om < bm)) {
            br = orv;
            bm = om;
          }
        }
        token = bm;
      }
      if (lane == 0) {
        p.token[b] = token;
        if (p.verified) p.verified[b] = open ? 1 : 0;
        if (p.gap) p.gap[b] = g;
      }
    }
    if (p.cand && t < ks) p.cand[(int64_t)b * ks + t] = key_row(s_best[t]);
    __syncthreads();                             // s_lead, s_cand, s_best, s_r are rewritten next
  }
  // the histograms are read: clear them for the next call
  for (int i = t; i < p.B * kHistWords; i += kSelThreads) p.hist[i] = 0u;
}

int g_head_sms = 0;
size_t g_select_smem = 0;       // dynamic shared-memory limit set on head_select_kernel

template <typename Kern>
cudaError_t raise_smem(Kern kernel, size_t bytes, size_t& set_bytes) {
  if (bytes <= set_bytes) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) set_bytes = bytes;
  return e;
}

template <int B>
cudaError_t launch_head_t(HeadParams p, cudaStream_t s) {
  static size_t set_proj = 0;    // per instance: head_kernel<B> is a kernel of its own
  const size_t smem = (size_t)kHeadWarps * kHeadList * 8 + (size_t)B * p.Kpad;
  cudaError_t e = raise_smem(head_kernel<B>, smem, set_proj);
  if (e != cudaSuccess) return e;
  // resident CTAs per SM, queried once per shared-memory size (a driver
  // call of about a microsecond)
  static int per_sm = 0;
  static size_t per_sm_smem = 0;
  if (per_sm == 0 || per_sm_smem != smem) {
    int n = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, head_kernel<B>, kHeadThreads, smem);
    if (e != cudaSuccess) return e;
    per_sm = n < 1 ? 1 : n;
    per_sm_smem = smem;
  }
  // one wave: every CTA resident at once
  int grid = g_head_sms * per_sm;
  const int need = (p.units + kHeadWarps - 1) / kHeadWarps;
  if (grid > need) grid = need;
  if (grid > kHeadMaxGrid) grid = kHeadMaxGrid;
  if (grid < 1) grid = 1;
  p.nlists = grid;
  e = launch_pdl(head_kernel<B>, dim3((unsigned)grid), dim3(kHeadThreads), smem, s, p);
  if (e != cudaSuccess) return e;

  const size_t sel_smem = (size_t)(grid * kLead > 16 * kHeadList ? grid * kLead : 16 * kHeadList) * 8;
  e = raise_smem(head_select_kernel, sel_smem, g_select_smem);   // one kernel for every B
  if (e != cudaSuccess) return e;
  return launch_pdl(head_select_kernel, dim3(1), dim3(kSelThreads), sel_smem, s, p);
}

}  // namespace

size_t head_workspace_bytes() { return kListBytes + kHistBytes; }

cudaError_t launch_head(const HeadArgs& a, cudaStream_t s) {
  if (g_head_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&g_head_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  HeadParams p;
  p.W = a.W;
  p.ldw = a.ldw;
  p.scale = a.scale;
  p.V = a.V;
  p.K = a.K;
  p.Kpad = (a.K + 511) / 512 * 512;
  p.units = (a.V + kHeadRows - 1) / kHeadRows;
  p.h = a.h;
  p.ldh = a.ldh;
  p.tau = a.tau;
  p.k_sel = a.k_sel;
  p.token = a.token;
  p.verified = a.verified;
  p.gap = a.gap;
  p.cand = a.cand;
  p.r = a.r;
  p.z = a.z;
  p.ld_z = a.ld_z;
  p.B = a.B;
  p.lists = static_cast<hkey*>(a.ws);
  p.hist = reinterpret_cast<uint32_t*>(static_cast<unsigned char*>(a.ws) + kListBytes);
  p.nlists = 0;
  switch (a.B) {
    case 1: return launch_head_t<1>(p, s);
    case 2: return launch_head_t<2>(p, s);
    case 3: return launch_head_t<3>(p, s);
    default: return launch_head_t<4>(p, s);
  }
}

}  // namespace sp
