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
// The selection is a tree of pairwise bitonic merges of 64-key lists.  The
// CTA merges its 8 warp lists in shared memory and writes one list to the
// workspace.  A second kernel, one cluster of 8 CTAs of 512 threads
// launched as the programmatic dependent of the first, merges those lists:
// CTA r the lists of projection CTAs r, r + 8, ... (stored contiguously, so
// one bulk copy brings them into shared memory), CTA 0 the eight results.  CTA 0 applies the gate, the
// cluster's 64 warps recompute one candidate each, and CTA 0 picks the token.
// Results move between the CTAs of the cluster by stores into the receiver's
// shared memory, each followed by a cluster barrier before the receiver
// reads.  The projection kernel is launched without clusters and with little
// shared memory: a cluster launch or a larger shared-memory carve-out slows
// its weight stream (fewer resident CTAs, less L1 for loads in flight).
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
constexpr int kHeadCluster = 8;               // CTAs of the selection kernel
constexpr int kSelThreads = 512;              // threads of a selection CTA
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kHeadGatherLists = 128;         // most lists one gather_ge call takes
constexpr int kHistBits = 12;                 // histogram bins: the keys' leading order bits
constexpr int kHistWords = 1 << kHistBits;    // bins of one hidden state
constexpr int kHeadMaxGrid = 1024;            // projection CTAs (lists) of one call
static_assert(kHeadList == 64, "a list is two keys per lane");
static_assert(SPIKE_PROJ_HEAD_MAX_K % (4 * 256) == 0, "the codes phase covers K in float4 per thread");
static_assert(kSelThreads * 8 == kHistWords, "hist_bound: 8 bins per selection thread");
static_assert(kHeadList == kHeadCluster * kHeadWarps, "one candidate per warp of a cluster");

typedef unsigned long long hkey;

// Workspace: the CTA lists (projection CTA c's list of hidden state b is
// list (b * 8 + c % 8) * ceil(nlists / 8) + c / 8), then per hidden state
// the histogram of the listed keys' 12 leading order bits (4096 bins, an
// eighth of an octave of z each), zero between calls.
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

// Scratch of gather_ge (shared memory).
struct GatherScratch {
  int off[kHeadGatherLists];       // keys per list that pass the bound, then offsets
  int total;
};

// Copies the keys >= T of the n sorted lists s[0 .. n) (64 keys each, in
// shared memory; a prefix of each) into buf and
// returns their number, or -1 (nothing copied) when more than cap pass.
// n <= kHeadGatherLists; every thread of the CTA calls it.
__device__ int gather_ge(const hkey* s, int n, hkey T, hkey* buf, int cap, GatherScratch& sc) {
  const int t = threadIdx.x, nt = blockDim.x;
  for (int l = t >> 5; l < n; l += nt >> 5) {    // a warp per list: its keys >= T, counted
    const hkey* L = s + (size_t)l * kHeadList;
    const uint32_t b0 = __ballot_sync(0xffffffffu, L[t & 31] >= T);
    const uint32_t b1 = __ballot_sync(0xffffffffu, L[32 + (t & 31)] >= T);
    if ((t & 31) == 0) sc.off[l] = __popc(b0) + __popc(b1);
  }
  __syncthreads();
  if (t < 32) {                                  // exclusive scan, 4 lists per lane
    int v[4], sum = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int l = 4 * t + e;
      v[e] = l < n ? sc.off[l] : 0;
      sum += v[e];
    }
    int inc = sum;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, inc, d);
      if (t >= d) inc += o;
    }
    int o = inc - sum;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int l = 4 * t + e;
      if (l < n) sc.off[l] = o;
      o += v[e];
    }
    if (t == 31) sc.total = inc;
  }
  __syncthreads();
  const int C = sc.total;
  if (C > cap) return -1;
  const int lane = t & 31;
  for (int l = t >> 5; l < n; l += nt >> 5) {    // a warp per list, a lane per key
    const int o = sc.off[l], c = (l + 1 < n ? sc.off[l + 1] : C) - o;
    for (int e = lane; e < c; e += 32) buf[o + e] = s[(size_t)l * kHeadList + e];
  }
  __syncthreads();
  return C;
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
// the need-th largest key, from a kHistWords-bin histogram in global memory
// (bin i counts the keys whose leading bits are i): thread t of a
// kSelThreads-thread CTA reads bins 8t .. 8t + 7, and the suffix sums meet in
// two barriers.  0 when the histogram holds fewer than need keys.  Every
// thread calls it.
__device__ uint32_t hist_bound(const uint32_t* h, uint32_t need, uint32_t* s_wtot, uint32_t& s_bin) {
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const uint4 q0 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * t);
  const uint4 q1 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * t + 1);
  const uint32_t c[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
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

__device__ __forceinline__ uint32_t peer_addr(const void* local, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(a)
               : "r"((uint32_t)__cvta_generic_to_shared(local)), "r"(rank));
  return a;
}
__device__ __forceinline__ void st_peer_key(uint32_t a, hkey v) {
  asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(a), "l"(v) : "memory");
}
__device__ __forceinline__ void st_peer_u32(uint32_t a, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Every thread of every CTA of the cluster: stores before it are visible to
// loads after it.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// r of candidate row m for hidden state hb: lane l sums the 16-byte chunks
// l, l + 32, ... in ascending k with fmaf, then the 5-level butterfly; loads
// of up to 4 chunks are in flight together.
__device__ __forceinline__ float verify_row(const HeadParams& p, const float* hb, int m, int lane) {
  const int8_t* wr = p.W + (int64_t)m * p.ldw;
  const int nch = (p.K + 511) / 512;
  float acc = 0.f;
  for (int c0 = 0; c0 < nch; c0 += 4) {
    uint4 v[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int k = 16 * (lane + 32 * (c0 + t));
      if (c0 + t < nch && k < p.K) v[t] = ld_weights16(wr + k);
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int k = 16 * (lane + 32 * (c0 + t));
      if (c0 + t < nch && k < p.K) {
        float x[16];
        load_x16(hb, k, p.K, x);
        const uint32_t ww[4] = {v[t].x ^ 0x80808080u, v[t].y ^ 0x80808080u, v[t].z ^ 0x80808080u,
                                v[t].w ^ 0x80808080u};
#pragma unroll
        for (int e = 0; e < 16; ++e) acc = fmaf(byte_to_float(ww[e >> 2], (uint32_t)(e & 3)), x[e], acc);
      }
    }
  }
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, d);
  return __fmul_rn(__ldg(p.scale + m), acc);
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

  // 1. activation scale and INT8 codes of each hidden state (zero past K):
  // thread t holds h[4t + 1024 i .. +3] in registers (one read of h), the
  // CTA's maximum |h| meets in one barrier, every thread derives s_x
#pragma unroll 1
  for (int b = 0; b < B; ++b) {
    const float* hb = p.h + (int64_t)b * p.ldh;
    constexpr int kHv = SPIKE_PROJ_HEAD_MAX_K / (4 * kHeadThreads);
    float4 hv[kHv];
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < kHv; ++i) {
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
    for (int i = 0; i < kHv; ++i) {
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
    const int n8 = (p.nlists + kHeadCluster - 1) / kHeadCluster;
    const int64_t slot = (int64_t)(b * kHeadCluster + (int)blockIdx.x % kHeadCluster) * n8 +
                         (int)blockIdx.x / kHeadCluster;
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

// Steps 3-6: one cluster of kHeadCluster CTAs.  Per hidden state, CTA r
// merges the lists of projection CTAs r, r + 8, ... and pushes the result
// into CTA 0's s_part[r]; CTA 0 merges those, applies the gate and pushes the
// final list; warps 0-7 of each CTA recompute one candidate each and push r
// to CTA 0, which picks the token.  A bulk copy that does not complete
// within the bounded wait leaves the CTA's share empty and the call reports
// token -1 (no candidate of an incomplete list is ever read).
__global__ void __launch_bounds__(kSelThreads, 1)
head_select_kernel(const __grid_constant__ HeadParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  hkey* s_mine = reinterpret_cast<hkey*>(smem);            // [ceil(nlists / 8)][64]
  __shared__ hkey s_part[kHeadCluster][kHeadList];
  __shared__ hkey s_best[kHeadList];
  __shared__ hkey s_buf[kSelThreads];
  __shared__ GatherScratch s_gs;
  __shared__ uint32_t s_wtot[kSelWarps];
  __shared__ uint32_t s_bin;
  __shared__ hkey s_final[kHeadList];
  __shared__ float s_r[kHeadList];
  __shared__ uint32_t s_open, s_bad, s_ok;
  __shared__ float s_gap;
  __shared__ __align__(8) uint64_t s_bar;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t rank = cluster_rank();
  const int csize = kHeadCluster;
  const int ks = p.k_sel;
  const int n8 = (p.nlists + csize - 1) / csize;
  const int mine = p.nlists > (int)rank ? (p.nlists - (int)rank + csize - 1) / csize : 0;
  if (threadIdx.x == 0) {
    mbar_init(&s_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    s_bad = 0;
  }
  __syncthreads();
  pdl_launch_dependents();
  pdl_wait();                                    // every CTA list is written
  for (int b = 0; b < p.B; ++b) {
    uint32_t* hc = p.hist + (int64_t)b * kHistWords;
    if (threadIdx.x == 0 && mine > 0) {
      // the previous hidden state's reads and writes of s_mine (generic
      // proxy) come before this copy's writes (async proxy)
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      const uint32_t bytes = (uint32_t)mine * kHeadList * 8;
      mbar_arrive_expect_tx(&s_bar, bytes);
      bulk_load(s_mine, p.lists + (int64_t)(b * csize + (int)rank) * n8 * kHeadList, bytes, &s_bar);
    }
    // while the lists arrive, the bound T: the histogram bin holding the
    // 64th best listed key (every CTA finds it; no key of the final 64 lies
    // below T)
    const uint32_t tb = hist_bound(hc, kHeadList, s_wtot, s_bin);
    const hkey T = tb ? (hkey)tb << 32 : 1ull;   // no bound: every key passes
    if (threadIdx.x == 0 && mine > 0 && !mbar_wait(&s_bar, (uint32_t)(b & 1))) s_bad = 1;
    __syncthreads();
    const int have = s_bad ? 0 : mine;
    // this CTA's best 64 of its keys >= T (all of them, more than
    // kSelThreads only for adversarial spreads: then the merge tree)
    const int C = gather_ge(s_mine, have, T, s_buf, kSelThreads, s_gs);
    if (C >= 0) {
      rank_place(s_buf, C, s_best);
    } else {
      tree_merge(s_mine, have, kSelWarps);
      if (threadIdx.x < kHeadList) s_best[threadIdx.x] = s_mine[threadIdx.x];
      __syncthreads();
    }
    if (threadIdx.x < kHeadList) st_peer_key(peer_addr(&s_part[rank][threadIdx.x], 0u), s_best[threadIdx.x]);
    if (threadIdx.x == 0 && s_bad) st_peer_u32(peer_addr(&s_bad, 0u), 1u);
    cluster_sync();                              // the partial results in CTA 0
    if (rank == 0) {
      const int C0 = gather_ge(&s_part[0][0], csize, 1ull, s_buf, kSelThreads, s_gs);
      rank_place(s_buf, C0, s_best);             // C0 <= 8 * 64 = kSelThreads
      const hkey* fin = s_best;
      // The 64 best keys >= T are the 64 best keys when at least min(V, 64)
      // keys pass T, which holds whenever the histogram counted exactly this
      // call's listed keys; fewer (a histogram left dirty by a call that
      // never reached this kernel) or a failed copy: token -1 (the histogram
      // is cleared at the end either way).
      const bool ok = s_bad == 0 && C0 >= min(p.V, kHeadList);
      const float g = __fsub_rn(key_z(fin[0]), key_z(fin[1]));
      const uint32_t open = ok && g < p.tau ? 1u : 0u;
      if (threadIdx.x < kHeadList) {
        const hkey k = fin[threadIdx.x];
        for (int r = 0; r < csize; ++r) st_peer_key(peer_addr(&s_final[threadIdx.x], (uint32_t)r), k);
      }
      if (threadIdx.x == 0) {
        for (int r = 0; r < csize; ++r) st_peer_u32(peer_addr(&s_open, (uint32_t)r), open);
        s_ok = ok ? 1u : 0u;
        s_gap = g;
      }
    }
    // (global stores come after the cluster barriers: a barrier's release
    // would wait for them)
    cluster_sync();                              // s_final and s_open everywhere
    if (s_open && warp < kHeadWarps) {
      const float* hb = p.h + (int64_t)b * p.ldh;
      for (int i = (int)rank + csize * warp; i < ks; i += csize * kHeadWarps) {
        const float rv = verify_row(p, hb, key_row(s_final[i]), lane);
        if (lane == 0) st_peer_u32(peer_addr(&s_r[i], 0u), __float_as_uint(rv));
      }
    }
    cluster_sync();                              // every r in CTA 0
    if (rank == 0) {
      if (threadIdx.x == 0) {
        if (!s_open) p.token[b] = s_ok ? key_row(s_final[0]) : -1;
        if (p.verified) p.verified[b] = (int)s_open;
        if (p.gap) p.gap[b] = s_gap;
      }
      if (p.cand && (int)threadIdx.x < ks) p.cand[(int64_t)b * ks + threadIdx.x] = key_row(s_final[threadIdx.x]);
    }
    if (rank == 0 && s_open && warp == 0) {
      // largest r, equal r: lower row (starting from candidate 0, so the
      // token is always a candidate)
      float br = s_r[0];
      int bm = key_row(s_final[0]);
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int i = lane + 32 * t;
        if (i < ks) {
          const float rv = s_r[i];
          const int m = key_row(s_final[i]);
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
      if (lane == 0) p.token[b] = bm;
    }
    // Before the next hidden state rewrites s_mine (bulk copy), s_part,
    // s_best, s_final, s_open and s_r, every reader of them must be done:
    // one more barrier.
    if (b + 1 < p.B) cluster_sync();
  }
  // every CTA has read the histograms: CTA r clears bins 512 r .. 512 r + 511
  // of each hidden state's for the next call
  for (int b = 0; b < p.B; ++b)
    for (int i = threadIdx.x; i < kHistWords / kHeadCluster; i += kSelThreads)
      p.hist[(int64_t)b * kHistWords + (int)rank * (kHistWords / kHeadCluster) + i] = 0u;
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
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, head_kernel<B>, kHeadThreads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  // one wave: every CTA resident at once
  int grid = g_head_sms * per_sm;
  const int need = (p.units + kHeadWarps - 1) / kHeadWarps;
  if (grid > need) grid = need;
  if (grid > kHeadMaxGrid) grid = kHeadMaxGrid;
  if (grid < 1) grid = 1;
  p.nlists = grid;
  e = launch_pdl(head_kernel<B>, dim3((unsigned)grid), dim3(kHeadThreads), smem, s, p);
  if (e != cudaSuccess) return e;

  const size_t sel_smem = (size_t)((grid + kHeadCluster - 1) / kHeadCluster) * kHeadList * 8;
  e = raise_smem(head_select_kernel, sel_smem, g_select_smem);   // one kernel for every B
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kHeadCluster, 1, 1);
  cfg.blockDim = dim3(kSelThreads, 1, 1);
  cfg.dynamicSmemBytes = sel_smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kHeadCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, head_select_kernel, p);
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
