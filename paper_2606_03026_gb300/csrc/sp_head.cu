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
constexpr int kHistWords = 256 + 65536;       // coarse and fine histograms of one hidden state
constexpr int kHeadMaxGrid = 1024;            // projection CTAs (lists) of one call
static_assert(kHeadList == 64, "a list is two keys per lane");
static_assert(kHeadList == kHeadCluster * kHeadWarps, "one candidate per warp of a cluster");

typedef unsigned long long hkey;

// Workspace: the CTA lists (projection CTA c's list of hidden state b is
// list (b * 8 + c % 8) * ceil(nlists / 8) + c / 8), then per hidden state
// the histograms of the listed keys' order bits: 256 coarse bins (bits
// 31-24) and 65536 fine bins (bits 31-16), zero between calls.
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
// shared memory; a prefix of each, found by binary search) into buf and
// returns their number, or -1 (nothing copied) when more than cap pass.
// n <= kHeadGatherLists; every thread of the CTA calls it.
__device__ int gather_ge(const hkey* s, int n, hkey T, hkey* buf, int cap, GatherScratch& sc) {
  const int t = threadIdx.x, nt = blockDim.x;
  for (int l = t; l < n; l += nt) {
    const hkey* L = s + (size_t)l * kHeadList;
    int lo = 0, hi = kHeadList;                  // first index with key < T
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (L[mid] >= T) lo = mid + 1; else hi = mid;
    }
    sc.off[l] = lo;
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

// Over a 256-bin histogram h in global memory (bin i counts the keys whose
// leading bits are i, so higher bins hold larger keys): the bin holding the
// need-th largest key and the number of keys in the bins above it; false
// when h holds fewer than need keys.  The 8 counts of lane l's bins
// 8l .. 8l + 7 are left in c.  One full warp calls it.
__device__ bool find_bin(const uint32_t* h, uint32_t need, int lane, uint32_t (&c)[8],
                         uint32_t& bin, uint32_t& above) {
  const uint4 q0 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * lane);
  const uint4 q1 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * lane + 1);
  c[0] = q0.x; c[1] = q0.y; c[2] = q0.z; c[3] = q0.w;
  c[4] = q1.x; c[5] = q1.y; c[6] = q1.z; c[7] = q1.w;
  uint32_t sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) sum += c[i];
  uint32_t S = sum;                              // keys in the bins of lanes >= this one
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t o = __shfl_down_sync(0xffffffffu, S, d);
    if (lane + d < 32) S += o;
  }
  const uint32_t hit = __ballot_sync(0xffffffffu, S >= need);
  if (hit == 0u) return false;
  const int L = 31 - __clz(hit);                 // the highest lane reaching need
  uint32_t cum = __shfl_sync(0xffffffffu, S - sum, L);
  bool found = false;
#pragma unroll
  for (int i = 7; i >= 0; --i) {
    const uint32_t ci = __shfl_sync(0xffffffffu, c[i], L);
    if (!found && cum + ci >= need) {
      bin = (uint32_t)(8 * L + i);
      above = cum;
      found = true;
    }
    cum += ci;
  }
  return true;
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

  // 1. activation scale and INT8 codes of each hidden state (zero past K)
#pragma unroll
  for (int b = 0; b < B; ++b) {
    const float* hb = p.h + (int64_t)b * p.ldh;
    float mx = 0.f;
    for (int k = threadIdx.x; k < p.K; k += kHeadThreads) mx = fmaxf(mx, fabsf(hb[k]));
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, d));
    if (lane == 0) s_red[warp] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
      float a = s_red[0];
      for (int w = 1; w < kHeadWarps; ++w) a = fmaxf(a, s_red[w]);
      s_sx[b] = __fdiv_rn(fmaxf(a, 1e-8f), 127.0f);
    }
    __syncthreads();
    const float sx = s_sx[b];
    for (int k = threadIdx.x; k < p.Kpad; k += kHeadThreads) {
      int c = 0;
      if (k < p.K) c = (int)fminf(fmaxf(rintf(__fdiv_rn(hb[k], sx)), -127.0f), 127.0f);
      s_codes[b * p.Kpad + k] = (int8_t)c;
    }
  }
  __syncthreads();

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
      // the listed keys into the histograms (equal bins of a warp summed
      // first): every key of the final selection is a listed key
      const uint32_t real = __ballot_sync(0xffffffffu, k != 0ull);
      if (k != 0ull) {
        uint32_t* hc = p.hist + (int64_t)b * kHistWords;
        const uint32_t ob = (uint32_t)(k >> 32);
        const uint32_t mf = __match_any_sync(real, ob >> 16);
        if (lane == __ffs(mf) - 1) atomicAdd(hc + 256 + (ob >> 16), (uint32_t)__popc(mf));
        const uint32_t mc = __match_any_sync(real, ob >> 24);
        if (lane == __ffs(mc) - 1) atomicAdd(hc + (ob >> 24), (uint32_t)__popc(mc));
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
  __shared__ uint32_t s_coarse[256];
  __shared__ hkey s_T;
  __shared__ hkey s_final[kHeadList];
  __shared__ float s_r[kHeadList];
  __shared__ uint32_t s_open, s_bad, s_dirty;
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
    if (warp == 1) {
      // the bound T: the fine bin holding the 64th best listed key (every
      // CTA finds it; no key of the final 64 lies below T)
      uint32_t c[8], cb = 0, above = 0;
      hkey T = 1ull;                             // fewer than 64 keys: all pass
      if (find_bin(hc, kHeadList, lane, c, cb, above)) {
        uint32_t cf[8], fb = 0, above2 = 0;
        if (find_bin(hc + 256 + cb * 256, kHeadList - above, lane, cf, fb, above2))
          T = (hkey)((cb << 24) | (fb << 16)) << 32;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) s_coarse[8 * lane + i] = c[i];
      if (lane == 0) s_T = T;
    }
    if (threadIdx.x == 0 && mine > 0) {
      // the previous hidden state's reads and writes of s_mine (generic
      // proxy) come before this copy's writes (async proxy)
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      const uint32_t bytes = (uint32_t)mine * kHeadList * 8;
      mbar_arrive_expect_tx(&s_bar, bytes);
      bulk_load(s_mine, p.lists + (int64_t)(b * csize + (int)rank) * n8 * kHeadList, bytes, &s_bar);
      if (!mbar_wait(&s_bar, (uint32_t)(b & 1))) s_bad = 1;
    }
    __syncthreads();
    const int have = s_bad ? 0 : mine;
    // this CTA's best 64 of its keys >= T (all of them, more than
    // kSelThreads only for adversarial spreads: then the merge tree)
    const int C = gather_ge(s_mine, have, s_T, s_buf, kSelThreads, s_gs);
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
      // keys pass T, which holds whenever the histograms counted exactly
      // this call's listed keys; fewer (histograms left dirty by a call that
      // never reached this kernel) or a failed copy: token -1, and every bin
      // is cleared below.
      const bool ok = s_bad == 0 && C0 >= min(p.V, kHeadList);
      const float g = __fsub_rn(key_z(fin[0]), key_z(fin[1]));
      const uint32_t open = ok && g < p.tau ? 1u : 0u;
      if (threadIdx.x < kHeadList) {
        const hkey k = fin[threadIdx.x];
        for (int r = 0; r < csize; ++r) st_peer_key(peer_addr(&s_final[threadIdx.x], (uint32_t)r), k);
      }
      if (threadIdx.x == 0) {
        for (int r = 0; r < csize; ++r) {
          st_peer_u32(peer_addr(&s_open, (uint32_t)r), open);
          st_peer_u32(peer_addr(&s_dirty, (uint32_t)r), ok ? 0u : 1u);
        }
        p.token[b] = ok ? key_row(fin[0]) : -1;  // replaced below when verified
        if (p.verified) p.verified[b] = (int)open;
        if (p.gap) p.gap[b] = g;
      }
      if (p.cand && (int)threadIdx.x < ks) p.cand[(int64_t)b * ks + threadIdx.x] = key_row(fin[threadIdx.x]);
    }
    cluster_sync();                              // s_final, s_open and s_dirty everywhere
    // every CTA has read the histograms: clear the fine bins of the coarse
    // bins r, r + 8, ... that counted keys (all of them after a failed
    // check), and CTA 0 the coarse bins, for the next call
    for (int i = threadIdx.x; i < (256 / kHeadCluster) * 256; i += kSelThreads) {
      const int cbin = (int)rank + kHeadCluster * (i >> 8);
      if (s_coarse[cbin] || s_dirty) hc[256 + cbin * 256 + (i & 255)] = 0u;
    }
    if (rank == 0 && threadIdx.x < 256) hc[threadIdx.x] = 0u;
    if (s_open && warp < kHeadWarps) {
      const float* hb = p.h + (int64_t)b * p.ldh;
      for (int i = (int)rank + csize * warp; i < ks; i += csize * kHeadWarps) {
        const float rv = verify_row(p, hb, key_row(s_final[i]), lane);
        if (lane == 0) st_peer_u32(peer_addr(&s_r[i], 0u), __float_as_uint(rv));
      }
    }
    cluster_sync();                              // every r in CTA 0
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
