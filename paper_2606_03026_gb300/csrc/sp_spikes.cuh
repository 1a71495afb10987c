// sp_spikes.cuh -- device helpers shared by the gather and union kernels:
// reading spike rows as 32-column words, compacting words into the ascending
// active-column list (Section 2.2: the active indices are collected first), and
// the byte-lane accumulation of INT8 columns.
#pragma once

#include "sp_internal.h"

namespace sp {

// --- spike words -------------------------------------------------------------

// Four u8 spikes (one per byte of v) -> the same four bytes as 0 / 1.
__device__ __forceinline__ uint32_t nonzero_bytes_to_01(uint32_t v) {
  v |= v >> 4;          // fold each byte onto its low bit; bits that leak in
  v |= v >> 2;          // from the next byte land above bit 3 of the byte and
  v |= v >> 1;          // are masked off below
  return v & 0x01010101u;
}
// Four u8 spikes (one per byte of v) -> four bits, byte b -> bit b.
__device__ __forceinline__ uint32_t nonzero_bytes_to_bits(uint32_t v) {
  return (nonzero_bytes_to_01(v) * 0x01020408u) >> 24;   // bit 0 of bytes 0..3 -> bits 0..3
}

// Word of the spike row covering columns [kw, kw + 32), bits at or past K
// cleared.  `row` points at the row's first element.  kw % 32 == 0.
__device__ __forceinline__ uint32_t spike_word(const void* row, int fmt, int K, int kw) {
  if (kw >= K) return 0u;
  uint32_t w;
  const int rem = K - kw;
  if (fmt == SP_SPIKES_BITS32) {
    w = __ldg(reinterpret_cast<const uint32_t*>(row) + (kw >> 5));
  } else {
    const uint8_t* x = reinterpret_cast<const uint8_t*>(row) + kw;
    w = 0u;
    if (rem >= 32 && (reinterpret_cast<uintptr_t>(x) & 3u) == 0) {
      uint32_t v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = __ldg(reinterpret_cast<const uint32_t*>(x) + i);
#pragma unroll
      for (int i = 0; i < 8; ++i) w |= nonzero_bytes_to_bits(v[i]) << (4 * i);
    } else {
      const int n = rem < 32 ? rem : 32;
      for (int i = 0; i < n; ++i) w |= (uint32_t)(__ldg(x + i) != 0) << i;
    }
  }
  if (rem < 32) w &= (1u << rem) - 1u;
  return w;
}

__device__ __forceinline__ const void* spike_row(const void* base, int fmt, int64_t row,
                                                  int64_t ld) {
  return fmt == SP_SPIKES_BITS32
             ? static_cast<const void*>(reinterpret_cast<const uint32_t*>(base) + row * ld)
             : static_cast<const void*>(reinterpret_cast<const uint8_t*>(base) + row * ld);
}

// Warp-cooperative compaction of nw <= 32 words into ascending column
// indices base_k + 32*i + bit.  Call with the whole warp; returns |list| to
// every lane.
__device__ __forceinline__ int compact_words(const uint32_t* words, int nw, int base_k,
                                             int* list) {
  const int lane = threadIdx.x & 31;
  uint32_t w = lane < nw ? words[lane] : 0u;
  const int c = __popc(w);
  int incl = c;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += v;
  }
  int off = incl - c;
  const int k = base_k + lane * 32;
  while (w) {
    list[off++] = k + __ffs(w) - 1;
    w &= w - 1u;
  }
  return __shfl_sync(0xffffffffu, incl, 31);
}

// --- byte-lane accumulation ----------------------------------------------------
// A 32-bit word holds four INT8 weights of four consecutive output channels.
// XOR with 0x80 maps q in [-128, 127] to q + 128 in [0, 255]; PRMT spreads
// bytes 0,2 and 1,3 into the 16-bit halves of two registers.  A 16-bit lane
// then holds sum(q) + 128 * n exactly while n <= 257 columns (255 * 257 <
// 2^16) -- the exact lower-width partial sum of Section 2.3 -- and
// unbias16() recovers the INT32 sum.
__device__ __forceinline__ void acc_bytes(uint32_t w, uint32_t& even, uint32_t& odd) {
  const uint32_t t = w ^ 0x80808080u;
  even += __byte_perm(t, 0u, 0x4240);   // bytes 0, 2 -> halves 0, 1
  odd += __byte_perm(t, 0u, 0x4341);    // bytes 1, 3 -> halves 0, 1
}

// Channels 4i+0..3 of the word whose lanes are (even, odd), after n columns.
__device__ __forceinline__ void unbias16(uint32_t even, uint32_t odd, int n, int out[4]) {
  const int bias = 128 * n;
  out[0] = (int)(even & 0xffffu) - bias;
  out[1] = (int)(odd & 0xffffu) - bias;
  out[2] = (int)(even >> 16) - bias;
  out[3] = (int)(odd >> 16) - bias;
}

// Streaming 16-byte load of weights: read once, keep out of L1.
__device__ __forceinline__ uint4 ld_weights16(const int8_t* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// y = s * float(acc): exact conversion (|acc| < 2^24), one RN multiply.
__device__ __forceinline__ float scale_out(float s, int acc) {
  return __fmul_rn(s, __int2float_rn(acc));
}

}  // namespace sp
