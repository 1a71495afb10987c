// sp_rows.cuh -- device helpers of the continuous-input (row-major) kernels:
// exact INT8 -> FP32 conversion and 16-float activation loads.
#pragma once

#include <stdint.h>

namespace sp {

// float(int8 byte e of w), exact: with w_biased = w ^ 0x80808080 each byte is
// w + 128, placed in the low mantissa byte of 2^23 and 2^23 + 128 subtracted.
__device__ __forceinline__ float byte_to_float(uint32_t w_biased, uint32_t e_sel) {
  return __int_as_float((int)__byte_perm(w_biased, 0x4B000000u, 0x7650u | e_sel)) - 8388736.0f;
}

// x[k .. k+15] of one activation row, zero at and past K (xr 16-byte aligned
// and k % 16 == 0 for the vector path).
__device__ __forceinline__ void load_x16(const float* __restrict__ xr, int k, int K, float (&v)[16]) {
  if (k + 16 <= K) {
    const float4* p = reinterpret_cast<const float4*>(xr + k);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldg(p + q);
      v[4 * q] = f.x;
      v[4 * q + 1] = f.y;
      v[4 * q + 2] = f.z;
      v[4 * q + 3] = f.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = (k + e < K) ? __ldg(xr + k + e) : 0.f;
  }
}

}  // namespace sp
