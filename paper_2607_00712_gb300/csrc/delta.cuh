// The bf16 pair that carries Delta = A_full - A_loc into the least-squares sums (Sec. 3.2):
// hi = bf16(Delta), lo = bf16(Delta - hi), so hi + lo equals Delta to about 2^-16 relative.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace ispa {

// Eight bf16 features of A_loc (a) and A_full (f).  Delta = f - a is exact in fp32 (both
// operands bf16, within 2^16 of each other in magnitude) and both halves round to nearest even.
__device__ __forceinline__ void split_delta8(const uint4 a, const uint4 f, uint4& hi, uint4& lo) {
  const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, fw[4] = {f.x, f.y, f.z, f.w};
  uint32_t hw[4], lw[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float d0 = __uint_as_float(fw[e] << 16) - __uint_as_float(aw[e] << 16);
    const float d1 = __uint_as_float(fw[e] & 0xFFFF0000u) - __uint_as_float(aw[e] & 0xFFFF0000u);
    __nv_bfloat162 h = __floats2bfloat162_rn(d0, d1);
    const uint32_t hb = *reinterpret_cast<uint32_t*>(&h);
    __nv_bfloat162 l = __floats2bfloat162_rn(d0 - __uint_as_float(hb << 16), d1 - __uint_as_float(hb & 0xFFFF0000u));
    hw[e] = hb;
    lw[e] = *reinterpret_cast<uint32_t*>(&l);
  }
  hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

}  // namespace ispa
