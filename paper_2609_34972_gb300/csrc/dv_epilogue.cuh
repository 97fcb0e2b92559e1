// Device helpers shared by the epilogues of the build kernels.
#pragma once
#include <cstdint>

#include "dv_internal.h"

namespace dv {

// Four 16-byte stores of 32 packed bf16 values.
__device__ __forceinline__ void store_row32(uint16_t* dst, const uint32_t (&pk)[16]) {
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  d[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
  d[2] = make_uint4(pk[8], pk[9], pk[10], pk[11]);
  d[3] = make_uint4(pk[12], pk[13], pk[14], pk[15]);
}

// Two 16-byte stores of 16 packed bf16 values.
__device__ __forceinline__ void store_row16(uint16_t* dst, const uint32_t (&pk)[8]) {
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  d[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
}

// sin and cos of the rotary angle pos * theta^(-2j/D_h). The product is kept as an
// unevaluated sum of two floats (fma residual, inverse frequency split in two floats), then
// reduced to [-pi, pi] by Cody-Waite subtraction of k * 2pi (2pi split in two floats) before
// the hardware sine/cosine, so the angle stays accurate to ~2e-7 rad at positions of a few
// thousand.
__device__ __forceinline__ void rope_sincos(float pos, float fhi, float flo, const EpiKV& kv,
                                            float& s, float& c) {
  const float a_hi = pos * fhi;
  const float a_lo = fmaf(pos, flo, fmaf(pos, fhi, -a_hi));
  const float k = rintf(a_hi * kv.inv_two_pi);
  float r = fmaf(-k, kv.two_pi_hi, a_hi);
  r = fmaf(-k, kv.two_pi_lo, r) + a_lo;
  __sincosf(r, &s, &c);
}

}  // namespace dv
