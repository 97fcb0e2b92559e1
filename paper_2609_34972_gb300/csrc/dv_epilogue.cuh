// Device helpers shared by the epilogues of the build kernels.
#pragma once
#include <cstdint>

#include "dv_internal.h"
#include "dv_ptx.cuh"

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

// H[t, n*BN + c] = bf16(SiLU(z)), SiLU(z) = z / (1 + e^-z)  (phi of Sec. 3.1 Eq. 4).
template <int BN>
__device__ __forceinline__ void epi_silu(const GemmParams& p, uint32_t tbase, int n, int t) {
  const bool valid = t < p.s.M;
  uint16_t* out = p.silu.H + static_cast<size_t>(valid ? t : 0) * p.silu.ldh +
                  static_cast<size_t>(n) * BN;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + c * 32, r);
    tmem_ld_wait();
    uint32_t pk[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const float z0 = __uint_as_float(r[2 * u]), z1 = __uint_as_float(r[2 * u + 1]);
      pk[u] = pack_bf16x2(z0 / (1.0f + __expf(-z0)), z1 / (1.0f + __expf(-z1)));
    }
    if (valid) store_row32(out + c * 32, pk);
  }
}

// ||m||^2 = ||x0||^2 + h . (2 x0 U^T + h G) with G = U U^T, so with acc = [x0 | h] [2U^T; G]
// the statistic of RMSNorm is rstd = 1 / sqrt((xx + h . acc) / d + eps).
template <int BN>
__device__ __forceinline__ void epi_norm(const GemmParams& p, uint32_t tbase, int l, int t) {
  const bool valid = t < p.s.M;
  const uint16_t* hrow = p.norm.H + static_cast<size_t>(valid ? t : 0) * p.norm.ldh +
                         static_cast<size_t>(l) * p.norm.r_pad;
  float dot = 0.0f;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + c * 32, r);
    tmem_ld_wait();
    if (valid) {
      const uint4* hv = reinterpret_cast<const uint4*>(hrow + c * 32);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 w = hv[q];
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          dot = fmaf(bf16_bits_to_float(ws[e] & 0xFFFFu), __uint_as_float(r[q * 8 + 2 * e]), dot);
          dot = fmaf(bf16_bits_to_float(ws[e] >> 16), __uint_as_float(r[q * 8 + 2 * e + 1]), dot);
        }
      }
    }
  }
  if (valid) {
    const float ss = fmaxf(p.norm.xx[t] + dot, 0.0f);
    p.norm.rstd[static_cast<size_t>(l) * p.norm.ld_rstd + t] =
        rsqrtf(fmaf(ss, p.norm.inv_d, p.norm.eps));
  }
}


// Row-per-thread K/V epilogue for an accumulator whose 256 columns are one 128-channel group
// of layer l: columns [0, 128) the K channels of the group (128 / HD heads), [128, 256) the
// same V channels (the Wkv packing). Thread = token t. k = rstd * acc + b_K rotated in
// rotate-half pairs (j, j + HD/2) of each head; v = rstd * acc + b_V.
template <int HD>
__device__ __forceinline__ void epi_kv_group(const GemmParams& p, uint32_t tbase, int l, int g,
                                             int t) {
  constexpr int kHalf = HD / 2;
  constexpr int kHeads = 128 / HD;
  const EpiKV& e = p.kv;
  const bool valid = t < p.s.M;
  const int tt = valid ? t : 0;
  const int b = tt / e.n_vis, i = tt - b * e.n_vis;
  const float rs = valid ? e.rstd[static_cast<size_t>(l) * e.ld_rstd + tt] : 0.0f;
  const int slot = e.slot ? e.slot[tt] : e.slot0 + i;
  const long long row0 = l * e.s_layer + b * e.s_batch + slot * e.s_seq;
  const int* pp = e.pos + static_cast<size_t>(b) * e.n_pos * e.n_vis + i;
  const float pt = static_cast<float>(pp[0]);
  const float ph = e.n_pos == 3 ? static_cast<float>(pp[e.n_vis]) : pt;
  const float pw = e.n_pos == 3 ? static_cast<float>(pp[2 * e.n_vis]) : pt;
  const float* bk = e.bk ? e.bk + static_cast<size_t>(l) * e.kv + g * 128 : nullptr;
  const float* bv = e.bv ? e.bv + static_cast<size_t>(l) * e.kv + g * 128 : nullptr;

#pragma unroll 1
  for (int c = 0; c < 128 / 64; ++c) {  // 2 blocks of 32 pairs: (head, first or second 32 j)
    const int hl = (c * 32) / kHalf, jb = (c * 32) % kHalf;
    const int col = hl * HD + jb;
    uint32_t lo[32], hi[32];
    __syncwarp();
    tmem_ld32(tbase + col, lo);
    tmem_ld32(tbase + col + kHalf, hi);
    tmem_ld_wait();
    uint32_t plo[16], phi[16];
#pragma unroll
    for (int u = 0; u < 32; u += 2) {
      float y1[2], y2[2];
#pragma unroll
      for (int w = 0; w < 2; ++w) {
        const int j = jb + u + w;
        float x1 = __uint_as_float(lo[u + w]) * rs;
        float x2 = __uint_as_float(hi[u + w]) * rs;
        if (bk) {
          x1 += bk[col + u + w];
          x2 += bk[col + kHalf + u + w];
        }
        const float pj = j < e.sec0 ? pt : (j < e.sec01 ? ph : pw);
        float s, cs;
        rope_sincos(pj, e.inv_freq_hi[j], e.inv_freq_lo[j], e, s, cs);
        y1[w] = x1 * cs - x2 * s;
        y2[w] = x2 * cs + x1 * s;
      }
      plo[u / 2] = pack_bf16x2(y1[0], y1[1]);
      phi[u / 2] = pack_bf16x2(y2[0], y2[1]);
    }
    if (valid) {
      uint16_t* krow = e.kc + row0 + static_cast<long long>(g * kHeads + hl) * e.s_head;
      store_row32(krow + jb, plo);
      store_row32(krow + kHalf + jb, phi);
    }
  }
#pragma unroll 1
  for (int c = 0; c < 4; ++c) {  // V: 4 blocks of 32 channels
    const int hl = (c * 32) / HD, jv = (c * 32) % HD;
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + 128 + c * 32, r);
    tmem_ld_wait();
    uint32_t pk[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      float v0 = __uint_as_float(r[2 * u]) * rs, v1 = __uint_as_float(r[2 * u + 1]) * rs;
      if (bv) {
        v0 += bv[c * 32 + 2 * u];
        v1 += bv[c * 32 + 2 * u + 1];
      }
      pk[u] = pack_bf16x2(v0, v1);
    }
    if (valid) {
      uint16_t* vrow = e.vc + row0 + static_cast<long long>(g * kHeads + hl) * e.s_head;
      store_row32(vrow + jv, pk);
    }
  }
}

}  // namespace dv
