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

// A warp's 32 x 32 block of an output in global memory: lane i holds row i. Stored through the
// warp's shared staging (kWarpStageFloats floats) so that each store instruction writes whole
// row segments (8 lanes x 16 bytes per fp32 row, 4 lanes per bf16 row) instead of 32 scattered
// 16-byte pieces: one L2 request per 128-byte line, not one per lane.
constexpr int kWarpStagePitch = 36;                      // floats per staged row (32 + 4 pad)
constexpr int kWarpStageFloats = 32 * kWarpStagePitch;   // 4608 bytes per warp

// fp32: rows [row0, row0 + rows) of dst (row stride ld floats) get lane-row's 32 values.
__device__ __forceinline__ void warp_store_f32(float* stage, const uint32_t (&r)[32], float* dst,
                                               long long ld, int rows) {
  const int lane = threadIdx.x & 31;
  float4* srow = reinterpret_cast<float4*>(stage + lane * kWarpStagePitch);
#pragma unroll
  for (int q = 0; q < 8; ++q)
    srow[q] = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                          __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
  __syncwarp();
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int row = 4 * k + (lane >> 3), c4 = lane & 7;
    const float4 v = reinterpret_cast<const float4*>(stage + row * kWarpStagePitch)[c4];
    if (row < rows) reinterpret_cast<float4*>(dst + row * ld)[c4] = v;
  }
  __syncwarp();
}

// bf16: rows [0, rows) of dst (row stride ld elements) get lane-row's 32 packed values.
__device__ __forceinline__ void warp_store_bf16(float* stage, const uint32_t (&pk)[16],
                                                uint16_t* dst, long long ld, int rows) {
  const int lane = threadIdx.x & 31;
  uint32_t* st = reinterpret_cast<uint32_t*>(stage);
  constexpr int kPitch = 20;  // words per staged row (16 + 4 pad)
  uint4* srow = reinterpret_cast<uint4*>(st + lane * kPitch);
#pragma unroll
  for (int q = 0; q < 4; ++q) srow[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
  __syncwarp();
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = 8 * k + (lane >> 2), c4 = lane & 3;
    const uint4 v = reinterpret_cast<const uint4*>(st + row * kPitch)[c4];
    if (row < rows) reinterpret_cast<uint4*>(dst + row * ld)[c4] = v;
  }
  __syncwarp();
}

// In-register transpose of a warp's 32 x 32 block: on entry lane i holds row i (r[j] = M[i][j]),
// on exit lane i holds column i (r[j] = M[j][i]). Five butterfly rounds: in the round of bit b,
// registers j and j + b (j without bit b) of lanes i and i ^ b swap the two off-diagonal
// b x b sub-blocks, one shuffle per register pair.
__device__ __forceinline__ void warp_transpose32(uint32_t (&r)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int b = 16; b >= 1; b >>= 1) {
    const bool upper = (lane & b) != 0;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      if (j & b) continue;
      const uint32_t send = upper ? r[j] : r[j + b];
      const uint32_t recv = __shfl_xor_sync(0xFFFFFFFFu, send, b);
      if (upper) r[j] = recv;
      else r[j + b] = recv;
    }
  }
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

// H[t, n*BN + c] = bf16(SiLU(z)) (phi of Sec. 3.1 Eq. 4); tiles past
// the down-projection columns store the raw fp32 product into C instead (the launch picks BN
// dividing n_h, so no tile straddles the two). t: this lane's token row; the warp's rows are
// t - lane .. t - lane + 31, written through the warp's staging `wstage`.
template <int BN>
__device__ __forceinline__ void epi_silu(const GemmParams& p, uint32_t tbase, int n, int t,
                                         float* wstage) {
  const int row0 = t - (threadIdx.x & 31);
  const int rows = p.s.M - row0;  // valid rows of this warp's block (may be <= 0)
  const int col0 = n * BN;
  if (col0 >= p.silu.n_h) {
    float* c0 = p.silu.C + static_cast<size_t>(rows > 0 ? row0 : 0) * p.silu.ldc + (col0 - p.silu.n_h);
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld32(tbase + c * 32, r);
      tmem_ld_wait();
      warp_store_f32(wstage, r, c0 + c * 32, p.silu.ldc, rows);
    }
    return;
  }
  uint16_t* h0 = p.silu.H + static_cast<size_t>(rows > 0 ? row0 : 0) * p.silu.ldh +
                 static_cast<size_t>(col0);
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
      pk[u] = pack_bf16x2(silu(z0), silu(z1));
    }
    warp_store_bf16(wstage, pk, h0 + c * 32, p.silu.ldh, rows);
  }
}

// ||m||^2 = ||x0||^2 + h . (2 x0 U^T + h G) with G = U U^T, so with acc = [x0 | h] [2U^T; G]
// the statistic of RMSNorm is rstd = 1 / sqrt((xx + h . acc) / d + eps). A tile of group l
// holds the lpt layers l * lpt + j in columns [j rn, j rn + r_pad) (the B operand's G blocks
// are block-diagonal against [h_{l lpt} | h_{l lpt + 1} | ...]); columns past r_pad within a
// layer's rn are zero rows and skipped.
template <int BN>
__device__ __forceinline__ void epi_norm(const GemmParams& p, uint32_t tbase, int l, int t) {
  const EpiNorm& e = p.norm;
  const bool valid = t < p.s.M;
  const uint16_t* hrow = e.H + static_cast<size_t>(valid ? t : 0) * e.ldh;
  float dot = 0.0f;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    const int j = (c * 32) / e.rn, n0 = (c * 32) % e.rn;
    const int layer = l * e.lpt + j;
    if (layer >= e.n_layers || n0 >= e.r_pad) continue;  // uniform over the warp
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + c * 32, r);
    tmem_ld_wait();
    if (valid) {
      const uint4* hv = reinterpret_cast<const uint4*>(hrow + static_cast<size_t>(layer) * e.r_pad + n0);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 w = hv[q];
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          dot = fmaf(bf16_bits_to_float(ws[u] & 0xFFFFu), __uint_as_float(r[q * 8 + 2 * u]), dot);
          dot = fmaf(bf16_bits_to_float(ws[u] >> 16), __uint_as_float(r[q * 8 + 2 * u + 1]), dot);
        }
      }
      if (n0 + 32 == e.r_pad) {  // the layer's last columns: its statistic is complete
        const float ss = fmaxf(e.xx[t] + dot, 0.0f);
        e.rstd[static_cast<size_t>(layer) * e.ld_rstd + t] = rsqrtf(fmaf(ss, e.inv_d, e.eps));
        dot = 0.0f;
      }
    }
  }
}

// Per-token context of the K/V store: cache row base, positions, rstd of one token.
struct KvToken {
  bool valid;
  long long row0;  // element offset of (layer, batch, slot) in the cache
  float rs, pt, ph, pw;
};

__device__ __forceinline__ KvToken kv_token(const GemmParams& p, int l, int t) {
  const EpiKV& e = p.kv;
  KvToken k;
  k.valid = t < p.s.M;
  const int tt = k.valid ? t : 0;
  const int b = tt / e.n_vis, i = tt - b * e.n_vis;
  k.rs = k.valid ? e.rstd[static_cast<size_t>(l) * e.ld_rstd + tt] : 0.0f;
  const int slot = e.slot ? e.slot[tt] : e.slot0 + i;
  k.row0 = static_cast<long long>(p.layer_map[l]) * e.s_layer + b * e.s_batch + slot * e.s_seq;
  const int* pp = e.pos + static_cast<size_t>(b) * e.n_pos * e.n_vis + i;
  k.pt = static_cast<float>(pp[0]);
  k.ph = e.n_pos == 3 ? static_cast<float>(pp[e.n_vis]) : k.pt;
  k.pw = e.n_pos == 3 ? static_cast<float>(pp[2 * e.n_vis]) : k.pt;
  return k;
}

// K values of block q (0..3) of a 128-channel group for one token: r[m] and r[16 + m]
// (m < 16) are the accumulators of rotate-half pair p = 16q + m (Wkv K-row permutation); the
// key channels are x1 = rstd * r[m] + b_K (channel j of head hl) and x2 = rstd * r[16 + m] + b_K
// (channel j + HD/2), j = (16q + m) mod HD/2.
template <int HD>
__device__ __forceinline__ void k_pair_values(const GemmParams& p, const KvToken& tk, int l,
                                              int g, int q, const uint32_t (&r)[32], int m,
                                              float& x1, float& x2) {
  constexpr int kHalf = HD / 2;
  const EpiKV& e = p.kv;
  const int hl = (16 * q) / kHalf, j0 = (16 * q) % kHalf;
  x1 = __uint_as_float(r[m]) * tk.rs;
  x2 = __uint_as_float(r[16 + m]) * tk.rs;
  if (e.bk) {
    const float* bk = e.bk + static_cast<size_t>(l) * e.kv + g * 128 + hl * HD + j0;
    x1 += bk[m];
    x2 += bk[kHalf + m];
  }
}

// Sum of squares of the 32 key channels of block q (the head's share for its K norm).
template <int HD>
__device__ __forceinline__ float kv_k16_sumsq(const GemmParams& p, const KvToken& tk, int l, int g,
                                              int q, const uint32_t (&r)[32]) {
  float ss = 0.0f;
#pragma unroll
  for (int m = 0; m < 16; ++m) {
    float x1, x2;
    k_pair_values<HD>(p, tk, l, g, q, r, m, x1, x2);
    ss = fmaf(x1, x1, ss);
    ss = fmaf(x2, x2, ss);
  }
  return ss;
}

// K block q (0..3) of a 128-channel group for one token: k = rstd * acc + b_K (k_pair_values),
// with the per-head K norm when enabled (kinv = 1 / sqrt(mean(k_h^2) + eps) of this head, times
// the gain of each channel), rotated, and written as two 32-byte runs of the head row.
template <int HD>
__device__ __forceinline__ void kv_store_k16(const GemmParams& p, const KvToken& tk, int l, int g,
                                             int q, const uint32_t (&r)[32], float kinv) {
  constexpr int kHalf = HD / 2;
  const EpiKV& e = p.kv;
  const int hl = (16 * q) / kHalf, j0 = (16 * q) % kHalf;
  const float* kg = e.kg ? e.kg + static_cast<size_t>(l) * HD : nullptr;
  uint32_t plo[8], phi[8];
#pragma unroll
  for (int m = 0; m < 16; m += 2) {
    float y1[2], y2[2];
#pragma unroll
    for (int w = 0; w < 2; ++w) {
      const int j = j0 + m + w;
      float x1, x2;
      k_pair_values<HD>(p, tk, l, g, q, r, m + w, x1, x2);
      if (kg) {
        x1 *= kinv * kg[j];
        x2 *= kinv * kg[kHalf + j];
      }
      const int ax = e.axis[j];
      const float pj = ax == 0 ? tk.pt : (ax == 1 ? tk.ph : tk.pw);
      float s, cs;
      rope_sincos(pj, e.inv_freq_hi[j], e.inv_freq_lo[j], e, s, cs);
      y1[w] = x1 * cs - x2 * s;
      y2[w] = x2 * cs + x1 * s;
    }
    plo[m / 2] = pack_bf16x2(y1[0], y1[1]);
    phi[m / 2] = pack_bf16x2(y2[0], y2[1]);
  }
  if (tk.valid) {
    uint16_t* krow = e.kc + tk.row0 + static_cast<long long>(g * (128 / HD) + hl) * e.s_head;
    store_row16(krow + j0, plo);
    store_row16(krow + kHalf + j0, phi);
  }
}

// V block q (0..3) of a 128-channel group for one token: r[u] is channel 32q + u.
template <int HD>
__device__ __forceinline__ void kv_store_v32(const GemmParams& p, const KvToken& tk, int l, int g,
                                             int q, const uint32_t (&r)[32]) {
  const EpiKV& e = p.kv;
  const int hl = (32 * q) / HD, jv = (32 * q) % HD;
  const float* bv = e.bv ? e.bv + static_cast<size_t>(l) * e.kv + g * 128 + 32 * q : nullptr;
  uint32_t pk[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) {
    float v0 = __uint_as_float(r[2 * u]) * tk.rs, v1 = __uint_as_float(r[2 * u + 1]) * tk.rs;
    if (bv) {
      v0 += bv[2 * u];
      v1 += bv[2 * u + 1];
    }
    pk[u] = pack_bf16x2(v0, v1);
  }
  if (tk.valid) {
    uint16_t* vrow = e.vc + tk.row0 + static_cast<long long>(g * (128 / HD) + hl) * e.s_head;
    store_row32(vrow + jv, pk);
  }
}

// Row-per-thread K/V epilogue (tokens as M): the thread's token row has 256 accumulator
// columns, the 128 K rows of group g (permuted, see kv_store_k16) then its 128 V rows.
template <int HD>
__device__ __forceinline__ void epi_kv_group(const GemmParams& p, uint32_t tbase, int l, int g,
                                             int t) {
  const KvToken tk = kv_token(p, l, t);
  // Per-head K norm: a first pass over the K blocks sums each head's squares (one head per
  // group for HD = 128, blocks {0, 1} and {2, 3} for HD = 64).
  float kinv0 = 1.0f, kinv1 = 1.0f;  // heads of blocks {0, 1} and {2, 3} (the same for HD = 128)
  if (p.kv.kg) {
    float ss0 = 0.0f, ss1 = 0.0f;
#pragma unroll 1
    for (int q = 0; q < 4; ++q) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld32(tbase + 32 * q, r);
      tmem_ld_wait();
      const float part = kv_k16_sumsq<HD>(p, tk, l, g, q, r);
      if (HD == 128 || q < 2) ss0 += part;
      else ss1 += part;
    }
    kinv0 = rsqrtf(fmaf(ss0, 1.0f / HD, p.kv.k_eps));
    kinv1 = HD == 128 ? kinv0 : rsqrtf(fmaf(ss1, 1.0f / HD, p.kv.k_eps));
  }
#pragma unroll 1
  for (int q = 0; q < 4; ++q) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + 32 * q, r);
    tmem_ld_wait();
    kv_store_k16<HD>(p, tk, l, g, q, r, (HD == 128 || q < 2) ? kinv0 : kinv1);
  }
#pragma unroll 1
  for (int q = 0; q < 4; ++q) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + 128 + 32 * q, r);
    tmem_ld_wait();
    kv_store_v32<HD>(p, tk, l, g, q, r);
  }
}

}  // namespace dv
