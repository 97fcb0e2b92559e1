// Persistent, warp-specialised 1-SM tcgen05 GEMM for the rank-r contractions of the
// visual-memory build, each with its own fused epilogue (the K/V contraction runs on CTA pairs,
// dv_kv2sm.cu / dv_pair_tm.cu):
//   EPI_SILU  H   = SiLU(x0 [D_1 ... D_L])          all L down-projections as one GEMM, since
//                                                    every layer reads only E (Sec. 3.1 Eq. 5)
//   EPI_NORM  rstd_l = (||M_l||^2 / d + eps)^-1/2    the RMS statistic of M_l = x0 + h_l U_l
//                                                    (Sec. 3.1 Eq. 4), from [x0 | h_l] times
//                                                    [2 U_l^T ; U_l U_l^T]
//   EPI_RESID M_l = M_{l-1} + h_l U_l                one step of the recurrent adapter
//                                                    (Sec. 3.1 Eq. 6), fp32 state in HBM
//
// CTA layout (192 threads, one CTA per SM):
//   warp 0      TMA producer: one lane streams 64-wide K slabs of A (128 token rows) and B
//               (BLOCK_N weight rows) into a ring of shared-memory stages
//   warp 1      owns the TMEM allocation; one lane issues tcgen05.mma (128 x BLOCK_N x 16)
//               into one of two TMEM accumulators
//   warps 2-5   epilogue: each thread owns one token row (TMEM lane) of the finished
//               accumulator, while the MMA warp fills the other accumulator
// Tiles are visited in (layer, n-block, m-block) order, m fastest, so the CTAs working at the
// same time share weight tiles through L2.
#include <cstdio>

#include "dv_epilogue.cuh"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {

constexpr int kNumThreads = 192;
constexpr int kEpiThreads = 128;
constexpr int kRingBytes = 192 * 1024;

template <int BN>
struct TileCfg {
  static constexpr int kABytes = kBlockM * kBlockK * 2;
  static constexpr int kBBytes = BN * kBlockK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStagesRaw = kRingBytes / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kEpiStageBytes = 4 * kWarpStageFloats * 4;  // one block per epilogue warp
  static constexpr int kSmemBytes = kStages * kStageBytes + kEpiStageBytes + 1024 + 256;
  static_assert(kStageBytes % 1024 == 0, "stage tiles must stay 1024-byte aligned");
  static_assert(kTmemCols >= 32 && kTmemCols <= 512 && (kTmemCols & (kTmemCols - 1)) == 0,
                "TMEM allocation must be a power of two in [32, 512]");
};

// Wait with a time limit only (used to drain in-flight work after an abort).
__device__ __forceinline__ bool wait_drain(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait(bar, parity, &never, timeout_ns);
}

// ------------------------------------------------------------------------------ epilogues

// EPI_SILU and EPI_NORM are shared with the pair engine (dv_epilogue.cuh); EPI_RESID, the
// recurrent step of the per-layer path, runs only here.

// The inverse of warp_store_f32, in two steps: warp_gather_f32 issues the loads of rows
// [0, rows) of src (row stride ld floats), a row segment per instruction (rows past `rows` read
// 0); warp_unstage_f32 then gives lane-row its 32 values through the warp's staging. Loads of
// the next block can be in flight while the current one is used.
__device__ __forceinline__ void warp_gather_f32(float4 (&g)[8], const float* src, long long ld,
                                                int rows) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int row = 4 * k + (lane >> 3), c4 = lane & 7;
    g[k] = row < rows ? reinterpret_cast<const float4*>(src + row * ld)[c4]
                      : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  }
}

__device__ __forceinline__ void warp_unstage_f32(float* stage, const float4 (&g)[8],
                                                 float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int row = 4 * k + (lane >> 3), c4 = lane & 7;
    reinterpret_cast<float4*>(stage + row * kWarpStagePitch)[c4] = g[k];
  }
  __syncwarp();
  const float4* srow = reinterpret_cast<const float4*>(stage + lane * kWarpStagePitch);
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 x = srow[q];
    v[4 * q] = x.x;
    v[4 * q + 1] = x.y;
    v[4 * q + 2] = x.z;
    v[4 * q + 3] = x.w;
  }
  __syncwarp();
}

// The same for a bf16 block, widened to fp32.
__device__ __forceinline__ void warp_load_bf16(float* stage, float (&v)[32], const uint16_t* src,
                                               long long ld, int rows) {
  const int lane = threadIdx.x & 31;
  uint32_t* st = reinterpret_cast<uint32_t*>(stage);
  constexpr int kPitch = 20;  // words per staged row (16 + 4 pad)
  uint4 g[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = 8 * k + (lane >> 2), c4 = lane & 3;
    g[k] = row < rows ? reinterpret_cast<const uint4*>(src + row * ld)[c4] : make_uint4(0, 0, 0, 0);
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = 8 * k + (lane >> 2), c4 = lane & 3;
    reinterpret_cast<uint4*>(st + row * kPitch)[c4] = g[k];
  }
  __syncwarp();
  const uint4* srow = reinterpret_cast<const uint4*>(st + lane * kPitch);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint4 w = srow[q];
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      v[q * 8 + 2 * u] = bf16_bits_to_float(ws[u] & 0xFFFFu);
      v[q * 8 + 2 * u + 1] = bf16_bits_to_float(ws[u] >> 16);
    }
  }
  __syncwarp();
}

// One step of the recurrent adapter (Sec. 3.1 Eq. 6) for token row t and columns
// [n*BN, (n+1)*BN): M = prev + h U^T with prev = x0 (first planned layer) or the fp32 state.
// Writes the new fp32 state, bf16(M) for the K/V GEMM (with the split chain also the bf16
// rounding of M - bf16(M), the low part the next down-projection reads), and the sum of M^2 over
// the tile. The state moves through the warp's staging a row segment per instruction (whole
// 128-byte lines), not a 16-byte piece per lane and row.
template <int BN>
__device__ __forceinline__ void epi_resid(const GemmParams& p, uint32_t tbase, int n, int t,
                                          float* stage) {
  const EpiResid& e = p.resid;
  const int lane = threadIdx.x & 31;
  const int t0 = t - lane;             // the warp's first row
  const int rows = p.s.M - t0;         // rows of the warp's block inside the build (may be <= 0)
  const size_t base = static_cast<size_t>(t0) * e.d + static_cast<size_t>(n) * BN;
  float ss = 0.0f;
  // the next two chunks of the fp32 state, loading while this chunk is used
  float4 g[2][8];
  if (!e.first) {
    warp_gather_f32(g[0], e.state + base, e.d, rows);
    if (BN / 32 > 1) warp_gather_f32(g[1], e.state + base + 32, e.d, rows);
  }
#pragma unroll 2
  for (int c = 0; c < BN / 32; ++c) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld32(tbase + c * 32, r);  // in flight while the previous M loads
    float mv[32];
    if (e.first) {
      warp_load_bf16(stage, mv, e.x0 + base + c * 32, e.d, rows);
    } else {
      warp_unstage_f32(stage, g[c & 1], mv);
      if (c + 2 < BN / 32) warp_gather_f32(g[c & 1], e.state + base + (c + 2) * 32, e.d, rows);
    }
    tmem_ld_wait();
    // the accumulator registers are used only past the wait (the empty statement redefines them)
    asm volatile(""
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                   "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                   "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                   "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                   "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                   "+r"(r[30]), "+r"(r[31]));
    uint32_t vb[32], pk[16];
#pragma unroll
    for (int u = 0; u < 32; ++u) {
      const float v = mv[u] + __uint_as_float(r[u]);
      ss = fmaf(v, v, ss);
      vb[u] = __float_as_uint(v);
    }
#pragma unroll
    for (int u = 0; u < 16; ++u)
      pk[u] = pack_bf16x2(__uint_as_float(vb[2 * u]), __uint_as_float(vb[2 * u + 1]));
    warp_store_f32(stage, vb, e.state + base + c * 32, e.d, rows);
    warp_store_bf16(stage, pk, e.mem + base + c * 32, e.d, rows);
    if (e.mem_lo) {  // split chain: the remainder M - bf16(M), rounded to bf16
      uint32_t lo[16];
#pragma unroll
      for (int u = 0; u < 16; ++u)
        lo[u] = pack_bf16x2(__uint_as_float(vb[2 * u]) - __uint_as_float(pk[u] << 16),
                            __uint_as_float(vb[2 * u + 1]) - __uint_as_float(pk[u] & 0xFFFF0000u));
      warp_store_bf16(stage, lo, e.mem_lo + base + c * 32, e.d, rows);
    }
  }
  if (t < p.s.M) e.part[static_cast<size_t>(n) * p.s.M + t] = ss;
}


// ------------------------------------------------------------------------------ the kernel

template <int EPI, int BN, int HD>
__global__ void __launch_bounds__(kNumThreads, 1)
    dv_gemm_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                   const __grid_constant__ CUtensorMap tmB, const __grid_constant__ GemmParams p) {
  using C = TileCfg<BN>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  uint8_t* ring_ptr = smem_raw + (ring - raw);
  float* epi_stage = reinterpret_cast<float*>(ring_ptr + S * C::kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring_ptr + S * C::kStageBytes + C::kEpiStageBytes);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * S + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * S + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t tmo = p.timeout_ns;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), kEpiThreads);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    if (p.s.k1_slabs > 0) tma_prefetch_desc(&tmA1);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  const int m_tiles = (p.s.M + kBlockM - 1) / kBlockM;
  const int n_tiles = p.s.n_per_layer / BN;
  const int num_tiles = m_tiles * n_tiles * p.s.n_layers;
  const int k_slabs = p.s.k0_slabs + p.s.k1_slabs;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      int stage = 0;
      uint32_t phase = 0, used = 0, issued_parity = 0;
      for (int tile = blockIdx.x; tile < num_tiles && !*abort_flag; tile += gridDim.x) {
        const int m = tile % m_tiles;
        const int rest = tile / m_tiles;
        const int n = rest % n_tiles;
        const int l = p.s.layer0 + rest / n_tiles;
        const int brow = l * p.s.n_per_layer + n * BN;
        const int arow = l * p.s.a0_rows_per_layer + m * kBlockM;
        for (int ks = 0; ks < k_slabs; ++ks) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, tmo)) break;
          const uint32_t a_dst = ring + stage * C::kStageBytes;
          const uint32_t b_dst = a_dst + C::kABytes;
          mbar_arrive_expect_tx(full_bar(stage), C::kStageBytes);
          if (ks < p.s.k0_slabs) {
            tma_load_2d(a_dst, &tmA0, full_bar(stage), ks * kBlockK, arow);
          } else {
            tma_load_2d(a_dst, &tmA1, full_bar(stage),
                        l * p.s.a1_cols_per_layer + (ks - p.s.k0_slabs) * kBlockK, m * kBlockM);
          }
          tma_load_2d(b_dst, &tmB, full_bar(stage), ks * kBlockK, brow);
          used |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*abort_flag) {  // let every copy still in flight land before the CTA exits
        for (int s = 0; s < S; ++s)
          if (used & (1u << s)) wait_drain(full_bar(s), (issued_parity >> s) & 1u, tmo);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      const uint32_t idesc = idesc_bf16_f32(kBlockM, BN);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool issued_any = false;
      for (int tile = blockIdx.x; tile < num_tiles && !*abort_flag; tile += gridDim.x) {
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, tmo)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        bool ok = true;
        for (int ks = 0; ks < k_slabs; ++ks) {
          if (!mbar_wait(full_bar(stage), phase, abort_flag, tmo)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = ring + stage * C::kStageBytes;
          const uint32_t b_s = a_s + C::kABytes;
#pragma unroll
          for (int k = 0; k < kBlockK / 16; ++k) {
            umma_bf16(d_tmem, sdesc_kmajor_sw128(a_s + 32u * k), sdesc_kmajor_sw128(b_s + 32u * k),
                      idesc, (ks | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(empty_bar(stage));
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(tfull_bar(acc));
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (*abort_flag && issued_any) {  // no TMEM release while an MMA may still run
        umma_commit(drain_bar);
        wait_drain(drain_bar, 0, tmo);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue warps
    const int q = warp & 3;  // the TMEM lane quarter this warp may access
    const int row = q * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      const int m = tile % m_tiles;
      const int rest = tile / m_tiles;
      const int n = rest % n_tiles;
      const int l = p.s.layer0 + rest / n_tiles;
      // the warp leaves together (its lanes meet in __syncwarp and the TMEM loads below)
      if (!__all_sync(0xFFFFFFFFu, mbar_wait(tfull_bar(acc), acc_phase, abort_flag, tmo))) break;
      tc_fence_after();
      const uint32_t tbase =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      const int t = m * kBlockM + row;
      if constexpr (EPI == EPI_SILU) {
        epi_silu<BN>(p, tbase, n, t, epi_stage + q * kWarpStageFloats);
      } else if constexpr (EPI == EPI_NORM) {
        epi_norm<BN>(p, tbase, l, t);
      } else {
        epi_resid<BN>(p, tbase, n, t, epi_stage + q * kWarpStageFloats);
      }
      tc_fence_before();
      mbar_arrive(tempty_bar(acc));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, 6 /* DV_ERR_DEVICE_TIMEOUT */);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::kTmemCols);
  }
}

// ------------------------------------------------------------------------------ launch

template <int EPI, int BN, int HD>
static cudaError_t launch_t(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                            const GemmParams& p, int num_sms, cudaStream_t stream) {
  using C = TileCfg<BN>;
  auto kern = dv_gemm_kernel<EPI, BN, HD>;
  cudaError_t err =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess) return err;
  const long long m_tiles = (p.s.M + kBlockM - 1) / kBlockM;
  const long long tiles = m_tiles * (p.s.n_per_layer / BN) * p.s.n_layers;
  if (tiles <= 0) return cudaSuccess;
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(kNumThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, kern, a0, a1, b, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

int gemm_smem_bytes(int block_n) {
  switch (block_n) {
    case 64: return TileCfg<64>::kSmemBytes;
    case 128: return TileCfg<128>::kSmemBytes;
    case 256: return TileCfg<256>::kSmemBytes;
    default: return -1;
  }
}

cudaError_t launch_gemm(int epi, int block_n, int head_dim, const CUtensorMap& a0,
                        const CUtensorMap& a1, const CUtensorMap& b, const GemmParams& p,
                        int num_sms, cudaStream_t stream) {
  if (epi == EPI_SILU) {
    if (block_n == 64) return launch_t<EPI_SILU, 64, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 128) return launch_t<EPI_SILU, 128, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 256) return launch_t<EPI_SILU, 256, 0>(a0, a1, b, p, num_sms, stream);
  } else if (epi == EPI_NORM) {
    if (block_n == 64) return launch_t<EPI_NORM, 64, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 128) return launch_t<EPI_NORM, 128, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 256) return launch_t<EPI_NORM, 256, 0>(a0, a1, b, p, num_sms, stream);
  } else if (epi == EPI_RESID) {
    if (block_n == 64) return launch_t<EPI_RESID, 64, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 128) return launch_t<EPI_RESID, 128, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 256) return launch_t<EPI_RESID, 256, 0>(a0, a1, b, p, num_sms, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace dv
