// 2-SM tcgen05 GEMM with the tokens as the M operand, used for all three contractions of the
// build when the token count is (close to) a multiple of 256:
//   EPI_SILU  H = SiLU(x0 [D_1 ... D_L])                  (Sec. 3.1 Eqs. 4-5)
//   EPI_NORM  rstd_l from [x0 | h_l] [2 U_l^T ; G_l]      (RMSNorm of M_l, Sec. 3.2 Eq. 7)
//   EPI_KV    K/V = rstd_l * ([x0 | h_l] Wkv_l^T) + b, RoPE on K, cache store (Sec. 3.2 Eq. 7)
//
// One CTA pair computes a 256 x BN tile: 256 tokens (128 in each CTA's TMEM lanes) times BN
// weight rows, of which each CTA stages half. With BN = 256 both operands of a CTA are 128 rows
// per 64-wide K slab, the balance at which the shared-memory traffic of the 2-SM MMA matches its
// tensor throughput. Each epilogue thread owns one token row of its CTA's accumulator, so RoPE
// pairs and head rows are in registers and go straight to 16-byte stores.
//
// Roles as in the other kernels: warp 0 lane 0 loads (both CTAs, two K slabs per pipeline
// step as one 3-D box per operand, completion counted on the leader's full barrier whose single
// expect_tx covers both CTAs), warp 1 owns TMEM and, in the leader, issues the MMAs with
// multicast commits, warps 2-5 drain the accumulator.
//
// Tile order: the tiles form a grid of token blocks (m) x weight tiles (w = layer * n_tiles +
// n). It is walked in super-blocks of group_m token blocks x group_w weight tiles (token block
// fastest inside), columns of super-blocks one after the other, so that the operands the
// running pairs touch fit in L2 together and each is read from DRAM a few times, not once per
// tile of the other operand.
#include "dv_epilogue.cuh"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {

constexpr int kTmThreads = 192;
constexpr int kTmSmemLimit = 232448;

template <int BN>
struct TmCfg {
  static constexpr int kASlab = 128 * kBlockK * 2;         // one K slab of 128 token rows
  static constexpr int kBSlab = (BN / 2) * kBlockK * 2;    // one K slab of BN / 2 weight rows
  static constexpr int kABytes = kSlabsPerStep * kASlab;
  static constexpr int kBBytes = kSlabsPerStep * kBSlab;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kEpiStageBytes = 4 * kWarpStageFloats * 4;  // one block per epilogue warp
  static constexpr int kStagesRaw = (kTmSmemLimit - kEpiStageBytes - 1024 - 512) / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kSmemBytes = kStages * kStageBytes + kEpiStageBytes + 1024 + 512;
  static constexpr int kTmemCols = 2 * BN < 32 ? 32 : 2 * BN;
  static_assert(BN == 64 || BN == 128 || BN == 256, "N tile");
  static_assert(kASlab % 1024 == 0 && kBSlab % 1024 == 0, "slab tiles must stay 1024-byte aligned");
  static_assert(kStages >= 2, "pipeline depth");
  static_assert((kTmemCols & (kTmemCols - 1)) == 0 && kTmemCols <= 512, "TMEM allocation");
};

// (m, w) of tile t in the super-blocked order described above.
__device__ __forceinline__ void tm_tile(int t, int m_blocks, int w_tiles, int gm, int gw, int& m,
                                        int& w) {
  const int sbw = t / (gw * m_blocks);  // every column before the last one is gw wide
  const int r = t - sbw * gw * m_blocks;
  const int gw_eff = min(gw, w_tiles - sbw * gw);
  const int sbm = r / (gm * gw_eff);
  const int r2 = r - sbm * gm * gw_eff;
  const int gm_eff = min(gm, m_blocks - sbm * gm);
  m = sbm * gm + r2 % gm_eff;
  w = sbw * gw + r2 / gm_eff;
}

template <int EPI, int BN, int HD>
__global__ void __launch_bounds__(kTmThreads, 1)
    dv_pair_tm_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                      const __grid_constant__ CUtensorMap tmB, const __grid_constant__ GemmParams p) {
  using C = TmCfg<BN>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  uint8_t* ring_ptr = smem_raw + (ring - raw);
  float* epi_stage = reinterpret_cast<float*>(ring_ptr + S * C::kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring_ptr + S * C::kStageBytes + C::kEpiStageBytes);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };                   // leader
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };            // both
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * S + a); };        // both
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * S + 2 + a); };   // leader
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint64_t tmo = p.timeout_ns;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 2 * 4);  // one lane of each epilogue warp of both CTAs
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
    tmem_alloc_pair(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // The K/V epilogue waits for the kernel before it (the RMS statistic) in its epilogue warps
  // only: its producer reads x0 or M, H and the weights, which every kernel before the statistic
  // has finished writing once this grid can start (each trigger follows its kernel's own wait).
  // The down-projection and the statistic wait here, before any access.
  if (EPI != EPI_KV) pdl_wait();
  pdl_trigger();

  const int m_tiles = (p.s.M + 255) / 256;
  const int n_tiles = p.s.n_per_layer / BN;
  const int w_tiles = n_tiles * p.s.n_layers;
  const int num_tiles = m_tiles * w_tiles;
  const int gm = p.s.group_m > 0 ? min(p.s.group_m, m_tiles) : m_tiles;
  const int gw = p.s.group_w > 0 ? min(p.s.group_w, w_tiles) : 1;
  const int k0 = p.s.k0_slabs, k1 = p.s.k1_slabs;
  const int n_steps = k_steps(k0, k1);
  const int pair = static_cast<int>(cluster_id_x());
  const int num_pairs = static_cast<int>(num_clusters_x());

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      const uint32_t leader_full0 = map_to_rank(full_bar(0), 0);
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = pair; tile < num_tiles && !*abort_flag; tile += num_pairs) {
        int m, w;
        tm_tile(tile, m_tiles, w_tiles, gm, gw, m, w);
        const int n = w % n_tiles;
        const int l = w / n_tiles;
        const int arow = m * 256 + static_cast<int>(rank) * 128;
        const int a0row = l * p.s.a0_rows_per_layer + arow;
        const int brow = l * p.s.n_per_layer + n * BN + static_cast<int>(rank) * (BN / 2);
        for (int j = 0; j < n_steps; ++j) {
          const KStep ks = k_step(j, k0, k1);
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, tmo)) break;
          const uint32_t a_dst = ring + stage * C::kStageBytes;
          const uint32_t b_dst = a_dst + C::kABytes;
          const uint32_t fb = leader_full0 + 8u * stage;
          if (rank == 0) mbar_arrive_expect_tx(full_bar(stage), 2 * C::kStageBytes);
          if (ks.seg == 0) {
            tma_load_3d_pair(a_dst, &tmA0, fb, a0row, ks.slab);
          } else {
            tma_load_3d_pair(a_dst, &tmA1, fb, arow,
                             l * (p.s.a1_cols_per_layer / kBlockK) + ks.slab);
          }
          tma_load_3d_pair(b_dst, &tmB, fb, brow, ks.seg == 0 ? ks.slab : k0 + ks.slab);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------------------------------------------------------- MMA issuer (leader)
      const uint32_t idesc = idesc_bf16_f32(256, BN);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool issued_any = false;
      for (int tile = pair; tile < num_tiles && !*abort_flag; tile += num_pairs) {
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, tmo)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        bool ok = true;
        for (int j = 0; j < n_steps; ++j) {
          const int n_used = k_step(j, k0, k1).n;
          if (!mbar_wait(full_bar(stage), phase, abort_flag, tmo)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = ring + stage * C::kStageBytes;
          const uint32_t b_s = a_s + C::kABytes;
#pragma unroll
          for (int sl = 0; sl < kSlabsPerStep; ++sl) {
            if (sl < n_used) {
#pragma unroll
              for (int k = 0; k < kBlockK / 16; ++k) {
                umma_bf16_pair(d_tmem, sdesc_kmajor_sw128(a_s + sl * C::kASlab + 32u * k),
                               sdesc_kmajor_sw128(b_s + sl * C::kBSlab + 32u * k), idesc,
                               (j | sl | k) != 0 ? 1u : 0u);
              }
            }
          }
          issued_any = true;
          umma_commit_pair(empty_bar(stage), 0x3);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair(tfull_bar(acc), 0x3);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (*abort_flag && issued_any) {  // no teardown while an MMA may still run
        umma_commit_pair(drain_bar, 0x1);
        int never = 0;
        mbar_wait(drain_bar, 0, &never, tmo);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue warps
    if (EPI == EPI_KV) pdl_wait();  // rstd and the cache are touched only after this
    const int q = warp & 3;  // TMEM lane quarter of this warp
    const uint32_t leader_tempty0 = map_to_rank(tempty_bar(0), 0);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = pair; tile < num_tiles; tile += num_pairs) {
      int m, w;
      tm_tile(tile, m_tiles, w_tiles, gm, gw, m, w);
      const int n = w % n_tiles;
      const int l = w / n_tiles;
      // the warp leaves together (its lanes meet in __syncwarp and the TMEM loads below)
      if (!__all_sync(0xFFFFFFFFu, mbar_wait(tfull_bar(acc), acc_phase, abort_flag, tmo))) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t tbase =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      const int t = m * 256 + static_cast<int>(rank) * 128 + q * 32 + lane;
      if constexpr (EPI == EPI_SILU) {
        epi_silu<BN>(p, tbase, n, t, epi_stage + q * kWarpStageFloats);
      } else if constexpr (EPI == EPI_NORM) {
        epi_norm<BN>(p, tbase, l, t);
      } else {
        epi_kv_group<HD>(p, tbase, l, n, t);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(leader_tempty0 + 8u * acc);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    // Let this CTA's own copies still in flight land before the pair is torn down.
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 200000ull) {
    }
    atomicExch(p.status, 6 /* DV_ERR_DEVICE_TIMEOUT */);
  }
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::kTmemCols);
  }
}

template <int EPI, int BN, int HD>
static cudaError_t launch_tm_t(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                               const GemmParams& p, int num_sms, cudaStream_t stream) {
  using C = TmCfg<BN>;
  auto kern = dv_pair_tm_kernel<EPI, BN, HD>;
  cudaError_t err =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess) return err;
  const long long tiles =
      static_cast<long long>((p.s.M + 255) / 256) * (p.s.n_per_layer / BN) * p.s.n_layers;
  if (tiles <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kTmThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int max_clusters = 0;
  cfg.gridDim = dim3(2 * (num_sms / 2), 1, 1);
  if (cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg) != cudaSuccess || max_clusters < 1) {
    cudaGetLastError();
    max_clusters = num_sms / 2;
  }
  const long long pairs = tiles < max_clusters ? tiles : max_clusters;
  cfg.gridDim = dim3(static_cast<unsigned>(2 * pairs), 1, 1);
  attr[1] = pdl_attribute();
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, kern, a0, a1, b, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_pair_tm(int epi, int block_n, int head_dim, const CUtensorMap& a0,
                           const CUtensorMap& a1, const CUtensorMap& b, const GemmParams& p,
                           int num_sms, cudaStream_t stream) {
  if (epi == EPI_SILU) {
    if (block_n == 64) return launch_tm_t<EPI_SILU, 64, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 128) return launch_tm_t<EPI_SILU, 128, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 256) return launch_tm_t<EPI_SILU, 256, 0>(a0, a1, b, p, num_sms, stream);
  } else if (epi == EPI_NORM) {
    if (block_n == 64) return launch_tm_t<EPI_NORM, 64, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 128) return launch_tm_t<EPI_NORM, 128, 0>(a0, a1, b, p, num_sms, stream);
    if (block_n == 256) return launch_tm_t<EPI_NORM, 256, 0>(a0, a1, b, p, num_sms, stream);
  } else if (epi == EPI_KV && block_n == 256) {
    if (head_dim == 64) return launch_tm_t<EPI_KV, 256, 64>(a0, a1, b, p, num_sms, stream);
    if (head_dim == 128) return launch_tm_t<EPI_KV, 256, 128>(a0, a1, b, p, num_sms, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace dv
