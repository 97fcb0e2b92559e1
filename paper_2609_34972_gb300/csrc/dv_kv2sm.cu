// K/V projection, RoPE and KV-cache store (Sec. 3.2 Eq. 7) as a 2-SM tcgen05 GEMM.
//
//   [K_l | V_l]^T = Wkv_l [x0 | h_l]^T,  then rstd_l * (.) + b, RoPE on K, bf16 into the cache
//
// The weights are the M operand and the tokens the N operand ("swap AB"), so the token count
// only has to be a multiple of the N tile (64..256 in steps of 64), not of 128 or 256 rows.
// One CTA pair (cluster of 2) computes a 256 x NT tile: 256 weight rows = the 128 K channels
// of a 128-channel group (leader CTA, TMEM lanes 0..127) and the same 128 V channels (peer
// CTA), times NT tokens. Each CTA stages only its own half of both operands (128 weight rows,
// NT/2 token rows), which halves the shared-memory traffic per MMA against a 1-SM tile.
//
// CTA roles (192 threads, one CTA per SM, both CTAs of a pair alike):
//   warp 0      TMA producer for this CTA's halves, two K slabs per pipeline step (one 3-D
//               box per operand: a TMA instruction has a fixed cost, and two-slab boxes let one
//               SM's copies keep pace with the MMA); completion is counted on the leader's full
//               barrier (cta_group::2 TMA), whose single expect_tx arrival (leader) announces
//               the bytes of both CTAs
//   warp 1      TMEM owner (cta_group::2 alloc in both CTAs); in the leader one lane issues the
//               256 x NT x 16 MMAs and multicasts its commits to both CTAs
//   warps 2-5   epilogue over this CTA's 128 weight rows: TMEM -> registers (lane = weight
//               row, 32 tokens), an in-register 32 x 32 transpose by xor-shuffles (lane = token,
//               the warp's 32 weight rows), then 16 complete RoPE pairs of K (the Wkv K rows are
//               permuted so that partners are 16 rows apart) or 32 channels of V per lane, as
//               32-byte runs. The transpose needs no shared memory, which leaves room for a
//               fourth two-slab pipeline step (the weights stream from HBM and need the depth);
//               only the per-head K norm exchanges one float per warp and token.
// Pair tiles run in (layer, group, token block) order, token block fastest, so the pairs
// running together share each weight tile through L2.
#include "dv_epilogue.cuh"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {

constexpr int kPairThreads = 192;
constexpr int kEpiPairThreads = 128;
constexpr int kSmemLimit = 232448;  // largest dynamic shared memory of one CTA on sm_103

template <int NT>
struct PairCfg {
  static constexpr int kHalfN = NT / 2;
  static constexpr int kASlab = 128 * kBlockK * 2;     // one K slab of this CTA's weight rows
  static constexpr int kBSlab = kHalfN * kBlockK * 2;  // one K slab of its token rows
  static constexpr int kABytes = kSlabsPerStep * kASlab;
  static constexpr int kBBytes = kSlabsPerStep * kBSlab;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kKnormBytes = 2 * 32 * 4 * 4;  // K-norm partial sums [2][token][warp]
  static constexpr int kRingBudget = kSmemLimit - kKnormBytes - 1024 - 512;
  static constexpr int kStagesRaw = kRingBudget / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kSmemBytes = kStages * kStageBytes + kKnormBytes + 1024 + 512;
  static constexpr int kTmemCols = 512;
  static_assert(NT % 64 == 0 && NT >= 64 && NT <= 256, "N tile");
  static_assert(kASlab % 1024 == 0 && kBSlab % 1024 == 0, "slab tiles must stay 1024-byte aligned");
  static_assert(kStages >= 2, "pipeline depth");
  static_assert(2 * NT <= kTmemCols, "two accumulators must fit in TMEM");
  static_assert(kSmemBytes <= kSmemLimit, "shared memory");
};

__device__ __forceinline__ bool wait_local_only(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait(bar, parity, &never, timeout_ns);
}

template <int HD, int NT>
__global__ void __launch_bounds__(kPairThreads, 1)
    dv_kv_pair_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                      const __grid_constant__ CUtensorMap tmH, const __grid_constant__ GemmParams p) {
  using C = PairCfg<NT>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  uint8_t* ring_ptr = smem_raw + (ring - raw);
  float* knorm_pad = reinterpret_cast<float*>(ring_ptr + S * C::kStageBytes);  // K-norm partials
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring_ptr + S * C::kStageBytes + C::kKnormBytes);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };            // used in the leader
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };     // both CTAs
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * S + a); };  // both CTAs
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * S + 2 + a); };  // leader
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint64_t tmo = p.timeout_ns;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);     // the leader's expect_tx covers the bytes of both CTAs
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 2 * kEpiPairThreads / 32);  // one lane per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    if (p.s.k1_slabs > 0) tma_prefetch_desc(&tmH);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialised, TMEM allocated in both
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Only the epilogue warps wait for the kernel before this one (the RMS statistic): the
  // producer and MMA warps read x0, H and the weights, which every kernel before the statistic
  // has finished writing once this grid can start (each trigger follows its kernel's own wait),
  // so the first tiles' loads and MMAs overlap the statistic's tail. rstd and the cache are
  // touched only after the epilogue's wait.
  pdl_trigger();

  const int tok_tiles = (p.s.M + NT - 1) / NT;
  const int groups = p.kv.kv / 128;
  const int num_tiles = tok_tiles * groups * p.s.n_layers;
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
        const int nt = tile % tok_tiles;
        const int rest = tile / tok_tiles;
        const int g = rest % groups;
        const int l = rest / groups;
        const int wrow = l * p.s.n_per_layer + g * 256 + static_cast<int>(rank) * 128;
        const int trow = nt * NT + static_cast<int>(rank) * C::kHalfN;
        const int xrow = l * p.s.a0_rows_per_layer + trow;
        for (int j = 0; j < n_steps; ++j) {
          const KStep ks = k_step(j, k0, k1);
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, tmo)) break;
          const uint32_t a_dst = ring + stage * C::kStageBytes;
          const uint32_t b_dst = a_dst + C::kABytes;
          const uint32_t fb = leader_full0 + 8u * stage;
          // Only the leader arrives (local, CTA scope) and announces both CTAs' bytes (whole
          // boxes, zero fill included); the peer's copies may complete on the barrier first
          // (the transaction count is signed).
          if (rank == 0) mbar_arrive_expect_tx(full_bar(stage), 2 * C::kStageBytes);
          tma_load_3d_pair(a_dst, &tmW, fb, wrow, ks.seg == 0 ? ks.slab : k0 + ks.slab);
          if (ks.seg == 0) {
            tma_load_3d_pair(b_dst, &tmX, fb, xrow, ks.slab);
          } else {
            tma_load_3d_pair(b_dst, &tmH, fb, trow,
                             l * (p.s.a1_cols_per_layer / kBlockK) + ks.slab);
          }
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
      const uint32_t idesc = idesc_bf16_f32(256, NT);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool issued_any = false;
      for (int tile = pair; tile < num_tiles && !*abort_flag; tile += num_pairs) {
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, tmo)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * NT);
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
        wait_local_only(drain_bar, 0, tmo);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue warps
    pdl_wait();
    const int q = warp & 3;  // TMEM lane quarter = block of 32 weight rows of this warp
    const uint32_t leader_tempty0 = map_to_rank(tempty_bar(0), 0);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = pair; tile < num_tiles; tile += num_pairs) {
      const int nt = tile % tok_tiles;
      const int rest = tile / tok_tiles;
      const int g = rest % groups;
      const int l = rest / groups;
      // All 128 epilogue threads take the same branch: they meet at named barriers below.
      const bool ready = named_barrier_and(
          1, kEpiPairThreads, mbar_wait(tfull_bar(acc), acc_phase, abort_flag, tmo));
      if (!ready) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                             static_cast<uint32_t>(acc * NT);
#pragma unroll 1
      for (int c = 0; c < NT / 32; ++c) {
        uint32_t r[32];
        __syncwarp();
        tmem_ld32(tbase + c * 32, r);  // lane i: weight row 32q + i, 32 tokens
        tmem_ld_wait();
        warp_transpose32(r);           // lane i: token 32c + i, weight rows 32q .. 32q + 31
        const KvToken tk = kv_token(p, l, nt * NT + c * 32 + lane);
        if (rank == 0) {
          float kinv = 1.0f;
          if (p.kv.kg) {
            // Per-head K norm: a head spans warps (4 blocks of 32 channels for HD = 128,
            // 2 for HD = 64). Each warp leaves its block's sum of squares for the token of each
            // lane; the head's blocks are summed in block order. Two buffers by chunk parity:
            // a warp rewrites one only after every warp has passed the next chunk's barrier.
            float* pad = knorm_pad + ((c & 1) * 32 + lane) * 4;
            pad[q] = kv_k16_sumsq<HD>(p, tk, l, g, q, r);
            named_barrier(1, kEpiPairThreads);
            const float ss = HD == 128 ? ((pad[0] + pad[1]) + pad[2]) + pad[3]
                                       : (q < 2 ? pad[0] + pad[1] : pad[2] + pad[3]);
            kinv = rsqrtf(fmaf(ss, 1.0f / HD, p.kv.k_eps));
          }
          kv_store_k16<HD>(p, tk, l, g, q, r, kinv);
        } else {
          kv_store_v32<HD>(p, tk, l, g, q, r);
        }
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
  cluster_sync();  // neither CTA leaves while its peer may still touch its memory
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::kTmemCols);
  }
}

// ------------------------------------------------------------------------------ launch

template <int HD, int NT>
static cudaError_t launch_pair_t(const CUtensorMap& w, const CUtensorMap& x, const CUtensorMap& h,
                                 const GemmParams& p, int num_sms, cudaStream_t stream) {
  using C = PairCfg<NT>;
  auto kern = dv_kv_pair_kernel<HD, NT>;
  cudaError_t err =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess) return err;
  const long long tiles = static_cast<long long>((p.s.M + NT - 1) / NT) * (p.kv.kv / 128) * p.s.n_layers;
  if (tiles <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kPairThreads, 1, 1);
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
  err = cudaLaunchKernelEx(&cfg, kern, w, x, h, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

int kv_pair_tile_n(long long tokens) {
  // Fewest padded tokens; per-tile fixed cost counted as 16 tokens; larger tiles win ties.
  const int cands[4] = {256, 192, 128, 64};
  int best = 256;
  long long best_cost = -1;
  for (int nt : cands) {
    const long long tiles = (tokens + nt - 1) / nt;
    const long long cost = tiles * (nt + 16);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = nt;
    }
  }
  return best;
}

int kv_pair_smem_bytes(int nt) {
  switch (nt) {
    case 64: return PairCfg<64>::kSmemBytes;
    case 128: return PairCfg<128>::kSmemBytes;
    case 192: return PairCfg<192>::kSmemBytes;
    case 256: return PairCfg<256>::kSmemBytes;
    default: return -1;
  }
}

cudaError_t launch_kv_pair(int head_dim, int nt, const CUtensorMap& w, const CUtensorMap& x,
                           const CUtensorMap& h, const GemmParams& p, int num_sms,
                           cudaStream_t stream) {
  if (head_dim == 128) {
    switch (nt) {
      case 64: return launch_pair_t<128, 64>(w, x, h, p, num_sms, stream);
      case 128: return launch_pair_t<128, 128>(w, x, h, p, num_sms, stream);
      case 192: return launch_pair_t<128, 192>(w, x, h, p, num_sms, stream);
      case 256: return launch_pair_t<128, 256>(w, x, h, p, num_sms, stream);
    }
  } else if (head_dim == 64) {
    switch (nt) {
      case 64: return launch_pair_t<64, 64>(w, x, h, p, num_sms, stream);
      case 128: return launch_pair_t<64, 128>(w, x, h, p, num_sms, stream);
      case 192: return launch_pair_t<64, 192>(w, x, h, p, num_sms, stream);
      case 256: return launch_pair_t<64, 256>(w, x, h, p, num_sms, stream);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace dv
