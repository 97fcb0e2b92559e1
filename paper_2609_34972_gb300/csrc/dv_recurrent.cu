// Down-projection of one layer of the recurrent adapter (Sec. 3.1 Eq. 6):
//   H[:, h_col0 + n] = bf16(SiLU(M_{l-1} D_l^T)),  n < r_pad,
// where M_{l-1} (bf16 [M][d]) is the layer's input state. Unlike the embedding adapter, the
// L down-projections cannot be stacked (each reads the previous layer's state), and one layer
// is a thin [M x d] x [d x r_pad] product: with 128-token blocks a small build has only a few
// tiles, each with a long K loop. So the K dimension (d) is split over the CTAs of a
// thread-block cluster:
//   - CTA s of the cluster owns K slabs [s*k/S, (s+1)*k/S) of token block m (the cluster id)
//     and accumulates its 128 x r_pad partial product in TMEM (tcgen05.mma, one thread
//     streams K slabs by TMA and issues the MMAs);
//   - the partial goes to the CTA's shared memory as fp32;
//   - after a cluster barrier, CTA s sums rows [s*128/S, (s+1)*128/S) over all S CTAs'
//     partials through distributed shared memory, in the fixed order 0..S-1 (the result does
//     not depend on scheduling), applies SiLU and stores bf16 H;
//   - a second cluster barrier keeps every CTA's shared memory alive until all reads are done.
// With the split chain the K loop runs twice over the CTA's slabs, first with the high and then
// with the low bf16 part of M_{l-1} (the second A map), against the same D_l slabs, and h is
// stored as its bf16 rounding plus the bf16 rounding of the remainder (H and Hlo), so that the
// up-projection can read it in two parts as well.
// Every wait is bounded; a CTA that gives up still passes both cluster barriers, flags the
// plan's status word and returns.
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {
namespace {

constexpr int kDownThreads = 128;

template <int RP>
struct DownCfg {
  static constexpr int kABytes = kBlockM * kBlockK * 2;
  static constexpr int kBBytes = RP * kBlockK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStagesRaw = (160 * 1024) / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kPitch = RP + 4;  // floats per partial row: conflict-free row writes
  static constexpr int kRedBytes = kBlockM * kPitch * 4;
  static constexpr int kRingBytes = kStages * kStageBytes;
  static constexpr int kRegion = kRingBytes > kRedBytes ? kRingBytes : kRedBytes;
  static constexpr int kSmemBytes = kRegion + 1024 + 256;
  static constexpr int kTmemCols = RP <= 64 ? 64 : (RP <= 128 ? 128 : 256);
  static_assert(kStageBytes % 1024 == 0, "stage tiles must stay 1024-byte aligned");
  static_assert(kStages >= 2, "at least two stages");
  static_assert(RP % 32 == 0 && RP <= 256, "r_pad is a multiple of 64 up to 256");
};

__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// 16-byte load from shared memory of a CTA of this cluster (shared::cluster address).
__device__ __forceinline__ float4 ld_cluster_f4(uint32_t caddr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(caddr)
               : "memory");
  return v;
}

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait(bar, parity, &never, timeout_ns);
}

template <int RP>
__global__ void __launch_bounds__(kDownThreads, 1)
    dv_down_split_kernel(const __grid_constant__ CUtensorMap tmA,
                         const __grid_constant__ CUtensorMap tmAlo,
                         const __grid_constant__ CUtensorMap tmB,
                         const __grid_constant__ DownParams p) {
  using C = DownCfg<RP>;
  constexpr int NS = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  uint8_t* ring_ptr = smem_raw + (ring - raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring_ptr + C::kRegion);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (NS + s); };
  const uint32_t done_bar = bar0 + 8u * (2 * NS);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * NS + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* red = reinterpret_cast<float*>(ring_ptr);  // partial sums, after the last MMA

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t tmo = p.timeout_ns;
  const int split = static_cast<int>(cluster_ctarank());
  const int S = static_cast<int>(cluster_nctarank());
  const int m = static_cast<int>(cluster_id_x());
  const int ks0 = split * p.k_slabs / S;
  const int n_own = (split + 1) * p.k_slabs / S - ks0;  // this CTA's K slabs of A (and of D_l)
  const int n_slabs = p.a_lo ? 2 * n_own : n_own;       // split chain: high, then low parts

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(done_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------ TMA producer and MMA issuer
      tma_prefetch_desc(&tmA);
      if (p.a_lo) tma_prefetch_desc(&tmAlo);
      tma_prefetch_desc(&tmB);
      const uint32_t idesc = idesc_bf16_f32(kBlockM, RP);
      const int arow = p.a_row0 + m * kBlockM;
      auto load = [&](int j) {
        const int s = j % NS;
        const uint32_t a_dst = ring + s * C::kStageBytes;
        mbar_arrive_expect_tx(full_bar(s), C::kStageBytes);
        const int kk = ks0 + (j < n_own ? j : j - n_own);
        if (j < n_own) {
          tma_load_2d(a_dst, &tmA, full_bar(s), kk * kBlockK, arow);
        } else {  // the low part of the state: one [M][d] buffer, token rows from 0
          tma_load_2d(a_dst, &tmAlo, full_bar(s), kk * kBlockK, m * kBlockM);
        }
        tma_load_2d(a_dst + C::kABytes, &tmB, full_bar(s), kk * kBlockK, p.b_row0);
      };
      int loaded = 0, consumed = 0;
      for (; loaded < n_slabs && loaded < NS; ++loaded) load(loaded);
      bool ok = true, any_mma = false;
      for (int j = 0; j < n_slabs; ++j) {
        const int s = j % NS;
        const uint32_t ph = static_cast<uint32_t>(j / NS) & 1u;
        if (!mbar_wait(full_bar(s), ph, abort_flag, tmo)) {
          ok = false;
          break;
        }
        consumed = j + 1;
        tc_fence_after();
        const uint32_t a_s = ring + s * C::kStageBytes;
        const uint32_t b_s = a_s + C::kABytes;
  #pragma unroll
        for (int k = 0; k < kBlockK / 16; ++k)
          umma_bf16(tmem, sdesc_kmajor_sw128(a_s + 32u * k), sdesc_kmajor_sw128(b_s + 32u * k),
                    idesc, (j | k) != 0 ? 1u : 0u);
        any_mma = true;
        umma_commit(empty_bar(s));
        if (loaded < n_slabs) {  // refill this stage once its MMAs have read it
          if (!mbar_wait(empty_bar(s), ph, abort_flag, tmo)) {
            ok = false;
            break;
          }
          load(loaded);
          ++loaded;
        }
      }
      if (any_mma) umma_commit(done_bar);
      else mbar_arrive(done_bar);
      if (!ok) {  // let the copies still in flight land and the MMAs finish before moving on
        for (int j = consumed; j < loaded; ++j)
          wait_bounded(full_bar(j % NS), static_cast<uint32_t>(j / NS) & 1u, tmo);
        wait_bounded(done_bar, 0, tmo);
      }
    }
    __syncwarp();  // the other lanes of warp 0 wait here, not in a spin
  }

  // ---------------------------------------------------------- partial product -> smem
  bool have = mbar_wait(done_bar, 0, abort_flag, tmo) && !*abort_flag;
  have = __all_sync(0xFFFFFFFFu, have);
  if (have) {
    tc_fence_after();
    const int row = warp * 32 + lane;
#pragma unroll 1
    for (int c = 0; c < RP / 32; ++c) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld32(tmem + (static_cast<uint32_t>(warp * 32) << 16) + c * 32, r);
      tmem_ld_wait();
      float4* dst = reinterpret_cast<float4*>(red + row * C::kPitch + c * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        dst[q] = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                             __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
    }
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync();

  // ---------------------------------------------------------- reduce over the splits
  {
    constexpr int kV4 = RP / 4;
    const int rows = kBlockM / S;
    const int row_lo = split * rows;
#pragma unroll 1
    for (int idx = threadIdx.x; idx < rows * kV4; idx += kDownThreads) {
      const int rr = row_lo + idx / kV4, c4 = idx % kV4;
      const int t = m * kBlockM + rr;
      if (t >= p.M) continue;
      const uint32_t laddr = smem_addr(red + rr * C::kPitch + c4 * 4);
      // all S loads first (independent, so their latencies overlap), then the sum in order
      float4 part[8];
#pragma unroll
      for (int s = 0; s < 8; ++s)
        if (s < S) part[s] = ld_cluster_f4(map_to_rank(laddr, static_cast<uint32_t>(s)));
      float4 z = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        if (s < S) {
          z.x += part[s].x;
          z.y += part[s].y;
          z.z += part[s].z;
          z.w += part[s].w;
        }
      }
      const float h[4] = {silu(z.x), silu(z.y), silu(z.z), silu(z.w)};
      uint2 out;
      out.x = pack_bf16x2(h[0], h[1]);
      out.y = pack_bf16x2(h[2], h[3]);
      const size_t o = static_cast<size_t>(t) * p.ldh + p.h_col0 + c4 * 4;
      *reinterpret_cast<uint2*>(p.H + o) = out;
      if (p.Hlo) {  // the remainder h - bf16(h), itself rounded to bf16
        uint2 lo;
        lo.x = pack_bf16x2(h[0] - __uint_as_float(out.x << 16), h[1] - __uint_as_float(out.x & 0xFFFF0000u));
        lo.y = pack_bf16x2(h[2] - __uint_as_float(out.y << 16), h[3] - __uint_as_float(out.y & 0xFFFF0000u));
        *reinterpret_cast<uint2*>(p.Hlo + o) = lo;
      }
    }
  }
  __syncwarp();
  cluster_sync();

  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, 6 /* DV_ERR_DEVICE_TIMEOUT */);
}

template <int RP>
cudaError_t launch_t(int splits, const CUtensorMap& a, const CUtensorMap& a_lo, const CUtensorMap& b,
                     const DownParams& p, cudaStream_t stream) {
  using C = DownCfg<RP>;
  auto kern = dv_down_split_kernel<RP>;
  cudaError_t err =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess) return err;
  const long long m_tiles = (p.M + kBlockM - 1) / kBlockM;
  if (m_tiles <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(splits);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(m_tiles * splits), 1, 1);
  cfg.blockDim = dim3(kDownThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, kern, a, a_lo, b, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace

int down_splits(long long m_tiles, int k_slabs, int num_sms) {
  // Waves of CTAs times the slabs each CTA streams, with two slabs' worth of fixed cost per
  // CTA (set-up, reduction, store); fewer splits win ties.
  int best = 1;
  long long best_cost = -1;
  for (int s : {1, 2, 4, 8}) {
    if (s > k_slabs) break;
    const long long waves = (m_tiles * s + num_sms - 1) / num_sms;
    const long long cost = waves * ((k_slabs + s - 1) / s + 2);
    if (best_cost < 0 || cost < best_cost) {
      best = s;
      best_cost = cost;
    }
  }
  return best;
}

cudaError_t launch_down_split(int r_pad, int splits, const CUtensorMap& a, const CUtensorMap& a_lo,
                              const CUtensorMap& b, const DownParams& p, cudaStream_t stream) {
  if (splits != 1 && splits != 2 && splits != 4 && splits != 8) return cudaErrorInvalidValue;
  if (splits > p.k_slabs) return cudaErrorInvalidValue;
  switch (r_pad) {
    case 64: return launch_t<64>(splits, a, a_lo, b, p, stream);
    case 128: return launch_t<128>(splits, a, a_lo, b, p, stream);
    case 192: return launch_t<192>(splits, a, a_lo, b, p, stream);
    case 256: return launch_t<256>(splits, a, a_lo, b, p, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace dv
