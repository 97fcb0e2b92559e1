// The recurrent adapter's chain (Sec. 3.1 Eq. 6) kept on chip: M_0 = E and
//   M_l = M_{l-1} + SiLU(M_{l-1} D_l) U_l,   l = 1 .. L,
// for one 128-token block per thread-block cluster, through all layers in one launch.
//
// The cluster's S CTAs split the hidden dimension: CTA s owns columns [s CW, (s + 1) CW).
//   - Its slice of the fp32 state M (128 rows x CW) lives in TMEM for the whole chain; the
//     up-projection MMA accumulates h_l U_l^T straight into it.
//   - Its bf16 copy of that slice sits in shared memory (128-byte-swizzled K-major slabs): the A
//     operand of its part of the down-projection and the source of the TMA store of M_l.
// Per layer:
//   1. down-projection partial: z_s = bf16(M_{l-1})[:, slice] D_l[:, slice]^T (TMEM, fp32);
//   2. the partial goes to shared memory: a region of its own where shared memory allows (r_pad
//      64), else the U buffer (r_pad 128; U_l then loads once every peer has acknowledged its z
//      rows). CTA s owns rows [s 128 / S, (s + 1) 128 / S): every CTA sends each peer the peer's
//      rows of its partial by bulk copies into the peer's D buffer (read by then), completing
//      on the peer's barrier. CTA s sums its rows over the S partials in the fixed order 0 .. S-1, applies
//      SiLU, writes bf16 h into its h tile (A operand of the up-projection) and sends its rows of
//      h to every peer's h tile the same way;
//   3. once all h rows have landed: state += h U_l[slice, :]^T (TMEM);
//   4. the state slice is read back, its bf16 rounding written over the bf16 slice (next layer's
//      A operand, then stored to the stacked M_l by TMA) and its rows' sums of squares written to
//      `part` (the K/V stage's RMS statistic adds the S partials).
// One cluster barrier per layer (arrival once the down MMA has read D_l, wait before sending z)
// keeps a CTA from sending into a peer's D buffer too early; every other ordering follows from
// the data: a CTA sends z_{l+1} only after it has all of h_l, so every receiver has finished
// with z_l, and so on. D_{l+1} loads once the z rows are summed; U_{l+1} after the up MMA, or
// (partial z in the U buffer) once layer l+1's z rows have left it.
// Only bf16 M_l and the partial sums of squares leave the chip; the state never does. Every
// wait is bounded; a CTA that gives up keeps passing the cluster barriers and keeps sending (so
// its peers' waits end and no copy lands after a CTA has exited), stops issuing MMAs and loads,
// drains what it issued and flags the plan's status word.
#include "../../include/dv.h"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {
namespace {

constexpr int kChainThreads = 128;

template <int RP, int SPC, bool SPLIT>
struct ChainCfg {
  static constexpr int CW = 64 * SPC;             // hidden columns per CTA
  static constexpr int kSlab = 128 * 128;         // [128 rows][64 bf16], 128-byte swizzle
  static constexpr int kA = SPC * kSlab;          // bf16 state slice
  static constexpr int kH = (RP / 64) * kSlab;    // bf16 h
  // split chain: the low bf16 parts of the state slice and of h, beside their high parts
  static constexpr int kAlo = SPLIT ? kA : 0;
  static constexpr int kHlo = SPLIT ? kH : 0;
  static constexpr int kDslab = RP * 128;         // D_l: RP rows x 64 columns
  static constexpr int kD = SPC * kDslab;
  static constexpr int kUslab = CW * 128;         // U_l: CW rows x 64 rank columns
  static constexpr int kU = (RP / 64) * kUslab;
  // The peers' z rows land in the D buffer and past it: (S - 1) ceil(128 / S) rows, at most
  // 130 (S = 14), of RP fp32.
  static constexpr int kRecvMax = 130 * RP * 4;
  static constexpr int kDRegion = kD > kRecvMax ? kD : kRecvMax;
  static constexpr int kOffA = 0;
  static constexpr int kOffAlo = kOffA + kA;
  static constexpr int kOffH = kOffAlo + kAlo;
  static constexpr int kOffHlo = kOffH + kH;
  static constexpr int kOffU = kOffHlo + kHlo;
  static constexpr int kOffD = kOffU + kU;
  // The fp32 partial z gets a region of its own where shared memory allows. Otherwise it takes
  // the U buffer: U_l then loads once the peers have acknowledged z (every copy out of the
  // partial has landed), still well before the up MMA. Either way the store of M_{l-1},
  // reading the bf16 slice, runs alongside the rest of the layer.
  static constexpr int kZ = 128 * RP * 4;
  static constexpr bool kZOwn = kOffD + kDRegion + kZ + 1024 + 256 <= 232448;
  static constexpr int kOffZ = kZOwn ? kOffD + kDRegion : kOffU;
  static constexpr int kEnd = kOffD + kDRegion + (kZOwn ? kZ : 0);
  static constexpr int kSmemBytes = kEnd + 1024 + 256;
  static constexpr int kTmemCols = CW + RP <= 256 ? 256 : 512;
  static_assert(kZOwn || kZ <= kU, "the partial z takes the U buffer");
  static_assert(kSmemBytes <= 232448, "shared memory of one CTA");
  static_assert(kDslab % 1024 == 0 && kUslab % 1024 == 0, "tiles stay 1024-byte aligned");
};

struct ChainParams {
  int M;              // tokens
  int L;              // planned layers
  int d;
  float* part;        // fp32 [L][part_ld / M][M]: partial sums of squares of M_l
  long long part_ld;  // layer stride of part
  uint16_t* H;        // bf16 [M][ldh]: h_l at columns l r_pad (kept for stage-wise checks)
  int ldh;
  int* status;
  unsigned long long timeout_ns;
};

__device__ __forceinline__ uint32_t n_cluster_ctas() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// Bulk copy of `bytes` from this CTA's shared memory to a shared::cluster address (a peer's),
// completing as transaction bytes on the peer's barrier `cbar`.
__device__ __forceinline__ void bulk_copy_to_peer(uint32_t dst_cluster, uint32_t src, uint32_t bytes,
                                                  uint32_t cbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst_cluster), "r"(src), "r"(bytes), "r"(cbar)
      : "memory");
}

__device__ __forceinline__ int chain_row_lo(int s, int S) { return s * 128 / S; }

// Arrive on an mbarrier given by a shared::cluster address (a peer's), with no release: the
// arrival publishes no data, and a release would first wait for this thread's global stores.
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t cbar) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cbar)
               : "memory");
}
__device__ __forceinline__ int peer_slot(int src, int self) { return src < self ? src : src - 1; }

// Registers -> TMEM: lane i of the warp writes TMEM lane (taddr.lane + i), 32 columns.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0],"
      " {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16,"
      " %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 3-D tiled store from shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int c0, int c1,
                                             int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(src), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async_cta() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait(bar, parity, &never, timeout_ns);
}

// Byte offset of 16-byte chunk `c` (8 bf16, c < 8) of row `row` in a 128-byte-swizzled slab.
__device__ __forceinline__ uint32_t sw128(int row, int c) {
  return static_cast<uint32_t>(row * 128 + ((c ^ (row & 7)) << 4));
}

template <int RP, int SPC, bool SPLIT>
__global__ void __launch_bounds__(kChainThreads, 1)
    dv_chain_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmD,
                    const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmM,
                    const __grid_constant__ ChainParams p) {
  using C = ChainCfg<RP, SPC, SPLIT>;
  constexpr int CW = C::CW;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + C::kEnd);
  const uint32_t bar0 = smem_addr(bars);
  const uint32_t bar_x = bar0, bar_d = bar0 + 8, bar_u = bar0 + 16, bar_z = bar0 + 24,
                 bar_up = bar0 + 32, bar_drain = bar0 + 40, bar_rz = bar0 + 48, bar_rh = bar0 + 56,
                 bar_zs = bar0 + 64;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 10);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint64_t tmo = p.timeout_ns;
  const int s = static_cast<int>(cluster_ctarank());
  const int S = static_cast<int>(n_cluster_ctas());
  const int m = static_cast<int>(cluster_id_x());
  const int col0 = s * CW, row0 = m * 128;
  const int t = row0 + tid;  // this thread's token row
  const int r_lo = chain_row_lo(s, S), n_rows = chain_row_lo(s + 1, S) - r_lo;  // rows summed here
  const uint32_t sA = base + C::kOffA, sH = base + C::kOffH, sD = base + C::kOffD,
                 sU = base + C::kOffU, sAlo = base + C::kOffAlo, sHlo = base + C::kOffHlo;
  float* zpart = reinterpret_cast<float*>(base_ptr + C::kOffZ);
  const uint32_t sZ = base + C::kOffZ;

  if (tid == 0) {
    mbar_init(bar_x, 1);
    mbar_init(bar_d, 1);
    mbar_init(bar_u, 1);
    mbar_init(bar_z, 1);
    mbar_init(bar_up, 1);
    mbar_init(bar_drain, 1);
    mbar_init(bar_rz, 1);  // the peers' z rows of this CTA, once per layer
    mbar_init(bar_rh, 1);  // the peers' h rows, once per layer
    // partial z in the U buffer: every peer acknowledges that this CTA's z rows have landed
    if (!C::kZOwn && S > 1) mbar_init(bar_zs, S - 1);
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
  pdl_wait();
  pdl_trigger();
  const uint32_t t_state = tmem, t_z = tmem + CW;
  const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;

  // thread 0's bookkeeping of async work, for the drain after an abort
  int d_loads = 0, d_waits = 0, u_loads = 0, u_waits = 0;
  bool mma_open = false;
  auto load_d = [&](int l) {
    mbar_arrive_expect_tx(bar_d, C::kD);
    for (int j = 0; j < SPC; ++j)
      tma_load_2d(sD + j * C::kDslab, &tmD, bar_d, col0 + 64 * j, l * RP);
    ++d_loads;
  };
  auto load_u = [&](int l) {
    mbar_arrive_expect_tx(bar_u, C::kU);
    for (int j = 0; j < RP / 64; ++j)
      tma_load_2d(sU + j * C::kUslab, &tmU, bar_u, 64 * j, l * p.d + col0);
    ++u_loads;
  };

  if (tid == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmD);
    tma_prefetch_desc(&tmU);
    tma_prefetch_desc(&tmM);
    mbar_arrive_expect_tx(bar_x, C::kA);
    for (int j = 0; j < SPC; ++j) tma_load_2d(sA + j * C::kSlab, &tmX, bar_x, col0 + 64 * j, row0);
    load_d(0);
    if (C::kZOwn) load_u(0);  // else once the layer's z rows have left the U buffer
  }

  // M_0 = E: the state slice in TMEM is the fp32 widening of the bf16 slice just loaded.
  bool ok = mbar_wait(bar_x, 0, abort_flag, tmo);
  if (__all_sync(0xFFFFFFFFu, ok)) {
#pragma unroll 1
    for (int c = 0; c < CW / 32; ++c) {
      const uint8_t* slab = base_ptr + C::kOffA + (c / 2) * C::kSlab;
      uint32_t r[32];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 w = *reinterpret_cast<const uint4*>(slab + sw128(tid, (c % 2) * 4 + q));
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          r[q * 8 + 2 * e] = ws[e] << 16;
          r[q * 8 + 2 * e + 1] = ws[e] & 0xFFFF0000u;
        }
      }
      tmem_st32(t_state + lane_base + c * 32, r);
    }
    tmem_st_wait();
  }
  tc_fence_before();
  ok = __syncthreads_and(ok) != 0;

  for (int l = 0; l < p.L; ++l) {
    const uint32_t ph = static_cast<uint32_t>(l) & 1u;
    if (tid == 0) {  // this layer's transfers into this CTA: the peers' z rows, then h rows
      mbar_arrive_expect_tx(bar_rz, static_cast<uint32_t>((S - 1) * n_rows * RP * 4));
      mbar_arrive_expect_tx(bar_rh, static_cast<uint32_t>((128 - n_rows) * RP * 2 * (SPLIT ? 2 : 1)));
    }

    // (1) down-projection partial z = bf16(M_{l-1})[:, slice] D_l[:, slice]^T; store M_{l-1}
    if (tid == 0 && ok && !*abort_flag) {
      tc_fence_after();
      fence_proxy_async_cta();  // the bf16 slice was written by the threads
      if (mbar_wait(bar_d, ph, abort_flag, tmo)) {
        ++d_waits;
        const uint32_t idesc = idesc_bf16_f32(128, RP);
        for (int j = 0; j < SPC; ++j)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_bf16(t_z, sdesc_kmajor_sw128(sA + j * C::kSlab + 32u * k),
                      sdesc_kmajor_sw128(sD + j * C::kDslab + 32u * k), idesc,
                      (j | k) != 0 ? 1u : 0u);
        if (SPLIT && l > 0) {  // the low part of M_{l-1} (E, at l = 0, is exact in bf16)
          for (int j = 0; j < SPC; ++j)
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(t_z, sdesc_kmajor_sw128(sAlo + j * C::kSlab + 32u * k),
                        sdesc_kmajor_sw128(sD + j * C::kDslab + 32u * k), idesc, 1u);
        }
        umma_commit(bar_z);
        mma_open = true;
      }
      if (l >= 1) {
        for (int j = 0; j < SPC; ++j)
          tma_store_3d(&tmM, sA + j * C::kSlab, col0 + 64 * j, row0, l - 1);
        bulk_commit();
      }
    }

    // (2) z partial -> shared memory (over the bf16 slice: once the down MMA and the store of
    // M_{l-1} have read it)
    bool zok = ok && mbar_wait(bar_z, ph, abort_flag, tmo);
    if (tid == 0) {
      if (zok) mma_open = false;
    }
    // The down MMA has read D_l (or this CTA issues no more MMAs): the D buffer may receive.
    // Relaxed: the arrival publishes no data, and a release would first wait for this thread's
    // earlier global stores (h rows, sums of squares) to complete, about 2 us.
    __syncwarp();
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    zok = __syncthreads_and(zok) != 0;
    if (zok) {
      tc_fence_after();
      float* zrow = zpart + tid * RP;
#pragma unroll 1
      for (int c = 0; c < RP / 32; ++c) {
        uint32_t r[32];
        __syncwarp();
        tmem_ld32(t_z + lane_base + c * 32, r);
        tmem_ld_wait();
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int c4 = c * 8 + q;
          reinterpret_cast<float4*>(zrow)[c4 ^ (tid & 7)] =
              make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                          __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
        }
      }
    }
    ok = zok;
    fence_proxy_async_cta();  // the partial is read by the bulk copies
    tc_fence_before();
    __syncthreads();
    __syncwarp();
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");  // every D buffer is free
    // Each peer's rows of this partial into its D buffer, slot peer_slot(s, peer): lane dd of
    // warp 0 sends to peer dd, so the copies issue in parallel. A CTA that gave up sends too, so
    // that every receiver's wait ends.
    if (warp == 0) {
      const int dd = tid;
      if (dd < S && dd != s) {
        const int lo = chain_row_lo(dd, S), n = chain_row_lo(dd + 1, S) - lo;
        const uint32_t rank = static_cast<uint32_t>(dd);
        bulk_copy_to_peer(
            map_to_rank(sD + static_cast<uint32_t>(peer_slot(s, dd) * n * RP * 4), rank),
            sZ + static_cast<uint32_t>(lo * RP * 4), static_cast<uint32_t>(n * RP * 4),
            map_to_rank(bar_rz, rank));
      }
    }

    // (3) rows [r_lo, r_lo + n_rows): sum the S partials in order (this CTA's own from its
    // partial, the peers' from the D buffer), SiLU, bf16 h into this CTA's h tile (8-byte
    // pieces, swizzled as the MMA reads them) and into H. Not cut short by the abort flag: the
    // copies into this CTA must land before it may exit.
    if (!wait_bounded(bar_rz, ph, tmo)) *abort_flag = 1;
    // Partial z in the U buffer: tell each peer that its z rows have landed here (thread i
    // < S - 1, one peer each; relaxed, as nothing is published).
    if (!C::kZOwn && tid < S - 1)
      mbar_arrive_cluster_relaxed(map_to_rank(bar_zs, static_cast<uint32_t>(tid < s ? tid : tid + 1)));
    {
      const int items = n_rows * (RP / 4);
#pragma unroll 1
      for (int it = tid; it < items; it += kChainThreads) {
        const int rr = it / (RP / 4), row = r_lo + rr, c4 = it % (RP / 4);
        const uint32_t chunk = static_cast<uint32_t>((c4 ^ (row & 7)) << 4);
        float4 z = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        for (int b = 0; b < S; ++b) {
          const uint32_t src =
              b == s ? sZ + static_cast<uint32_t>(row * RP * 4) + chunk
                     : sD + static_cast<uint32_t>((peer_slot(b, s) * n_rows + rr) * RP * 4) + chunk;
          const float4 v = *reinterpret_cast<const float4*>(__cvta_shared_to_generic(src));
          z.x += v.x;
          z.y += v.y;
          z.z += v.z;
          z.w += v.w;
        }
        const float h0 = silu(z.x), h1 = silu(z.y), h2 = silu(z.z), h3 = silu(z.w);
        uint2 hv;
        hv.x = pack_bf16x2(h0, h1);
        hv.y = pack_bf16x2(h2, h3);
        // columns 4 c4 .. 4 c4 + 3: slab c4 / 16, 16-byte chunk (c4 % 16) / 2, half c4 % 2
        const uint32_t hoff = static_cast<uint32_t>((c4 / 16) * C::kSlab + sw128(row, (c4 % 16) / 2) +
                                                    (c4 % 2) * 8);
        *reinterpret_cast<uint2*>(base_ptr + C::kOffH + hoff) = hv;
        if (SPLIT) {  // the remainder h - bf16(h), itself in bf16, at the same place of its tile
          uint2 lv;
          lv.x = pack_bf16x2(h0 - __uint_as_float(hv.x << 16), h1 - __uint_as_float(hv.x & 0xFFFF0000u));
          lv.y = pack_bf16x2(h2 - __uint_as_float(hv.y << 16), h3 - __uint_as_float(hv.y & 0xFFFF0000u));
          *reinterpret_cast<uint2*>(base_ptr + C::kOffHlo + hoff) = lv;
        }
        if (row0 + row < p.M)
          *reinterpret_cast<uint2*>(p.H + static_cast<long long>(row0 + row) * p.ldh + l * RP +
                                    c4 * 4) = hv;
      }
    }
    fence_proxy_async_cta();  // this CTA's h rows: read by the bulk copies and the up MMA
    __syncthreads();
    if (warp == 0) {
      // this CTA's rows of h into every peer's h tile (the same bytes of each 64-column slab),
      // lane dd to peer dd
      const int dd = tid;
      if (dd < S && dd != s) {
        const uint32_t rank = static_cast<uint32_t>(dd), cbar = map_to_rank(bar_rh, rank);
        for (int j = 0; j < RP / 64; ++j) {
          const uint32_t off = sH + static_cast<uint32_t>(j * C::kSlab + r_lo * 128);
          bulk_copy_to_peer(map_to_rank(off, rank), off, static_cast<uint32_t>(n_rows * 128), cbar);
          if (SPLIT) {
            const uint32_t lo = sHlo + static_cast<uint32_t>(j * C::kSlab + r_lo * 128);
            bulk_copy_to_peer(map_to_rank(lo, rank), lo, static_cast<uint32_t>(n_rows * 128), cbar);
          }
        }
      }
      if (tid == 0 && ok && !*abort_flag && l + 1 < p.L) load_d(l + 1);  // the z rows are summed
    }
    if (!C::kZOwn && tid == 0) {  // every copy out of the partial has landed: U_l may load
      if (S > 1 && !wait_bounded(bar_zs, ph, tmo)) *abort_flag = 1;
      if (ok && !*abort_flag) load_u(l);
    }

    // (4) state += h U_l[slice, :]^T, once every peer's h rows have landed. The readback after
    // it overwrites the bf16 slice: the store of M_{l-1} must have read it (every thread's
    // readback waits for this MMA).
    if (tid == 0) {
      if (!wait_bounded(bar_rh, ph, tmo)) *abort_flag = 1;
      bulk_wait_read0();
      if (ok && !*abort_flag) {
        tc_fence_after();
        if (mbar_wait(bar_u, ph, abort_flag, tmo)) {
          ++u_waits;
          const uint32_t idesc = idesc_bf16_f32(128, CW);
          for (int j = 0; j < RP / 64; ++j)
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(t_state, sdesc_kmajor_sw128(sH + j * C::kSlab + 32u * k),
                        sdesc_kmajor_sw128(sU + j * C::kUslab + 32u * k), idesc, 1u);
          if (SPLIT)  // and the low part of h
            for (int j = 0; j < RP / 64; ++j)
#pragma unroll
              for (int k = 0; k < 4; ++k)
                umma_bf16(t_state, sdesc_kmajor_sw128(sHlo + j * C::kSlab + 32u * k),
                          sdesc_kmajor_sw128(sU + j * C::kUslab + 32u * k), idesc, 1u);
          umma_commit(bar_up);
          mma_open = true;
        }
      }
    }
    bool uok = ok && mbar_wait(bar_up, ph, abort_flag, tmo);
    if (tid == 0 && uok) {
      mma_open = false;
      if (C::kZOwn && l + 1 < p.L) load_u(l + 1);  // the U buffer is free
    }
    // (5) state -> bf16 slice (next A operand, stored next layer) and sums of squares
    if (__all_sync(0xFFFFFFFFu, uok)) {
      tc_fence_after();
      float ss = 0.0f;
#pragma unroll 1
      for (int c2 = 0; c2 < CW / 64; ++c2) {  // one 64-column slab: two TMEM loads in flight
        uint32_t r[2][32];
        __syncwarp();
        tmem_ld32(t_state + lane_base + c2 * 64, r[0]);
        tmem_ld32(t_state + lane_base + c2 * 64 + 32, r[1]);
        tmem_ld_wait();
        uint8_t* slab = base_ptr + C::kOffA + c2 * C::kSlab;
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          uint32_t pk[16];
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const float a = __uint_as_float(r[h2][2 * u]), b = __uint_as_float(r[h2][2 * u + 1]);
            ss = fmaf(a, a, ss);
            ss = fmaf(b, b, ss);
            pk[u] = pack_bf16x2(a, b);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q)
            *reinterpret_cast<uint4*>(slab + sw128(tid, h2 * 4 + q)) =
                make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
          if (SPLIT) {  // the low part M - bf16(M), the next down-projection's second operand
            uint8_t* lslab = base_ptr + C::kOffAlo + c2 * C::kSlab;
            uint32_t lo[16];
#pragma unroll
            for (int u = 0; u < 16; ++u)
              lo[u] = pack_bf16x2(__uint_as_float(r[h2][2 * u]) - __uint_as_float(pk[u] << 16),
                                  __uint_as_float(r[h2][2 * u + 1]) - __uint_as_float(pk[u] & 0xFFFF0000u));
#pragma unroll
            for (int q = 0; q < 4; ++q)
              *reinterpret_cast<uint4*>(lslab + sw128(tid, h2 * 4 + q)) =
                  make_uint4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
          }
        }
      }
      if (t < p.M) p.part[l * p.part_ld + static_cast<long long>(s) * p.M + t] = ss;
    }
    fence_proxy_async_cta();
    tc_fence_before();
    ok = __syncthreads_and(uok) != 0;
  }

  if (tid == 0) {
    if (ok && !*abort_flag && p.L > 0) {
      for (int j = 0; j < SPC; ++j)
        tma_store_3d(&tmM, sA + j * C::kSlab, col0 + 64 * j, row0, p.L - 1);
      bulk_commit();
    }
    bulk_wait0();
    if (!ok || *abort_flag) {  // let issued loads land and issued MMAs finish
      if (d_loads > d_waits) wait_bounded(bar_d, static_cast<uint32_t>(d_loads - 1) & 1u, tmo);
      if (u_loads > u_waits) wait_bounded(bar_u, static_cast<uint32_t>(u_loads - 1) & 1u, tmo);
      if (mma_open) {
        umma_commit(bar_drain);
        wait_bounded(bar_drain, 0, tmo);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  __syncwarp();
  cluster_sync();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
  if (tid == 0 && (!ok || *abort_flag)) atomicExch(p.status, DV_ERR_DEVICE_TIMEOUT);
}

template <int RP, int SPC, bool SPLIT = false>
cudaError_t launch_t(int S, long long blocks, const CUtensorMap& x, const CUtensorMap& dmap,
                     const CUtensorMap& umap, const CUtensorMap& mmap, const ChainParams& p,
                     cudaStream_t stream) {
  using C = ChainCfg<RP, SPC, SPLIT>;
  auto kern = dv_chain_kernel<RP, SPC, SPLIT>;
  cudaError_t err =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err == cudaSuccess && S > 8)
    err = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (err != cudaSuccess || blocks <= 0) return err;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(S);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(blocks * S), 1, 1);
  cfg.blockDim = dim3(kChainThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess || clusters < 1) {
    cudaGetLastError();
    return cudaErrorNotSupported;  // the caller falls back to the per-layer launches
  }
  attr[1] = pdl_attribute();
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, kern, x, dmap, umap, mmap, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

template <int RP, int SPC, bool SPLIT = false>
int resident_t(int S) {
  using C = ChainCfg<RP, SPC, SPLIT>;
  auto kern = dv_chain_kernel<RP, SPC, SPLIT>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
          cudaSuccess ||
      (S > 8 && cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                    cudaSuccess)) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(S);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(S), 1, 1);
  cfg.blockDim = dim3(kChainThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return clusters;
}

}  // namespace

int chain_resident_clusters(int d, int r_pad, bool split) {
  int spc = 0, S = 0;
  if (!chain_shape(d, r_pad, &spc, &S)) return 0;
  if (split) {
    if (r_pad == 64 && spc == 2) return resident_t<64, 2, true>(S);
    if (r_pad == 64 && spc == 3) return resident_t<64, 3, true>(S);
    if (r_pad == 64 && spc == 4) return resident_t<64, 4, true>(S);
    return 0;
  }
  if (r_pad == 64 && spc == 2) return resident_t<64, 2>(S);
  if (r_pad == 64 && spc == 3) return resident_t<64, 3>(S);
  if (r_pad == 64 && spc == 4) return resident_t<64, 4>(S);
  if (r_pad == 128 && spc == 4) return resident_t<128, 4>(S);
  return 0;
}

bool chain_shape(int d, int r_pad, int* spc_out, int* s_out) {
  if (r_pad != 64 && r_pad != 128) return false;
  const int k_slabs = d / 64;
  const int min_spc = r_pad == 128 ? 4 : 2;  // the fp32 partial z must fit over the bf16 slice
  for (int spc = min_spc; spc <= 4; ++spc) {
    if (k_slabs % spc) continue;
    const int S = k_slabs / spc;
    if (S < 1 || S > 16) continue;
    *spc_out = spc;
    *s_out = S;
    return true;
  }
  return false;
}

cudaError_t launch_chain(int r_pad, int spc, int S, long long tokens, int n_layers, int d,
                         const CUtensorMap& x, const CUtensorMap& dmap, const CUtensorMap& umap,
                         const CUtensorMap& mmap, float* part, long long part_ld, uint16_t* H,
                         int* status, unsigned long long timeout_ns, cudaStream_t stream,
                         bool split) {
  ChainParams p;
  p.H = H;
  p.ldh = n_layers * r_pad;
  p.M = static_cast<int>(tokens);
  p.L = n_layers;
  p.d = d;
  p.part = part;
  p.part_ld = part_ld;
  p.status = status;
  p.timeout_ns = timeout_ns;
  const long long blocks = (tokens + 127) / 128;
  if (split) {  // the low parts fit beside the state at r_pad 64 only
    if (r_pad == 64 && spc == 2) return launch_t<64, 2, true>(S, blocks, x, dmap, umap, mmap, p, stream);
    if (r_pad == 64 && spc == 3) return launch_t<64, 3, true>(S, blocks, x, dmap, umap, mmap, p, stream);
    if (r_pad == 64 && spc == 4) return launch_t<64, 4, true>(S, blocks, x, dmap, umap, mmap, p, stream);
    return cudaErrorInvalidValue;
  }
  if (r_pad == 64 && spc == 2) return launch_t<64, 2>(S, blocks, x, dmap, umap, mmap, p, stream);
  if (r_pad == 64 && spc == 3) return launch_t<64, 3>(S, blocks, x, dmap, umap, mmap, p, stream);
  if (r_pad == 64 && spc == 4) return launch_t<64, 4>(S, blocks, x, dmap, umap, mmap, p, stream);
  if (r_pad == 128 && spc == 4) return launch_t<128, 4>(S, blocks, x, dmap, umap, mmap, p, stream);
  return cudaErrorInvalidValue;
}

}  // namespace dv
