// The recurrent adapter (Sec. 3.1 Eq. 6) through an exact rearrangement of its chain. With rows
// of M, D_l [r][d] and U_l [d][r] (nn.Linear layout):
//   M_0 = E,   M_l = M_{l-1} + h_l U_l^T,   h_l = SiLU(z_l),   z_l = M_{l-1} D_l^T.
// Unrolling M_{l-1} = E + sum_{j<l} h_j U_j^T gives
//   z_l = E D_l^T + sum_{j<l} h_j Q_lj^T,   Q_lj = D_l U_j (r x r, formed once per weight set),
// so the chain splits into three parts, none of which moves the d-wide state between layers:
//   (1) C = E [D_1 ... D_L]^T, one fp32 GEMM over all layers on the GEMM engines;
//   (2) dv_hchain_kernel: per 128-token block, the recurrence over the r-wide vectors,
//         z_l = C_l + [h_1 .. h_{l-1}] [Q_l1 .. Q_l,l-1]^T,
//       one tcgen05 GEMM per layer whose accumulator starts at C_l and whose K grows by r_pad
//       each layer, SiLU in its epilogue;
//   (3) dv_accum_kernel: per two 128-token blocks and hidden slice, M_l = E + sum_{j<=l} h_j U_j^T
//       as a running sum in TMEM, bf16 M_l stored for the K/V GEMM with its rows' sums of
//       squares for the RMS statistic.
// Only (2) runs layer after layer, and each of its layers is a GEMM of N = r_pad with no
// exchange between CTAs. The sums differ from the chain's only in rounding (the same products,
// grouped differently). With the split chain, h_j and Q_lj are each read as a high and a low
// bf16 part in (2), and h_j in both parts in (3).
#include "../../include/dv.h"
#include "dv_epilogue.cuh"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {

// ------------------------------------------------------------------------------ kernels

namespace {

constexpr int kFoldThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM, warps 2-5 epilogue
constexpr int kEpi = 128;
constexpr int kAccumWarps = 2;     // epilogue warps per TMEM lane quarter of the running sum
constexpr int kSlabA = 128 * 128;  // [128 token rows][64] bf16, 128-byte swizzle

// Byte offset of 16-byte chunk `c` (c < 8) of row `row` in a 128-byte-swizzled slab.
__device__ __forceinline__ uint32_t swz(int row, int c) {
  return static_cast<uint32_t>(row * 128 + ((c ^ (row & 7)) << 4));
}

__device__ __forceinline__ bool wait_only(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait(bar, parity, &never, timeout_ns);
}

// Registers -> TMEM: lane i of the warp writes TMEM lane (taddr.lane + i), 32 columns.
__device__ __forceinline__ void tmem_st32x(uint32_t taddr, const uint32_t (&r)[32]) {
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

// ---------------------------------------------------------------- (2) the h recurrence

// 3-D tiled load of a slab-map box {64 columns, rows, slabs} at (0, row, slab).
__device__ __forceinline__ void tma_load_slabs(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                               int row, int slab) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(0), "r"(row), "r"(slab)
      : "memory");
}

// 2-D tiled store of a shared-memory box to global memory (bulk-group completion), and the
// group's commit and wait (writes complete: the source may be rewritten and the data is in
// global memory).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void bulk_commit_wait() {
  asm volatile("cp.async.bulk.commit_group;\n\tcp.async.bulk.wait_group 0;" ::: "memory");
}

template <int RP, int KS, int STAGES, bool SPLIT, bool PAIR>
struct HCfg {
  static constexpr int R = RP / 64;              // 64-wide K slabs per r_pad
  // [RP rows of Pf][64] bf16; on CTA pairs each CTA stages its half of the rows
  static constexpr int kSlabB = (PAIR ? RP / 2 : RP) * 128;
  static constexpr int kA = KS * kSlabA;         // one box of KS slabs of A
  static constexpr int kB = KS * kSlabB;         // one box of KS slabs of B
  static constexpr int kStage = kA + kB;
  static constexpr int kOffH = STAGES * kStage;  // h_{l-1} as the A operand of layer l's last slabs
  static constexpr int kOffL = kOffH + R * kSlabA;  // split: the low part of h_{l-1}
  static constexpr int kEnd = kOffL + (SPLIT ? R * kSlabA : 0);
  static constexpr int kSmemBytes = kEnd + 1024 + 256;
  static constexpr int kTmemCols = 2 * RP <= 128 ? 128 : (2 * RP <= 256 ? 256 : 512);
  static_assert(kSlabB % 1024 == 0, "stage tiles stay 1024-byte aligned");
  static_assert(kSmemBytes <= 232448, "shared memory of one CTA");
};

struct HChainParams {
  int M;           // tokens
  int L;           // planned layers
  const float* C;  // fp32 [M][ldc]: E D_l^T at columns l r_pad
  int ldc;
  uint16_t* H;     // bf16 [M][ldh]: h_l at columns l r_pad
  uint16_t* Hlo;   // split: bf16(h_l - bf16(h_l)), the same layout; else null
  int ldh;
  int* status;
  unsigned long long timeout_ns;
};

// Segment `seg` of layer l's K loop (l >= 1): n slabs, the first at slab a0 of its A source and
// at slab b0 of the layer's rows of its B source. A: 0 H, 1 Hlo, 2 the h tile, 3 the low h tile;
// B: 0 Pf, 1 Pf_lo. h_0 .. h_{l-2} come from global memory (A 0 / 1), h_{l-1} from the tiles the
// epilogue has just written (A 2 / 3). Without the split: (H, Pf), (h tile, Pf). With it, each
// product in three parts, h_hi Q_hi + h_lo Q_hi + h_hi Q_lo, for the older h_j and for h_{l-1}.
struct HSeg {
  int n, a0, b0, asrc, bsrc;
};
template <bool SPLIT>
__device__ __forceinline__ HSeg hseg(int l, int seg, int R) {
  const int n_old = l >= 2 ? (l - 1) * R : 0, b_new = (l - 1) * R;
  if (!SPLIT) return seg == 0 ? HSeg{n_old, 0, 0, 0, 0} : HSeg{R, 0, b_new, 2, 0};
  switch (seg) {
    case 0: return {n_old, 0, 0, 0, 0};
    case 1: return {n_old, 0, 0, 1, 0};
    case 2: return {n_old, 0, 0, 0, 1};
    case 3: return {R, 0, b_new, 2, 0};
    case 4: return {R, 0, b_new, 3, 0};
    default: return {R, 0, b_new, 2, 1};
  }
}

// One CTA per 128-token block, all layers. Layer l's accumulator starts as C_l, written into TMEM
// by the epilogue warps (tcgen05.st) while the tensor cores still work on earlier layers; the
// layer's GEMM then adds h_j Q_lj^T for every j < l over l R slabs of 64 in the segments of hseg
// (two; six with the split). A pipeline step moves KS consecutive slabs of one segment as one TMA box per operand (a
// TMA instruction has a fixed cost that one 16 KB slab does not amortise); the last step of a
// segment uses the slabs it needs of its box (the rest is zero fill or data the MMA does not
// read). Two accumulators alternate by layer: layer l's MMAs over the older h_j run while the
// epilogue of layer l - 1 still works. The epilogue applies SiLU (layer 0 straight from C_0),
// writes bf16 h_l to the h tile (the A operand of layer l + 1's last segments; with the split, its
// low part to a second tile), loads C_{l+2} into the accumulator it has just read, and stores
// its rows of the tiles to H by TMA (read back by TMA from layer l + 2 on, and by the running
// sum). The per-layer chain (accumulator full -> readback -> h tile -> layer l + 1's last MMAs)
// sets the pace, so everything else stays off it: at r_pad <= 128 C_{l+2} is fetched into
// registers a layer ahead, and the producer waits for h_{l-2} in H only before the box that
// reads it, the last of the older segment.
// Barriers (all waits bounded): stage full / empty; accumulator full; accumulator loaded with C;
// the h tile written (once per layer); h_l in global memory, alternating between two barriers by
// layer parity so that the producer, which may run up to two layers ahead of the epilogue, never
// waits on a phase that has wrapped. The accumulator barriers of layer l complete for the
// ((l - 1) / 2)-th time (integer division) at that layer, on accumulator l mod 2.
// PAIR: a cluster of two CTAs (token blocks 2c and 2c + 1) runs each layer's GEMM as one 2-SM
// MMA (M = 256, tcgen05 cta_group::2) issued by the leader: each CTA stages its own 128 rows of
// h and half of the layer's rows of Pf, so an SM moves half the B bytes per MMA through shared
// memory. The leader's stage-full barrier counts both CTAs' bytes; its commits arrive on both
// CTAs' stage-empty and accumulator-full barriers; both CTAs' epilogue warps arrive on the
// leader's accumulator-loaded and h-tile barriers (one lane per warp, 8 arrivals).
template <int RP, int KS, int STAGES, bool SPLIT, bool PAIR>
__global__ void __launch_bounds__(kFoldThreads, 1)
    dv_hchain_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmHlo,
                     const __grid_constant__ CUtensorMap tmP, const __grid_constant__ CUtensorMap tmPlo,
                     const __grid_constant__ CUtensorMap tmHst, const __grid_constant__ CUtensorMap tmHlost,
                     const __grid_constant__ HChainParams p) {
  using C = HCfg<RP, KS, STAGES, SPLIT, PAIR>;
  constexpr int kSegs = SPLIT ? 6 : 2;
  constexpr int kFirstNew = SPLIT ? 3 : 1;  // the first segment that reads the h tiles
  constexpr int R = C::R;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + C::kEnd);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto accf_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
  auto init_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
  auto hpub_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 4 + a); };
  const uint32_t htile_bar = bar0 + 8u * (2 * STAGES + 6);
  const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 7);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t ring = base, htile = base + C::kOffH, ltile = base + C::kOffL;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t tmo = p.timeout_ns;
  const int row0 = blockIdx.x * 128;  // with pairs: cluster c, rank r -> block 2c + r
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  // arrivals on the accumulator-loaded and h-tile barriers: every epilogue thread, or with pairs
  // one lane per epilogue warp of both CTAs on the leader's
  constexpr int kEpiArrivals = PAIR ? 8 : kEpi;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accf_bar(a), 1);
      mbar_init(init_bar(a), kEpiArrivals);
      mbar_init(hpub_bar(a), kEpi);
    }
    mbar_init(htile_bar, kEpiArrivals);
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmH);
    tma_prefetch_desc(&tmP);
    if (SPLIT) {
      tma_prefetch_desc(&tmHlo);
      tma_prefetch_desc(&tmPlo);
    }
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(smem_addr(tmem_slot), C::kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (PAIR)
    cluster_sync();  // both CTAs' barriers exist before any remote arrival or pair load
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      const uint32_t leader_full0 = PAIR ? map_to_rank(full_bar(0), 0) : full_bar(0);
      int stage = 0;
      uint32_t phase = 0, used = 0, issued_parity = 0;
      bool ok = true;
      for (int l = 1; l < p.L && ok; ++l) {
        bool newest_in_h = false;
        for (int seg = 0; seg < kSegs && ok; ++seg) {
          const HSeg g = hseg<SPLIT>(l, seg, R);
          for (int s0 = 0; s0 < g.n; s0 += KS) {
            // h_{l-2}, the newest layer the older segments read, fills their last R slabs: wait
            // until it is in global memory before the first box that covers one of them (the
            // layers before it were published earlier)
            if (g.asrc < 2 && !newest_in_h && s0 + KS > (l - 2) * R) {
              if (!mbar_wait(hpub_bar((l - 2) & 1), static_cast<uint32_t>((l - 2) >> 1) & 1u,
                             abort_flag, tmo)) {
                ok = false;
                break;
              }
              newest_in_h = true;
            }
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, tmo)) {
              ok = false;
              break;
            }
            const uint32_t a_dst = ring + stage * C::kStage, b_dst = a_dst + C::kA;
            const uint32_t bytes = g.asrc >= 2 ? C::kB : C::kStage;
            const CUtensorMap* am = g.asrc == 0 ? &tmH : &tmHlo;
            const CUtensorMap* bm = g.bsrc == 0 ? &tmP : &tmPlo;
            if (PAIR) {
              // both CTAs' copies complete on the leader's barrier, which expects both
              const uint32_t fb = leader_full0 + 8u * stage;
              if (rank == 0) mbar_arrive_expect_tx(full_bar(stage), 2 * bytes);
              if (g.asrc < 2) tma_load_3d_pair(a_dst, am, fb, row0, g.a0 + s0);
              tma_load_3d_pair(b_dst, bm, fb, l * RP + static_cast<int>(rank) * (RP / 2), g.b0 + s0);
            } else {
              mbar_arrive_expect_tx(full_bar(stage), bytes);
              if (g.asrc < 2) tma_load_slabs(a_dst, am, full_bar(stage), row0, g.a0 + s0);
              tma_load_slabs(b_dst, bm, full_bar(stage), l * RP, g.b0 + s0);
            }
            used |= 1u << stage;
            issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      // every copy still in flight lands before the CTA exits (pairs: their copies complete on
      // the leader's barriers; the teardown waits instead)
      if (!PAIR && *abort_flag) {
        for (int s = 0; s < STAGES; ++s)
          if (used & (1u << s)) wait_only(full_bar(s), (issued_parity >> s) & 1u, tmo);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------------------------------------------------------- MMA issuer (the leader)
      const uint32_t idesc = idesc_bf16_f32(PAIR ? 256 : 128, RP);
      int stage = 0;
      uint32_t phase = 0;
      bool issued_any = false, ok = true;
      for (int l = 1; l < p.L && ok; ++l) {
        const int acc = l & 1;
        const uint32_t par = static_cast<uint32_t>((l - 1) >> 1) & 1u;
        if (!mbar_wait(init_bar(acc), par, abort_flag, tmo)) break;  // C_l is in the accumulator
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * RP);
        for (int seg = 0; seg < kSegs && ok; ++seg) {
          const HSeg g = hseg<SPLIT>(l, seg, R);
          if (seg == kFirstNew &&
              !mbar_wait(htile_bar, static_cast<uint32_t>(l - 1) & 1u, abort_flag, tmo)) {
            ok = false;
            break;
          }
          for (int s0 = 0; s0 < g.n; s0 += KS) {
            if (!mbar_wait(full_bar(stage), phase, abort_flag, tmo)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t st = ring + stage * C::kStage;
            const int n_use = g.n - s0 < KS ? g.n - s0 : KS;
            for (int u = 0; u < n_use; ++u) {
              const uint32_t a_s =
                  g.asrc >= 2 ? (g.asrc == 2 ? htile : ltile) + static_cast<uint32_t>((s0 + u) * kSlabA)
                              : st + static_cast<uint32_t>(u * kSlabA);
              const uint32_t b_s = st + C::kA + static_cast<uint32_t>(u * C::kSlabB);
#pragma unroll
              for (int k = 0; k < 4; ++k) {  // the accumulator starts from C_l
                if (PAIR)
                  umma_bf16_pair(d_tmem, sdesc_kmajor_sw128(a_s + 32u * k),
                                 sdesc_kmajor_sw128(b_s + 32u * k), idesc, 1u);
                else
                  umma_bf16(d_tmem, sdesc_kmajor_sw128(a_s + 32u * k),
                            sdesc_kmajor_sw128(b_s + 32u * k), idesc, 1u);
              }
            }
            issued_any = true;
            if (PAIR)
              umma_commit_pair(empty_bar(stage), 0x3);
            else
              umma_commit(empty_bar(stage));
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
        if (!ok) break;
        if (PAIR)
          umma_commit_pair(accf_bar(acc), 0x3);
        else
          umma_commit(accf_bar(acc));
      }
      if (*abort_flag && issued_any) {  // no TMEM release while an MMA may still run
        if (PAIR)
          umma_commit_pair(drain_bar, 0x1);
        else
          umma_commit(drain_bar);
        wait_only(drain_bar, 0, tmo);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue warps
    const int qq = warp & 3;  // the TMEM lane quarter this warp may access
    const int row = qq * 32 + lane;
    const int t = row0 + row;
    const bool live = t < p.M;
    const uint32_t tl = tmem + (static_cast<uint32_t>(qq * 32) << 16);
    const float* crow = p.C + static_cast<long long>(live ? t : 0) * p.ldc;
    uint8_t* hrow = base_ptr + C::kOffH;
    uint8_t* lrow = base_ptr + C::kOffL;
    // At r_pad <= 128 a row of C_{l+2} (r_pad fp32) is fetched into registers one layer before it
    // goes into TMEM, so its global-memory latency is not on the per-layer chain.
    constexpr bool kAhead = RP <= 128;
    uint32_t cnext[kAhead ? RP / 32 : 1][32];
    // this row's 32 columns c*32 .. of C_lc (zero past the build's tokens)
    auto load_c = [&](int lc, int c, uint32_t (&r)[32]) {
      const float4* src = reinterpret_cast<const float4*>(crow + lc * RP + c * 32);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float4 v = live ? src[k] : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        r[4 * k] = __float_as_uint(v.x);
        r[4 * k + 1] = __float_as_uint(v.y);
        r[4 * k + 2] = __float_as_uint(v.z);
        r[4 * k + 3] = __float_as_uint(v.w);
      }
    };
    auto fetch_c = [&](int lc) {
      if constexpr (kAhead) {
#pragma unroll
        for (int c = 0; c < RP / 32; ++c) load_c(lc, c, cnext[c]);
      }
    };
    auto loaded = [&](int a) {  // accumulator a holds its C
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();
      if (PAIR) {  // one lane per warp on the leader's barrier, for the warp's 32 rows
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(map_to_rank(init_bar(a), 0));
      } else {
        mbar_arrive(init_bar(a));
      }
    };
    // C_lc into accumulator a, the starting value of layer lc's GEMM: from the registers fetched
    // a layer ahead, else straight from global memory
    auto put_c = [&](int lc, int a) {
      if constexpr (kAhead) {
        (void)lc;
#pragma unroll
        for (int c = 0; c < RP / 32; ++c) {
          __syncwarp();
          tmem_st32x(tl + static_cast<uint32_t>(a * RP + c * 32), cnext[c]);
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < RP / 32; ++c) {
          uint32_t r[32];
          load_c(lc, c, r);
          __syncwarp();
          tmem_st32x(tl + static_cast<uint32_t>(a * RP + c * 32), r);
        }
      }
      loaded(a);
    };
    // SiLU of the 32 columns c*32 .. of z into the h tile (bf16, swizzled as the MMA reads it);
    // split: the remainder h - bf16(h), itself in bf16, into the low tile
    auto put_h = [&](int c, const uint32_t (&r)[32]) {
      uint32_t pk[16], lo[16];
#pragma unroll
      for (int v = 0; v < 16; ++v) {
        const float a = silu(__uint_as_float(r[2 * v])), b = silu(__uint_as_float(r[2 * v + 1]));
        pk[v] = pack_bf16x2(a, b);
        if (SPLIT)
          lo[v] = pack_bf16x2(a - __uint_as_float(pk[v] << 16), b - __uint_as_float(pk[v] & 0xFFFF0000u));
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t off = static_cast<uint32_t>((c / 2) * kSlabA) + swz(row, (c % 2) * 4 + k);
        *reinterpret_cast<uint4*>(hrow + off) = make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]);
        if (SPLIT)
          *reinterpret_cast<uint4*>(lrow + off) = make_uint4(lo[4 * k], lo[4 * k + 1], lo[4 * k + 2], lo[4 * k + 3]);
      }
    };
    for (int l = 0; l < p.L; ++l) {
      if (l == 0) {  // z_0 = C_0
#pragma unroll 1
        for (int c = 0; c < RP / 32; ++c) {
          uint32_t r[32];
          load_c(0, c, r);
          put_h(c, r);
        }
      } else {
        const int acc = l & 1;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(accf_bar(acc), static_cast<uint32_t>((l - 1) >> 1) & 1u,
                                               abort_flag, tmo)))
          break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < RP / 32; ++c) {
          uint32_t r[32];
          __syncwarp();
          tmem_ld32(tl + static_cast<uint32_t>(acc * RP + c * 32), r);
          tmem_ld_wait();
          put_h(c, r);
        }
      }
      // The h tile first: layer l + 1's last MMAs wait for it (async proxy reads).
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      if (PAIR) {
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(map_to_rank(htile_bar, 0));
      } else {
        mbar_arrive(htile_bar);
      }
      // Then the accumulator just read starts layer l + 2 (before layer 1 both start), and the
      // C of the layer after that is fetched.
      if (l == 0) {
        if constexpr (kAhead) {
          if (p.L > 1) {
            fetch_c(1);
            put_c(1, 1);
          }
          if (p.L > 2) {
            fetch_c(2);
            put_c(2, 0);
          }
        } else {
          if (p.L > 1) put_c(1, 1);
          if (p.L > 2) put_c(2, 0);
        }
        if (p.L > 3) fetch_c(3);
      } else {
        if (l + 2 < p.L) put_c(l + 2, l & 1);
        if (l + 3 < p.L) fetch_c(l + 3);
      }
      // Last, the warp's 32 rows of h_l (and of its low part) go from the tiles to H by TMA;
      // complete before the tiles are rewritten and before the producer may read them back.
      // Rows past the build's tokens are clipped; a warp with none of them stores nothing.
      __syncwarp();
      if (lane == 0 && row0 + qq * 32 < p.M) {
#pragma unroll
        for (int sl = 0; sl < R; ++sl) {
          const uint32_t src = static_cast<uint32_t>(sl * kSlabA + qq * 32 * 128);
          tma_store_2d(&tmHst, htile + src, l * RP + 64 * sl, row0 + qq * 32);
          if (SPLIT) tma_store_2d(&tmHlost, ltile + src, l * RP + 64 * sl, row0 + qq * 32);
        }
        bulk_commit_wait();
      }
      __syncwarp();
      mbar_arrive(hpub_bar(l & 1));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) {
    if (PAIR) {  // this CTA's own copies still in flight land before the pair is torn down
      const uint64_t t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 200000ull) {
      }
    }
    atomicExch(p.status, DV_ERR_DEVICE_TIMEOUT);
  }
  if (PAIR) cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem, C::kTmemCols);
    else
      tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ---------------------------------------------------------------- (3) the running sum

// Shared staging of one warp's 32 x 32 bf16 block for its TMA store: 32 rows of 64 bytes, the
// 16-byte chunk q of row r at chunk q ^ ((r / 2) mod 4) (the tensor map's 64-byte swizzle). Two
// per warp, alternating, so that a block is staged while the previous one is still being read.
constexpr int kStageBytes = 32 * 64;

template <int RP, int CW, int STAGES, int EW>
struct ACfg {
  static constexpr int R = RP / 64;
  static constexpr int kThreads = 64 + 128 * EW;     // TMA warp, MMA warp, EW warps per lane quarter
  static constexpr int kEpiThreads = 128 * EW;
  static constexpr int kCols = CW / EW;              // hidden columns of one epilogue warp
  static constexpr int kSlabB = CW * 128;            // [CW rows of U_l][64] bf16
  static constexpr int kStage = 2 * kSlabA + kSlabB; // h slabs of the two token blocks, U slab
  static constexpr int kOffWarp = STAGES * kStage;   // per-warp staging of the M_l stores
  static constexpr int kEnd = kOffWarp + 4 * EW * 2 * kStageBytes;
  static_assert(kCols % 32 == 0 && CW / 64 >= EW, "whole 32-column chunks; parts fit d / 64");
  static constexpr int kSmemBytes = kEnd + 1024 + 256;
  static constexpr int kTmemCols = 2 * CW <= 256 ? 256 : 512;
  static_assert(kSlabB % 1024 == 0, "stage tiles stay 1024-byte aligned");
  static_assert(kSmemBytes <= 232448, "shared memory of one CTA");
};

struct AccumParams {
  int M;               // tokens
  int L;               // planned layers
  int d;
  int S;               // hidden slices (d / CW)
  const uint16_t* x0;  // bf16 [M][d]
  float* part;         // fp32 [L][part_ld / M][M]: sums of squares of M_l per CW / EW columns
  long long part_ld;
  int split;           // 1: h_l in two bf16 parts (H, then Hlo), both against U_l
  int* status;
  unsigned long long timeout_ns;
};

// CTA (pair of token blocks b, slice s) of the grid b * S + s: token blocks 2b and 2b + 1 (128
// rows each) and hidden columns [s CW, (s+1) CW); one TMEM accumulator per block. Each
// accumulator starts as the fp32 widening of E's slice (tcgen05.st); layer l adds h_l U_l^T
// (K = r_pad, the U slab staged once for both blocks) and is read back: bf16 M_l stored through
// the warp's staging (whole row segments per store instruction) and the row's sum of M_l^2 over
// the warp's CW / EW columns to part (slot s EW + e). EW warps share each TMEM lane quarter,
// each with its own columns, so that the loads, conversions and stores of several warps overlap
// on every SM sub-partition. Each block has its own barriers, so one block's next MMAs run while
// the other block's readback and stores go on.
template <int RP, int CW, int STAGES, int EW>
__global__ void __launch_bounds__(ACfg<RP, CW, STAGES, EW>::kThreads, 1)
    dv_accum_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmHlo,
                    const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmM,
                    const __grid_constant__ AccumParams p) {
  using C = ACfg<RP, CW, STAGES, EW>;
  constexpr int R = C::R;
  const int nq = p.split ? 2 * R : R;  // K slabs per layer: h_l (and its low part), 64 wide
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + C::kEnd);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto accf_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + b); };
  auto accr_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t ring = base;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t tmo = p.timeout_ns;
  const int pb = blockIdx.x / p.S, sl = blockIdx.x % p.S;
  const int row0 = pb * 256, col0 = sl * CW;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(accr_bar(b), C::kEpiThreads);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmH);
    tma_prefetch_desc(&tmU);
    if (p.split) tma_prefetch_desc(&tmHlo);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      int stage = 0;
      uint32_t phase = 0, used = 0, issued_parity = 0;
      bool ok = true;
      for (int l = 0; l < p.L && ok; ++l) {
        for (int q = 0; q < nq; ++q) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, tmo)) {
            ok = false;
            break;
          }
          const uint32_t dst = ring + stage * C::kStage;
          const CUtensorMap* ha = q < R ? &tmH : &tmHlo;
          const int kq = q % R;
          mbar_arrive_expect_tx(full_bar(stage), C::kStage);
          tma_load_2d(dst, ha, full_bar(stage), l * RP + 64 * kq, row0);
          tma_load_2d(dst + kSlabA, ha, full_bar(stage), l * RP + 64 * kq, row0 + 128);
          tma_load_2d(dst + 2 * kSlabA, &tmU, full_bar(stage), 64 * kq, l * p.d + col0);
          used |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*abort_flag) {
        for (int s = 0; s < STAGES; ++s)
          if (used & (1u << s)) wait_only(full_bar(s), (issued_parity >> s) & 1u, tmo);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      const uint32_t idesc = idesc_bf16_f32(128, CW);
      int stage = 0;
      uint32_t phase = 0;
      bool issued_any = false, ok = true;
      for (int l = 0; l < p.L && ok; ++l) {
        for (int q = 0; q < nq && ok; ++q) {
          if (!mbar_wait(full_bar(stage), phase, abort_flag, tmo)) {
            ok = false;
            break;
          }
          const uint32_t a0 = ring + stage * C::kStage, b_s = a0 + 2 * kSlabA;
          for (int b = 0; b < 2; ++b) {
            // block b's accumulator holds E (l = 0) or M_{l-1}, and its readback has left TMEM
            if (q == 0 && !mbar_wait(accr_bar(b), static_cast<uint32_t>(l) & 1u, abort_flag, tmo)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_s = a0 + static_cast<uint32_t>(b * kSlabA);
            const uint32_t d_tmem = tmem + static_cast<uint32_t>(b * CW);
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(d_tmem, sdesc_kmajor_sw128(a_s + 32u * k), sdesc_kmajor_sw128(b_s + 32u * k),
                        idesc, 1u);
            issued_any = true;
            if (q == nq - 1) umma_commit(accf_bar(b));
          }
          if (!ok) break;
          umma_commit(empty_bar(stage));
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*abort_flag && issued_any) {
        umma_commit(drain_bar);
        wait_only(drain_bar, 0, tmo);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue warps
    const int qq = warp & 3;          // the TMEM lane quarter this warp may access
    const int eh = (warp - 2) >> 2;   // which CW / EW columns of the quarter's rows
    const int row = qq * 32 + lane;
    const int cw0 = eh * C::kCols;    // the warp's first column in the slice
    const uint32_t tl = tmem + (static_cast<uint32_t>(qq * 32) << 16) + static_cast<uint32_t>(cw0);
    const uint32_t wstage = base + static_cast<uint32_t>(C::kOffWarp + (warp - 2) * 2 * kStageBytes);
    uint8_t* wstage_ptr = base_ptr + C::kOffWarp + (warp - 2) * 2 * kStageBytes;
    int nstored = 0;  // blocks this warp has stored: the staging buffer alternates with it
    // M_0 = E: the fp32 widening of this row's columns of E into both accumulators
#pragma unroll 1
    for (int b = 0; b < 2; ++b) {
      const int t = row0 + b * 128 + row;
      const uint16_t* xr = p.x0 + static_cast<long long>(t < p.M ? t : 0) * p.d + col0 + cw0;
#pragma unroll 1
      for (int c = 0; c < C::kCols / 32; ++c) {
        uint32_t r[32];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint4 w = t < p.M ? reinterpret_cast<const uint4*>(xr + c * 32)[k] : make_uint4(0, 0, 0, 0);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            r[k * 8 + 2 * e] = ws[e] << 16;
            r[k * 8 + 2 * e + 1] = ws[e] & 0xFFFF0000u;
          }
        }
        __syncwarp();
        tmem_st32x(tl + static_cast<uint32_t>(b * CW + c * 32), r);
      }
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    tc_fence_before();
    mbar_arrive(accr_bar(0));
    mbar_arrive(accr_bar(1));
    bool ok = true;
    for (int l = 0; l < p.L && ok; ++l) {
#pragma unroll 1
      for (int b = 0; b < 2; ++b) {
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(accf_bar(b), static_cast<uint32_t>(l) & 1u, abort_flag, tmo));
        if (!ok) break;
        tc_fence_after();
        // the warp's whole row segment leaves TMEM first, so the next layer's MMA can start
        uint32_t pk[C::kCols / 32][16];
        float ss = 0.0f;
#pragma unroll
        for (int c = 0; c < C::kCols / 32; ++c) {
          uint32_t r[32];
          __syncwarp();
          tmem_ld32(tl + static_cast<uint32_t>(b * CW + c * 32), r);
          tmem_ld_wait();
#pragma unroll
          for (int v = 0; v < 16; ++v) {
            const float x = __uint_as_float(r[2 * v]), y = __uint_as_float(r[2 * v + 1]);
            ss = fmaf(x, x, ss);
            ss = fmaf(y, y, ss);
            pk[c][v] = pack_bf16x2(x, y);
          }
        }
        tc_fence_before();
        mbar_arrive(accr_bar(b));
        const int t0 = row0 + b * 128 + qq * 32;  // the warp's first row
        // each 32 x 32 block: staged (lane i's row i, swizzled), then one TMA store by lane 0
        // (rows past the build's tokens are clipped by the map); before a buffer is restaged,
        // the store issued from it two blocks earlier has finished reading it
#pragma unroll
        for (int c = 0; c < C::kCols / 32; ++c, ++nstored) {
          const int sb = nstored & 1;
          if (lane == 0 && nstored >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
          __syncwarp();
          uint8_t* st = wstage_ptr + sb * kStageBytes;
#pragma unroll
          for (int q = 0; q < 4; ++q)
            *reinterpret_cast<uint4*>(st + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4)) =
                make_uint4(pk[c][4 * q], pk[c][4 * q + 1], pk[c][4 * q + 2], pk[c][4 * q + 3]);
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncwarp();
          if (lane == 0 && t0 < p.M) {
            asm volatile(
                "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                    reinterpret_cast<uint64_t>(&tmM)),
                "r"(wstage + static_cast<uint32_t>(sb * kStageBytes)), "r"(col0 + cw0 + c * 32), "r"(t0), "r"(l)
                : "memory");
          }
          if (lane == 0) asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        }
        if (t0 + lane < p.M)
          p.part[l * p.part_ld + static_cast<long long>(sl * EW + eh) * p.M + t0 + lane] = ss;
      }
    }
    // every store has left shared memory and reached global memory before the CTA exits
    if (lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, DV_ERR_DEVICE_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int RP, int KS, int ST, bool SPLIT>
cudaError_t hchain_t(long long blocks, const CUtensorMap& h, const CUtensorMap& hlo,
                     const CUtensorMap& pf, const CUtensorMap& pflo, const CUtensorMap& hst,
                     const CUtensorMap& hlost, const HChainParams& p, cudaStream_t stream) {
  // CTA pairs: two token blocks per cluster (the last pair may hold a block past the build)
  using C = HCfg<RP, KS, ST, SPLIT, true>;
  auto kern = dv_hchain_kernel<RP, KS, ST, SPLIT, true>;
  cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess || blocks <= 0) return err;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = pdl_attribute();
  cfg.gridDim = dim3(static_cast<unsigned>((blocks + 1) / 2 * 2), 1, 1);
  cfg.blockDim = dim3(kFoldThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, kern, h, hlo, pf, pflo, hst, hlost, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

template <int RP, int CW, int ST, int EW>
cudaError_t accum_t(long long ctas, const CUtensorMap& h, const CUtensorMap& hlo,
                    const CUtensorMap& u, const CUtensorMap& m, const AccumParams& p,
                    cudaStream_t stream) {
  using C = ACfg<RP, CW, ST, EW>;
  auto kern = dv_accum_kernel<RP, CW, ST, EW>;
  cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (err != cudaSuccess || ctas <= 0) return err;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas), 1, 1);
  cfg.blockDim = dim3(C::kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, kern, h, hlo, u, m, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace

int hchain_box_slabs(int r_pad, bool split) {
  return r_pad == 256 || (split && r_pad == 192) ? 1 : 2;
}

// A CTA of the running sum covers two token blocks and 256 hidden columns (128 where d is not a
// multiple of 256): the U slab it stages serves both blocks, and the two accumulators fill TMEM.
int fold_slice_cols(int d) {
  for (int cw : {256, 128})
    if (d % cw == 0) return cw;
  return 0;
}

// Two epilogue warps share each TMEM lane quarter of the running sum, each with half of the
// slice's columns and its own sum-of-squares slot: d / CW * 2 slots per layer.
int fold_sum_parts(int d) {
  const int cw = fold_slice_cols(d);
  return cw > 0 ? d / cw * kAccumWarps : 0;
}

cudaError_t launch_hchain(int r_pad, bool split, long long tokens, int n_layers, const float* C,
                          int ldc, const CUtensorMap& h, const CUtensorMap& hlo,
                          const CUtensorMap& pf, const CUtensorMap& pflo, const CUtensorMap& hst,
                          const CUtensorMap& hlost, uint16_t* H, uint16_t* Hlo, int ldh, int* status,
                          unsigned long long timeout_ns, cudaStream_t stream) {
  HChainParams p;
  p.M = static_cast<int>(tokens);
  p.L = n_layers;
  p.C = C;
  p.ldc = ldc;
  p.H = H;
  p.Hlo = Hlo;
  p.ldh = ldh;
  p.status = status;
  p.timeout_ns = timeout_ns;
  const long long blocks = (tokens + 127) / 128;
  // slabs per box (hchain_box_slabs) and pipeline stages; the split keeps a low h tile beside
  // the high one
  if (split) {
    switch (r_pad) {
      case 64: return hchain_t<64, 2, 4, true>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
      case 128: return hchain_t<128, 2, 3, true>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
      case 192: return hchain_t<192, 1, 4, true>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
      case 256: return hchain_t<256, 1, 3, true>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (r_pad) {
    case 64: return hchain_t<64, 2, 5, false>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
    case 128: return hchain_t<128, 2, 4, false>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
    case 192: return hchain_t<192, 2, 3, false>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
    case 256: return hchain_t<256, 1, 5, false>(blocks, h, hlo, pf, pflo, hst, hlost, p, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_accum(int r_pad, int cw, long long tokens, int n_layers, int d,
                         const void* x0, const CUtensorMap& h, const CUtensorMap& hlo, bool split,
                         const CUtensorMap& u, const CUtensorMap& mem, float* part, long long part_ld,
                         int* status, unsigned long long timeout_ns, cudaStream_t stream) {
  AccumParams p;
  p.M = static_cast<int>(tokens);
  p.L = n_layers;
  p.d = d;
  p.S = d / cw;
  p.x0 = static_cast<const uint16_t*>(x0);
  p.part = part;
  p.part_ld = part_ld;
  p.split = split ? 1 : 0;
  p.status = status;
  p.timeout_ns = timeout_ns;
  const long long ctas = (tokens + 255) / 256 * p.S;
#define DV_ACCUM(RPV, CWV, STV) \
  if (r_pad == RPV && cw == CWV) return accum_t<RPV, CWV, STV, kAccumWarps>(ctas, h, hlo, u, mem, p, stream);
  DV_ACCUM(64, 256, 3) DV_ACCUM(64, 128, 4)
  DV_ACCUM(128, 256, 3) DV_ACCUM(128, 128, 4)
  DV_ACCUM(192, 256, 3) DV_ACCUM(192, 128, 4)
  DV_ACCUM(256, 256, 3) DV_ACCUM(256, 128, 4)
#undef DV_ACCUM
  return cudaErrorInvalidValue;
}

}  // namespace dv
