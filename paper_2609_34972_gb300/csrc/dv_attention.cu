// Consumer of the visual memory (Sec. 3.2): the text queries of one layer attend causally to
// the keys/values of a KV cache that holds the visual K/V written by the build (and whatever
// text K/V the caller stored), O = softmax(scale * Q K^T, causal) V, as a tcgen05 flash-
// attention kernel. It reads the cache in place, through 4-D tensor maps over its strides
// (head_dim, kv head, slot, batch), so it checks the build's cache layout end to end.
//
// One cluster of S CTAs (S = 1, 2, 4 or 8) handles 128 query rows of one (batch, kv head):
// the rows of the kv head's query group (query head-major, then text token). The cluster's
// key range (up to the last slot any of its rows may see) is split into S runs of 128-key
// blocks. For each block a CTA:
//   1. loads the K and V tiles by TMA (rows = slots, 128 B per 64 channels, 128-byte swizzle);
//   2. one thread issues S = Q K^T (M = 128 rows, N = 128 keys, K = head_dim) into TMEM;
//   3. each thread owns one query row: it reads the row's 128 scores from TMEM at once, keeps
//      the running maximum m and sum l, and writes the row's probabilities exp2(scaled score -
//      m) as bf16 pairs back into TMEM over the first 64 score columns;
//   4. one thread issues O += P V (N = head_dim) with P (the A operand) read from TMEM and V
//      read as it lies ([keys][channels] rows, an MN-major B operand, no transpose). O stays in
//      TMEM over the CTA's key run; m is only moved (and O rescaled in TMEM) when the block
//      maximum exceeds it by more than 2^8, a bound on the probabilities, since O / l is the
//      same for any common reference maximum.
// With two stages the next block's K and V load during this block; with one stage the next K
// loads once the score MMA has read K, the next V once the P V MMA has read V.
// The partial (O, m, l) rows then go to the CTA that combines them, staged in shared memory and
// moved by bulk copies that complete on the receiver's barrier. CTA s combines rows
// [s * 128 / S, (s + 1) * 128 / S) over the S partials, in the fixed order 0..S-1, and stores
// bf16 rows: with two stages from a receive region of its own, with one stage (S = 2, two CTAs
// per SM) from its own registers and the peer's rows received over Q and K. Every wait is
// bounded; a CTA that gives up still passes the cluster barriers and flags the status word.
#include <cmath>
#include <mutex>

#include "../../include/dv.h"
#include "dv_internal.h"
#include "dv_ptx.cuh"

namespace dv {
namespace {

constexpr int kAttnThreads = 128;
constexpr int kKeyBlock = 128;

struct AttnParams {
  int Hq, Hkv, Nt, G;
  int rows_per_group;  // G * Nt query rows per kv head
  int q_blocks;        // 128-row blocks of one group
  int max_keys;
  const int* n_keys;   // [B]
  const int* q_slot;   // [B][Nt]
  float scale_log2;    // softmax scale * log2(e): scores are kept in base 2
  uint16_t* out;       // bf16 [B][Hq][Nt][head_dim]
  unsigned long long timeout_ns;
};

// Device status word of the attention launches on this device (DV_ERR_DEVICE_TIMEOUT when a
// wait gave up); read and cleared by dv_text_attention_status.
__device__ int g_attn_status;

// NST = 2: two stages of [K | V] (the next block loads during this one), one CTA per SM.
// NST = 1: one stage, small enough for two CTAs per SM; used in clusters of 2 where two stages
// could not split the keys at all.
template <int HD, int NST>
struct AttnCfg {
  static constexpr int kSlabs = HD / 64;
  static constexpr int kTile = 128 * 128;        // 128 rows x 64 bf16 (one 128-byte-swizzled slab)
  static constexpr int kKV = kSlabs * kTile;     // one K or V tile of 128 keys
  static constexpr int kOffQ = 0;
  static constexpr int kOffStage = kOffQ + kKV;  // NST stages of [K | V]
  static constexpr int kStage = 2 * kKV;
  static constexpr int kEnd = kOffStage + NST * kStage;  // P lives in TMEM, not here
  // TMEM: two score buffers (block j + 1's score MMA runs while block j finishes) and O at one
  // CTA per SM; one score buffer and O at two.
  static constexpr int kSBuf = NST == 2 ? 2 : 1;
  static constexpr int kTmemCols = NST == 2 ? 512 : 256;
  static constexpr int kTmemO = 128 * kSBuf;
  static constexpr int kMisc = 2048;                      // barriers, m, l, key end
  // Partial outputs received from the cluster: 128 rows of HD fp32 (16-byte chunks swizzled by
  // the row, no padding). With two stages they get a region of their own, so peers may write
  // them while this CTA still computes; the one-stage variant reuses Q and its stage.
  static constexpr int kRecvBytes = 128 * HD * 4;
  static constexpr bool kRecvOwn = NST == 2;
  static constexpr int kOffRecv = kRecvOwn ? kEnd + kMisc : kOffQ;
  static constexpr int kSmemBytes = kEnd + kMisc + (kRecvOwn ? kRecvBytes : 0) + 1024;
  static_assert(kRecvOwn || kRecvBytes <= kKV + NST * kStage, "partials reuse Q and the stage");
  // Two stages: the rows sent to peers are staged in Q and the stages (free after the key run),
  // their maxima and sums right after them.
  static constexpr int kOffSendML = kOffQ + kRecvBytes;
  static_assert(kOffSendML + 1024 <= kKV + NST * kStage, "staged partials fit Q and the stages");
  // One stage (S = 2): 64 rows received over Q and K, 64 staged after them; their m and l lists
  // at kEnd + 256 and kEnd + 1280 (512 bytes each).
  static_assert(NST == 2 || 2 * 64 * HD * 4 <= kKV + kStage, "one-stage exchange fits Q, K, V");
  static constexpr int kOffSendML1 = kEnd + 1280;
  static_assert(kKV % 1024 == 0, "tiles stay 1024-byte aligned");
  static_assert(kSmemBytes <= 232448, "shared memory of one CTA");
};

// 4-D tiled load (c0 innermost); completion counted as transaction bytes on `bar`.
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}

// 4-D tiled prefetch of one box into L2 (no shared memory, no completion).
__device__ __forceinline__ void tma_prefetch_l2_4d(const CUtensorMap* map, int c0, int c1, int c2,
                                                   int c3) {
  asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}

// Shared-memory descriptor of an MN-major operand written by TMA with 128-byte swizzling, as V
// lies in shared memory for the P V MMA: each 128-byte row holds 64 consecutive N elements
// (channels) of one K index (key); 8-row (8-key) swizzle atoms are 1024 B apart along K (stride
// byte offset) and the next 64 N elements sit `n_stride` bytes further (leading byte offset).
__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr, uint32_t n_stride) {
  uint64_t desc = 0;
  desc |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  desc |= static_cast<uint64_t>((n_stride >> 4) & 0x3FFFu) << 16;
  desc |= static_cast<uint64_t>(1024 >> 4) << 32;
  desc |= static_cast<uint64_t>(1) << 46;
  desc |= static_cast<uint64_t>(2) << 61;
  return desc;
}

// Orders this thread's generic-proxy shared-memory writes before later async-proxy reads
// (tcgen05.mma operands) of the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// D (+)= A B with A (M x 16, K-major, bf16) in TMEM at `a_tmem` (lane = row, column c = the
// bf16 pair k = 2c, 2c + 1) and B from shared memory.
__device__ __forceinline__ void umma_bf16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Largest growth (base 2) of a row's maximum absorbed without rescaling O: probabilities
// relative to a stale maximum stay <= 2^8, far inside bf16 and fp32 range.
constexpr float kRescaleLog2 = 8.0f;

__device__ __forceinline__ float ex2_approx(float x) {  // 2^x (PTX ex2.approx, -inf -> +0)
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t (&chunk32(uint32_t* r, int c))[32] {
  return *reinterpret_cast<uint32_t(*)[32]>(r + 32 * c);
}

// Uses of registers loaded by tcgen05.ld stay after tcgen05.wait::ld: the empty statement
// (ordered after the wait like every volatile asm) redefines them.
__device__ __forceinline__ void reg_fence32(uint32_t (&r)[32]) {
  asm volatile(""
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                 "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                 "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                 "+r"(r[30]), "+r"(r[31]));
}

// Warp-wide registers -> TMEM, the inverse of tmem_ld32 (lane i writes TMEM lane taddr.lane + i).
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

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  int never = 0;
  return mbar_wait<false>(bar, parity, &never, timeout_ns);
}

// Partial rows travel between the CTAs of a cluster as fp32 rows of HD / 4 16-byte chunks,
// chunk c of row R stored at chunk position c ^ rev3(R mod 8) (rev3 reverses 3 bits). Eight
// consecutive rows writing one chunk, and the combine's reads (S threads of a row on
// consecutive chunks, 8 / S rows per quarter warp), then touch 8 distinct bank groups.
__device__ __forceinline__ uint32_t chunk_swizzle(int R) {
  return static_cast<uint32_t>(((R & 1) << 2) | (R & 2) | ((R >> 2) & 1));
}

// Thread `tid` holds query row tid of this CTA's key run: (o, m, l). Row tid is combined by CTA
// d = tid / rows (rows = 128 / S, a multiple of 8, so a row's chunk swizzle is that of tid mod
// rows); its maximum and sum travel as lists [source][m | l][row].
__device__ __forceinline__ void bulk_copy_to_peer(uint32_t dst_cluster, uint32_t src, uint32_t bytes,
                                                  uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst_cluster), "r"(src), "r"(bytes), "r"(bar_cluster)
      : "memory");
}

// Two-stage variant: receive rows R = source * rows + row in a region of their own. Rows for a
// peer are staged in this CTA's shared memory (`send`, `send_ml`, laid out as the peer will hold
// them), this CTA's own rows go straight into its receive rows, and one thread moves each
// peer's share with two bulk copies, which complete on the peer's receive barrier. Bulk copies
// move the 16 KB shares about twice as fast as per-thread remote stores. Precondition: every
// CTA of the cluster has initialised its receive barrier (the caller's cluster wait).
template <int HD>
__device__ __forceinline__ void stage_partial(const float* o, float m_run, float l_run,
                                              uint32_t recv, uint32_t recv_ml, uint32_t send,
                                              uint32_t send_ml, int split, int S) {
  const int tid = threadIdx.x, rows = 128 / S;
  const int d = tid / rows, rr = tid % rows;
  const uint32_t sw = chunk_swizzle(tid);
  const bool mine = d == split;
  const uint32_t row = mine ? recv + static_cast<uint32_t>(split * rows + rr) * (HD * 4)
                            : send + static_cast<uint32_t>(tid) * (HD * 4);
  const uint32_t ml = (mine ? recv_ml + 4u * (2 * split * rows) : send_ml + 4u * (2 * d * rows)) +
                      4u * rr;
#pragma unroll
  for (int c = 0; c < HD / 4; ++c) {
    float4* dst = reinterpret_cast<float4*>(__cvta_shared_to_generic(row + ((c ^ sw) << 4)));
    *dst = make_float4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
  }
  *reinterpret_cast<float*>(__cvta_shared_to_generic(ml)) = m_run;
  *reinterpret_cast<float*>(__cvta_shared_to_generic(ml + 4u * rows)) = l_run;
  fence_proxy_async_smem();  // the staged rows are read by the bulk copies (async proxy)
}

// Query rows of its 128 / S that CTA d combines and stores: those of the tile's `tile_rows`
// valid rows (rows past the query group are never stored, so they are neither sent nor
// combined). Sender and receiver use this same count.
__device__ __forceinline__ int rows_combined(int tile_rows, int d, int S) {
  const int rows = 128 / S;
  return max(0, min(rows, tile_rows - d * rows));
}

// Bytes CTA `d` receives from each peer: its valid rows, then all m and l of its rows.
template <int HD>
__device__ __forceinline__ uint32_t bytes_from_peer(int tile_rows, int d, int S) {
  const int n = rows_combined(tile_rows, d, S);
  return n > 0 ? static_cast<uint32_t>(n * HD * 4 + 8 * (128 / S)) : 0u;
}

template <int HD>
__device__ __forceinline__ void send_partial(uint32_t recv, uint32_t recv_ml, uint32_t send,
                                             uint32_t send_ml, uint32_t bar_recv, int split,
                                             int S, int tile_rows) {
  const int rows = 128 / S;
  for (int dd = 0; dd < S; ++dd) {
    const int n = rows_combined(tile_rows, dd, S);
    if (dd == split || n == 0) continue;
    const uint32_t rank = static_cast<uint32_t>(dd), cbar = map_to_rank(bar_recv, rank);
    bulk_copy_to_peer(map_to_rank(recv + static_cast<uint32_t>(split * rows) * (HD * 4), rank),
                      send + static_cast<uint32_t>(dd * rows) * (HD * 4),
                      static_cast<uint32_t>(n * HD * 4), cbar);
    bulk_copy_to_peer(map_to_rank(recv_ml + 4u * (2 * split * rows), rank),
                      send_ml + 4u * (2 * dd * rows), static_cast<uint32_t>(8 * rows), cbar);
  }
}

// One-stage variant (S = 2, the shared memory of two CTAs per SM): a CTA's own rows stay in
// the registers of the threads that hold them, so it receives only its S - 1 peers' rows, in
// slots of `rows` rows (peer s in slot s, or s - 1 past this CTA's rank), over Q and the K slot
// (free once every key run of the cluster has ended). Rows for peer d are staged after them,
// in slots numbered the same way (d, or d - 1 past this CTA's rank).
__device__ __forceinline__ int peer_slot(int s, int self) { return s < self ? s : s - 1; }

template <int HD>
__device__ __forceinline__ void stage_peer_rows(const float* o, float m_run, float l_run,
                                                uint32_t send, uint32_t send_ml, int split, int S) {
  const int tid = threadIdx.x, rows = 128 / S;
  const int d = tid / rows, rr = tid % rows;
  if (d == split) return;
  const int di = peer_slot(d, split);
  const uint32_t sw = chunk_swizzle(rr);
  const uint32_t row = send + static_cast<uint32_t>(di * rows + rr) * (HD * 4);
#pragma unroll
  for (int c = 0; c < HD / 4; ++c) {
    float4* dst = reinterpret_cast<float4*>(__cvta_shared_to_generic(row + ((c ^ sw) << 4)));
    *dst = make_float4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
  }
  const uint32_t ml = send_ml + 4u * (2 * di * rows + rr);
  *reinterpret_cast<float*>(__cvta_shared_to_generic(ml)) = m_run;
  *reinterpret_cast<float*>(__cvta_shared_to_generic(ml + 4u * rows)) = l_run;
  fence_proxy_async_smem();  // the staged rows are read by the bulk copies (async proxy)
}

template <int HD>
__device__ __forceinline__ void send_peer_rows(uint32_t recv, uint32_t recv_ml, uint32_t send,
                                               uint32_t send_ml, uint32_t bar_recv, int split,
                                               int S, int tile_rows) {
  const int rows = 128 / S;
  for (int dd = 0; dd < S; ++dd) {
    const int n = rows_combined(tile_rows, dd, S);
    if (dd == split || n == 0) continue;
    const int di = peer_slot(dd, split), slot = peer_slot(split, dd);
    const uint32_t rank = static_cast<uint32_t>(dd), cbar = map_to_rank(bar_recv, rank);
    bulk_copy_to_peer(map_to_rank(recv + static_cast<uint32_t>(slot * rows) * (HD * 4), rank),
                      send + static_cast<uint32_t>(di * rows) * (HD * 4),
                      static_cast<uint32_t>(n * HD * 4), cbar);
    bulk_copy_to_peer(map_to_rank(recv_ml + 4u * (2 * slot * rows), rank),
                      send_ml + 4u * (2 * di * rows), static_cast<uint32_t>(8 * rows), cbar);
  }
}

// The threads holding this CTA's own rows combine them: own partial from registers, the peers'
// from the receive slots, summed in the fixed order of the sources 0 .. S-1.
template <int HD, int S>
__device__ __forceinline__ void combine_own_rows(const float* o, float m_run, float l_run,
                                                 uint32_t recv, const float* recv_ml, int split,
                                                 int qb, int h, int b, const AttnParams& p) {
  constexpr int kRows = 128 / S;
  const int tid = threadIdx.x;
  if (tid / kRows != split) return;
  const int rr = tid % kRows, ii = qb * 128 + tid;
  if (ii >= p.rows_per_group) return;
  const uint32_t sw = chunk_swizzle(rr);
  float ms[S], ls[S], w[S];
  uint32_t prow[S];
#pragma unroll
  for (int s = 0; s < S; ++s) {
    if (s == split) {
      ms[s] = m_run;
      ls[s] = l_run;
      prow[s] = 0;
    } else {
      const int slot = peer_slot(s, split);
      ms[s] = recv_ml[(2 * slot) * kRows + rr];
      ls[s] = recv_ml[(2 * slot + 1) * kRows + rr];
      prow[s] = recv + static_cast<uint32_t>(slot * kRows + rr) * (HD * 4);
    }
  }
  float M = -INFINITY;
#pragma unroll
  for (int s = 0; s < S; ++s) M = fmaxf(M, ms[s]);
  float L = 0.0f;
#pragma unroll
  for (int s = 0; s < S; ++s) {
    w[s] = ms[s] != -INFINITY ? exp2f(ms[s] - M) : 0.0f;
    L = fmaf(w[s], ls[s], L);
  }
  const float inv = L > 0.0f ? 1.0f / L : 0.0f;
  const int hq = h * p.G + ii / p.Nt, t = ii % p.Nt;
  uint16_t* orow = p.out + ((static_cast<size_t>(b) * p.Hq + hq) * p.Nt + t) * HD;
#pragma unroll
  for (int c2 = 0; c2 < HD / 8; ++c2) {
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
#pragma unroll
    for (int s = 0; s < S; ++s) {
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int c = 2 * c2 + h2;
        float4 v;
        if (s == split) {
          v = make_float4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
        } else {
          v = *reinterpret_cast<const float4*>(
              __cvta_shared_to_generic(prow[s] + ((static_cast<uint32_t>(c) ^ sw) << 4)));
        }
        acc[4 * h2] = fmaf(w[s], v.x, acc[4 * h2]);
        acc[4 * h2 + 1] = fmaf(w[s], v.y, acc[4 * h2 + 1]);
        acc[4 * h2 + 2] = fmaf(w[s], v.z, acc[4 * h2 + 2]);
        acc[4 * h2 + 3] = fmaf(w[s], v.w, acc[4 * h2 + 3]);
      }
    }
    uint4 out;
    out.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
    out.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
    out.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
    out.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
    *reinterpret_cast<uint4*>(orow + c2 * 8) = out;
  }
}

// Combine of the S key runs of a cluster from this CTA's receive rows: CTA `split` owns query
// rows [split * 128 / S, (split + 1) * 128 / S); S threads per row, thread j taking chunks j,
// j + S, j + 2 S, ...; the S partials are summed in the fixed order 0 .. S-1.
template <int HD, int S>
__device__ __forceinline__ void combine_rows(uint32_t recv, const float* recv_ml, int split,
                                             int qb, int h, int b, const AttnParams& p) {
  constexpr int kRows = 128 / S, kTpr = kAttnThreads / kRows, kPer = HD / 4 / kTpr;
  const int tid = threadIdx.x;
  const int rr = tid / kTpr, j = tid % kTpr;
  const int ii = qb * 128 + split * kRows + rr;
  if (ii >= p.rows_per_group) return;
  const uint32_t sw = chunk_swizzle(rr);  // rows R = s * kRows + rr share rr mod 8
  float ms[S], ls[S], w[S];
#pragma unroll
  for (int s = 0; s < S; ++s) {
    ms[s] = recv_ml[(2 * s) * kRows + rr];
    ls[s] = recv_ml[(2 * s + 1) * kRows + rr];
  }
  float M = -INFINITY;
#pragma unroll
  for (int s = 0; s < S; ++s) M = fmaxf(M, ms[s]);
  float L = 0.0f;
#pragma unroll
  for (int s = 0; s < S; ++s) {
    w[s] = ms[s] != -INFINITY ? exp2f(ms[s] - M) : 0.0f;
    L = fmaf(w[s], ls[s], L);
  }
  const float inv = L > 0.0f ? 1.0f / L : 0.0f;
  const int hq = h * p.G + ii / p.Nt, t = ii % p.Nt;
  uint16_t* orow = p.out + ((static_cast<size_t>(b) * p.Hq + hq) * p.Nt + t) * HD;
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int c = i * kTpr + j;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const uint32_t a = recv + static_cast<uint32_t>(s * kRows + rr) * (HD * 4) +
                         ((static_cast<uint32_t>(c) ^ sw) << 4);
      const float4 v = *reinterpret_cast<const float4*>(__cvta_shared_to_generic(a));
      acc.x = fmaf(w[s], v.x, acc.x);
      acc.y = fmaf(w[s], v.y, acc.y);
      acc.z = fmaf(w[s], v.z, acc.z);
      acc.w = fmaf(w[s], v.w, acc.w);
    }
    uint2 out;
    out.x = pack_bf16x2(acc.x * inv, acc.y * inv);
    out.y = pack_bf16x2(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(orow + c * 4) = out;
  }
}

template <int HD, int NST>
__global__ void __launch_bounds__(kAttnThreads, 1)
    dv_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnParams p) {
  using C = AttnCfg<HD, NST>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + C::kEnd);
  const uint32_t bar0 = smem_addr(bars);
  // barriers: Q, K of stage 0/1, V of stage 0/1, scores ready, block output ready, drain
  const uint32_t bar_q = bar0, bar_s = bar0 + 40, bar_o = bar0 + 48, bar_drain = bar0 + 56;
  const uint32_t bar_recv = bar0 + 80;  // partial rows received from the peers
  auto bar_k = [&](int st) { return bar0 + 8u + 8u * st; };
  auto bar_v = [&](int st) { return bar0 + 24u + 8u * st; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* key_end = reinterpret_cast<int*>(tmem_slot + 2);
  float* recv_ml = reinterpret_cast<float*>(base_ptr + C::kEnd + 256);  // [S][m | l][128 / S]
  const uint32_t recv = base + C::kOffRecv;

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint64_t tmo = p.timeout_ns;
  const int split = static_cast<int>(cluster_ctarank());
  const int S = static_cast<int>(cluster_size());
  const int unit = static_cast<int>(cluster_id_x());
  const int qb = unit % p.q_blocks;
  const int h = (unit / p.q_blocks) % p.Hkv;
  const int b = unit / (p.q_blocks * p.Hkv);
  const int tile_rows = min(128, p.rows_per_group - qb * 128);  // valid query rows of the tile

  if (tid == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    mbar_init(bar_q, 1);
    for (int st = 0; st < 2; ++st) {
      mbar_init(bar_k(st), 1);
      mbar_init(bar_v(st), 1);
    }
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_drain, 1);
    mbar_init(bar_recv, 1);
    mbar_arrive_expect_tx(bar_recv,
                          static_cast<uint32_t>(S - 1) * bytes_from_peer<HD>(tile_rows, split, S));
    *abort_flag = 0;
    *key_end = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // Peers send into this CTA's receive rows and barrier as soon as their own key runs end; this
  // arrival (waited for before they send) tells them that the barrier is initialised.
  if (C::kRecvOwn) asm volatile("barrier.cluster.arrive.aligned;" ::: "memory");
  // The launch may start while the previous kernel of the stream still runs (dependent launch):
  // the prologue above touches no global memory; everything below comes after its completion.
  pdl_wait();
  pdl_trigger();

  // Q does not depend on the key range: it loads while the range is found. So does the first
  // K/V block this CTA would take if the keys filled the cache (max_keys), prefetched into L2;
  // a wrong guess costs only L2 bandwidth.
  const int q_row0 = (b * p.Hq + h * p.G) * p.Nt + qb * 128;
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_q, C::kKV);
    for (int ds = 0; ds < C::kSlabs; ++ds)
      tma_load_2d(base + C::kOffQ + ds * C::kTile, &tmQ, bar_q, ds * 64, q_row0);
    const int nb_guess = (p.max_keys + kKeyBlock - 1) / kKeyBlock;
    const int kb_guess = split * nb_guess / S;
    if (kb_guess < (split + 1) * nb_guess / S) {
      for (int ds = 0; ds < C::kSlabs; ++ds) {
        tma_prefetch_l2_4d(&tmK, ds * 64, h, kb_guess * kKeyBlock, b);
        tma_prefetch_l2_4d(&tmV, ds * 64, h, kb_guess * kKeyBlock, b);
      }
    }
  }

  // This thread's query row and the last slot it may see; the CTA's key end is the maximum.
  const int i = qb * 128 + tid;
  const int nk = min(p.n_keys[b], p.max_keys);
  int last = -1;
  if (i < p.rows_per_group) last = min(p.q_slot[b * p.Nt + i % p.Nt], nk - 1);
  const int warp_end = __reduce_max_sync(0xFFFFFFFFu, last + 1);
  if ((tid & 31) == 0) atomicMax(key_end, warp_end);
  __syncthreads();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_o = tmem + C::kTmemO;
  auto t_s = [&](int j) { return tmem + static_cast<uint32_t>((j % C::kSBuf) * 128); };
  const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
  const int n_blocks = (*key_end + kKeyBlock - 1) / kKeyBlock;
  const int kb0 = split * n_blocks / S, kb1 = (split + 1) * n_blocks / S;

  const uint32_t sQ = base + C::kOffQ;
  auto sK = [&](int st) { return base + C::kOffStage + st * C::kStage; };
  auto sV = [&](int st) { return base + C::kOffStage + st * C::kStage + C::kKV; };
  // K or V of block kb0 + j into stage j % NST (thread 0); last_k / last_v: the latest blocks
  // whose K and V loads were issued, waited for before the memory is reused after an abort.
  int last_k = -1, last_v = -1;
  auto load_k = [&](int j) {
    const int st = j % NST, kb = kb0 + j;
    mbar_arrive_expect_tx(bar_k(st), C::kKV);
    for (int ds = 0; ds < C::kSlabs; ++ds)
      tma_load_4d(sK(st) + ds * C::kTile, &tmK, bar_k(st), ds * 64, h, kb * kKeyBlock, b);
    last_k = j;
  };
  auto load_v = [&](int j) {
    const int st = j % NST, kb = kb0 + j;
    mbar_arrive_expect_tx(bar_v(st), C::kKV);
    for (int ds = 0; ds < C::kSlabs; ++ds)
      tma_load_4d(sV(st) + ds * C::kTile, &tmV, bar_v(st), ds * 64, h, kb * kKeyBlock, b);
    last_v = j;
  };
  auto issue_s = [&](int j) {  // thread 0: S_j = Q K_j^T into score buffer j % kSBuf
    const int st = j % NST;
    if (mbar_wait<false>(bar_q, 0, abort_flag, tmo) &&
        mbar_wait<false>(bar_k(st), static_cast<uint32_t>(j / NST) & 1u, abort_flag, tmo)) {
      tc_fence_after();
      const uint32_t idesc = idesc_bf16_f32(128, kKeyBlock);
      for (int ds = 0; ds < C::kSlabs; ++ds)
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_bf16(t_s(j), sdesc_kmajor_sw128(sQ + ds * C::kTile + 32u * k),
                    sdesc_kmajor_sw128(sK(st) + ds * C::kTile + 32u * k), idesc,
                    (ds | k) != 0 ? 1u : 0u);
      umma_commit(bar_s);
    }
  };

  float m_run = -INFINITY, l_run = 0.0f;

  const int n_mine = kb1 - kb0;
  if (tid == 0 && n_mine > 0) {
    load_k(0);
    load_v(0);
    issue_s(0);
  }

  bool ok = true;
  for (int j = 0; j < n_mine && ok; ++j) {
    const int st = j % NST, kb = kb0 + j;
    const uint32_t sph = static_cast<uint32_t>(j / NST) & 1u;  // phase of this stage's barriers
    const uint32_t ph = static_cast<uint32_t>(j) & 1u;        // phase of bar_s / bar_o
    // Two stages: the other stage was freed by the previous block. One stage: K of this block
    // was issued once the previous score MMA had read K, V once the previous P V MMA had read V.
    // S_j itself was issued with the previous block (or before the loop).
    if (NST == 2 && tid == 0 && j + 1 < n_mine) {
      load_k(j + 1);
      load_v(j + 1);
    }

    // Scores -> probabilities (this thread: query row tid).
    ok = mbar_wait<false>(bar_s, ph, abort_flag, tmo);
    if (NST == 1 && tid == 0 && ok && j + 1 < n_mine) load_k(j + 1);  // K slot read
    if (__all_sync(0xFFFFFFFFu, ok)) {
      tc_fence_after();
      // the row's 128 scores in one TMEM round trip; keys past the row's last slot are masked
      uint32_t r[kKeyBlock];
#pragma unroll
      for (int c = 0; c < kKeyBlock / 32; ++c) tmem_ld32(t_s(j) + lane_base + c * 32, chunk32(r, c));
      tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < kKeyBlock / 32; ++c) reg_fence32(chunk32(r, c));
      // raw scores; the scale (> 0) is applied after the maximum and inside the exponent
      const int n_valid = last - kb * kKeyBlock + 1;
      float x[kKeyBlock];
      if (n_valid >= kKeyBlock) {
#pragma unroll
        for (int u = 0; u < kKeyBlock; ++u) x[u] = __uint_as_float(r[u]);
      } else {
#pragma unroll
        for (int u = 0; u < kKeyBlock; ++u) x[u] = u < n_valid ? __uint_as_float(r[u]) : -INFINITY;
      }
      float mx[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx[u] = x[u];
#pragma unroll
      for (int u = 8; u < kKeyBlock; ++u) mx[u % 8] = fmaxf(mx[u % 8], x[u]);
      const float mb = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                             fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7]))) *
                       p.scale_log2;
      const float m_new = fmaxf(m_run, mb);
      // The row keeps its reference maximum while the new scores exceed it by at most
      // kRescaleLog2 (probabilities stay <= 2^kRescaleLog2); O and l only need the same
      // reference, so O in TMEM is rescaled only when the maximum grows by more than that.
      // A row that has seen no key yet (m_run = -inf) has O = 0 and l = 0: it takes the new
      // maximum with nothing to rescale.
      float alpha = 1.0f, m_use = m_run;
      if (m_run == -INFINITY) {
        m_use = m_new;
      } else if (m_new > m_run + kRescaleLog2) {
        alpha = ex2_approx(m_run - m_new);
        m_use = m_new;
      }
      if (__any_sync(0xFFFFFFFFu, alpha != 1.0f)) {  // rows of this warp whose reference moved
#pragma unroll 1
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t q[32];
          tmem_ld32(t_o + lane_base + c * 32, q);
          tmem_ld_wait();
          reg_fence32(q);
#pragma unroll
          for (int u = 0; u < 32; ++u) q[u] = __float_as_uint(__uint_as_float(q[u]) * alpha);
          tmem_st32(t_o + lane_base + c * 32, q);
        }
        tmem_st_wait();
      }
      const float m_sub = m_use == -INFINITY ? 0.0f : m_use;
      // P as bf16 pairs (keys 2c, 2c + 1 in column c) over the first 64 score columns: the A
      // operand of the P V MMA, read from TMEM (the scores are all in registers by now).
      float lb[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int c = 0; c < kKeyBlock / 64; ++c) {
        uint32_t pk[32];
#pragma unroll
        for (int u = 0; u < 64; u += 2) {
          const float p0 = ex2_approx(fmaf(x[c * 64 + u], p.scale_log2, -m_sub));
          const float p1 = ex2_approx(fmaf(x[c * 64 + u + 1], p.scale_log2, -m_sub));
          lb[(u / 2) % 4] += p0 + p1;
          pk[u / 2] = pack_bf16x2(p0, p1);
        }
        tmem_st32(t_s(j) + lane_base + c * 32, pk);
      }
      tmem_st_wait();
      l_run = alpha * l_run + ((lb[0] + lb[1]) + (lb[2] + lb[3]));
      m_run = m_use;
    }
    tc_fence_before();
    ok = __syncthreads_and(ok) != 0;

    // O (+)= P V in TMEM; the CTA's first block initialises O. V is read as it lies ([keys]
    // [channels], an MN-major B operand); P (A, K-major) from TMEM, 16 keys = 8 columns.
    if (ok && tid == 0 && mbar_wait<false>(bar_v(st), sph, abort_flag, tmo)) {
      tc_fence_after();
      const uint32_t idesc = idesc_bf16_f32(128, HD) | (1u << 16);
#pragma unroll
      for (int kk = 0; kk < kKeyBlock / 16; ++kk)
        umma_bf16_tmem_a(t_o, t_s(j) + kk * 8,
                         sdesc_mnmajor_sw128(sV(st) + kk * 16 * 128, C::kTile), idesc,
                         (j | kk) != 0 ? 1u : 0u);
      umma_commit(bar_o);
      // Two score buffers: S_{j+1} runs behind P V (its buffer's P_{j-1} was read by the previous
      // P V, which has completed).
      if (C::kSBuf == 2 && j + 1 < n_mine) issue_s(j + 1);
    }
    ok = ok && mbar_wait<false>(bar_o, ph, abort_flag, tmo);
    if (NST == 1 && tid == 0 && ok && j + 1 < n_mine) {
      load_v(j + 1);  // V slot read
      issue_s(j + 1);  // P_j (in the one score buffer) read
    }
    tc_fence_before();
    ok = __syncthreads_and(ok) != 0;
  }

  // This CTA's partial output rows (O relative to m_run, unnormalised) out of TMEM.
  float o[HD];
  if (ok && n_mine > 0) {
    tc_fence_after();
    uint32_t ob[HD];
#pragma unroll
    for (int c = 0; c < HD / 32; ++c) tmem_ld32(t_o + lane_base + c * 32, chunk32(ob, c));
    tmem_ld_wait();
#pragma unroll
    for (int c = 0; c < HD / 32; ++c) reg_fence32(chunk32(ob, c));
#pragma unroll
    for (int d = 0; d < HD; ++d) o[d] = __uint_as_float(ob[d]);
  } else {
#pragma unroll
    for (int d = 0; d < HD; ++d) o[d] = 0.0f;
  }

  if (!ok && tid == 0) {
    // Let the copies in flight (the last block issued on each stage) land and every issued MMA
    // finish before the memory is reused; each wait targets its stage's latest phase.
    for (int jj = last_k; jj >= 0 && jj > last_k - NST; --jj)
      wait_bounded(bar_k(jj % NST), static_cast<uint32_t>(jj / NST) & 1u, tmo);
    for (int jj = last_v; jj >= 0 && jj > last_v - NST; --jj)
      wait_bounded(bar_v(jj % NST), static_cast<uint32_t>(jj / NST) & 1u, tmo);
    umma_commit(bar_drain);
    wait_bounded(bar_drain, 0, tmo);
  }
  // Q was loaded in every CTA; its memory is reused below.
  if (tid == 0) wait_bounded(bar_q, 0, tmo);
  __syncthreads();

  // Partial (O, m, l) of this CTA's key run -> the CTA that combines each row, by bulk copies
  // that complete on the receiver's barrier; the waits for them are not cut short by the abort
  // flag, since the copies into a CTA must land before it may exit. Once every CTA has seen
  // its copies land (the cluster barrier before exit), no copy touches any CTA's memory.
  if (C::kRecvOwn) {
    stage_partial<HD>(o, m_run, l_run, recv, smem_addr(recv_ml), base + C::kOffQ,
                      base + C::kOffSendML, split, S);
    __syncthreads();
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");  // peers' barriers initialised
    if (tid == 0)
      send_partial<HD>(recv, smem_addr(recv_ml), base + C::kOffQ, base + C::kOffSendML, bar_recv,
                       split, S, tile_rows);
    if (!wait_bounded(bar_recv, 0, tmo)) *abort_flag = 1;
    __syncwarp();
    asm volatile("barrier.cluster.arrive.aligned;" ::: "memory");
    switch (S) {  // the cluster size: 1, 2, 4 or 8
      case 1: combine_rows<HD, 1>(recv, recv_ml, split, qb, h, b, p); break;
      case 2: combine_rows<HD, 2>(recv, recv_ml, split, qb, h, b, p); break;
      case 4: combine_rows<HD, 4>(recv, recv_ml, split, qb, h, b, p); break;
      default: combine_rows<HD, 8>(recv, recv_ml, split, qb, h, b, p); break;
    }
  } else {  // one stage: S = 2
    const int rows = 128 / S;
    const uint32_t send = base + static_cast<uint32_t>((128 - rows) * HD * 4);
    const uint32_t send_ml = base + C::kOffSendML1;
    stage_peer_rows<HD>(o, m_run, l_run, send, send_ml, split, S);
    __syncthreads();
    cluster_sync();  // every key run of the cluster has ended: Q and K may receive
    if (tid == 0)
      send_peer_rows<HD>(recv, smem_addr(recv_ml), send, send_ml, bar_recv, split, S, tile_rows);
    if (!wait_bounded(bar_recv, 0, tmo)) *abort_flag = 1;
    __syncwarp();
    asm volatile("barrier.cluster.arrive.aligned;" ::: "memory");
    combine_own_rows<HD, 2>(o, m_run, l_run, recv, recv_ml, split, qb, h, b, p);
  }
  __syncwarp();
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");

  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
  if (tid == 0 && *abort_flag) atomicExch(&g_attn_status, DV_ERR_DEVICE_TIMEOUT);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* q = nullptr;
    cudaDriverEntryPointQueryResult r;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &q, 12000, cudaEnableDefault,
                                         &r) == cudaSuccess &&
        r == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(q);
  });
  return fn;
}

// Cache layer as a 4-D bf16 tensor (head_dim, kv head, slot, batch), boxes of 64 channels x
// 1 head x 128 slots x 1 batch element with 128-byte swizzle; slots past max_keys read zero.
bool encode_cache_4d(CUtensorMap* map, const void* ptr, int HD, int Hkv, int keys, int B,
                     long long s_head, long long s_seq, long long s_batch) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  // strides of dimensions of extent 1 are never used; any valid multiple of 16 bytes will do
  const long long sh = Hkv > 1 ? s_head : 8, sb = B > 1 ? s_batch : 8;
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(HD), static_cast<cuuint64_t>(Hkv),
                        static_cast<cuuint64_t>(keys), static_cast<cuuint64_t>(B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(sh * 2), static_cast<cuuint64_t>(s_seq * 2),
                           static_cast<cuuint64_t>(sb * 2)};
  cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(kKeyBlock), 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int device_ok() {
  static int state[64] = {};  // 0 unknown, 1 sm_103, 2 other
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return DV_ERR_CUDA;
  if (state[dev] == 0) {
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return DV_ERR_CUDA;
    state[dev] = (prop.major == 10 && prop.minor == 3) ? 1 : 2;
  }
  return state[dev] == 1 ? DV_OK : DV_ERR_UNSUPPORTED_DEVICE;
}

int num_sms_of_device() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (sms[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 148;
    sms[dev] = n;
  }
  return sms[dev];
}

template <int HD, int NST>
cudaError_t launch_attn(int splits, int units, const CUtensorMap& q, const CUtensorMap& k,
                        const CUtensorMap& v, const AttnParams& p, cudaStream_t stream) {
  using C = AttnCfg<HD, NST>;
  auto kern = dv_attn_kernel<HD, NST>;
  static bool attr_set[64] = {};  // the shared-memory opt-in, once per device
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!attr_set[dev]) {
    err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
    if (err != cudaSuccess) return err;
    attr_set[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(splits);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = pdl_attribute();
  cfg.gridDim = dim3(static_cast<unsigned>(units * splits), 1, 1);
  cfg.blockDim = dim3(kAttnThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, kern, q, k, v, p);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

bool al16(const void* x) { return (reinterpret_cast<uintptr_t>(x) & 15u) == 0; }

}  // namespace
}  // namespace dv

extern "C" int dv_text_attention(const void* q, int batch, int n_q_heads, int n_kv_heads,
                                 int n_text, int head_dim, const dv_kv_cache* cache, int layer,
                                 int max_keys, const int* n_keys, const int* q_slot, float scale,
                                 void* out, void* stream) {
  using namespace dv;
  if (batch < 0 || n_text < 0) return DV_ERR_INVALID_ARG;
  if (batch == 0 || n_text == 0) return DV_OK;
  if (!q || !cache || !cache->k || !cache->v || !n_keys || !q_slot || !out) return DV_ERR_INVALID_ARG;
  if (n_q_heads <= 0 || n_kv_heads <= 0 || n_q_heads % n_kv_heads != 0 || layer < 0 ||
      max_keys <= 0 || !(scale > 0.0f) || !std::isfinite(scale))
    return DV_ERR_INVALID_ARG;
  if (head_dim != 64 && head_dim != 128) return DV_ERR_UNSUPPORTED_SHAPE;
  const long long rows = static_cast<long long>(batch) * n_q_heads * n_text;
  if (rows > (1LL << 30) || max_keys > (1 << 24) || n_kv_heads > 4096 || batch > 65535)
    return DV_ERR_UNSUPPORTED_SHAPE;
  if (!al16(q) || !al16(out) || !al16(cache->k) || !al16(cache->v)) return DV_ERR_ALIGNMENT;
  if ((reinterpret_cast<uintptr_t>(n_keys) & 3u) || (reinterpret_cast<uintptr_t>(q_slot) & 3u))
    return DV_ERR_ALIGNMENT;
  const long long st[4] = {cache->s_layer, cache->s_batch, cache->s_seq, cache->s_head};
  for (long long x : st) {
    if (x < 0) return DV_ERR_INVALID_ARG;
    if (x % 8 != 0) return DV_ERR_ALIGNMENT;
  }
  if (cache->s_seq == 0) return DV_ERR_INVALID_ARG;
  int rc = device_ok();
  if (rc != DV_OK) return rc;
  if (!encode_fn()) return DV_ERR_CUDA;

  const long long off = static_cast<long long>(layer) * cache->s_layer;
  const uint16_t* kl = static_cast<const uint16_t*>(cache->k) + off;
  const uint16_t* vl = static_cast<const uint16_t*>(cache->v) + off;
  CUtensorMap tq, tk, tv;
  {
    EncodeTiledFn fn = encode_fn();
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(head_dim), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(head_dim) * 2};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t estr[2] = {1, 1};
    if (fn(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(q), dims, strides, box,
           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return DV_ERR_UNSUPPORTED_SHAPE;
  }
  if (!encode_cache_4d(&tk, kl, head_dim, n_kv_heads, max_keys, batch, cache->s_head,
                       cache->s_seq, cache->s_batch) ||
      !encode_cache_4d(&tv, vl, head_dim, n_kv_heads, max_keys, batch, cache->s_head,
                       cache->s_seq, cache->s_batch))
    return DV_ERR_UNSUPPORTED_SHAPE;

  AttnParams p;
  p.Hq = n_q_heads;
  p.Hkv = n_kv_heads;
  p.Nt = n_text;
  p.G = n_q_heads / n_kv_heads;
  p.rows_per_group = p.G * n_text;
  p.q_blocks = (p.rows_per_group + 127) / 128;
  p.max_keys = max_keys;
  p.n_keys = n_keys;
  p.q_slot = q_slot;
  p.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634);
  p.out = static_cast<uint16_t*>(out);
  p.timeout_ns = 2000000000ull;

  const long long units = static_cast<long long>(batch) * n_kv_heads * p.q_blocks;
  if (units > (1LL << 30)) return DV_ERR_UNSUPPORTED_SHAPE;
  const int blocks_max = (max_keys + kKeyBlock - 1) / kKeyBlock;
  // Key splits (cluster size): as many as the key blocks allow while the CTAs fit in one wave,
  // with two stages and one CTA per SM, or with one stage and two CTAs per SM when that
  // allows more splits (each CTA then has few blocks, so losing the prefetch costs little).
  const int sms = num_sms_of_device();
  int split2 = 1, split1 = 1;
  for (int s : {2, 4, 8}) {
    if (s <= blocks_max && units * s <= sms) split2 = s;
    if (s == 2 && s <= blocks_max && units * s <= 2LL * sms) split1 = s;
  }
  // One stage (two CTAs per SM, clusters of 2) only where two stages cannot split the keys at
  // all: measured on GB300 it then beats unsplit key runs (16.0 vs 18.0 us per layer at 128
  // clusters of 6 key blocks), while clusters of 4 lose to two stages in clusters of 2 (18.3 vs
  // 17.1 us at 64 clusters of 11 blocks).
  const bool one_stage = split2 == 1 && split1 == 2;
  const int splits = one_stage ? split1 : split2;
  const cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int u = static_cast<int>(units);
  cudaError_t err;
  if (head_dim == 128)
    err = one_stage ? launch_attn<128, 1>(splits, u, tq, tk, tv, p, cs)
                    : launch_attn<128, 2>(splits, u, tq, tk, tv, p, cs);
  else
    err = one_stage ? launch_attn<64, 1>(splits, u, tq, tk, tv, p, cs)
                    : launch_attn<64, 2>(splits, u, tq, tk, tv, p, cs);
  return err == cudaSuccess ? DV_OK : DV_ERR_CUDA;
}

extern "C" int dv_text_attention_status(void) {
  int st = 0;
  if (cudaDeviceSynchronize() != cudaSuccess) return DV_ERR_CUDA;
  if (cudaMemcpyFromSymbol(&st, dv::g_attn_status, sizeof(int)) != cudaSuccess) return DV_ERR_CUDA;
  if (st != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(dv::g_attn_status, &zero, sizeof(int)) != cudaSuccess) return DV_ERR_CUDA;
  }
  return st;
}
