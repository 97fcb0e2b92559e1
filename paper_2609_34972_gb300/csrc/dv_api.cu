// C ABI of the visual-memory build (include/dv.h): argument validation, the plan (repacked
// weights, workspace, TMA descriptors) and the per-build launch sequence.
//
// Plan-time repacking (once per weight set). With r_pad = r rounded up to 64:
//   Dst  [L*r_pad][d]         stacked down-projections, zero rows past r
//   Bn   [G*256][d+lpt*r_pad]  the statistic's B operand, lpt layers per 256-row group (norm_group):
//                             row j*rn + n of group g (layer l = g*lpt + j): [2 U_l[n,:] | 0 ..
//                             G_l[n,:] at columns d + j*r_pad .. | 0], G_l = U_l U_l^T
//   Wkv  [L*2kv][d+r_pad]     per layer, per group of 128 channels: the 128 K rows (permuted so
//                             that RoPE partners are 16 rows apart, see wkv_row), then the 128
//                             V rows of the same channels, each
//                             [W[c,:] * gamma_l | (W diag(gamma_l) U_l^T)[c,:]]
// so that, with A_l = [x0 | h_l] (h_l = SiLU(x0 D_l), Sec. 3.1 Eq. 4):
//   A_l Bn_l^T   = 2 x0 U_l^T + h_l G_l        -> ||M_l||^2 = ||x0||^2 + h_l . (that)
//   A_l Wkv_l^T  = (x0 + h_l U_l) diag(gamma_l) W^T = gamma_l * M_l projected (Sec. 3.2 Eq. 7)
// and K/V = rstd_l * (A_l Wkv_l^T) + b is exactly W RMSNorm(M_l) + b, without M_l ever being
// formed. Per build: (0) ||x0||^2 per token, (1) H = SiLU(x0 Dst^T), (2) rstd, (3) K/V.
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <utility>
#include <vector>

#include "../../include/dv.h"
#include "dv_internal.h"
#include "dv_ptx.cuh"

using dv::GemmParams;

struct dv_plan {
  dv_config cfg;
  int device = 0;
  int num_sms = 0;
  int r_pad = 0, kv = 0, k_total = 0, max_tokens = 0;
  int bn_lpt = 0, bn_rn = 0, bn_groups = 0, bn_k = 0;  // Bn layout (norm_group)
  uint16_t* Dst = nullptr;
  uint16_t* Bn = nullptr;
  uint16_t* Wkv = nullptr;
  uint16_t* Uup = nullptr;     // recurrent adapter: U_l as [L*d][uup_ld] (split chain: [U_l | U_l])
  uint16_t* Pf = nullptr;      // recurrent adapter, refactored chain: [L*r_pad][L*r_pad]
                               // (k_fold_products), or null
  uint16_t* Pf_lo = nullptr;   // its low bf16 part with split_chain, or null
  bool fold = false;           // recurrent builds may run the refactored chain (dv_fold.cu)
  int chain_clusters = 0;      // recurrent: clusters of the on-chip chain resident at once
  int uup_ld = 0;              // r_pad, or 2 r_pad with the split chain
  float* bk = nullptr;
  float* bv = nullptr;
  float* kg = nullptr;         // per-head K-norm gain fp32 [L][head_dim] (k_norm)
  float* Gf = nullptr;         // embedding adapter: G_l = U_l^T U_l, fp32 [L][r_pad][r_pad]
  void* ws = nullptr;          // workspace of a build of max_tokens tokens (carve_workspace)
  long long last_tokens = 0;   // tokens of the last build (layout of the workspace)
  int* status = nullptr;
  void* scratch = nullptr;     // static scratch of the no-allocation entry on this device
  CUtensorMap tm_Dst[3];       // boxes of 64, 128, 256 rows
  CUtensorMap tm_Dst_half[3];  // slab maps, boxes of 32, 64, 128 rows (halves for CTA pairs)
  CUtensorMap tm_Bn;           // boxes of 256 rows (one layer group)
  CUtensorMap tm_Bn_half;      // slab map, boxes of 128 rows (CTA-pair halves)
  CUtensorMap tm_Wkv;          // slab map, boxes of 128 rows
  CUtensorMap tm_Dst_rp, tm_Uup;  // recurrent adapter
  CUtensorMap tm_Pf, tm_Pf_lo;    // recurrent adapter: Pf (and Pf_lo) with r_pad-row boxes
  int resid_bn = 0;
  double inv_freq[dv::kMaxHalfHead];
  unsigned char mode[dv::kMaxLayers];  // DV_LAYER_* per layer
  int n_active = 0;                    // layers not dropped
  int16_t active[dv::kMaxLayers];      // their indices
  // per-stage timing
  bool timing = false;
  std::vector<cudaEvent_t> ev;  // kMaxTimed * kStages1
  int timed = 0;
};

namespace {

constexpr int kStages = 4;
constexpr int kEvPerBuild = kStages + 1;
constexpr int kMaxTimed = 4096;
constexpr unsigned long long kTimeoutNs = 2000000000ull;  // 2 s per device-side wait

// ------------------------------------------------------------------------------ driver entry

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// bf16 2-D tensor [rows][cols] (row stride in elements), 128-byte-swizzled boxes of
// 64 columns x box_rows rows; out-of-range elements read as zero.
bool encode_2d(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint64_t ld,
               uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(dv::kBlockK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 [rows][cols] (row stride ld elements) viewed as {64 columns, rows, cols / 64 slabs} for
// the 2-SM kernels: one box = box_rows rows x box_slabs (default kSlabsPerStep) consecutive K
// slabs, each slab a 128-byte-swizzled [box_rows][64] tile. cols must be a multiple of 64; slabs past the end of
// the matrix read as zero.
bool encode_slabs(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint64_t ld,
                  uint32_t box_rows, uint32_t box_slabs = dv::kSlabsPerStep) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || cols % dv::kBlockK != 0) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(dv::kBlockK), rows, cols / dv::kBlockK};
  cuuint64_t strides[2] = {ld * 2, static_cast<cuuint64_t>(dv::kBlockK) * 2};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(dv::kBlockK), box_rows, box_slabs};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 3-D tensor [L][rows][cols] (rows x cols per layer, packed), boxes of 64 columns x
// box_rows rows x 1 layer with 128-byte swizzle: a store past `rows` is clipped per layer.
bool encode_3d(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint64_t layers,
               uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {cols, rows, layers};
  cuuint64_t strides[2] = {cols * 2, cols * rows * 2};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(dv::kBlockK), box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same [L][rows][cols] bf16 tensor for stores of one warp's 32 x 32 block: boxes of 32
// columns x 32 rows x 1 layer with 64-byte swizzle (a 16-byte chunk q of staged row r sits at
// chunk q ^ ((r / 2) mod 4) of its 64-byte row); a store past `rows` is clipped per layer.
bool encode_3d_warp_store(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows,
                          uint64_t layers) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {cols, rows, layers};
  cuuint64_t strides[2] = {cols * 2, cols * rows * 2};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Launch of a build kernel with programmatic stream serialization (dv::pdl_attribute); the
// kernel calls dv::pdl_wait() before touching global memory, except where it states otherwise
// (k_row_sumsq).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1] = {dv::pdl_attribute()};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// ------------------------------------------------------------------------------ small kernels

__device__ __forceinline__ float bf(uint16_t b) { return __uint_as_float(static_cast<uint32_t>(b) << 16); }

__device__ __forceinline__ uint16_t to_bf16(float f) {
  return static_cast<uint16_t>(dv::pack_bf16x2(f, 0.0f) & 0xFFFFu);
}

// Planned layer i of the repacked weights comes from source layer src[i]. A layer whose
// adapter is skipped (DV_LAYER_IDENTITY, zero_du[i] != 0) is packed as if D_l = U_l = 0, which
// makes every adapter term of the fold vanish: M_l = E exactly (Sec. 3.1, U = 0 is the
// identity). Passed by value (768 bytes of kernel parameters).
struct PackLayers {
  int16_t src[dv::kMaxLayers];
  unsigned char zero_du[dv::kMaxLayers];
};

// Dst[i*r_pad + k][j] = D[src[i]][k][j] for k < r, else 0 (row stride ld).
__global__ void k_pack_down(const uint16_t* __restrict__ D, uint16_t* __restrict__ Dst, int L,
                            int r, int r_pad, int d, int ld, PackLayers pl) {
  const long long total = static_cast<long long>(L) * r_pad * d;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(e % d);
    const long long row = e / d;
    const int k = static_cast<int>(row % r_pad), i = static_cast<int>(row / r_pad);
    Dst[row * ld + j] =
        (k < r && !pl.zero_du[i]) ? D[(static_cast<long long>(pl.src[i]) * r + k) * d + j] : 0;
  }
}

// Bn row j*rn + n of group g (planned layer i = g*lpt + j): columns [0, d) hold 2 U[src[i]][:][n]
// for n < r and i < L; everything else is zero here. The G blocks are written by
// k_rank_product.
__global__ void k_pack_norm_u(const uint16_t* __restrict__ U, uint16_t* __restrict__ Bn, int L,
                              int r, int d, int lpt, int rn, int groups, int bn_k, PackLayers pl) {
  const long long total = static_cast<long long>(groups) * 256 * bn_k;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(e % bn_k);
    const long long row = e / bn_k;
    const int jr = static_cast<int>(row % 256), g = static_cast<int>(row / 256);
    const int n = jr % rn, i = g * lpt + jr / rn;
    float v = 0.0f;
    if (j < d && n < r && i < L && !pl.zero_du[i])
      v = 2.0f * bf(U[(static_cast<long long>(pl.src[i]) * d + j) * r + n]);
    Bn[e] = to_bf16(v);
  }
}

// Dst[row0 + i*r_pad + n][j] = 2 U[src[i]][j][n] (n < r), else 0: the x0 (2 U_l)^T part of the
// statistic of M_l, stacked after the down-projections so that one GEMM over x0 forms both.
__global__ void k_pack_2u(const uint16_t* __restrict__ U, uint16_t* __restrict__ Dst, int L, int r,
                          int r_pad, int d, int ld, PackLayers pl) {
  const long long total = static_cast<long long>(L) * r_pad * d;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(e % d);
    const long long row = e / d;
    const int n = static_cast<int>(row % r_pad), i = static_cast<int>(row / r_pad);
    float v = 0.0f;
    if (n < r && !pl.zero_du[i]) v = 2.0f * bf(U[(static_cast<long long>(pl.src[i]) * d + j) * r + n]);
    Dst[row * ld + j] = to_bf16(v);
  }
}

// Row rl of layer l in Wkv: group rl / 256 of 128 channels, K (first 128) or V (next 128).
// V rows are in channel order. K rows are permuted so that rows 32q + i and 32q + 16 + i
// (i < 16) are the two channels (j, j + HD/2) of rotate-half pair p = 16q + i of the group: a
// warp that reads 32 consecutive rows (TMEM lanes) or columns then holds 16 complete RoPE pairs.
__device__ __forceinline__ void wkv_row(int rl, int HD, int& part, int& c) {
  part = (rl >> 7) & 1;
  const int i = rl & 127;
  int within = i;
  if (part == 0) {
    const int half = HD / 2;
    const int p = 16 * (i >> 5) + (i & 15);
    within = (p / half) * HD + p % half + ((i & 16) ? half : 0);
  }
  c = (rl >> 8) * 128 + within;
}

// Wkv rows: per planned layer, per 128-channel group, 128 K rows then 128 V rows; columns
// [0, d) hold W[c][j] * gamma[l][j] of source layer l = src[i]; columns [d, k_total) are filled
// by k_rank_product (zero past r).
__global__ void k_pack_kv(const uint16_t* __restrict__ Wk, const uint16_t* __restrict__ Wv,
                          const uint16_t* __restrict__ gamma, uint16_t* __restrict__ Wkv, int L,
                          int kv, int HD, int d, int k_total, PackLayers pl) {
  const long long total = static_cast<long long>(L) * 2 * kv * k_total;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(e % k_total);
    const long long row = e / k_total;
    const int rl = static_cast<int>(row % (2 * kv));
    const int l = pl.src[row / (2 * kv)];
    int part, c;
    wkv_row(rl, HD, part, c);
    float v = 0.0f;
    if (j < d) {
      const uint16_t* W = part ? Wv : Wk;
      v = bf(W[(static_cast<long long>(l) * kv + c) * d + j]) * bf(gamma[static_cast<long long>(l) * d + j]);
    }
    Wkv[e] = to_bf16(v);
  }
}

// out[p][i][n] = sum_j A(l, i, j) * U[l][j][n] for n < r, accumulated in fp32 over j < d, for
// planned layer p = blockIdx.z of source layer l = src[p] (U taken as zero where zero_du[p]);
// in MODE 1 the fp32 result also goes to gout[p][i][n] when gout is given:
//   MODE 0 (fold):  A(l, i, j) = W_part[l][c][j] * gamma[l][j], i indexes the 2*kv Wkv rows
//                   of the layer; the result goes to Wkv row (p, i), column d + n
//   MODE 1 (gram):  A(l, i, j) = U[l][j][i], i < r; the result goes to Bn row
//                   (p / lpt) * 256 + (p % lpt) * rn + i, column d + (p % lpt) * r_pad + n
// 64 x 64 output tile per block, 256 threads with 4 x 4 outputs each, j in steps of 32.
template <int MODE>
__global__ void __launch_bounds__(256) k_rank_product(const uint16_t* __restrict__ Wk,
                                                      const uint16_t* __restrict__ Wv,
                                                      const uint16_t* __restrict__ gamma,
                                                      const uint16_t* __restrict__ U,
                                                      uint16_t* __restrict__ out, int rows, int r,
                                                      int d, int kv, int HD, int r_pad,
                                                      int k_total, PackLayers pl,
                                                      float* __restrict__ gout, int lpt, int rn) {
  __shared__ float As[32][65];
  __shared__ float Us[32][65];
  const int p = blockIdx.z, l = pl.src[p];
  const bool zero_u = pl.zero_du[p] != 0;
  const int i0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  const uint16_t* Ul = U + static_cast<long long>(l) * d * r;
  for (int j0 = 0; j0 < d; j0 += 32) {
    for (int e = threadIdx.x; e < 64 * 32; e += 256) {
      const int ii = e / 32, jj = e % 32;
      const int i = i0 + ii, j = j0 + jj;
      float a = 0.0f;
      if (i < rows && j < d) {
        if (MODE == 0) {
          int part, c;
          wkv_row(i, HD, part, c);
          const uint16_t* W = part ? Wv : Wk;
          a = bf(W[(static_cast<long long>(l) * kv + c) * d + j]) *
              bf(gamma[static_cast<long long>(l) * d + j]);
        } else {
          a = zero_u ? 0.0f : bf(Ul[static_cast<long long>(j) * r + i]);
        }
      }
      As[jj][ii] = a;
      const int nn = e % 64, jk = e / 64;
      const int n = n0 + nn, j2 = j0 + jk;
      Us[jk][nn] = (n < r && j2 < d && !zero_u) ? bf(Ul[static_cast<long long>(j2) * r + n]) : 0.0f;
    }
    __syncthreads();
#pragma unroll 8
    for (int jj = 0; jj < 32; ++jj) {
      float a[4], u[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        a[q] = As[jj][ty * 4 + q];
        u[q] = Us[jj][tx * 4 + q];
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int w = 0; w < 4; ++w) acc[q][w] = fmaf(a[q], u[w], acc[q][w]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = i0 + ty * 4 + q;
    if (i >= rows) continue;
    const long long orow = MODE == 0 ? static_cast<long long>(p) * 2 * kv + i
                                     : static_cast<long long>(p / lpt) * 256 + (p % lpt) * rn + i;
    const int ocol = MODE == 0 ? d : d + (p % lpt) * r_pad;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int n = n0 + tx * 4 + w;
      if (n >= r) continue;
      if (out) out[orow * k_total + ocol + n] = to_bf16(acc[q][w]);
      if (MODE == 1 && gout) gout[(static_cast<long long>(p) * r_pad + i) * r_pad + n] = acc[q][w];
    }
  }
}

// out[i][c] = b[src[i]][c] in fp32 (K/V biases, K-norm gains: c < kv).
__global__ void k_bias_to_f32(const uint16_t* __restrict__ b, float* __restrict__ out, int L,
                              int kv, PackLayers pl) {
  const long long n = static_cast<long long>(L) * kv;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<long long>(gridDim.x) * blockDim.x)
    out[e] = bf(b[static_cast<long long>(pl.src[e / kv]) * kv + e % kv]);
}

// Recurrent adapter, refactored chain (dv_fold.cu). Pf [L r_pad][L r_pad]: row i r_pad + a,
// columns j r_pad + b with j < i hold bf16 of Q_ij[a][b] = sum_e D_i[a][e] U_j[e][b] (a, b < r;
// zero where layer i or j is an identity layer), and Pf_lo (split chain, or null) the bf16 of
// Q_ij - bf16(Q_ij); the caller zeroes the rest.
// Q_ij blocks: grid (r_pad / 64 b-tiles, (L) * (r_pad / 64) (j, a-tile), L (i)); blocks with
// j >= i return. 64 x 64 outputs per block, 256 threads with 4 x 4 each, fp32 accumulation
// over e in steps of 32 (a fixed order).
__global__ void __launch_bounds__(256) k_fold_products(const uint16_t* __restrict__ D,
                                                       const uint16_t* __restrict__ U,
                                                       uint16_t* __restrict__ Pf,
                                                       uint16_t* __restrict__ Pf_lo, int L, int r,
                                                       int r_pad, int d, long long pld,
                                                       PackLayers pl) {
  const int at_n = r_pad / 64;
  const int i = blockIdx.z, j = blockIdx.y / at_n, at = blockIdx.y % at_n;
  if (j >= i) return;
  const bool zero = pl.zero_du[i] || pl.zero_du[j];
  const int li = pl.src[i], lj = pl.src[j];
  const int a0 = at * 64, b0 = blockIdx.x * 64;
  __shared__ float Ds[32][65];
  __shared__ float Us[32][65];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int e0 = 0; e0 < d; e0 += 32) {
    for (int e = threadIdx.x; e < 64 * 32; e += 256) {
      const int aa = e / 32, ee = e % 32;  // D row a0 + aa, contiguous in e
      Ds[ee][aa] = (a0 + aa < r && !zero)
                       ? bf(D[(static_cast<long long>(li) * r + a0 + aa) * d + e0 + ee]) : 0.0f;
      const int bb = e % 64, ek = e / 64;  // U row e0 + ek, contiguous in b
      Us[ek][bb] = (b0 + bb < r && !zero)
                       ? bf(U[(static_cast<long long>(lj) * d + e0 + ek) * r + b0 + bb]) : 0.0f;
    }
    __syncthreads();
#pragma unroll 8
    for (int ee = 0; ee < 32; ++ee) {
      float av[4], uv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        av[q] = Ds[ee][ty * 4 + q];
        uv[q] = Us[ee][tx * 4 + q];
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int w = 0; w < 4; ++w) acc[q][w] = fmaf(av[q], uv[w], acc[q][w]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const long long row = static_cast<long long>(i) * r_pad + a0 + ty * 4 + q;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const long long e = row * pld + static_cast<long long>(j) * r_pad + b0 + tx * 4 + w;
      const uint16_t hi = to_bf16(acc[q][w]);
      Pf[e] = hi;
      if (Pf_lo) Pf_lo[e] = to_bf16(acc[q][w] - bf(hi));  // split: the remainder, in bf16
    }
  }
}

// Uup[i*d + j][n] = U[src[i]][j][n mod r_pad] for (n mod r_pad) < r, else 0: the up-projection
// of the recurrent adapter as a K-major B operand (rows = output channels j, K = bottleneck n),
// with ld = r_pad, or ld = 2 r_pad for the split chain (U twice: once for the low and once for
// the high bf16 part of h).
__global__ void k_pack_up(const uint16_t* __restrict__ U, uint16_t* __restrict__ Uup, int L, int r,
                          int r_pad, int d, int ld, PackLayers pl) {
  const long long total = static_cast<long long>(L) * d * ld;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int n = static_cast<int>(e % ld) % r_pad;
    const long long row = e / ld;
    const int j = static_cast<int>(row % d), i = static_cast<int>(row / d);
    Uup[e] = (n < r && !pl.zero_du[i]) ? U[(static_cast<long long>(pl.src[i]) * d + j) * r + n] : 0;
  }
}

// rstd[i][t] = 1 / sqrt(sum_n part[i][n][t] / d + eps), the partial sums of squares of the
// recurrent state M_i summed in column-tile order (n < n_parts; layer stride ld_part).
__global__ void k_rstd_parts(const float* __restrict__ part, int L, long long T, int n_parts,
                             long long ld_part, float inv_d, float eps, float* __restrict__ rstd) {
  dv::pdl_wait();
  dv::pdl_trigger();
  const long long total = static_cast<long long>(L) * T;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long i = e / T, t = e % T;
    const float* pp = part + i * ld_part + t;
    float ss = 0.0f;
    for (int n = 0; n < n_parts; ++n) ss += pp[static_cast<long long>(n) * T];
    rstd[e] = rsqrtf(fmaf(ss, inv_d, eps));
  }
}

// Statistic of M_l = x0 + h_l U_l for small token counts: ||M_l||^2 = ||x0||^2 +
// h_l . (c_l + G_l h_l), with c_l = x0 (2 U_l)^T (fp32, from the stacked GEMM) and
// G_l = U_l^T U_l (fp32, from the plan), so rstd_l = ((xx + h . (c + G h)) / d + eps)^-1/2.
// One block of 64 threads per (layer, 64 tokens): thread (tg, k) keeps u_n = c_n + (G h)_n for
// the 4 tokens 4 tg .. 4 tg + 3 and n in quarter k ([16 k, 16 k + 16)) in registers. G is
// symmetric, so row m scales h_m into all sums; G_l sits in shared memory with each row's
// quarters interleaved (float4 n4 of quarter k at word 16 n4 + 4 k) so that the four quarters
// read together fall in distinct banks, and h as [m][token], read as float4 over 4 tokens. The
// four partial dots of a token are summed with two shuffles (fixed order).
template <int RP>
__global__ void __launch_bounds__(64) k_rstd_hc(const uint16_t* __restrict__ H, int ldh,
                                                const float* __restrict__ C, int ldc,
                                                const float* __restrict__ xx,
                                                const float* __restrict__ Gf, int T, float inv_d,
                                                float eps, float* __restrict__ rstd) {
  static_assert(RP == 64, "one quarter = 16 sums = 4 float4");
  dv::pdl_wait();
  dv::pdl_trigger();
  __shared__ __align__(16) float g[RP * RP];
  __shared__ __align__(16) float hs[RP][64];
  const int l = blockIdx.y, tid = threadIdx.x;
  const int tg = tid >> 2, k = tid & 3;
  const float* gl = Gf + static_cast<long long>(l) * RP * RP;
  {  // all 16 loads of this thread first, then the stores (interleaved quarters)
    float4 gv[RP * RP / 4 / 64];
    const float4* gl4 = reinterpret_cast<const float4*>(gl);
#pragma unroll
    for (int i = 0; i < RP * RP / 4 / 64; ++i) gv[i] = gl4[tid + 64 * i];
#pragma unroll
    for (int i = 0; i < RP * RP / 4 / 64; ++i) {
      const int e = 4 * (tid + 64 * i);  // e = m*64 + n, n a multiple of 4
      const int m = e >> 6, n = e & 63, kk = n >> 4, n4 = (n >> 2) & 3;
      *reinterpret_cast<float4*>(g + m * RP + n4 * 16 + kk * 4) = gv[i];
    }
  }
  {  // token tid, all RP channels: 8 independent 16-byte loads, then the widening stores
    const int t = min(static_cast<int>(blockIdx.x) * 64 + tid, T - 1);
    const uint4* hrow = reinterpret_cast<const uint4*>(H + static_cast<long long>(t) * ldh + l * RP);
    uint4 hw[RP / 8];
#pragma unroll
    for (int c8 = 0; c8 < RP / 8; ++c8) hw[c8] = hrow[c8];
#pragma unroll
    for (int c8 = 0; c8 < RP / 8; ++c8) {
      const uint32_t ws[4] = {hw[c8].x, hw[c8].y, hw[c8].z, hw[c8].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        hs[c8 * 8 + 2 * q][tid] = __uint_as_float(ws[q] << 16);
        hs[c8 * 8 + 2 * q + 1][tid] = __uint_as_float(ws[q] & 0xFFFF0000u);
      }
    }
  }
  __syncthreads();
  float u[4][16];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int t = min(blockIdx.x * 64 + tg * 4 + i, T - 1);
    const float4* cr = reinterpret_cast<const float4*>(C + static_cast<long long>(t) * ldc + l * RP + k * 16);
#pragma unroll
    for (int n4 = 0; n4 < 4; ++n4) {
      const float4 c4 = cr[n4];
      u[i][4 * n4] = c4.x;
      u[i][4 * n4 + 1] = c4.y;
      u[i][4 * n4 + 2] = c4.z;
      u[i][4 * n4 + 3] = c4.w;
    }
  }
#pragma unroll 2
  for (int m = 0; m < RP; ++m) {
    const float4 hm = *reinterpret_cast<const float4*>(&hs[m][tg * 4]);
    const float hv[4] = {hm.x, hm.y, hm.z, hm.w};
#pragma unroll
    for (int n4 = 0; n4 < 4; ++n4) {
      const float4 gv = *reinterpret_cast<const float4*>(g + m * RP + n4 * 16 + k * 4);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        u[i][4 * n4] = fmaf(gv.x, hv[i], u[i][4 * n4]);
        u[i][4 * n4 + 1] = fmaf(gv.y, hv[i], u[i][4 * n4 + 1]);
        u[i][4 * n4 + 2] = fmaf(gv.z, hv[i], u[i][4 * n4 + 2]);
        u[i][4 * n4 + 3] = fmaf(gv.w, hv[i], u[i][4 * n4 + 3]);
      }
    }
  }
  float dot[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    const float4 hn = *reinterpret_cast<const float4*>(&hs[k * 16 + n][tg * 4]);
    dot[0] = fmaf(hn.x, u[0][n], dot[0]);
    dot[1] = fmaf(hn.y, u[1][n], dot[1]);
    dot[2] = fmaf(hn.z, u[2][n], dot[2]);
    dot[3] = fmaf(hn.w, u[3][n], dot[3]);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    dot[i] += __shfl_xor_sync(0xFFFFFFFFu, dot[i], 1);
    dot[i] += __shfl_xor_sync(0xFFFFFFFFu, dot[i], 2);
  }
  if (k == 0) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = blockIdx.x * 64 + tg * 4 + i;
      if (t < T) {
        const float ss = fmaxf(xx[t] + dot[i], 0.0f);
        rstd[static_cast<long long>(l) * T + t] = rsqrtf(fmaf(ss, inv_d, eps));
      }
    }
  }
}

// xx[t] = sum_j x0[t][j]^2 (fp32), one warp per token row, 16-byte loads; the row also goes to
// x0p[t] (row pitch ldp elements), the copy of E that the RMS statistic and the K/V GEMM read:
// a pitch of d + 64 elements is not a power of two, which spreads a TMA box's rows over the L2
// (the caller's E has pitch d, a power of two on the 7B shapes).
// Launched right after the down-projection and run beside it, on the SMs that its tiles leave
// free. Its reads of x0 and its writes of xx and x0p come before its dependency wait. That is
// safe: a dependent grid starts only once every CTA of the grid before it has triggered, and the
// down-projection triggers after its own wait, so every earlier writer of x0 and every earlier
// reader of xx and x0p (the previous build's statistic and K/V GEMM) has finished. The wait comes
// last, so that this grid completes only after the down-projection has, and the kernel after it,
// which waits on this grid alone, still sees H.
__global__ void k_row_sumsq(const uint16_t* __restrict__ x0, int T, int d, float* __restrict__ xx,
                            uint16_t* __restrict__ x0p, long long ldp) {
  dv::pdl_trigger();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp < T) {
    const uint4* row = reinterpret_cast<const uint4*>(x0 + static_cast<long long>(warp) * d);
    uint4* prow = x0p ? reinterpret_cast<uint4*>(x0p + static_cast<long long>(warp) * ldp) : nullptr;
    float s = 0.0f;
#pragma unroll 8
    for (int c = lane; c < d / 8; c += 32) {
      const uint4 v = row[c];
      if (prow) prow[c] = v;
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = __uint_as_float(w[e] << 16), b = __uint_as_float(w[e] & 0xFFFF0000u);
        s = fmaf(a, a, s);
        s = fmaf(b, b, s);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    if (lane == 0) xx[warp] = s;
  }
  dv::pdl_wait();
}

// Failure-detection self-test: waits on a barrier nothing completes; gives up after the limit.
__global__ void k_wait_timeout(int* status, unsigned long long timeout_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int abort_flag;
  if (threadIdx.x != 0) return;
  const uint32_t b = dv::smem_addr(&bar);
  dv::mbar_init(b, 1);
  dv::fence_barrier_init();
  abort_flag = 0;
  if (!dv::mbar_wait(b, 0, &abort_flag, timeout_ns)) atomicExch(status, DV_ERR_DEVICE_TIMEOUT);
}

// ------------------------------------------------------------------------------ host helpers

int grid_for(long long n) {
  long long g = (n + 255) / 256;
  if (g > 65535LL * 16) g = 65535LL * 16;
  return static_cast<int>(g < 1 ? 1 : g);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned2(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 1u) == 0; }

}  // namespace

// Position axis (0 t, 1 h, 2 w) of rotary frequency pair j: contiguous M-RoPE sections, or
// the interleaved layout (j = 1 mod 3 below 3 s_h -> h, j = 2 mod 3 below 3 s_w -> w, else t).
int dv::rope_axis(int rope, const int* sec, int j) {
  if (rope == DV_ROPE_MROPE) return j < sec[0] ? 0 : (j < sec[0] + sec[1] ? 1 : 2);
  if (rope == DV_ROPE_MROPE_INTERLEAVED) {
    if (j % 3 == 1 && j < 3 * sec[1]) return 1;
    if (j % 3 == 2 && j < 3 * sec[2]) return 2;
  }
  return 0;
}

namespace {

int check_config(const dv_config* c) {
  if (!c) return DV_ERR_INVALID_ARG;
  if (c->act != DV_ACT_SILU) return DV_ERR_INVALID_ARG;
  if (c->rope != DV_ROPE_1D && c->rope != DV_ROPE_MROPE && c->rope != DV_ROPE_MROPE_INTERLEAVED)
    return DV_ERR_INVALID_ARG;
  if (c->k_norm != 0 && c->k_norm != 1) return DV_ERR_INVALID_ARG;
  if (!(c->k_norm_eps >= 0.0f) || !std::isfinite(c->k_norm_eps)) return DV_ERR_INVALID_ARG;
  if (c->d <= 0 || c->n_layers <= 0 || c->n_kv_heads <= 0 || c->head_dim <= 0 || c->rank <= 0 ||
      c->max_batch <= 0 || c->max_n_vis <= 0)
    return DV_ERR_INVALID_ARG;
  if (!(c->rope_theta > 0.0f) || !(c->rms_eps >= 0.0f) || !std::isfinite(c->rope_theta) ||
      !std::isfinite(c->rms_eps))
    return DV_ERR_INVALID_ARG;
  if (c->has_kv_bias != 0 && c->has_kv_bias != 1) return DV_ERR_INVALID_ARG;
  if (c->adapter != DV_ADAPTER_EMBEDDING && c->adapter != DV_ADAPTER_RECURRENT)
    return DV_ERR_INVALID_ARG;
  if (c->split_chain != 0 && c->split_chain != 1) return DV_ERR_INVALID_ARG;
  if (c->split_chain && c->adapter != DV_ADAPTER_RECURRENT) return DV_ERR_INVALID_ARG;
  if (c->recurrent_path != DV_RECURRENT_AUTO && c->recurrent_path != DV_RECURRENT_CHAIN &&
      c->recurrent_path != DV_RECURRENT_REARRANGED)
    return DV_ERR_INVALID_ARG;
  if (c->recurrent_path != DV_RECURRENT_AUTO && c->adapter != DV_ADAPTER_RECURRENT)
    return DV_ERR_INVALID_ARG;
  if (c->recurrent_path == DV_RECURRENT_REARRANGED && dv::fold_slice_cols(c->d) == 0)
    return DV_ERR_UNSUPPORTED_SHAPE;
  if (c->d % 64 != 0 || c->d > 16384) return DV_ERR_UNSUPPORTED_SHAPE;
  if (c->rank > 256) return DV_ERR_UNSUPPORTED_SHAPE;
  if (c->head_dim != 64 && c->head_dim != 128) return DV_ERR_UNSUPPORTED_SHAPE;
  if (static_cast<long long>(c->n_kv_heads) * c->head_dim > 8192) return DV_ERR_UNSUPPORTED_SHAPE;
  if ((c->n_kv_heads * c->head_dim) % 128 != 0) return DV_ERR_UNSUPPORTED_SHAPE;
  if (c->n_layers > 256) return DV_ERR_UNSUPPORTED_SHAPE;
  if (static_cast<long long>(c->max_batch) * c->max_n_vis > (1LL << 24)) return DV_ERR_UNSUPPORTED_SHAPE;
  if (c->rope == DV_ROPE_MROPE || c->rope == DV_ROPE_MROPE_INTERLEAVED) {
    const int* s = c->mrope_section;
    if (s[0] < 0 || s[1] < 0 || s[2] < 0) return DV_ERR_INVALID_ARG;
    if (s[0] + s[1] + s[2] != c->head_dim / 2) return DV_ERR_UNSUPPORTED_SHAPE;
    int count[3] = {0, 0, 0};
    for (int j = 0; j < c->head_dim / 2; ++j) ++count[dv::rope_axis(c->rope, s, j)];
    if (count[0] != s[0] || count[1] != s[1] || count[2] != s[2]) return DV_ERR_UNSUPPORTED_SHAPE;
  }
  return DV_OK;
}

void free_plan_memory(dv_plan* p) {
  void* ptrs[] = {p->Dst, p->Bn, p->Wkv, p->Uup, p->Pf, p->Pf_lo, p->bk, p->bv, p->kg, p->Gf,
                  p->ws, p->status};
  for (void* q : ptrs)
    if (q) cudaFree(q);
  for (cudaEvent_t e : p->ev) cudaEventDestroy(e);
  p->ev.clear();
}

template <typename T>
bool dmalloc(T** out, size_t bytes) {
  void* q = nullptr;
  if (cudaMalloc(&q, bytes) != cudaSuccess) {
    cudaGetLastError();
    *out = nullptr;
    return false;
  }
  *out = static_cast<T*>(q);
  return true;
}

}  // namespace

namespace dv {

int check_build_args(const void* x0, int batch, int n_vis, const int* pos, const int* slot,
                     int slot0, const dv_kv_cache* out) {
  if (batch < 0 || n_vis < 0 || slot0 < 0) return DV_ERR_INVALID_ARG;
  if (static_cast<long long>(batch) * n_vis == 0) return DV_OK;
  if (!x0 || !pos || !out || !out->k || !out->v) return DV_ERR_INVALID_ARG;
  if (!aligned16(x0) || !aligned16(out->k) || !aligned16(out->v)) return DV_ERR_ALIGNMENT;
  const long long s[4] = {out->s_layer, out->s_batch, out->s_seq, out->s_head};
  for (long long x : s) {
    if (x < 0) return DV_ERR_INVALID_ARG;
    if (x % 8 != 0) return DV_ERR_ALIGNMENT;
  }
  if ((reinterpret_cast<uintptr_t>(pos) & 3u) || (slot && (reinterpret_cast<uintptr_t>(slot) & 3u)))
    return DV_ERR_ALIGNMENT;
  return DV_OK;
}

// Orientation of the GEMMs. The 2-SM kernels with 256-token M blocks balance shared-memory
// traffic against tensor throughput best, but pad the token count to a multiple of 256; they
// are used when that padding costs at most 6 % over the 128-token blocks of the 1-SM kernel
// (rank-r GEMMs) or over the token tile of the weights-as-M K/V kernel.
static bool prefer_256(long long padded256, long long padded_other) {
  return padded256 * 100 <= padded_other * 106;
}

// L2 super-blocks of the tokens-as-M kernels (see dv_pair_tm.cu): about kGroupBytes of token
// blocks and as much of weight tiles. When all token blocks fit in that budget, the token
// blocks of each weight tile run together and the weights stream from DRAM once.
constexpr long long kGroupBytes = 32ll << 20;  // 16-64 MB measured within 2 % of each other
static void tm_groups(GemmShape& s, int block_n, long long tokens) {
  const long long k = static_cast<long long>(s.k0_slabs + s.k1_slabs) * kBlockK * 2;  // bytes/row
  const long long m_blocks = (tokens + 255) / 256;
  const long long w_tiles = static_cast<long long>(s.n_per_layer / block_n) * s.n_layers;
  long long gm = kGroupBytes / (256 * k), gw = kGroupBytes / (block_n * k);
  if (m_blocks * 256 * k <= kGroupBytes) {
    gm = m_blocks;
    gw = 1;
  }
  s.group_m = static_cast<int>(gm < 1 ? 1 : (gm > m_blocks ? m_blocks : gm));
  s.group_w = static_cast<int>(gw < 1 ? 1 : (gw > w_tiles ? w_tiles : gw));
}

// Epilogue constants of the K/V stage: biases, positions, cache, RoPE frequencies.
static void fill_epi_kv(const PlanView& v, const BuildArgs& a, long long T, EpiKV& e) {
  const int HD = v.head_dim;
  e.rstd = a.rstd;
  e.ld_rstd = static_cast<int>(T);
  e.bk = v.bk;
  e.bv = v.bv;
  e.kv = v.kv;
  e.pos = a.pos;
  e.slot = a.slot;
  e.slot0 = a.slot0;
  e.n_vis = a.n_vis;
  e.n_pos = v.rope == DV_ROPE_1D ? 1 : 3;
  for (int j = 0; j < HD / 2; ++j) e.axis[j] = static_cast<uint8_t>(rope_axis(v.rope, v.mrope_section, j));
  e.kg = v.kg;
  e.k_eps = v.k_eps;
  e.kc = static_cast<uint16_t*>(const_cast<void*>(a.kc));
  e.vc = static_cast<uint16_t*>(const_cast<void*>(a.vc));
  e.s_layer = a.s_layer;
  e.s_batch = a.s_batch;
  e.s_seq = a.s_seq;
  e.s_head = a.s_head;
  const double two_pi = 6.283185307179586476925286766559;
  e.two_pi_hi = static_cast<float>(two_pi);
  e.two_pi_lo = static_cast<float>(two_pi - static_cast<double>(e.two_pi_hi));
  e.inv_two_pi = static_cast<float>(1.0 / two_pi);
  for (int j = 0; j < HD / 2; ++j) {
    e.inv_freq_hi[j] = static_cast<float>(v.inv_freq[j]);
    e.inv_freq_lo[j] = static_cast<float>(v.inv_freq[j] - static_cast<double>(e.inv_freq_hi[j]));
  }
}

// K/V stage over all planned layers: K/V = rstd_l * (A_l [| h_l] Wkv_l^T) + b, RoPE on K,
// stored into the cache. gp.s holds the operand schedule; the engine is chosen by token count
// (tokens-as-M pairs when 256-token blocks pad little, else weights-as-M pairs). The token
// operands are slab maps: a_full / h_full with 128-row boxes, a_half / h_half (made here) with
// nt / 2-row boxes.
static cudaError_t launch_kv_stage(const PlanView& v, GemmParams& gp, long long T,
                                   const void* a_ptr, uint64_t a_rows, uint64_t a_ld,
                                   const CUtensorMap& a_full, const void* h_ptr, uint64_t h_cols,
                                   uint64_t h_ld, const CUtensorMap& h_full, cudaStream_t st) {
  const int nt = kv_pair_tile_n(T);
  const long long pad256 = (T + 255) / 256 * 256, pad_nt = (T + nt - 1) / nt * nt;
  if (prefer_256(pad256, pad_nt)) {
    tm_groups(gp.s, 256, T);
    return launch_pair_tm(EPI_KV, 256, v.head_dim, a_full, h_full, *v.tm_Wkv, gp, v.num_sms, st);
  }
  CUtensorMap a_half, h_half;
  if (!encode_slabs(&a_half, a_ptr, v.d, a_rows, a_ld, nt / 2)) return cudaErrorInvalidValue;
  if (h_ptr && !encode_slabs(&h_half, h_ptr, h_cols, static_cast<uint64_t>(T), h_ld, nt / 2))
    return cudaErrorInvalidValue;
  return launch_kv_pair(v.head_dim, nt, *v.tm_Wkv, a_half, h_ptr ? h_half : a_half, gp, v.num_sms,
                        st);
}

// K/V stage of a recurrent build: every layer in one launch, A = the stacked M_l (tm_mem_s: its
// slab map with 128-row boxes).
template <typename Mark>
static cudaError_t launch_recurrent_kv(const PlanView& v, const BuildArgs& a, long long T,
                                       const CUtensorMap& tm_mem_s, cudaStream_t st, Mark& mark) {
  const int L = v.n_layers, d = v.d;
  GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.status = v.status;
  gp.timeout_ns = kTimeoutNs;
  for (int i = 0; i < L; ++i) gp.layer_map[i] = v.active[i];
  gp.s = {static_cast<int>(T), L, 2 * v.kv, d / 64, 0, 0, 0, 0, 0, static_cast<int>(T)};
  fill_epi_kv(v, a, T, gp.kv);
  const cudaError_t err = launch_kv_stage(v, gp, T, a.mem, static_cast<uint64_t>(L) * T,
                                          static_cast<uint64_t>(d), tm_mem_s, nullptr, 0, 0,
                                          tm_mem_s, st);
  mark(4);
  return err;
}

// Recurrent builds of this plan may run the refactored chain (dv_fold.cu): its workspace holds
// the two parts of E D^T instead of the per-layer path's fp32 state.
static bool uses_fold(const PlanView& v) { return v.tm_Pf != nullptr; }

// The refactored chain runs a build unless its token blocks fit in one wave of on-chip chain
// clusters: the chain spreads each block over a cluster of 14-16 SMs, where the refactored
// recurrence keeps a block on one SM.
static bool fold_build(const PlanView& v, long long tokens) {
  return uses_fold(v) && (tokens + kBlockM - 1) / kBlockM > v.chain_clusters;
}

// Recurrent adapter by the refactored chain (dv_fold.cu): (1) C = E [D_1 .. D_L]^T in fp32, one
// GEMM on the engine the embedding adapter's down-projection would use; (2) the
// recurrence h_l = SiLU(C_l + sum_{j<l} h_j Q_lj^T) per 128-token block; (3) the running sum
// M_l = E + sum_{j<=l} h_j U_j^T with the rows' sums of squares; then the RMS statistics and one
// K/V launch over all layers, as in the chain below.
static cudaError_t enqueue_fold(const PlanView& v, const BuildArgs& a, cudaStream_t st) {
  const long long T = static_cast<long long>(a.batch) * a.n_vis;
  const int L = v.n_layers, d = v.d;
  const long long n1 = static_cast<long long>(L) * v.r_pad;
  const int cw = fold_slice_cols(d);
  auto mark = [&](int i) {
    if (a.marks) cudaEventRecord(a.marks[i], st);
  };
  const bool split = v.split_chain != 0;
  const uint32_t ks = static_cast<uint32_t>(hchain_box_slabs(v.r_pad, split));
  // tm_hst: the recurrence's stores of h_l, 32 rows (one epilogue warp) per box; tm_mem_w: the
  // running sum's stores of M_l, one warp's 32 x 32 block per box
  CUtensorMap tm_x0, tm_x0_s, tm_hs, tm_h, tm_hst, tm_u, tm_mem_s, tm_mem_w;
  if (!encode_2d(&tm_x0, a.x0, d, static_cast<uint64_t>(T), d, kBlockM) ||
      !encode_slabs(&tm_x0_s, a.x0, d, static_cast<uint64_t>(T), d, kBlockM) ||
      !encode_slabs(&tm_hs, a.H, n1, static_cast<uint64_t>(T), a.hld, kBlockM, ks) ||
      !encode_2d(&tm_h, a.H, n1, static_cast<uint64_t>(T), a.hld, kBlockM) ||
      !encode_2d(&tm_hst, a.H, n1, static_cast<uint64_t>(T), a.hld, 32) ||
      !encode_2d(&tm_u, v.Uup, v.r_pad, static_cast<uint64_t>(L) * d, v.uup_ld, cw) ||
      !encode_slabs(&tm_mem_s, a.mem, d, static_cast<uint64_t>(L) * T, d, kBlockM) ||
      !encode_3d_warp_store(&tm_mem_w, a.mem, d, static_cast<uint64_t>(T), L))
    return cudaErrorInvalidValue;
  // split chain: the low parts of h (its own buffer, H's pitch) and of the products
  CUtensorMap tm_hlo_s = tm_hs, tm_hlo = tm_h, tm_hlo_st = tm_hst;
  if (split && (!encode_slabs(&tm_hlo_s, a.Hlo, n1, static_cast<uint64_t>(T), a.hld, kBlockM, ks) ||
                !encode_2d(&tm_hlo, a.Hlo, n1, static_cast<uint64_t>(T), a.hld, kBlockM) ||
                !encode_2d(&tm_hlo_st, a.Hlo, n1, static_cast<uint64_t>(T), a.hld, 32)))
    return cudaErrorInvalidValue;
  const CUtensorMap& tm_pf_lo = split ? *v.tm_Pf_lo : *v.tm_Pf;
  mark(0);
  // (1) C = E [D_1 .. D_L]^T, every column in fp32
  GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.status = v.status;
  gp.timeout_ns = kTimeoutNs;
  for (int i = 0; i < L; ++i) gp.layer_map[i] = v.active[i];
  gp.s = {static_cast<int>(T), 1, static_cast<int>(n1), d / 64, 0, 0, 0, 0, 0, 0};
  gp.silu = {nullptr, 0, 0, a.c, static_cast<int>(n1)};
  const long long pad128 = (T + 127) / 128 * 128, pad256 = (T + 255) / 256 * 256;
  cudaError_t err;
  if (prefer_256(pad256, pad128)) {
    const long long pairs = v.num_sms / 2;
    int bn = 64;
    for (int cand : {256, 128})
      if (n1 % cand == 0 && (pad256 / 256) * (n1 / cand) >= pairs) {
        bn = cand;
        break;
      }
    tm_groups(gp.s, bn, T);
    err = launch_pair_tm(EPI_SILU, bn, 0, tm_x0_s, tm_x0_s,
                         v.tm_Dst_half[bn == 64 ? 0 : (bn == 128 ? 1 : 2)], gp, v.num_sms, st);
  } else {
    int bn = 64;
    for (int cand : {256, 128})
      if (n1 % cand == 0 && (pad128 / 128) * (n1 / cand) >= v.num_sms) {
        bn = cand;
        break;
      }
    err = launch_gemm(EPI_SILU, bn, 0, tm_x0, tm_x0, v.tm_Dst[bn == 64 ? 0 : (bn == 128 ? 1 : 2)],
                      gp, v.num_sms, st);
  }
  mark(1);
  // (2) the recurrence over the rank-r vectors, (3) the running sum of the memories
  const long long part_ld = static_cast<long long>(d / 64) * T;
  if (err == cudaSuccess)
    err = launch_hchain(v.r_pad, split, T, L, a.c, static_cast<int>(n1), tm_hs, tm_hlo_s, *v.tm_Pf,
                        tm_pf_lo, tm_hst, tm_hlo_st, a.H, split ? a.Hlo : nullptr,
                        static_cast<int>(a.hld), v.status, kTimeoutNs, st);
  if (err == cudaSuccess)
    err = launch_accum(v.r_pad, cw, T, L, d, a.x0, tm_h, tm_hlo, split, tm_u, tm_mem_w, a.part, part_ld,
                       v.status, kTimeoutNs, st);
  mark(2);
  if (err == cudaSuccess)
    err = launch_pdl(k_rstd_parts, dim3(grid_for(static_cast<long long>(L) * T)), dim3(256), st,
                     a.part, L, T, fold_sum_parts(d), part_ld, 1.0f / d, v.rms_eps, a.rstd);
  mark(3);
  return err == cudaSuccess ? launch_recurrent_kv(v, a, T, tm_mem_s, st, mark) : err;
}

// Recurrent adapter (Sec. 3.1 Eq. 6): the chain M_i = M_{i-1} + SiLU(M_{i-1} D_i) U_i runs
// layer by layer (a split-K down-projection, then the up-projection whose epilogue adds the
// fp32 state and writes bf16 M_i and partial sums of squares); the RMS statistics of all
// layers follow in one kernel, and one K/V launch covers every layer, reading M_i as A.
static cudaError_t enqueue_recurrent(const PlanView& v, const BuildArgs& a, cudaStream_t st) {
  if (fold_build(v, static_cast<long long>(a.batch) * a.n_vis)) return enqueue_fold(v, a, st);
  const long long T = static_cast<long long>(a.batch) * a.n_vis;
  const int L = v.n_layers, d = v.d;
  const long long n1 = static_cast<long long>(L) * v.r_pad;
  auto mark = [&](int i) {
    if (a.marks) cudaEventRecord(a.marks[i], st);
  };
  CUtensorMap tm_x0, tm_mem, tm_H, tm_mem_s;
  if (!encode_2d(&tm_x0, a.x0, d, static_cast<uint64_t>(T), d, kBlockM) ||
      !encode_2d(&tm_mem, a.mem, d, static_cast<uint64_t>(L) * T, d, kBlockM) ||
      !encode_2d(&tm_H, a.H, n1, static_cast<uint64_t>(T), n1, kBlockM) ||
      !encode_slabs(&tm_mem_s, a.mem, d, static_cast<uint64_t>(L) * T, d, kBlockM))
    return cudaErrorInvalidValue;

  mark(0);
  mark(1);
  const long long part_ld = static_cast<long long>(d / 64) * T;
  cudaError_t err = cudaSuccess;
  // On chip: one cluster per 128-token block runs the whole chain with the state in TMEM. With
  // the split chain only at r_pad 64: at larger r_pad its low operand parts do not fit beside it.
  int spc = 0, S = 0;
  if ((!v.split_chain || v.r_pad == 64) && chain_shape(d, v.r_pad, &spc, &S)) {
    CUtensorMap tm_u, tm_m3;
    // U_l as [L d][r_pad] (its first copy when the split chain packs [U_l | U_l])
    if (!encode_2d(&tm_u, v.Uup, v.r_pad, static_cast<uint64_t>(L) * d, v.uup_ld, 64 * spc) ||
        !encode_3d(&tm_m3, a.mem, d, static_cast<uint64_t>(T), L, kBlockM))
      return cudaErrorInvalidValue;
    err = launch_chain(v.r_pad, spc, S, T, L, d, tm_x0, *v.tm_Dst_rp, tm_u, tm_m3, a.part, part_ld,
                       a.H, v.status, kTimeoutNs, st, v.split_chain != 0);
    if (err == cudaSuccess) {
      mark(2);
      err = launch_pdl(k_rstd_parts, dim3(grid_for(static_cast<long long>(L) * T)), dim3(256), st,
                       a.part, L, T, S, part_ld, 1.0f / d, v.rms_eps, a.rstd);
      mark(3);
      return err == cudaSuccess ? launch_recurrent_kv(v, a, T, tm_mem_s, st, mark) : err;
    }
    if (err != cudaErrorNotSupported) return err;
    cudaGetLastError();
    // no cluster of that size fits: the refactored chain, or the per-layer launches below
    if (uses_fold(v)) return enqueue_fold(v, a, st);
    err = cudaSuccess;
  }
  const long long m_tiles = (T + kBlockM - 1) / kBlockM;
  const int splits = down_splits(m_tiles, d / kBlockK, v.num_sms);
  DownParams dp;
  std::memset(&dp, 0, sizeof(dp));
  dp.M = static_cast<int>(T);
  dp.k_slabs = d / kBlockK;
  dp.H = a.H;
  dp.ldh = static_cast<int>(n1);
  dp.status = v.status;
  dp.timeout_ns = kTimeoutNs;

  GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.status = v.status;
  gp.timeout_ns = kTimeoutNs;
  // up-projection step: A = h_i (H columns from i * r_pad), B = U_i ([d][r_pad] rows i * d).
  // Split chain: A = [low part of h_i | h_i] (the low part as A0 through a per-layer map) and
  // B = [U_i | U_i], so each product reads h_i in two bf16 parts.
  const bool split = v.split_chain != 0;
  const int kh = v.r_pad / 64;
  gp.s = {static_cast<int>(T), 1, d, split ? kh : 0, kh, v.r_pad, 0, 0, 0, 0};
  CUtensorMap tm_mem_lo = tm_x0;  // split chain: the low part of M_{i-1} (one [T][d] buffer)
  if (split && !encode_2d(&tm_mem_lo, a.mem_lo, d, static_cast<uint64_t>(T), d, kBlockM))
    return cudaErrorInvalidValue;
  dp.Hlo = split ? a.Hlo : nullptr;
  // Large builds at r_pad 256 (one 256-token tile per CTA pair is enough to fill the pairs, so
  // no K split): the down-projection runs on CTA pairs, each SM staging half of D_l instead of
  // every CTA reading all of it from L2. Its maps start at the layer's rows: the previous
  // state (x0 for the first layer) and layer i's rows of the stacked D.
  const bool down_pairs = v.r_pad == 256 && splits == 1 && !split;
  GemmParams gd;
  std::memset(&gd, 0, sizeof(gd));
  gd.status = v.status;
  gd.timeout_ns = kTimeoutNs;
  gd.s = {static_cast<int>(T), 1, v.r_pad, d / 64, 0, 0, 0, 0, 0, 0};
  tm_groups(gd.s, 256, T);
  for (int i = 0; i < L && err == cudaSuccess; ++i) {
    if (down_pairs) {
      CUtensorMap tm_a, tm_b;
      const uint16_t* a_ptr = i == 0 ? static_cast<const uint16_t*>(a.x0)
                                     : a.mem + static_cast<size_t>(i - 1) * T * d;
      if (!encode_slabs(&tm_a, a_ptr, d, static_cast<uint64_t>(T), d, kBlockM) ||
          !encode_slabs(&tm_b, v.Dst + static_cast<size_t>(i) * v.r_pad * v.dst_ld, d, v.r_pad,
                        v.dst_ld, 128))
        return cudaErrorInvalidValue;
      gd.silu = {a.H + static_cast<size_t>(i) * v.r_pad, static_cast<int>(n1), v.r_pad, nullptr, 0};
      err = launch_pair_tm(EPI_SILU, 256, 0, tm_a, tm_a, tm_b, gd, v.num_sms, st);
    } else {
      dp.a_row0 = i == 0 ? 0 : static_cast<int>((i - 1) * T);
      dp.b_row0 = i * v.r_pad;
      dp.h_col0 = i * v.r_pad;
      dp.a_lo = split && i > 0 ? 1 : 0;  // E (layer 0) is exact in bf16: no low part
      err = launch_down_split(v.r_pad, splits, i == 0 ? tm_x0 : tm_mem, tm_mem_lo, *v.tm_Dst_rp,
                              dp, st);
    }
    if (err != cudaSuccess) break;
    gp.s.layer0 = i;
    gp.resid = {static_cast<const uint16_t*>(a.x0), a.state,
                a.mem + static_cast<size_t>(i) * T * d, a.part + static_cast<size_t>(i) * part_ld,
                d, i == 0 ? 1 : 0, split ? a.mem_lo : nullptr};
    CUtensorMap tm_a0 = tm_H;
    if (split && !encode_2d(&tm_a0, a.Hlo + static_cast<size_t>(i) * v.r_pad, v.r_pad,
                            static_cast<uint64_t>(T), n1, kBlockM))
      return cudaErrorInvalidValue;
    err = launch_gemm(EPI_RESID, v.resid_bn, 0, tm_a0, tm_H, *v.tm_Uup, gp, v.num_sms, st);
  }
  mark(2);
  if (err == cudaSuccess) {
    err = launch_pdl(k_rstd_parts, dim3(grid_for(static_cast<long long>(L) * T)), dim3(256), st,
                     a.part, L, T, d / v.resid_bn, part_ld, 1.0f / d, v.rms_eps, a.rstd);
  }
  mark(3);
  return err == cudaSuccess ? launch_recurrent_kv(v, a, T, tm_mem_s, st, mark) : err;
}

cudaError_t enqueue_build(const PlanView& v, const BuildArgs& a, cudaStream_t st) {
  if (v.adapter == DV_ADAPTER_RECURRENT) return enqueue_recurrent(v, a, st);
  const long long T = static_cast<long long>(a.batch) * a.n_vis;
  const int L = v.n_layers, d = v.d;
  const long long n1 = static_cast<long long>(L) * v.r_pad;
  auto mark = [&](int i) {
    if (a.marks) cudaEventRecord(a.marks[i], st);
  };
  const long long pad128 = (T + 127) / 128 * 128, pad256 = (T + 255) / 256 * 256;
  const bool rank_pairs = prefer_256(pad256, pad128);

  // 2-D maps for the 1-SM kernel, slab maps (two K slabs per box) for the CTA-pair kernels. The
  // down-projection reads the caller's E; the statistic and the K/V GEMM read the row sums'
  // copy of it (x0p, pitch d + 64), and H has pitch hld = L r_pad + 64 (see k_row_sumsq).
  const long long hld = a.hld, xld = a.x0p_ld;
  CUtensorMap tm_x0, tm_H, tm_x0_s, tm_H_s, tm_xp, tm_xp_s;
  if (!encode_2d(&tm_x0, a.x0, d, static_cast<uint64_t>(T), d, kBlockM) ||
      !encode_2d(&tm_H, a.H, n1, static_cast<uint64_t>(T), hld, kBlockM) ||
      !encode_slabs(&tm_x0_s, a.x0, d, static_cast<uint64_t>(T), d, kBlockM) ||
      !encode_slabs(&tm_H_s, a.H, n1, static_cast<uint64_t>(T), hld, kBlockM) ||
      !encode_2d(&tm_xp, a.x0p, d, static_cast<uint64_t>(T), xld, kBlockM) ||
      !encode_slabs(&tm_xp_s, a.x0p, d, static_cast<uint64_t>(T), xld, kBlockM))
    return cudaErrorInvalidValue;

  GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.status = v.status;
  gp.timeout_ns = kTimeoutNs;
  for (int i = 0; i < L; ++i) gp.layer_map[i] = v.active[i];

  // xx = row sums of squares of x0, launched after the down-projection (see k_row_sumsq).
  auto row_sumsq = [&]() {
    return launch_pdl(k_row_sumsq, dim3(static_cast<unsigned>((T + 7) / 8)), dim3(256), st,
                      static_cast<const uint16_t*>(a.x0), static_cast<int>(T), d, a.xx, a.x0p, xld);
  };
  mark(0);
  cudaError_t err = cudaSuccess;

  // (1) H = SiLU(x0 [D_1 ... D_L]) — one GEMM over all layers' down-projections.
  gp.s = {static_cast<int>(T), 1, static_cast<int>(n1), d / 64, 0, 0, 0, 0, 0, 0};
  gp.silu = {a.H, static_cast<int>(hld), static_cast<int>(n1), nullptr, 0};
  if (!rank_pairs && a.c) {
    // Small or awkward token counts: x0 [D_1 .. D_L | 2U_1 .. 2U_L]^T as one GEMM (the
    // down-projections get SiLU, the second half is c_l = x0 (2 U_l)^T in fp32), then the
    // statistic of M_l from h_l, c_l and G_l in a small kernel: one tensor-core pass over x0
    // instead of two GEMMs of long K over few token blocks.
    // On CTA pairs (256-token blocks, each SM staging half of the weight rows): the K loop is
    // long and the tiles few, so the bytes each SM must stage per slab, not the MMA work, set the
    // time; the 256-token padding only adds MMA work.
    const long long n2 = 2 * n1;
    // a tile is either all down-projection columns or all c columns: bn divides n1
    const int bn = n1 % 256 == 0 ? 256 : (n1 % 128 == 0 ? 128 : 64);
    gp.s = {static_cast<int>(T), 1, static_cast<int>(n2), d / 64, 0, 0, 0, 0, 0, 0};
    gp.silu = {a.H, static_cast<int>(hld), static_cast<int>(n1), a.c, static_cast<int>(n1)};
    tm_groups(gp.s, bn, T);
    const CUtensorMap& tmD = v.tm_Dst_half[bn == 64 ? 0 : (bn == 128 ? 1 : 2)];
    if (err == cudaSuccess) err = launch_pair_tm(EPI_SILU, bn, 0, tm_x0_s, tm_x0_s, tmD, gp, v.num_sms, st);
    mark(1);
    if (err == cudaSuccess) err = row_sumsq();
    mark(2);
    if (err == cudaSuccess) {
      dim3 grid(static_cast<unsigned>((T + 63) / 64), static_cast<unsigned>(L));
      err = launch_pdl(k_rstd_hc<64>, grid, dim3(64), st, static_cast<const uint16_t*>(a.H),
                       static_cast<int>(hld), static_cast<const float*>(a.c), static_cast<int>(n1),
                       static_cast<const float*>(a.xx), v.Gf, static_cast<int>(T), 1.0f / d,
                       v.rms_eps, a.rstd);
    }
    mark(3);
  } else {
  if (rank_pairs) {
    const long long pairs = v.num_sms / 2;
    int bn = 64;
    for (int cand : {256, 128}) {
      if (n1 % cand == 0 && (pad256 / 256) * (n1 / cand) >= pairs) {
        bn = cand;
        break;
      }
    }
    const CUtensorMap& tmD = v.tm_Dst_half[bn == 64 ? 0 : (bn == 128 ? 1 : 2)];
    tm_groups(gp.s, bn, T);
    if (err == cudaSuccess) err = launch_pair_tm(EPI_SILU, bn, 0, tm_x0_s, tm_x0_s, tmD, gp, v.num_sms, st);
  } else {
    const long long m_tiles = pad128 / 128;
    int bn = 64;
    for (int cand : {256, 128}) {
      if (n1 % cand == 0 && m_tiles * (n1 / cand) >= v.num_sms) {
        bn = cand;
        break;
      }
    }
    const CUtensorMap& tmD = v.tm_Dst[bn == 64 ? 0 : (bn == 128 ? 1 : 2)];
    if (err == cudaSuccess) err = launch_gemm(EPI_SILU, bn, 0, tm_x0, tm_x0, tmD, gp, v.num_sms, st);
  }
  mark(1);
  if (err == cudaSuccess) err = row_sumsq();
  mark(2);

  // (2) rstd_l from ||x0||^2 + h_l . ([x0 | h_l] [2 U_l^T ; G_l]): 256-column tiles of lpt
  // layers each, A = [x0 | h of the group's layers] (contiguous H columns), B = the group's
  // Bn rows (block-diagonal G).
  const int lpt = v.bn_lpt;
  gp.s = {static_cast<int>(T), v.bn_groups, 256, d / 64, lpt * v.r_pad / 64, lpt * v.r_pad, 0, 0, 0, 0};
  if (rank_pairs) tm_groups(gp.s, 256, T);
  gp.norm = {a.H, static_cast<int>(hld), v.r_pad, lpt, v.bn_rn, L, a.xx, a.rstd,
             static_cast<int>(T), 1.0f / d, v.rms_eps};
  if (err == cudaSuccess) {
    err = rank_pairs ? launch_pair_tm(EPI_NORM, 256, 0, tm_xp_s, tm_H_s, *v.tm_Bn_half, gp, v.num_sms, st)
                     : launch_gemm(EPI_NORM, 256, 0, tm_xp, tm_H, *v.tm_Bn, gp, v.num_sms, st);
  }
  mark(3);
  }

  // (3) K/V = rstd_l * ([x0 | h_l] Wkv_l^T) + b, RoPE on K, stored into the cache.
  gp.s = {static_cast<int>(T), L, 2 * v.kv, d / 64, v.r_pad / 64, v.r_pad, 0, 0, 0, 0};
  fill_epi_kv(v, a, T, gp.kv);
  if (err == cudaSuccess)
    err = launch_kv_stage(v, gp, T, a.x0p, static_cast<uint64_t>(T), static_cast<uint64_t>(xld),
                          tm_xp_s, a.H, static_cast<uint64_t>(n1), static_cast<uint64_t>(hld),
                          tm_H_s, st);
  mark(4);
  return err;
}

size_t carve_workspace(const PlanView& v, long long T, void* base, BuildArgs* a) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) / 256 * 256;
    return o;
  };
  const size_t L = static_cast<size_t>(v.n_layers), t = static_cast<size_t>(T);
  const size_t d = static_cast<size_t>(v.d);
  const bool rec = v.adapter == DV_ADAPTER_RECURRENT;
  // Embedding adapter: H rows and the copy of E get a pitch 64 elements (128 bytes) past their
  // width, so that no row pitch is a power of two (see k_row_sumsq).
  const size_t hld = L * v.r_pad + (rec ? 0 : 64), xld = d + 64;
  const size_t oH = take(t * hld * 2), oR = take(L * t * 4), oX = take(t * 4);
  const size_t oXp = rec ? 0 : take(t * xld * 2);
  size_t oS = 0, oM = 0, oP = 0, oC = 0, oHl = 0, oMl = 0;
  // fp32 [tokens][L r_pad]: x0 (2 U_l)^T of the embedding adapter at small token counts (see
  // enqueue_build), or E D_l^T of the recurrent adapter's refactored chain, which needs no fp32
  // state
  const bool fold = rec && uses_fold(v);
  const bool small_path = !rec && v.r_pad == 64;
  if (small_path || fold) oC = take(t * L * v.r_pad * 4);
  if (rec) {
    if (!fold) oS = take(t * d * 4);
    oM = take(L * t * d * 2);
    oP = take(L * (d / 64) * t * 4);
    if (v.split_chain) {  // low bf16 parts of h_l (every layer) and of the last M_l
      oHl = take(t * L * v.r_pad * 2);
      oMl = take(t * d * 2);
    }
  }
  if (base && a) {
    unsigned char* b = static_cast<unsigned char*>(base);
    a->H = reinterpret_cast<uint16_t*>(b + oH);
    a->hld = static_cast<long long>(hld);
    a->x0p = rec ? nullptr : reinterpret_cast<uint16_t*>(b + oXp);
    a->x0p_ld = static_cast<long long>(xld);
    a->rstd = reinterpret_cast<float*>(b + oR);
    a->xx = reinterpret_cast<float*>(b + oX);
    a->state = rec && !fold ? reinterpret_cast<float*>(b + oS) : nullptr;
    a->mem = rec ? reinterpret_cast<uint16_t*>(b + oM) : nullptr;
    a->part = rec ? reinterpret_cast<float*>(b + oP) : nullptr;
    a->c = small_path || fold ? reinterpret_cast<float*>(b + oC) : nullptr;
    const bool split = rec && v.split_chain;
    a->Hlo = split ? reinterpret_cast<uint16_t*>(b + oHl) : nullptr;
    a->mem_lo = split ? reinterpret_cast<uint16_t*>(b + oMl) : nullptr;
  }
  return off;
}

bool plan_view(const dv_plan* p, PlanView* v) {
  if (!p || !v) return false;
  const dv_config& c = p->cfg;
  v->d = c.d;
  v->n_layers = p->n_active;
  v->adapter = c.adapter;
  v->kg = p->kg;
  v->k_eps = c.k_norm_eps;
  v->head_dim = c.head_dim;
  v->rope = c.rope;
  for (int i = 0; i < 3; ++i) v->mrope_section[i] = c.mrope_section[i];
  v->rms_eps = c.rms_eps;
  v->num_sms = p->num_sms;
  v->r_pad = p->r_pad;
  v->kv = p->kv;
  v->k_total = p->k_total;
  v->bk = p->bk;
  v->bv = p->bv;
  v->status = p->status;
  v->tm_Dst = p->tm_Dst;
  v->Gf = p->Gf;
  v->tm_Dst_half = p->tm_Dst_half;
  v->tm_Bn = &p->tm_Bn;
  v->bn_lpt = p->bn_lpt;
  v->bn_rn = p->bn_rn;
  v->bn_groups = p->bn_groups;
  v->tm_Bn_half = &p->tm_Bn_half;
  v->tm_Wkv = &p->tm_Wkv;
  v->tm_Dst_rp = &p->tm_Dst_rp;
  v->tm_Uup = &p->tm_Uup;
  v->Uup = p->Uup;
  v->tm_Pf = p->fold ? &p->tm_Pf : nullptr;
  v->tm_Pf_lo = p->fold && c.split_chain ? &p->tm_Pf_lo : nullptr;
  v->chain_clusters = p->chain_clusters;
  v->uup_ld = p->uup_ld;
  v->split_chain = p->cfg.split_chain;
  v->Dst = p->Dst;
  v->dst_ld = c.d + 64;  // as the plan allocates Dst
  v->resid_bn = p->resid_bn;
  v->inv_freq = p->inv_freq;
  v->Wkv = p->Wkv;
  v->active = p->active;
  return true;
}

const dv_config* plan_config(const dv_plan* p) { return p ? &p->cfg : nullptr; }
void* plan_scratch(const dv_plan* p) { return p ? p->scratch : nullptr; }

bool encode_bf16_2d(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint64_t ld,
                    uint32_t box_rows) {
  return encode_2d(map, ptr, cols, rows, ld, box_rows);
}

}  // namespace dv

namespace {

// CUDA loads modules and kernels lazily, on first use, and loading takes device memory for their
// code. The plan loads every kernel its builds can launch, so that builds allocate nothing (the
// no-allocation entry relies on this). Each launcher, given no tokens, sets its kernel's
// attributes (which loads it) and returns without launching; the dispatchers cover every
// instantiation a build of this plan can pick.
cudaError_t preload_build_kernels(const dv_plan* p) {
  GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  CUtensorMap m;
  std::memset(&m, 0, sizeof(m));
  cudaError_t err = cudaSuccess;
  auto keep = [&](cudaError_t e) {
    if (err == cudaSuccess) err = e;
  };
  const int hd = p->cfg.head_dim;
  for (int bn : {64, 128, 256}) {
    keep(dv::launch_gemm(dv::EPI_SILU, bn, 0, m, m, m, gp, 1, nullptr));
    keep(dv::launch_gemm(dv::EPI_NORM, bn, 0, m, m, m, gp, 1, nullptr));
    keep(dv::launch_gemm(dv::EPI_RESID, bn, 0, m, m, m, gp, 1, nullptr));
    keep(dv::launch_pair_tm(dv::EPI_SILU, bn, 0, m, m, m, gp, 1, nullptr));
    keep(dv::launch_pair_tm(dv::EPI_NORM, bn, 0, m, m, m, gp, 1, nullptr));
  }
  keep(dv::launch_pair_tm(dv::EPI_KV, 256, hd, m, m, m, gp, 1, nullptr));
  for (int nt : {64, 128, 192, 256}) keep(dv::launch_kv_pair(hd, nt, m, m, m, gp, 1, nullptr));
  if (p->fold) {
    const int cw = dv::fold_slice_cols(p->cfg.d);
    keep(dv::launch_hchain(p->r_pad, p->cfg.split_chain != 0, 0, 1, nullptr, 0, m, m, m, m, m, m,
                           nullptr, nullptr, 0, nullptr, 0, nullptr));
    keep(dv::launch_accum(p->r_pad, cw, 0, 1, p->cfg.d, nullptr, m, m, false, m, m, nullptr, 0,
                          nullptr, 0, nullptr));
  }
  if (p->cfg.adapter == DV_ADAPTER_RECURRENT) {
    dv::DownParams dp;
    std::memset(&dp, 0, sizeof(dp));
    dp.k_slabs = 8;
    for (int s : {1, 2, 4, 8}) keep(dv::launch_down_split(p->r_pad, s, m, m, m, dp, nullptr));
    int spc = 0, S = 0;
    if (dv::chain_shape(p->cfg.d, p->r_pad, &spc, &S) && (!p->cfg.split_chain || p->r_pad == 64))
      keep(dv::launch_chain(p->r_pad, spc, S, 0, 1, p->cfg.d, m, m, m, m, nullptr, 0, nullptr,
                            nullptr, 0, nullptr, p->cfg.split_chain != 0));
  }
  return err;
}

}  // namespace

// ================================================================================== C ABI

extern "C" {

const char* dv_error_string(int s) {
  switch (s) {
    case DV_OK: return "ok";
    case DV_ERR_INVALID_ARG: return "invalid argument";
    case DV_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
    case DV_ERR_ALIGNMENT: return "pointer or stride not 16-byte aligned";
    case DV_ERR_OOM: return "device out of memory";
    case DV_ERR_CUDA: return "CUDA call failed";
    case DV_ERR_DEVICE_TIMEOUT: return "a device-side wait timed out";
    case DV_ERR_UNSUPPORTED_DEVICE: return "device is not an sm_103 GPU";
    default: return "unknown status";
  }
}

int dv_memory_plan(const dv_config* cfg, const dv_weights* w, void* stream, dv_plan** out) {
  if (!out) return DV_ERR_INVALID_ARG;
  *out = nullptr;
  int rc = check_config(cfg);
  if (rc != DV_OK) return rc;
  if (!w || !w->D || !w->U || !w->gamma || !w->Wk || !w->Wv) return DV_ERR_INVALID_ARG;
  if (cfg->has_kv_bias && (!w->bk || !w->bv)) return DV_ERR_INVALID_ARG;
  const void* wp[] = {w->D, w->U, w->gamma, w->Wk, w->Wv};
  for (const void* q : wp)
    if (!aligned2(q)) return DV_ERR_ALIGNMENT;
  if (cfg->has_kv_bias && (!aligned2(w->bk) || !aligned2(w->bv))) return DV_ERR_ALIGNMENT;
  if (cfg->k_norm && !w->k_norm_gamma) return DV_ERR_INVALID_ARG;
  if (cfg->k_norm && !aligned2(w->k_norm_gamma)) return DV_ERR_ALIGNMENT;

  int n_active = 0;
  for (int l = 0; l < cfg->n_layers; ++l) {
    const unsigned char m = w->layer_mode ? w->layer_mode[l] : DV_LAYER_ADAPTER;
    if (m != DV_LAYER_ADAPTER && m != DV_LAYER_IDENTITY && m != DV_LAYER_DROP) return DV_ERR_INVALID_ARG;
    if (m != DV_LAYER_DROP) ++n_active;
  }
  if (n_active == 0) return DV_ERR_INVALID_ARG;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DV_ERR_CUDA;
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return DV_ERR_CUDA;
  if (prop.major != 10 || prop.minor != 3) return DV_ERR_UNSUPPORTED_DEVICE;
  if (!encode_fn()) return DV_ERR_CUDA;

  // The build's small kernels ask for the same shared-memory carveout as its GEMMs (all of it),
  // so that consecutive launches need no L1 / shared-memory reconfiguration between them.
  {
    const void* small[] = {reinterpret_cast<const void*>(k_row_sumsq),
                           reinterpret_cast<const void*>(k_rstd_parts),
                           reinterpret_cast<const void*>(k_rstd_hc<64>)};
    for (const void* f : small)
      if (cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout,
                               cudaSharedmemCarveoutMaxShared) != cudaSuccess)
        cudaGetLastError();
  }

  dv_plan* p = new (std::nothrow) dv_plan();
  if (!p) return DV_ERR_OOM;
  p->cfg = *cfg;
  p->device = dev;
  p->num_sms = prop.multiProcessorCount;
  const int d = cfg->d, r = cfg->rank, HD = cfg->head_dim;
  for (int l = 0; l < cfg->n_layers; ++l) {
    p->mode[l] = w->layer_mode ? w->layer_mode[l] : DV_LAYER_ADAPTER;
    if (p->mode[l] != DV_LAYER_DROP) p->active[p->n_active++] = static_cast<int16_t>(l);
  }
  // The plan holds the layers that are not dropped, compacted: planned layer i is cache layer
  // active[i]; dropped layers take no weight or workspace memory.
  const int L = p->n_active;
  const bool rec = cfg->adapter == DV_ADAPTER_RECURRENT;
  p->r_pad = (r + 63) / 64 * 64;
  p->kv = cfg->n_kv_heads * HD;
  // Embedding adapter: K/V weights carry the folded rank-r columns. Recurrent: the K/V GEMM
  // reads M_l itself, so only the d columns of W diag(gamma).
  p->k_total = rec ? d : d + p->r_pad;
  dv::norm_group(p->r_pad, &p->bn_lpt, &p->bn_rn);
  p->bn_groups = (L + p->bn_lpt - 1) / p->bn_lpt;
  p->bn_k = d + p->bn_lpt * p->r_pad;
  p->resid_bn = d % 256 == 0 ? 256 : (d % 128 == 0 ? 128 : 64);
  p->uup_ld = cfg->split_chain ? 2 * p->r_pad : p->r_pad;
  p->max_tokens = cfg->max_batch * cfg->max_n_vis;
  const long long T = p->max_tokens;
  // Recurrent adapter: the refactored chain (dv_fold.cu); builds whose token blocks fit in one
  // wave of on-chip chain clusters take the chain instead (DV_RECURRENT_AUTO).
  p->fold = rec && dv::fold_slice_cols(d) > 0 && cfg->recurrent_path != DV_RECURRENT_CHAIN;
  p->chain_clusters = rec && cfg->recurrent_path != DV_RECURRENT_REARRANGED
                          ? dv::chain_resident_clusters(d, p->r_pad, cfg->split_chain != 0)
                          : 0;
  const long long pf_ld = static_cast<long long>(L) * p->r_pad;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The recurrent K/V GEMM addresses the stacked M_l as L * T rows (32-bit TMA coordinates).
  if (rec && static_cast<long long>(L) * T + dv::kBlockM >= (1LL << 31)) {
    delete p;
    return DV_ERR_UNSUPPORTED_SHAPE;
  }
  dv::PlanView pv;
  dv::plan_view(p, &pv);
  const size_t ws_bytes = dv::carve_workspace(pv, T, nullptr, nullptr);

  // Embedding adapter: Dst stacks 2 U^T under D (rows [L r_pad, 2 L r_pad)) for the small-token
  // path, which forms the statistic of M_l from x0 (2 U_l)^T and the fp32 G_l.
  const int dst_rows = (rec ? 1 : 2) * L * p->r_pad;
  // Rows padded by 64 elements: a stride that is not a power of two spreads the rows of a
  // 128-row TMA box over the L2 (the K/V weights' d + r_pad stride does the same).
  const int dst_ld = d + 64;
  bool ok = dmalloc(&p->Dst, sizeof(uint16_t) * dst_rows * dst_ld) &&
            (rec ? dmalloc(&p->Uup, sizeof(uint16_t) * static_cast<size_t>(L) * d * p->uup_ld)
                 : dmalloc(&p->Bn, sizeof(uint16_t) * p->bn_groups * 256 * p->bn_k)) &&
            dmalloc(&p->Wkv, sizeof(uint16_t) * static_cast<size_t>(L) * 2 * p->kv * p->k_total) &&
            dmalloc(&p->ws, ws_bytes) && dmalloc(&p->status, sizeof(int));
  if (ok && cfg->has_kv_bias)
    ok = dmalloc(&p->bk, sizeof(float) * L * p->kv) && dmalloc(&p->bv, sizeof(float) * L * p->kv);
  if (ok && cfg->k_norm) ok = dmalloc(&p->kg, sizeof(float) * L * HD);
  if (ok && !rec) ok = dmalloc(&p->Gf, sizeof(float) * L * p->r_pad * p->r_pad);
  const size_t pf_bytes = sizeof(uint16_t) * static_cast<size_t>(L) * p->r_pad * pf_ld;
  if (ok && p->fold) ok = dmalloc(&p->Pf, pf_bytes);
  if (ok && p->fold && cfg->split_chain) ok = dmalloc(&p->Pf_lo, pf_bytes);
  if (!ok) {
    free_plan_memory(p);
    delete p;
    return DV_ERR_OOM;
  }

  PackLayers pl;
  std::memset(&pl, 0, sizeof(pl));
  for (int i = 0; i < L; ++i) {
    pl.src[i] = p->active[i];
    pl.zero_du[i] = p->mode[p->active[i]] == DV_LAYER_IDENTITY;
  }
  const uint16_t* D = static_cast<const uint16_t*>(w->D);
  const uint16_t* U = static_cast<const uint16_t*>(w->U);
  const uint16_t* G = static_cast<const uint16_t*>(w->gamma);
  const uint16_t* Wk = static_cast<const uint16_t*>(w->Wk);
  const uint16_t* Wv = static_cast<const uint16_t*>(w->Wv);
  cudaMemsetAsync(p->status, 0, sizeof(int), st);
  k_pack_down<<<grid_for(1LL * L * p->r_pad * d), 256, 0, st>>>(D, p->Dst, L, r, p->r_pad, d,
                                                                dst_ld, pl);
  k_pack_kv<<<grid_for(1LL * L * 2 * p->kv * p->k_total), 256, 0, st>>>(Wk, Wv, G, p->Wkv, L, p->kv,
                                                                        HD, d, p->k_total, pl);
  if (rec) {
    k_pack_up<<<grid_for(1LL * L * d * p->uup_ld), 256, 0, st>>>(U, p->Uup, L, r, p->r_pad, d,
                                                                 p->uup_ld, pl);
    if (p->fold) {
      cudaMemsetAsync(p->Pf, 0, pf_bytes, st);
      if (p->Pf_lo) cudaMemsetAsync(p->Pf_lo, 0, pf_bytes, st);
      if (L > 1) {
        const dim3 gq(p->r_pad / 64, L * (p->r_pad / 64), L);
        k_fold_products<<<gq, 256, 0, st>>>(D, U, p->Pf, p->Pf_lo, L, r, p->r_pad, d, pf_ld, pl);
      }
    }
  } else {
    k_pack_2u<<<grid_for(1LL * L * p->r_pad * d), 256, 0, st>>>(
        U, p->Dst + static_cast<size_t>(L) * p->r_pad * dst_ld, L, r, p->r_pad, d, dst_ld, pl);
    cudaMemsetAsync(p->Gf, 0, sizeof(float) * L * p->r_pad * p->r_pad, st);
    k_pack_norm_u<<<grid_for(1LL * p->bn_groups * 256 * p->bn_k), 256, 0, st>>>(
        U, p->Bn, L, r, d, p->bn_lpt, p->bn_rn, p->bn_groups, p->bn_k, pl);
    dim3 g1((r + 63) / 64, (r + 63) / 64, L);
    k_rank_product<1><<<g1, 256, 0, st>>>(Wk, Wv, G, U, p->Bn, r, r, d, p->kv, HD, p->r_pad,
                                          p->bn_k, pl, p->Gf, p->bn_lpt, p->bn_rn);
    dim3 g0((r + 63) / 64, (2 * p->kv + 63) / 64, L);
    k_rank_product<0><<<g0, 256, 0, st>>>(Wk, Wv, G, U, p->Wkv, 2 * p->kv, r, d, p->kv, HD,
                                          p->r_pad, p->k_total, pl, nullptr, 1, 0);
  }
  if (cfg->has_kv_bias) {
    k_bias_to_f32<<<grid_for(1LL * L * p->kv), 256, 0, st>>>(static_cast<const uint16_t*>(w->bk),
                                                             p->bk, L, p->kv, pl);
    k_bias_to_f32<<<grid_for(1LL * L * p->kv), 256, 0, st>>>(static_cast<const uint16_t*>(w->bv),
                                                             p->bv, L, p->kv, pl);
  }
  if (cfg->k_norm)
    k_bias_to_f32<<<grid_for(1LL * L * HD), 256, 0, st>>>(
        static_cast<const uint16_t*>(w->k_norm_gamma), p->kg, L, HD, pl);
  cudaError_t err = cudaGetLastError();
  if (err == cudaSuccess) err = cudaStreamSynchronize(st);
  if (err != cudaSuccess) {
    free_plan_memory(p);
    delete p;
    return DV_ERR_CUDA;
  }

  bool enc = encode_2d(&p->tm_Dst[0], p->Dst, d, dst_rows, dst_ld, 64) &&
             encode_2d(&p->tm_Dst[1], p->Dst, d, dst_rows, dst_ld, 128) &&
             encode_2d(&p->tm_Dst[2], p->Dst, d, dst_rows, dst_ld, 256) &&
             encode_slabs(&p->tm_Dst_half[0], p->Dst, d, dst_rows, dst_ld, 32) &&
             encode_slabs(&p->tm_Dst_half[1], p->Dst, d, dst_rows, dst_ld, 64) &&
             encode_slabs(&p->tm_Dst_half[2], p->Dst, d, dst_rows, dst_ld, 128) &&
             encode_slabs(&p->tm_Wkv, p->Wkv, p->k_total, 1ull * L * 2 * p->kv, p->k_total, 128);
  if (enc && rec) {
    enc = encode_2d(&p->tm_Dst_rp, p->Dst, d, 1ull * L * p->r_pad, dst_ld, p->r_pad) &&
          encode_2d(&p->tm_Uup, p->Uup, p->uup_ld, 1ull * L * d, p->uup_ld, p->resid_bn);
    if (enc && p->fold)
      // boxes of r_pad / 2 rows: each CTA of a recurrence pair stages half of a layer's rows
      enc = encode_slabs(&p->tm_Pf, p->Pf, pf_ld, 1ull * L * p->r_pad, pf_ld, p->r_pad / 2,
                         static_cast<uint32_t>(dv::hchain_box_slabs(p->r_pad, cfg->split_chain)));
    if (enc && p->Pf_lo)
      enc = encode_slabs(&p->tm_Pf_lo, p->Pf_lo, pf_ld, 1ull * L * p->r_pad, pf_ld, p->r_pad / 2,
                         static_cast<uint32_t>(dv::hchain_box_slabs(p->r_pad, true)));
  } else if (enc) {
    enc = encode_slabs(&p->tm_Bn_half, p->Bn, p->bn_k, 256ull * p->bn_groups, p->bn_k, 128) &&
          encode_2d(&p->tm_Bn, p->Bn, p->bn_k, 256ull * p->bn_groups, p->bn_k, 256);
  }
  if (!enc) {
    free_plan_memory(p);
    delete p;
    return DV_ERR_CUDA;
  }
  for (int j = 0; j < HD / 2; ++j)
    p->inv_freq[j] = std::pow(static_cast<double>(cfg->rope_theta), -2.0 * j / HD);
  if (preload_build_kernels(p) != cudaSuccess) {
    cudaGetLastError();
    free_plan_memory(p);
    delete p;
    return DV_ERR_CUDA;
  }
  // The no-allocation entry's scratch array: looked up (and so reserved) now. If that fails the
  // plan still serves the other entry points; dv_build_visual_memory_noalloc then reports it.
  if (dv::noalloc_scratch(&p->scratch) != DV_OK) {
    cudaGetLastError();
    p->scratch = nullptr;
  }
  *out = p;
  return DV_OK;
}

int dv_kv_engine(const dv_plan* p, long long tokens) {
  if (!p || tokens <= 0) return 0;
  const int nt = dv::kv_pair_tile_n(tokens);
  const long long pad256 = (tokens + 255) / 256 * 256, pad_nt = (tokens + nt - 1) / nt * nt;
  return dv::prefer_256(pad256, pad_nt) ? DV_KV_ENGINE_TOKENS_AS_M : DV_KV_ENGINE_WEIGHTS_AS_M;
}

// Embedding adapter: row sums, stacked down-projection, RMS statistics, K/V. Recurrent: two
// launches per planned layer, the RMS statistics and K/V.
int dv_kernels_per_build(const dv_plan* p) {
  if (!p) return 0;
  if (p->cfg.adapter != DV_ADAPTER_RECURRENT) return kStages;
  // recurrent, at the plan's full size: the rearranged chain (E D^T, the recurrence, the running
  // sum, statistics, K/V), the on-chip chain (chain, statistics, K/V) or the per-layer launches
  const long long blocks = (p->max_tokens + dv::kBlockM - 1) / dv::kBlockM;
  if (p->fold && blocks > p->chain_clusters) return 5;
  if (p->chain_clusters > 0) return 3;
  return p->fold ? 5 : 2 * p->n_active + 2;
}

int dv_build_visual_memory(dv_plan* p, const void* x0, int batch, int n_vis, const int* pos,
                           const int* slot, int slot0, const dv_kv_cache* out, void* stream) {
  if (!p) return DV_ERR_INVALID_ARG;
  int rc = dv::check_build_args(x0, batch, n_vis, pos, slot, slot0, out);
  if (rc != DV_OK) return rc;
  const long long T = static_cast<long long>(batch) * n_vis;
  if (T == 0) return DV_OK;
  if (batch > p->cfg.max_batch || n_vis > p->cfg.max_n_vis || T > p->max_tokens)
    return DV_ERR_UNSUPPORTED_SHAPE;
  dv::PlanView v;
  dv::plan_view(p, &v);
  dv::BuildArgs a;
  a.x0 = x0;
  a.batch = batch;
  a.n_vis = n_vis;
  a.pos = pos;
  a.slot = slot;
  a.slot0 = slot0;
  a.kc = out->k;
  a.vc = out->v;
  a.s_layer = out->s_layer;
  a.s_batch = out->s_batch;
  a.s_seq = out->s_seq;
  a.s_head = out->s_head;
  dv::carve_workspace(v, T, p->ws, &a);
  p->last_tokens = T;
  a.marks = (p->timing && p->timed < kMaxTimed) ? &p->ev[static_cast<size_t>(p->timed++) * kEvPerBuild]
                                                : nullptr;
  return dv::enqueue_build(v, a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? DV_OK
                                                                                   : DV_ERR_CUDA;
}

int dv_plan_status(dv_plan* p) {
  if (!p) return DV_ERR_INVALID_ARG;
  int s = 0;
  if (cudaDeviceSynchronize() != cudaSuccess) return DV_ERR_CUDA;
  if (cudaMemcpy(&s, p->status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return DV_ERR_CUDA;
  if (s != 0 && cudaMemset(p->status, 0, sizeof(int)) != cudaSuccess) return DV_ERR_CUDA;
  return s;
}

void dv_free(dv_plan* p) {
  if (!p) return;
  cudaDeviceSynchronize();
  free_plan_memory(p);
  delete p;
}

int dv_timing_enable(dv_plan* p, int on) {
  if (!p) return DV_ERR_INVALID_ARG;
  p->timing = on != 0;
  p->timed = 0;
  if (on && p->ev.empty()) {
    p->ev.resize(static_cast<size_t>(kMaxTimed) * kEvPerBuild);
    for (auto& e : p->ev)
      if (cudaEventCreate(&e) != cudaSuccess) return DV_ERR_CUDA;
  }
  return DV_OK;
}

int dv_timing_read(dv_plan* p, double* ms, int n_stages, int* n_builds) {
  if (!p || !ms || !n_builds || n_stages < 0 || n_stages > kStages) return DV_ERR_INVALID_ARG;
  for (int s = 0; s < n_stages; ++s) ms[s] = 0.0;
  for (int b = 0; b < p->timed; ++b) {
    cudaEvent_t* ev = &p->ev[static_cast<size_t>(b) * kEvPerBuild];
    if (cudaEventSynchronize(ev[kStages]) != cudaSuccess) return DV_ERR_CUDA;
    for (int s = 0; s < n_stages; ++s) {
      float t = 0.0f;
      if (cudaEventElapsedTime(&t, ev[s], ev[s + 1]) != cudaSuccess) return DV_ERR_CUDA;
      ms[s] += t;
    }
  }
  *n_builds = p->timed;
  return DV_OK;
}

int dv_debug_wait_timeout(dv_plan* p, int timeout_us, void* stream) {
  if (!p || timeout_us < 1 || timeout_us > 2000000) return DV_ERR_INVALID_ARG;
  k_wait_timeout<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      p->status, static_cast<unsigned long long>(timeout_us) * 1000ull);
  return cudaGetLastError() == cudaSuccess ? DV_OK : DV_ERR_CUDA;
}

int dv_debug_copy_workspace(dv_plan* p, int tokens, void* H, void* rstd, void* xx,
                            int* r_pad_out, void* stream) {
  if (!p || tokens < 0 || tokens > p->last_tokens) return DV_ERR_INVALID_ARG;
  if (r_pad_out) *r_pad_out = p->r_pad;
  if (tokens == 0) return DV_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dv::PlanView v;
  dv::plan_view(p, &v);
  dv::BuildArgs a;
  dv::carve_workspace(v, p->last_tokens, p->ws, &a);  // the layout of the last build
  const int L = p->n_active;  // the workspace holds the planned (not dropped) layers
  const size_t hrow = static_cast<size_t>(L) * p->r_pad;
  const size_t T = static_cast<size_t>(p->last_tokens);
  cudaError_t err = cudaSuccess;
  if (H)
    err = cudaMemcpy2DAsync(H, sizeof(uint16_t) * hrow, a.H, sizeof(uint16_t) * a.hld,
                            sizeof(uint16_t) * hrow, tokens, cudaMemcpyDeviceToDevice, st);
  if (rstd && err == cudaSuccess)
    err = cudaMemcpy2DAsync(rstd, sizeof(float) * tokens, a.rstd, sizeof(float) * T,
                            sizeof(float) * tokens, L, cudaMemcpyDeviceToDevice, st);
  if (xx && err == cudaSuccess)
    err = cudaMemcpyAsync(xx, a.xx, sizeof(float) * tokens, cudaMemcpyDeviceToDevice, st);
  return err == cudaSuccess ? DV_OK : DV_ERR_CUDA;
}

int dv_debug_copy_memory(dv_plan* p, int tokens, void* mem, void* stream) {
  if (!p || !mem || tokens < 0 || tokens > p->last_tokens) return DV_ERR_INVALID_ARG;
  if (p->cfg.adapter != DV_ADAPTER_RECURRENT) return DV_ERR_INVALID_ARG;
  if (tokens == 0) return DV_OK;
  dv::PlanView v;
  dv::plan_view(p, &v);
  dv::BuildArgs a;
  dv::carve_workspace(v, p->last_tokens, p->ws, &a);
  const size_t row = sizeof(uint16_t) * p->cfg.d;
  const size_t T = static_cast<size_t>(p->last_tokens);
  return cudaMemcpy2DAsync(mem, row * tokens, a.mem, row * T, row * tokens, p->n_active,
                           cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DV_OK
             : DV_ERR_CUDA;
}

}  // extern "C"
