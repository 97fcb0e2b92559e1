// Internal interface between the C-ABI / plan code (dv_api.cu) and the tcgen05 kernels
// (dv_gemm.cu, dv_kv2sm.cu, dv_pair_tm.cu, dv_recurrent.cu). Not part of the public ABI.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

struct dv_plan;
struct dv_kv_cache;
struct dv_config;

namespace dv {

constexpr int kBlockM = 128;         // UMMA M: one TMEM lane per token row
constexpr int kBlockK = 64;          // bf16 elements per 128-byte swizzled row of a K slab
constexpr int kMaxHalfHead = 64;     // head_dim <= 128
constexpr int kMaxLayers = 256;

enum Epilogue : int {
  EPI_SILU = 0,  // stacked down-projection: H = bf16(SiLU(acc))
  EPI_NORM = 1,  // RMS statistic: rstd = (||x0||^2 + h . acc) / d + eps) ^ -1/2
  EPI_KV = 2,    // K/V: rstd * acc + bias, RoPE on K, bf16 cache store
  EPI_RESID = 3, // recurrent step: M_l = M_{l-1} + acc (fp32 state), bf16 M_l, sums of squares
};

// Operand schedule shared by all GEMMs. The A operand of a tile is the 128-row token block of
// [A0 | H_l]: k0_slabs 64-wide slabs of A0 starting at row layer * a0_rows_per_layer (x0 for
// every layer, or the stacked per-layer M_l of the recurrent adapter), then k1_slabs slabs of
// H starting at column layer * a1_cols_per_layer (tensor map A1). B is one stacked weight
// matrix whose rows for layer l start at l * n_per_layer; its columns follow the same slab
// order as A. "layer" counts from layer0 (1-SM kernel only; 0 elsewhere).
struct GemmShape {
  int M;                  // tokens in this build
  int n_layers;           // groups (layers)
  int n_per_layer;        // output columns per layer (multiple of BLOCK_N)
  int k0_slabs;           // d / 64
  int k1_slabs;           // r_pad / 64, or 0
  int a1_cols_per_layer;  // r_pad
  int group_m;            // tokens-as-M kernels: token blocks per L2 super-block (0: all)
  int group_w;            // tokens-as-M kernels: weight tiles per L2 super-block (0: 1)
  int layer0;             // first planned layer of the launch
  int a0_rows_per_layer;  // 0: one A0 for every layer; else A0 rows of layer l start at l * it
};

// The 2-SM kernels move two K slabs per pipeline step: one 3-D TMA box per operand and step
// (a TMA instruction has a fixed cost that 16 KB boxes do not amortise). A step stays inside
// one segment of the K schedule (A0, then A1); the last step of a segment with an odd slab
// count uses its first slab only (the box's second slab is zero fill or unused data).
constexpr int kSlabsPerStep = 2;

struct KStep {
  int seg;   // 0: A0 slabs (x0 or M_l), 1: A1 slabs (h_l)
  int slab;  // first slab of the step within its segment
  int n;     // slabs of the step that the MMA uses: 1 or 2
};

__host__ __device__ inline int k_steps(int k0_slabs, int k1_slabs) {
  return (k0_slabs + 1) / 2 + (k1_slabs + 1) / 2;
}

__host__ __device__ inline KStep k_step(int j, int k0_slabs, int k1_slabs) {
  const int s0 = (k0_slabs + 1) / 2;
  KStep r;
  if (j < s0) {
    r.seg = 0;
    r.slab = 2 * j;
    r.n = k0_slabs - 2 * j < 2 ? k0_slabs - 2 * j : 2;
  } else {
    r.seg = 1;
    r.slab = 2 * (j - s0);
    r.n = k1_slabs - r.slab < 2 ? k1_slabs - r.slab : 2;
  }
  return r;
}

// Columns [0, n_h) of the product are down-projections: H = bf16(SiLU(acc)). Columns from n_h
// on (x0 (2 U_l)^T when the statistic of M_l is formed outside a GEMM) go to C as fp32.
struct EpiSilu {
  uint16_t* H;   // bf16 [M][ldh]
  int ldh;
  int n_h;       // columns that are down-projections
  float* C;      // fp32 [M][ldc] or null
  int ldc;
};

// Launch attribute of the build's kernels: programmatic stream serialization (see pdl_wait in
// dv_ptx.cuh for what a kernel launched with it may touch before its wait).
inline cudaLaunchAttribute pdl_attribute() {
  cudaLaunchAttribute a;
  a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  a.val.programmaticStreamSerializationAllowed = 1;
  return a;
}

// Layers of the statistic GEMM per 256-column tile: its B operand (Bn) groups `lpt` layers, a
// layer's rows `rn` apart: r_pad <= 64: 4 layers of 64 rows; <= 128: 2 of 128; else 1 of 256
// (r_pad = 192 leaves 64 zero rows).
__host__ __device__ inline void norm_group(int r_pad, int* lpt, int* rn) {
  *lpt = r_pad <= 64 ? 4 : (r_pad <= 128 ? 2 : 1);
  *rn = 256 / *lpt;
}

struct EpiNorm {
  const uint16_t* H;  // bf16 [M_ld][ldh], h_l at columns l * r_pad
  int ldh;
  int r_pad;
  int lpt, rn;        // layers per 256-column tile and their row stride (norm_group)
  int n_layers;       // planned layers (the last group may hold fewer)
  const float* xx;    // [M] row sums of squares of x0
  float* rstd;        // [L][ld_rstd]
  int ld_rstd;
  float inv_d;
  float eps;
};

struct EpiKV {
  const float* rstd;  // [L][ld_rstd]
  int ld_rstd;
  const float* bk;    // fp32 [L][kv] or null
  const float* bv;
  int kv;
  const int* pos;     // int32 [B][P][n_vis]
  const int* slot;    // int32 [B][n_vis] or null
  int slot0;
  int n_vis;
  int n_pos;          // 1 or 3
  const float* kg;    // per-head K-norm gain fp32 [L][head_dim], or null (no K norm)
  float k_eps;
  uint8_t axis[kMaxHalfHead];  // position axis (0 t, 1 h, 2 w) of each frequency pair
  uint16_t* kc;
  uint16_t* vc;
  long long s_layer, s_batch, s_seq, s_head;
  float two_pi_hi, two_pi_lo, inv_two_pi;
  float inv_freq_hi[kMaxHalfHead];  // theta^(-2j/D_h) split into two floats
  float inv_freq_lo[kMaxHalfHead];
};

// Recurrent step of one layer (Sec. 3.1 Eq. 6): for token row t and the tile's columns,
// M = prev + acc with prev = x0 (first planned layer) or the fp32 state; the state is
// overwritten with M, bf16(M) goes to the layer's slice of the stacked memories, and the
// tile's sum of M^2 over its columns to part[n][t].
struct EpiResid {
  const uint16_t* x0;  // bf16 [M][d]
  float* state;        // fp32 [M][d]
  uint16_t* mem;       // bf16 [M][d]: this layer's M_l
  float* part;         // fp32 [d / BLOCK_N][M]: this layer's partial sums of squares
  int d;
  int first;           // 1: prev = x0
  uint16_t* mem_lo;    // split chain: bf16(M - bf16(M)) [M][d], or null
};

struct GemmParams {
  GemmShape s;
  // The plan holds the layers that are not dropped, in order; logical layer i of a launch (its
  // weights, H columns, rstd rows and biases) writes cache layer layer_map[i].
  int16_t layer_map[kMaxLayers];
  EpiSilu silu;
  EpiNorm norm;
  EpiKV kv;
  EpiResid resid;
  int* status;              // device status word
  unsigned long long timeout_ns;
};

// Launches one persistent warp-specialised 1-SM tcgen05 GEMM (EPI_SILU, EPI_NORM or
// EPI_RESID, block_n 64/128/256). Returns a cudaError_t value.
cudaError_t launch_gemm(int epi, int block_n, int head_dim, const CUtensorMap& a0,
                        const CUtensorMap& a1, const CUtensorMap& b, const GemmParams& p,
                        int num_sms, cudaStream_t stream);

// Shared-memory bytes one CTA of that GEMM asks for (for validation and reporting).
int gemm_smem_bytes(int block_n);

// K/V projection + RoPE + cache store on CTA pairs (2-SM UMMA). All maps are slab maps (two K
// slabs per box): w: Wkv with 128-row boxes; x / h: x0 and H with boxes of nt/2 token rows. nt
// from kv_pair_tile_n.
cudaError_t launch_kv_pair(int head_dim, int nt, const CUtensorMap& w, const CUtensorMap& x,
                           const CUtensorMap& h, const GemmParams& p, int num_sms,
                           cudaStream_t stream);

// 2-SM GEMM with 256-token M blocks (tokens as M): EPI_SILU / EPI_NORM with block_n 64/128/256
// (b: weights with boxes of block_n / 2 rows), EPI_KV with block_n 256 (b: Wkv, 128-row boxes).
// a0 / a1: x0 and H with 128-row boxes. All maps are slab maps (two K slabs per box).
cudaError_t launch_pair_tm(int epi, int block_n, int head_dim, const CUtensorMap& a0,
                           const CUtensorMap& a1, const CUtensorMap& b, const GemmParams& p,
                           int num_sms, cudaStream_t stream);

// Recurrent down-projection of one layer: H[:, h_col0 + n] = bf16(SiLU(A B^T)) with A the
// layer's input state (bf16 [M][k_slabs * 64], rows from a_row0) and B the layer's r_pad rows
// of the stacked down-projection (from b_row0). The K dimension is split over the CTAs of a
// thread-block cluster (size `splits`, 1/2/4/8) and the fp32 partials are summed in a fixed
// order through distributed shared memory.
struct DownParams {
  int M;
  int a_row0;
  int b_row0;
  int k_slabs;
  uint16_t* H;
  int ldh;
  int h_col0;
  int a_lo;      // split chain: 1 = the second A map holds the low bf16 part of A (rows a_row0..)
  uint16_t* Hlo; // split chain: bf16(h - bf16(h)) at the same place as H, or null
  int* status;
  unsigned long long timeout_ns;
};
cudaError_t launch_down_split(int r_pad, int splits, const CUtensorMap& a, const CUtensorMap& a_lo,
                              const CUtensorMap& b, const DownParams& p, cudaStream_t stream);
// K splits (1, 2, 4 or 8) for m_tiles token blocks of 128 rows and k_slabs slabs.
int down_splits(long long m_tiles, int k_slabs, int num_sms);

// The recurrent chain on chip (dv_chain.cu): one cluster of S CTAs per 128-token block runs all
// layers with the fp32 state in TMEM. chain_shape gives the slabs per CTA (spc) and S for a
// hidden size and r_pad, or false when the chain does not fit (then the per-layer launches
// run). launch_chain returns cudaErrorNotSupported when no cluster of that size can be resident.
// split: the split chain (hi + lo bf16 operands), available on chip at r_pad 64 only.
// x: x0 (128-row boxes); dmap: stacked D (r_pad-row boxes); umap: U as [L d][r_pad] (64 spc-row
// boxes); mmap: the stacked M_l as a 3-D (d, tokens, L) map with (64, 128, 1) boxes.
bool chain_shape(int d, int r_pad, int* spc_out, int* s_out);
// Clusters of the on-chip chain that can be resident at once on the current device (0: the
// chain does not fit or does not apply).
int chain_resident_clusters(int d, int r_pad, bool split);
cudaError_t launch_chain(int r_pad, int spc, int S, long long tokens, int n_layers, int d,
                         const CUtensorMap& x, const CUtensorMap& dmap, const CUtensorMap& umap,
                         const CUtensorMap& mmap, float* part, long long part_ld, uint16_t* H,
                         int* status, unsigned long long timeout_ns, cudaStream_t stream,
                         bool split);

// The recurrent adapter by the refactored chain (dv_fold.cu). With C = E [D_1 .. D_L]^T (fp32
// [tokens][ldc], C_l at columns l r_pad) and the plan's Pf ([L r_pad][L r_pad], block (l, j) =
// Q_lj = D_l U_j for j < l):
//   launch_hchain: h_l = SiLU(C_l + sum_{j<l} h_j Q_lj^T) into H ([tokens][ldh], h_l at columns
//     l r_pad), one CTA per 128-token block. Maps: h: slab map over H with 128-row boxes; pf:
//     slab map over Pf with r_pad-row boxes; hst: H as a 2-D map with 32-row boxes (the
//     stores of h_l).
//   launch_accum: M_l = E + sum_{j<=l} h_j U_j^T, bf16 into the stacked memories ([L][tokens][d],
//     stored through mem: a 3-D map over them with 32 x 32 boxes and 64-byte swizzle) and each
//     row's partial sums of M_l^2 into part (fold_sum_parts(d) partials per layer, at most
//     d / 64). h: H with 128-row boxes; u: U as [L d][r_pad] with cw-row boxes; x0: E, bf16
//     [tokens][d].
// fold_slice_cols: the slice width cw (256 or 128 dividing d), or 0.
// fold_sum_parts: the partial sums of squares per token and layer that launch_accum writes.
// hchain_box_slabs: K slabs per TMA box of launch_hchain's maps (h and pf are slab maps,
// encode_slabs, with boxes of that many slabs).
// split (split_chain): h_l also as its low bf16 part Hlo (hlo, hlost: its maps, as h's and hst's), and Pf_lo
// (pflo: its map, as pf's), the low part of the products: each product is taken in three parts,
// h_hi Q_hi + h_lo Q_hi + h_hi Q_lo, and the running sum adds h_hi U + h_lo U. Without the split
// hlo, hlost and pflo are not used.
int fold_slice_cols(int d);
int fold_sum_parts(int d);
int hchain_box_slabs(int r_pad, bool split);
cudaError_t launch_hchain(int r_pad, bool split, long long tokens, int n_layers, const float* C,
                          int ldc, const CUtensorMap& h, const CUtensorMap& hlo,
                          const CUtensorMap& pf, const CUtensorMap& pflo, const CUtensorMap& hst,
                          const CUtensorMap& hlost, uint16_t* H, uint16_t* Hlo, int ldh, int* status,
                          unsigned long long timeout_ns, cudaStream_t stream);
cudaError_t launch_accum(int r_pad, int cw, long long tokens, int n_layers, int d,
                         const void* x0, const CUtensorMap& h, const CUtensorMap& hlo, bool split,
                         const CUtensorMap& u, const CUtensorMap& mem, float* part, long long part_ld,
                         int* status, unsigned long long timeout_ns, cudaStream_t stream);

// Token tile (64, 128, 192 or 256) of the pair kernel for a build of `tokens` tokens.
int kv_pair_tile_n(long long tokens);
int kv_pair_smem_bytes(int nt);

// Position axis (0 t, 1 h, 2 w) of rotary frequency pair j for rope mode `rope` (DV_ROPE_*)
// and M-RoPE sections `sec` (t, h, w).
int rope_axis(int rope, const int* sec, int j);

// Read-only view of a plan's repacked weights and shape, for build variants outside dv_api.cu.
struct PlanView {
  int d, n_layers, head_dim, rope, mrope_section[3];  // n_layers: layers the plan holds
  int adapter;                                         // DV_ADAPTER_*
  float rms_eps;
  const float* kg;                 // per-head K-norm gain [L][head_dim], or null
  float k_eps;
  int num_sms, r_pad, kv, k_total;
  const float* bk;
  const float* bv;
  int* status;
  const CUtensorMap* tm_Dst;       // three maps: boxes of 64, 128, 256 rows; embedding adapter:
                                   // rows [0, L r_pad) D, rows [L r_pad, 2 L r_pad) 2 U^T
  const float* Gf;                 // embedding adapter: G_l = U_l^T U_l, fp32 [L][r_pad][r_pad]
  const CUtensorMap* tm_Dst_half;  // three slab maps: boxes of 32, 64, 128 rows (pair halves)
  const CUtensorMap* tm_Bn;        // boxes of 256 rows (one layer group, norm_group)
  const CUtensorMap* tm_Bn_half;   // slab map, boxes of 128 rows
  int bn_lpt, bn_rn, bn_groups;    // statistic GEMM: layers per group, their row stride, groups
  const CUtensorMap* tm_Wkv;       // slab map, boxes of 128 rows
  const CUtensorMap* tm_Dst_rp;    // recurrent: boxes of r_pad rows (one layer's D)
  const uint16_t* Dst;             // stacked D (and 2 U^T): rows of dst_ld elements
  int dst_ld;
  const CUtensorMap* tm_Uup;       // recurrent: [L*d][r_pad], boxes of resid_bn rows
  const uint16_t* Uup;             // recurrent: U_l as [L*d][r_pad] ([U_l | U_l] when split)
  const CUtensorMap* tm_Pf;        // recurrent, refactored chain: Pf with r_pad-row boxes, or null
  const CUtensorMap* tm_Pf_lo;     // the same for Pf_lo (split chain), or null
  int chain_clusters;              // recurrent: resident clusters of the on-chip chain (0: none)
  int split_chain;                 // recurrent: hi + lo bf16 operands in the chain's GEMMs
  int uup_ld;                      // row pitch of Uup: r_pad, or 2 r_pad with the split chain
  int resid_bn;                    // recurrent: column tile of the up-projection step
  const double* inv_freq;     // head_dim / 2 values
  const uint16_t* Wkv;        // repacked K/V weights [L*2kv][k_total]
  const int16_t* active;      // cache layer of each planned layer
};
bool plan_view(const dv_plan* p, PlanView* out);

// The configuration a plan was made with (null for a null plan).
const ::dv_config* plan_config(const dv_plan* p);

// Device address of the static build scratch of dv_build_visual_memory_noalloc on the current
// device and context (dv_noalloc.cu). Looking it up loads that file's module, which reserves the
// array; the plan does this once, so that the entry point itself allocates nothing.
int noalloc_scratch(void** out);
// The scratch address the plan looked up when it was made (null if that failed).
void* plan_scratch(const dv_plan* p);

// Everything one build needs besides the plan: caller tensors and where the intermediates go.
struct BuildArgs {
  const void* x0;
  int batch, n_vis;
  const int* pos;
  const int* slot;
  int slot0;
  const void* kc;
  const void* vc;
  long long s_layer, s_batch, s_seq, s_head;
  uint16_t* H;          // [tokens][hld] bf16, h_l at columns l * r_pad
  long long hld;        // row pitch of H: L * r_pad (+ 64 for the embedding adapter)
  uint16_t* x0p;        // embedding adapter: copy of E with row pitch x0p_ld (k_row_sumsq)
  long long x0p_ld;     // d + 64
  float* rstd;          // [L][tokens]
  float* xx;            // [tokens]
  float* c;             // fp32 [tokens][L * r_pad]: embedding adapter at small token counts,
                        // x0 (2 U_l)^T; recurrent adapter, refactored chain: E D_l^T
  float* state;         // recurrent: fp32 [tokens][d]
  uint16_t* mem;        // recurrent: bf16 [L][tokens][d]
  float* part;          // recurrent: fp32 [L][d / 64][tokens]
  uint16_t* Hlo;        // split chain: low bf16 parts of h, [tokens][L * r_pad]
  uint16_t* mem_lo;     // split chain: low bf16 part of the last M_l, [tokens][d]
  cudaEvent_t* marks;   // 5 events around the 4 stages, or null
};

// Bytes of the intermediates of a build of `tokens` tokens (each part 256-byte aligned). With
// a non-null base, also points the intermediates of `a` into [base, base + bytes).
size_t carve_workspace(const PlanView& v, long long tokens, void* base, BuildArgs* a);

// Argument checks shared by the build entry points (dv_status value; DV_OK for an empty build).
int check_build_args(const void* x0, int batch, int n_vis, const int* pos, const int* slot,
                     int slot0, const ::dv_kv_cache* out);

// Enqueue the four stages of one build on `stream` (arguments already validated).
// Returns a cudaError_t value.
cudaError_t enqueue_build(const PlanView& v, const BuildArgs& a, cudaStream_t stream);

// bf16 [rows][cols] (row stride ld elements) tensor map with 128-byte-swizzled boxes of
// 64 columns x box_rows rows; out-of-range elements read as zero.
bool encode_bf16_2d(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint64_t ld,
                    uint32_t box_rows);

}  // namespace dv
