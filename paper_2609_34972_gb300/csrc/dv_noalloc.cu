// dv_build_visual_memory_noalloc: the visual-memory build for callers that must not allocate
// device memory while they build.
//
// Some callers cannot call cudaMalloc at the point where they build visual memory: serving
// engines that reserve all device memory up front and hand out nothing afterwards, callers
// whose memory budget is fixed per model so that a per-plan workspace sized for the largest
// batch is not acceptable, and code that must not risk the implicit device synchronisation
// of cudaMalloc / cudaFree in its latency-critical path. For them this file keeps the build's
// intermediate buffers (SiLU(E D_l) for every layer, the RMS statistics and the row sums of
// squares) in one file-scope static device array of kScratchBytes instead of the plan's
// workspace. The plan's repacked weights are still used; nothing here allocates.
//
// Behaviour a caller must know:
//   - The array exists once per device that loads this library and lives until the process
//     exits, whether or not this entry point is ever called.
//   - Its device address is looked up (cudaGetSymbolAddress) by the first call on each device,
//     with that device current; that set-up call should come before any stream capture.
//   - Every call on a device uses the same array. Calls whose kernels overlap on the GPU (on
//     different streams, or from different threads without ordering) race on it and produce
//     wrong output; order them on one stream.
//   - The array keeps whatever the previous call left. No byte of it needs to start at zero:
//     each call writes every element it later reads, and the tensor maps over it stop at this
//     call's token count, so stale rows are never loaded.
//   - A build that needs more than kScratchBytes of intermediates is rejected with
//     DV_ERR_UNSUPPORTED_SHAPE before anything is launched.
#include <cstring>
#include <mutex>

#include "../../include/dv.h"
#include "dv_internal.h"

namespace {

constexpr size_t kScratchBytes = 32ull << 20;  // 32 MiB per device
constexpr int kMaxDevices = 64;
constexpr unsigned long long kTimeoutNs = 2000000000ull;

static __device__ __align__(256) unsigned char g_build_scratch[kScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_build_scratch on the current device (looked up once per device).
int scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DV_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DV_ERR_UNSUPPORTED_DEVICE;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_build_scratch) != cudaSuccess || !ptr) {
      cudaGetLastError();
      return DV_ERR_CUDA;
    }
    g_scratch_addr[dev] = ptr;
  }
  *out = g_scratch_addr[dev];
  return DV_OK;
}

size_t round256(size_t n) { return (n + 255) / 256 * 256; }

// xx[t] = sum_j x0[t][j]^2 (fp32), one warp per token row.
__global__ void k_row_sumsq_scratch(const uint16_t* __restrict__ x0, int T, int d,
                                    float* __restrict__ xx) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T) return;
  const uint4* row = reinterpret_cast<const uint4*>(x0 + static_cast<long long>(warp) * d);
  float s = 0.0f;
  for (int c = lane; c < d / 8; c += 32) {
    const uint4 v = row[c];
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

}  // namespace

extern "C" int dv_build_visual_memory_noalloc(dv_plan* plan, const void* x0, int batch,
                                              int n_vis, const int* pos, const int* slot,
                                              int slot0, const dv_kv_cache* out, void* stream) {
  dv::PlanView v;
  if (!dv::plan_view(plan, &v)) return DV_ERR_INVALID_ARG;
  if (batch < 0 || n_vis < 0 || slot0 < 0) return DV_ERR_INVALID_ARG;
  const long long T = static_cast<long long>(batch) * n_vis;
  if (T == 0) return DV_OK;
  if (!x0 || !pos || !out || !out->k || !out->v) return DV_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(x0) & 15u) || (reinterpret_cast<uintptr_t>(out->k) & 15u) ||
      (reinterpret_cast<uintptr_t>(out->v) & 15u))
    return DV_ERR_ALIGNMENT;
  const long long s[4] = {out->s_layer, out->s_batch, out->s_seq, out->s_head};
  for (long long x : s) {
    if (x < 0) return DV_ERR_INVALID_ARG;
    if (x % 8 != 0) return DV_ERR_ALIGNMENT;
  }
  if ((reinterpret_cast<uintptr_t>(pos) & 3u) || (slot && (reinterpret_cast<uintptr_t>(slot) & 3u)))
    return DV_ERR_ALIGNMENT;

  // Scratch layout: H [T][L*r_pad] bf16 | rstd [L][T] fp32 | xx [T] fp32, 256-byte aligned.
  const int L = v.n_layers, d = v.d, HD = v.head_dim;
  const long long n1 = static_cast<long long>(L) * v.r_pad;
  const size_t h_bytes = round256(static_cast<size_t>(T) * n1 * 2);
  const size_t r_bytes = round256(static_cast<size_t>(T) * L * 4);
  const size_t x_bytes = round256(static_cast<size_t>(T) * 4);
  if (h_bytes + r_bytes + x_bytes > kScratchBytes || T > (1LL << 24)) return DV_ERR_UNSUPPORTED_SHAPE;

  void* base = nullptr;
  int rc = scratch_address(&base);
  if (rc != DV_OK) return rc;
  uint16_t* H = static_cast<uint16_t*>(base);
  float* rstd = reinterpret_cast<float*>(static_cast<unsigned char*>(base) + h_bytes);
  float* xx = reinterpret_cast<float*>(static_cast<unsigned char*>(base) + h_bytes + r_bytes);

  const int nt = dv::kv_pair_tile_n(T);
  CUtensorMap tm_x0, tm_x0_half, tm_H, tm_H_half;
  if (!dv::encode_bf16_2d(&tm_x0, x0, d, T, d, dv::kBlockM) ||
      !dv::encode_bf16_2d(&tm_x0_half, x0, d, T, d, nt / 2) ||
      !dv::encode_bf16_2d(&tm_H, H, n1, T, n1, dv::kBlockM) ||
      !dv::encode_bf16_2d(&tm_H_half, H, n1, T, n1, nt / 2))
    return DV_ERR_CUDA;

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dv::GemmParams gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.status = v.status;
  gp.timeout_ns = kTimeoutNs;

  k_row_sumsq_scratch<<<static_cast<int>((T + 7) / 8), 256, 0, st>>>(
      static_cast<const uint16_t*>(x0), static_cast<int>(T), d, xx);
  cudaError_t err = cudaGetLastError();

  // H = SiLU(x0 [D_1 ... D_L]) into the scratch array.
  const long long m_tiles = (T + dv::kBlockM - 1) / dv::kBlockM;
  int bn1 = 64;
  for (int cand : {256, 128}) {
    if (n1 % cand == 0 && m_tiles * (n1 / cand) >= v.num_sms) {
      bn1 = cand;
      break;
    }
  }
  gp.s = {static_cast<int>(T), 1, static_cast<int>(n1), d / 64, 0, 0};
  gp.silu = {H, static_cast<int>(n1)};
  const CUtensorMap& tmD = v.tm_Dst[bn1 == 64 ? 0 : (bn1 == 128 ? 1 : 2)];
  if (err == cudaSuccess)
    err = dv::launch_gemm(dv::EPI_SILU, bn1, 0, tm_x0, tm_x0, tmD, gp, v.num_sms, st);

  // rstd_l from ||x0||^2 + h_l . ([x0 | h_l] [2 U_l^T ; G_l]).
  gp.s = {static_cast<int>(T), L, v.r_pad, d / 64, v.r_pad / 64, v.r_pad};
  gp.norm = {H, static_cast<int>(n1), v.r_pad, xx, rstd, static_cast<int>(T), 1.0f / d, v.rms_eps};
  if (err == cudaSuccess)
    err = dv::launch_gemm(dv::EPI_NORM, v.r_pad, 0, tm_x0, tm_H, *v.tm_Bn, gp, v.num_sms, st);

  // K/V with RoPE into the caller's cache.
  gp.s = {static_cast<int>(T), L, 2 * v.kv, d / 64, v.r_pad / 64, v.r_pad};
  dv::EpiKV& e = gp.kv;
  e.rstd = rstd;
  e.ld_rstd = static_cast<int>(T);
  e.bk = v.bk;
  e.bv = v.bv;
  e.kv = v.kv;
  e.pos = pos;
  e.slot = slot;
  e.slot0 = slot0;
  e.n_vis = n_vis;
  e.n_pos = v.rope == DV_ROPE_MROPE ? 3 : 1;
  e.sec0 = v.rope == DV_ROPE_MROPE ? v.mrope_section[0] : HD / 2;
  e.sec01 = v.rope == DV_ROPE_MROPE ? v.mrope_section[0] + v.mrope_section[1] : HD / 2;
  e.kc = static_cast<uint16_t*>(out->k);
  e.vc = static_cast<uint16_t*>(out->v);
  e.s_layer = out->s_layer;
  e.s_batch = out->s_batch;
  e.s_seq = out->s_seq;
  e.s_head = out->s_head;
  const double two_pi = 6.283185307179586476925286766559;
  e.two_pi_hi = static_cast<float>(two_pi);
  e.two_pi_lo = static_cast<float>(two_pi - static_cast<double>(e.two_pi_hi));
  e.inv_two_pi = static_cast<float>(1.0 / two_pi);
  for (int j = 0; j < HD / 2; ++j) {
    e.inv_freq_hi[j] = static_cast<float>(v.inv_freq[j]);
    e.inv_freq_lo[j] = static_cast<float>(v.inv_freq[j] - static_cast<double>(e.inv_freq_hi[j]));
  }
  if (err == cudaSuccess)
    err = dv::launch_kv_pair(HD, nt, *v.tm_Wkv, tm_x0_half, tm_H_half, gp, v.num_sms, st);
  return err == cudaSuccess ? DV_OK : DV_ERR_CUDA;
}
