// dv_build_visual_memory_noalloc: the visual-memory build for callers that must not allocate
// device memory while they build.
//
// Some callers cannot call cudaMalloc at the point where they build visual memory: serving
// engines that reserve all device memory up front and hand out nothing afterwards, callers
// whose memory budget is fixed per model so that a per-plan workspace sized for the largest
// batch is not acceptable, and code that must not risk the implicit device synchronisation
// of cudaMalloc / cudaFree in its latency-critical path. For them this file keeps the build's
// intermediate buffers (SiLU(E D_l) for every layer, the RMS statistics and the row sums of
// squares; for the recurrent adapter also M_l of every layer, partial sums of squares, and the
// fp32 state or, for the rearranged chain, the fp32 E D_l^T) in one file-scope static device
// array of kScratchBytes instead of the plan's
// workspace. The plan's repacked weights are still used; nothing here allocates.
//
// Behaviour a caller must know:
//   - The array exists once per device (and context) that loads this file's module, and lives
//     until the process exits. CUDA loads modules lazily, so the array is reserved when the
//     first plan on a device is made: dv_memory_plan looks up the array's device address
//     (cudaGetSymbolAddress, with the plan's device current), which loads the module, and also
//     loads every kernel a build can launch. The entry point therefore allocates nothing, even
//     on its first call, and needs no set-up step of its own.
//   - Every call on a device uses the same array. Calls whose kernels overlap on the GPU (on
//     different streams, or from different threads without ordering) race on it and produce
//     wrong output; order them on one stream.
//   - The array keeps whatever the previous call left. No byte of it needs to start at zero:
//     each call writes every element it later reads, and the tensor maps over it stop at this
//     call's token count, so stale rows are never loaded.
//   - A build that needs more than kScratchBytes of intermediates is rejected with
//     DV_ERR_UNSUPPORTED_SHAPE before anything is launched.
//   - The address belongs to the CUDA context the plan was made in; cudaDeviceReset ends that
//     context and invalidates plans and the array alike.
#include "../../include/dv.h"
#include "dv_internal.h"

namespace {

constexpr size_t kScratchBytes = 32ull << 20;  // 32 MiB per device

static __device__ __align__(256) unsigned char g_build_scratch[kScratchBytes];

}  // namespace

// In host code g_build_scratch names a host-side stand-in, not device memory: kernels get the
// address that cudaGetSymbolAddress returns for the current device.
int dv::noalloc_scratch(void** out) {
  void* ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_build_scratch) != cudaSuccess || !ptr) {
    cudaGetLastError();
    return DV_ERR_CUDA;
  }
  *out = ptr;
  return DV_OK;
}

extern "C" int dv_build_visual_memory_noalloc(dv_plan* plan, const void* x0, int batch,
                                              int n_vis, const int* pos, const int* slot,
                                              int slot0, const dv_kv_cache* out, void* stream) {
  dv::PlanView v;
  if (!dv::plan_view(plan, &v)) return DV_ERR_INVALID_ARG;
  int rc = dv::check_build_args(x0, batch, n_vis, pos, slot, slot0, out);
  if (rc != DV_OK) return rc;
  const long long T = static_cast<long long>(batch) * n_vis;
  if (T == 0) return DV_OK;

  // Scratch layout: the build's intermediates as carve_workspace lays them out for T tokens.
  const size_t bytes = dv::carve_workspace(v, T, nullptr, nullptr);
  if (bytes > kScratchBytes || T > (1LL << 24)) return DV_ERR_UNSUPPORTED_SHAPE;
  // the recurrent K/V GEMM addresses the stacked M_l with 32-bit TMA row coordinates (the
  // plan applies the same limit to its own workspace)
  if (v.adapter == DV_ADAPTER_RECURRENT &&
      static_cast<long long>(v.n_layers) * T + dv::kBlockM >= (1LL << 31))
    return DV_ERR_UNSUPPORTED_SHAPE;

  // looked up when the plan was made (see above); null if the array could not be reserved then
  void* base = dv::plan_scratch(plan);
  if (!base) return DV_ERR_OOM;

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
  dv::carve_workspace(v, T, base, &a);
  a.marks = nullptr;
  return dv::enqueue_build(v, a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? DV_OK
                                                                                   : DV_ERR_CUDA;
}
