// End-to-end builds from host memory: dv_host_pipeline_create / dv_build_visual_memory_host /
// dv_host_pipeline_wait / dv_host_pipeline_join / dv_host_pipeline_free (include/dv.h).
//
// A caller whose visual embeddings E sit in host memory, and who wants the K/V entries of the
// visual memory (Sec. 3.2 Eq. 7) back in host memory, submits builds to a pipeline. Each build
// moves through three streams of the pipeline:
//   copy-in   E and the positions, host -> the device staging set s
//   build     dv_build_visual_memory of set s's E into set s's staging cache
//   copy-out  the built layers' K and V, set s's staging cache -> the caller's host buffers
// with `depth` staging sets taken round-robin, so the copy-out of build i runs while build
// i + 1 computes and the copy-in of build i + 2 lands. Events order the reuse of a set:
//   copy-in of set s waits for the build that last read set s's E        (built[s])
//   the build of set s waits for its copy-in (in[s]) and for the copy-out that last read set
//   s's cache (out[s])
//   copy-out of set s waits for its build                                (built[s])
// Every copy is one cudaMemcpyAsync of a contiguous range: E, the positions, and one range of K
// and one of V per run of consecutive built layers. The staging cache is dense
// [n_layers][batch][n_vis][n_kv_heads][head_dim], as are the caller's host K and V.
#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "../../include/dv.h"
#include "dv_internal.h"

namespace {

constexpr int kMaxDepth = 4;

struct StagingSet {
  void* x0 = nullptr;   // bf16 [batch][n_vis][d]
  int* pos = nullptr;   // int32 [batch][P][n_vis]
  void* k = nullptr;    // bf16 [n_layers][batch][n_vis][n_kv_heads][head_dim]
  void* v = nullptr;
  cudaEvent_t in = nullptr, built = nullptr, out = nullptr;
  long long ticket = -1;  // last build that used this set
};

}  // namespace

struct dv_host_pipeline {
  dv_plan* plan = nullptr;
  int device = 0;
  int batch = 0, n_vis = 0, n_pos = 1, depth = 0;
  size_t x0_bytes = 0, pos_bytes = 0, layer_bytes = 0;
  long long s_layer = 0, s_batch = 0, s_seq = 0, s_head = 0;  // staging cache strides (elements)
  std::vector<int> run_first, run_count;                      // runs of consecutive built layers
  cudaStream_t s_in = nullptr, s_build = nullptr, s_out = nullptr;
  cudaEvent_t fork = nullptr;
  StagingSet set[kMaxDepth];
  long long submitted = 0;
  std::mutex mu;  // submissions from several host threads are serialised
};

namespace {

void release(dv_host_pipeline* p) {
  if (p->s_in) cudaStreamSynchronize(p->s_in);
  if (p->s_build) cudaStreamSynchronize(p->s_build);
  if (p->s_out) cudaStreamSynchronize(p->s_out);
  for (StagingSet& s : p->set) {
    void* bufs[] = {s.x0, s.pos, s.k, s.v};
    for (void* b : bufs)
      if (b) cudaFree(b);
    cudaEvent_t evs[] = {s.in, s.built, s.out};
    for (cudaEvent_t e : evs)
      if (e) cudaEventDestroy(e);
  }
  if (p->fork) cudaEventDestroy(p->fork);
  cudaStream_t sts[] = {p->s_in, p->s_build, p->s_out};
  for (cudaStream_t s : sts)
    if (s) cudaStreamDestroy(s);
}

bool current_device_is(int dev) {
  int cur = -1;
  return cudaGetDevice(&cur) == cudaSuccess && cur == dev;
}

}  // namespace

extern "C" {

int dv_host_pipeline_create(dv_plan* plan, int batch, int n_vis, int depth,
                            dv_host_pipeline** out) {
  if (!out) return DV_ERR_INVALID_ARG;
  *out = nullptr;
  const dv_config* c = dv::plan_config(plan);
  if (!c || batch < 1 || n_vis < 1 || depth < 1 || depth > kMaxDepth) return DV_ERR_INVALID_ARG;
  if (batch > c->max_batch || n_vis > c->max_n_vis ||
      static_cast<long long>(batch) * n_vis > static_cast<long long>(c->max_batch) * c->max_n_vis)
    return DV_ERR_UNSUPPORTED_SHAPE;
  dv::PlanView v;
  if (!dv::plan_view(plan, &v)) return DV_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DV_ERR_CUDA;

  dv_host_pipeline* p = new (std::nothrow) dv_host_pipeline();
  if (!p) return DV_ERR_OOM;
  p->plan = plan;
  p->device = dev;
  p->batch = batch;
  p->n_vis = n_vis;
  p->depth = depth;
  p->n_pos = c->rope == DV_ROPE_1D ? 1 : 3;
  const long long T = static_cast<long long>(batch) * n_vis;
  const long long kv = static_cast<long long>(c->n_kv_heads) * c->head_dim;
  p->x0_bytes = static_cast<size_t>(T) * c->d * 2;
  p->pos_bytes = static_cast<size_t>(T) * p->n_pos * 4;
  p->layer_bytes = static_cast<size_t>(T * kv) * 2;
  p->s_head = c->head_dim;
  p->s_seq = kv;
  p->s_batch = n_vis * kv;
  p->s_layer = T * kv;
  // runs of consecutive cache layers the plan builds (layers in DV_LAYER_DROP are not copied)
  for (int i = 0; i < v.n_layers; ++i) {
    const int l = v.active[i];
    if (!p->run_first.empty() && p->run_first.back() + p->run_count.back() == l) {
      ++p->run_count.back();
    } else {
      p->run_first.push_back(l);
      p->run_count.push_back(1);
    }
  }

  bool ok = cudaStreamCreateWithFlags(&p->s_in, cudaStreamNonBlocking) == cudaSuccess &&
            cudaStreamCreateWithFlags(&p->s_build, cudaStreamNonBlocking) == cudaSuccess &&
            cudaStreamCreateWithFlags(&p->s_out, cudaStreamNonBlocking) == cudaSuccess &&
            cudaEventCreateWithFlags(&p->fork, cudaEventDisableTiming) == cudaSuccess;
  int rc = ok ? DV_OK : DV_ERR_CUDA;
  const size_t cache_bytes = p->layer_bytes * static_cast<size_t>(c->n_layers);
  for (int i = 0; i < depth && rc == DV_OK; ++i) {
    StagingSet& s = p->set[i];
    if (cudaMalloc(&s.x0, p->x0_bytes) != cudaSuccess ||
        cudaMalloc(reinterpret_cast<void**>(&s.pos), p->pos_bytes) != cudaSuccess ||
        cudaMalloc(&s.k, cache_bytes) != cudaSuccess || cudaMalloc(&s.v, cache_bytes) != cudaSuccess) {
      cudaGetLastError();
      rc = DV_ERR_OOM;
      break;
    }
    if (cudaEventCreateWithFlags(&s.in, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&s.built, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&s.out, cudaEventDisableTiming) != cudaSuccess)
      rc = DV_ERR_CUDA;
  }
  if (rc != DV_OK) {
    cudaGetLastError();
    release(p);
    delete p;
    return rc;
  }
  *out = p;
  return DV_OK;
}

int dv_build_visual_memory_host(dv_host_pipeline* p, const void* x0_host, const int* pos_host,
                                void* k_host, void* v_host, void* stream, long long* ticket) {
  if (!p || !x0_host || !pos_host || !k_host || !v_host) return DV_ERR_INVALID_ARG;
  if (!current_device_is(p->device)) return DV_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(pos_host) & 3u) || (reinterpret_cast<uintptr_t>(x0_host) & 1u) ||
      (reinterpret_cast<uintptr_t>(k_host) & 1u) || (reinterpret_cast<uintptr_t>(v_host) & 1u))
    return DV_ERR_ALIGNMENT;
  std::lock_guard<std::mutex> lock(p->mu);
  const long long id = p->submitted;
  StagingSet& s = p->set[id % p->depth];
  cudaStream_t user = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaEventRecord(p->fork, user);
  // copy-in: after the caller's earlier work on `stream`, and once the build that last read
  // this set's E has run
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_in, p->fork, 0);
  if (e == cudaSuccess && s.ticket >= 0) e = cudaStreamWaitEvent(p->s_in, s.built, 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(s.x0, x0_host, p->x0_bytes, cudaMemcpyHostToDevice, p->s_in);
  if (e == cudaSuccess) e = cudaMemcpyAsync(s.pos, pos_host, p->pos_bytes, cudaMemcpyHostToDevice, p->s_in);
  if (e == cudaSuccess) e = cudaEventRecord(s.in, p->s_in);
  // build: after its copy-in, and once the copy-out that last read this set's cache is done
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_build, s.in, 0);
  if (e == cudaSuccess && s.ticket >= 0) e = cudaStreamWaitEvent(p->s_build, s.out, 0);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return DV_ERR_CUDA;
  }
  dv_kv_cache cache;
  cache.k = s.k;
  cache.v = s.v;
  cache.s_layer = p->s_layer;
  cache.s_batch = p->s_batch;
  cache.s_seq = p->s_seq;
  cache.s_head = p->s_head;
  const int rc = dv_build_visual_memory(p->plan, s.x0, p->batch, p->n_vis, s.pos, nullptr, 0, &cache,
                                        p->s_build);
  if (rc != DV_OK) return rc;
  e = cudaEventRecord(s.built, p->s_build);
  // copy-out: the built layers' K and V, one range per run of consecutive layers
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_out, s.built, 0);
  for (size_t r = 0; r < p->run_first.size() && e == cudaSuccess; ++r) {
    const size_t off = p->layer_bytes * static_cast<size_t>(p->run_first[r]);
    const size_t bytes = p->layer_bytes * static_cast<size_t>(p->run_count[r]);
    e = cudaMemcpyAsync(static_cast<char*>(k_host) + off, static_cast<char*>(s.k) + off, bytes,
                        cudaMemcpyDeviceToHost, p->s_out);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(static_cast<char*>(v_host) + off, static_cast<char*>(s.v) + off, bytes,
                          cudaMemcpyDeviceToHost, p->s_out);
  }
  if (e == cudaSuccess) e = cudaEventRecord(s.out, p->s_out);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return DV_ERR_CUDA;
  }
  s.ticket = id;
  p->submitted = id + 1;
  if (ticket) *ticket = id;
  return DV_OK;
}

int dv_host_pipeline_wait(dv_host_pipeline* p, long long ticket) {
  if (!p || ticket < 0) return DV_ERR_INVALID_ARG;
  cudaEvent_t ev = nullptr;
  {
    std::lock_guard<std::mutex> lock(p->mu);
    if (ticket >= p->submitted) return DV_ERR_INVALID_ARG;
    // The set's event now marks its latest copy-out, which the copy-out stream orders after
    // this ticket's: waiting for it is waiting at least as long as needed.
    ev = p->set[ticket % p->depth].out;
  }
  return cudaEventSynchronize(ev) == cudaSuccess ? DV_OK : DV_ERR_CUDA;
}

int dv_host_pipeline_join(dv_host_pipeline* p, void* stream) {
  if (!p) return DV_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lock(p->mu);
  if (p->submitted == 0) return DV_OK;
  const StagingSet& last = p->set[(p->submitted - 1) % p->depth];
  return cudaStreamWaitEvent(static_cast<cudaStream_t>(stream), last.out, 0) == cudaSuccess
             ? DV_OK
             : DV_ERR_CUDA;
}

void dv_host_pipeline_free(dv_host_pipeline* p) {
  if (!p) return;
  release(p);
  delete p;
}

}  // extern "C"
