/*
 * dv.h — C ABI of the GB300 (sm_103a) visual-memory build for delta-Vision
 * ("Just MLPs: Efficient Visual State Reconstruction for Multimodal Language Models").
 *
 * The library builds, for every visual token and every layer l, the key/value cache entries
 * that text tokens read:
 *     M_l = E + SiLU(E D_l) U_l                 (Sec. 3.1, Eqs. 4-5: embedding adapter)
 *  or M_0 = E, M_l = M_{l-1} + SiLU(M_{l-1} D_l) U_l
 *                                               (Sec. 3.1, Eq. 6: recurrent adapter)
 *     K_l = RoPE(W_K,l RMSNorm_l(M_l) [+ b_K,l]),  V_l = W_V,l RMSNorm_l(M_l) [+ b_V,l]
 *                                               (Sec. 3.2, Eq. 7; RMSNorm per App. K; RoPE
 *                                                at the original visual positions)
 * (with k_norm, each head of K is RMS-normalised with a learned gain before RoPE), and stores
 * them as bf16 into a caller-owned KV cache. Visual tokens get no query,
 * attention output or feed-forward update (Sec. 3.2), so K/V entries are the only output.
 *
 * Conventions for every entry point:
 *   - Tensor arguments are DEVICE pointers on the current CUDA device, owned by the caller.
 *   - bf16 tensors are IEEE bfloat16 bit patterns, row-major, innermost index last.
 *   - Every call returns a dv_status; no exception or abort crosses the ABI. Arguments are
 *     validated before anything is launched: a call that returns an error launched nothing
 *     (except DV_ERR_CUDA, which reports a failed launch or allocation).
 *   - Builds are stream-ordered and asynchronous: they enqueue kernels on `stream` (a
 *     cudaStream_t passed as void*, NULL = legacy default stream) and never synchronise.
 */
#ifndef DV_H
#define DV_H

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DV_OK = 0,
  DV_ERR_INVALID_ARG = 1,        /* null pointer, negative size, bad enum value */
  DV_ERR_UNSUPPORTED_SHAPE = 2,  /* a shape outside what the kernels are built for */
  DV_ERR_ALIGNMENT = 3,          /* a pointer or stride misses its 16-byte alignment */
  DV_ERR_OOM = 4,                /* device allocation failed */
  DV_ERR_CUDA = 5,               /* a CUDA runtime or driver call failed */
  DV_ERR_DEVICE_TIMEOUT = 6,     /* a device-side wait gave up (see dv_plan_status) */
  DV_ERR_UNSUPPORTED_DEVICE = 7  /* the current device is not an sm_103 GPU */
} dv_status;

enum { DV_ACT_SILU = 0 };                  /* phi of Sec. 3.1 Eq. 4 */
/* Per-layer treatment of the visual memory (App. J, layer-wise adapter skipping). */
enum {
  DV_LAYER_ADAPTER = 0,   /* M_l = E + SiLU(E D_l) U_l: the embedding adapter (Sec. 3.1 Eq. 5) */
  DV_LAYER_IDENTITY = 1,  /* adapter skipped, M_l = E: visual K/V still built from E */
  DV_LAYER_DROP = 2       /* adapter and visual memory skipped: no K/V entries for this layer */
};
/* Rotary embedding of visual keys: 1-D positions, or M-RoPE (t, h, w) with the frequency
 * pairs split into contiguous sections (t first, then h, then w) or interleaved as in
 * Qwen3-VL backbones (pair j follows h when j = 1 mod 3 and j < 3 s_h, w when j = 2 mod 3
 * and j < 3 s_w, t otherwise). */
enum { DV_ROPE_1D = 0, DV_ROPE_MROPE = 1, DV_ROPE_MROPE_INTERLEAVED = 2 };
/* How M_l is formed from the visual embeddings E (Sec. 3.1). */
enum {
  DV_ADAPTER_EMBEDDING = 0,  /* M_l = A_l(E) for every layer (Eq. 5) */
  DV_ADAPTER_RECURRENT = 1   /* M_0 = E, M_l = A_l(M_{l-1}) through the planned layers (Eq. 6) */
};
/* How the recurrent adapter's chain is evaluated (the same function either way, Sec. 3.1 Eq. 6):
 * the chain in the paper's order, z_l = M_{l-1} D_l^T layer after layer (on chip, a cluster of
 * SMs per 128-token block, where such a cluster fits; else per-layer launches), or rearranged,
 * z_l = E D_l^T + sum_{j<l} h_j (D_l U_j)^T and M_l = E + sum_{j<=l} h_j U_j^T, whose only
 * sequential part is r wide. */
enum {
  DV_RECURRENT_AUTO = 0,        /* the on-chip chain for builds whose token blocks fit in one
                                   wave of its clusters, the rearranged chain for larger ones */
  DV_RECURRENT_CHAIN = 1,       /* the chain in the paper's order for every build */
  DV_RECURRENT_REARRANGED = 2   /* the rearranged chain for every build */
};

/* Model shape and build limits. Supported (else DV_ERR_UNSUPPORTED_SHAPE):
 *   d % 64 == 0, 64 <= d <= 16384;  1 <= rank <= 256;  head_dim in {64, 128};
 *   1 <= n_kv_heads, n_kv_heads * head_dim <= 8192 and a multiple of 128;
 *   1 <= n_layers <= 256;
 *   act == DV_ACT_SILU;  rope_theta > 0;  rms_eps >= 0;
 *   DV_ROPE_MROPE / DV_ROPE_MROPE_INTERLEAVED: mrope_section[i] >= 0 and their sum ==
 *   head_dim / 2 (interleaved: the layout must give each axis exactly its section's count);
 *   k_norm in {0, 1}; k_norm_eps >= 0;
 *   adapter in {DV_ADAPTER_EMBEDDING, DV_ADAPTER_RECURRENT};
 *   split_chain in {0, 1}, and 1 only with DV_ADAPTER_RECURRENT;
 *   recurrent_path a DV_RECURRENT_* value, not AUTO only with DV_ADAPTER_RECURRENT,
 *   REARRANGED only with d % 128 == 0;
 *   max_batch * max_n_vis >= 1 and <= 2^24 (the tokens one build may carry). */
typedef struct dv_config {
  int d;                 /* hidden size of the language model */
  int n_layers;          /* L: layers that receive visual K/V */
  int n_kv_heads;        /* H_kv */
  int head_dim;          /* D_h */
  int rank;              /* r: adapter bottleneck (Sec. 3.1) */
  int act;               /* DV_ACT_SILU */
  int rope;              /* DV_ROPE_1D or DV_ROPE_MROPE */
  float rope_theta;      /* RoPE base */
  int mrope_section[3];  /* frequency pairs per axis (t, h, w); M-RoPE modes only */
  float rms_eps;         /* epsilon inside the RMSNorm square root */
  int max_batch;         /* largest batch a build may pass */
  int max_n_vis;         /* largest number of visual tokens per batch element */
  int has_kv_bias;       /* 1: weights carry b_K, b_V; 0: no bias */
  int adapter;           /* DV_ADAPTER_EMBEDDING or DV_ADAPTER_RECURRENT */
  int k_norm;            /* 1: each key head is RMS-normalised before RoPE, with the gain
                            dv_weights.k_norm_gamma (the per-head K norm of Qwen3-VL backbones,
                            applied after the bias) */
  float k_norm_eps;      /* epsilon inside that norm's square root */
  int split_chain;       /* recurrent adapter only (0 otherwise): 1 = each bf16 operand of the
                            chain's two GEMMs (M_{l-1} into the down-projection, h_l into the
                            up-projection) is read as a high and a low bf16 part, two MMAs per
                            product, so the state M_l keeps about fp32 accuracy through deep
                            chains (in the rearranged chain: h_j and the products D_l U_j in two
                            parts each); the chain in the paper's order then runs on chip only
                            at rank <= 64, else as per-layer launches.
                            0 = one bf16 operand (faster).
                            Either way, with DV_RECURRENT_AUTO, builds whose 128-token blocks fit
                            in one wave of on-chip chain clusters run the chain, larger ones (and
                            every build the on-chip chain does not fit) the rearranged chain,
                            which forms each layer's down-projection input from E D_l^T and the
                            earlier h_j through the r x r products D_l U_j (the same sum). */
  int recurrent_path;    /* recurrent adapter only: DV_RECURRENT_AUTO (0), _CHAIN or
                            _REARRANGED */
} dv_config;

/* Weights of all L layers, bf16, device pointers. Read only during dv_memory_plan: the plan
 * keeps repacked copies, so the caller may free or change these after it returns.
 *   D      [L][r][d]    down-projection D_l (Sec. 3.1 Eq. 4) as an nn.Linear weight [out][in]
 *   U      [L][d][r]    up-projection U_l, nn.Linear layout [out][in]
 *   gamma  [L][d]       gain of the frozen input RMSNorm LN_l (Sec. 3.2 Eq. 7)
 *   Wk, Wv [L][kv][d]   frozen key / value projections W_K,l, W_V,l (kv = n_kv_heads*head_dim)
 *   bk, bv [L][kv]      biases, or NULL when has_kv_bias == 0
 *   k_norm_gamma [L][head_dim]  gain of the per-head K norm when k_norm == 1, else NULL
 *   layer_mode          HOST array of L DV_LAYER_* values, or NULL for DV_LAYER_ADAPTER at every
 *                       layer (App. J skips the adapters of early and late layers). Layers in
 *                       DV_LAYER_DROP get no K/V entries: builds leave their cache rows untouched,
 *                       and the plan keeps neither repacked weights nor workspace for them.
 *                       At least one layer must not be DV_LAYER_DROP. With the recurrent
 *                       adapter a skipped layer passes its input state on unchanged
 *                       (M_l = M_{l-1}), whether it is DV_LAYER_IDENTITY or DV_LAYER_DROP. */
typedef struct dv_weights {
  const void* D;
  const void* U;
  const void* gamma;
  const void* Wk;
  const void* Wv;
  const void* bk;
  const void* bv;
  const unsigned char* layer_mode;
  const void* k_norm_gamma;
} dv_weights;

/* Destination KV cache (bf16, caller-owned). Element (layer l, batch b, slot s, head h, j) of
 * K lives at k[l*s_layer + b*s_batch + s*s_seq + h*s_head + j], j < head_dim contiguous; the
 * same for V. Strides are in elements and must be multiples of 8 (16 bytes); k and v must be
 * 16-byte aligned. */
typedef struct dv_kv_cache {
  void* k;
  void* v;
  long long s_layer;
  long long s_batch;
  long long s_seq;
  long long s_head;
} dv_kv_cache;

typedef struct dv_plan dv_plan;

/*
 * dv_memory_plan — validate the configuration, allocate the plan and its workspace on the
 * current device, and repack the weights for the build kernels. Embedding adapter: all L
 * down-projections stacked into one matrix, since every layer reads only E (Sec. 3.1: the
 * memories are conditionally independent across layers given E), and the RMSNorm gain and
 * the rank-r update folded into the K/V weights. Recurrent adapter: per-layer down- and
 * up-projections, and the RMSNorm gain folded into the K/V weights.
 *   cfg     shape and limits (copied)
 *   w       device weights (read on `stream` before this call returns; not retained)
 *   stream  cudaStream_t as void*; the repack kernels run on it and this call waits for them
 *   out     receives the plan; *out is set to NULL on any error
 * Errors: DV_ERR_INVALID_ARG, DV_ERR_UNSUPPORTED_SHAPE, DV_ERR_UNSUPPORTED_DEVICE,
 * DV_ERR_OOM, DV_ERR_CUDA. On error nothing stays allocated.
 */
int dv_memory_plan(const dv_config* cfg, const dv_weights* w, void* stream, dv_plan** out);

/*
 * dv_build_visual_memory — the hot path. For batch*n_vis visual tokens writes K^v_l and V^v_l
 * of every layer (Sec. 3.1 Eqs. 4-6, Sec. 3.2 Eq. 7) into the cache. With the recurrent
 * adapter the state M_l is carried in fp32 from layer to layer (on chip, or as the running sum
 * E + sum_{j<=l} h_j U_j^T of the rearranged chain); each layer's K/V read its bf16 rounding.
 *   x0     bf16 [batch][n_vis][d]: the visual embeddings E (Sec. 2 Eq. 1); 16-byte aligned
 *   pos    int32 [batch][P][n_vis], P = 1 (DV_ROPE_1D) or 3 (M-RoPE modes: t, h, w): the
 *          original positions of the visual tokens (Sec. 1 and App. H keep them unchanged)
 *   slot   int32 [batch][n_vis] cache slot of each token, or NULL for slot0 + i
 *   slot0  first slot when slot == NULL
 *   out    destination cache; token i of batch element b goes to slot slot[b][i] (or slot0+i)
 *   stream cudaStream_t as void*
 * batch*n_vis == 0 is a no-op. Concurrent builds with the same plan must be ordered on one
 * stream (they share the plan's workspace). The caller keeps slots in range of its cache.
 * Errors: DV_ERR_INVALID_ARG, DV_ERR_UNSUPPORTED_SHAPE (more tokens than the plan's limit),
 * DV_ERR_ALIGNMENT, DV_ERR_CUDA.
 */
int dv_build_visual_memory(dv_plan* plan, const void* x0, int batch, int n_vis, const int* pos,
                           const int* slot, int slot0, const dv_kv_cache* out, void* stream);

/*
 * dv_build_visual_memory_noalloc — the same build as dv_build_visual_memory (same arguments,
 * same output), for callers that must not allocate device memory when they build: engines
 * that reserve all device memory at start-up and cannot give a plan a workspace sized for
 * their largest batch, or code that must not risk the device-wide synchronisation that
 * cudaMalloc / cudaFree can cause. The paper has no counterpart to this entry point; it
 * only changes where the build keeps its intermediates.
 *   - It allocates nothing: the intermediates (SiLU(E D_l) of every layer, the RMS statistics
 *     and the row sums of squares) go to one static device array of 32 MiB that every device
 *     loading this library holds until the process exits. The plan's own workspace is not
 *     used, so its max_batch / max_n_vis do not bound this call.
 *   - Limit: with T = batch * n_vis, r_pad = rank rounded up to 64 and L the planned layers,
 *     the intermediates (each part rounded up to 256 bytes) must fit in 32 MiB:
 *       embedding adapter  T * ((L * r_pad + 64) * 2 + L * 4 + 4 + (d + 64) * 2) bytes (h of
 *                          every layer, RMS statistics, row sums, a copy of E), plus
 *                          T * L * r_pad * 4 when r_pad = 64 (the fp32 x0 (2 U_l)^T of the
 *                          small-token path);
 *       recurrent adapter  T * (L * r_pad * 2 + L * 4 + 4 + L * (2 d + 4 d / 64)) bytes
 *                          (h, RMS statistics, bf16 M_l of every layer, partial sums of
 *                          squares), plus T * L * r_pad * 4 (the fp32 E D_l^T of the
 *                          rearranged chain) without split_chain, or T * 4 d (the fp32 state)
 *                          and T * (L * r_pad + d) * 2 with it.
 *     Larger builds return DV_ERR_UNSUPPORTED_SHAPE and launch nothing.
 *   - dv_memory_plan reserves the array on the plan's device (CUDA loads the module that
 *     holds it when the plan looks up its address) and loads every kernel a build can launch,
 *     so this entry point allocates nothing, even on its first call.
 *   - All calls on a device share the array and find it as the last call left it (nothing in
 *     it needs to start at zero). Calls that overlap on the GPU race on it: order them on one
 *     stream.
 * Errors: as dv_build_visual_memory, plus DV_ERR_UNSUPPORTED_SHAPE for builds over the limit
 * and DV_ERR_OOM when the array could not be reserved when the plan was made.
 */
int dv_build_visual_memory_noalloc(dv_plan* plan, const void* x0, int batch, int n_vis,
                                   const int* pos, const int* slot, int slot0,
                                   const dv_kv_cache* out, void* stream);

/*
 * End-to-end builds from host memory. The visual memory is the K/V entries that text tokens
 * read (Sec. 3.2 Eq. 7); a caller that keeps E and its KV cache in host memory submits builds
 * to a pipeline that copies E and the positions in, runs dv_build_visual_memory, and copies the
 * built K/V out, with the copy-out of one build overlapping the next build.
 *
 * dv_host_pipeline_create — device staging for builds of exactly batch x n_vis tokens with
 * `plan`: `depth` (1..4) sets of E, positions and a dense K/V cache, and three CUDA streams
 * (copy-in, build, copy-out) on the current device. This call allocates (cudaMalloc) all of
 * it; builds allocate nothing more. Staging sets are used round-robin: with depth >= 2 the
 * copy-out of build i overlaps build i + 1. The plan must outlive the pipeline, and no other
 * build with the same plan may run while the pipeline's builds are in flight (they share the
 * plan's workspace).
 * Errors: DV_ERR_INVALID_ARG, DV_ERR_UNSUPPORTED_SHAPE (beyond the plan's max_batch /
 * max_n_vis), DV_ERR_OOM, DV_ERR_CUDA. On error nothing stays allocated and *out is NULL.
 */
typedef struct dv_host_pipeline dv_host_pipeline;
int dv_host_pipeline_create(dv_plan* plan, int batch, int n_vis, int depth,
                            dv_host_pipeline** out);

/*
 * dv_build_visual_memory_host — one end-to-end build, asynchronous. HOST pointers:
 *   x0_host  bf16 [batch][n_vis][d]   E
 *   pos_host int32 [batch][P][n_vis]  positions, P = 1 (DV_ROPE_1D) or 3 (M-RoPE modes)
 *   k_host, v_host  bf16 [n_layers][batch][n_vis][n_kv_heads][head_dim] (dense): receive K and V
 *            of every built layer; the rows of DV_LAYER_DROP layers are left untouched
 *   stream   cudaStream_t as void*: the copy-in starts after the work enqueued on it before
 *            this call (use dv_host_pipeline_join for the other direction)
 *   ticket   receives the build's sequence number (may be NULL)
 * The caller must not change x0_host / pos_host, nor read k_host / v_host, until
 * dv_host_pipeline_wait(ticket) returns. Page-locked host memory (cudaHostAlloc or
 * cudaHostRegister) lets the copies run asynchronously and overlap the builds; pageable memory
 * gives the same result, but the driver stages those copies and they do not overlap.
 * Each build moves batch*n_vis*(2 d + 4 P) bytes in and 2 * n_built * batch*n_vis*kv*2 bytes
 * out, one cudaMemcpyAsync per contiguous range.
 * Errors: DV_ERR_INVALID_ARG (NULL pointer, or the pipeline's device is not current),
 * DV_ERR_ALIGNMENT (pos_host not 4-byte, bf16 buffers not 2-byte aligned), DV_ERR_CUDA.
 */
int dv_build_visual_memory_host(dv_host_pipeline* pipe, const void* x0_host, const int* pos_host,
                                void* k_host, void* v_host, void* stream, long long* ticket);

/* dv_host_pipeline_wait — blocks the calling thread until the host buffers of build `ticket`
 * hold its K/V. DV_ERR_INVALID_ARG for a ticket not yet issued. Device-side timeouts of the
 * build are reported by dv_plan_status on the pipeline's plan. */
int dv_host_pipeline_wait(dv_host_pipeline* pipe, long long ticket);

/* dv_host_pipeline_join — makes work enqueued on `stream` after this call wait until every
 * build submitted so far has finished its copy-out (stream-ordered, does not block the host). */
int dv_host_pipeline_join(dv_host_pipeline* pipe, void* stream);

/* dv_host_pipeline_free — waits for the pipeline's builds, then releases its device buffers,
 * streams and events. NULL is a no-op. */
void dv_host_pipeline_free(dv_host_pipeline* pipe);

/*
 * dv_plan_status — synchronises the device, reads and clears the plan's device status word.
 * Returns DV_OK, DV_ERR_DEVICE_TIMEOUT when a kernel of an earlier build gave up on a wait
 * (its outputs are then incomplete), or DV_ERR_INVALID_ARG for a NULL plan.
 */
int dv_plan_status(dv_plan* plan);

/*
 * dv_text_attention — the consumer of the visual memory (Sec. 3.2): the text queries of one
 * layer attend jointly to the visual keys/values the build wrote and the text context, with
 * the original causal structure: O = Attn(Q^t, [K^v; K^t], [V^v; V^t]). Reads the cache in
 * place; needs no plan and allocates nothing.
 *   q         bf16 [batch][n_q_heads][n_text][head_dim]: the text queries, already rotated
 *   cache     the KV cache (the strides of dv_kv_cache); `layer` selects the layer
 *   max_keys  slots per batch element the cache holds (slots >= max_keys are never read)
 *   n_keys    int32 [batch]: slots 0 .. n_keys[b] - 1 hold keys (visual and text, in sequence
 *             order); later slots are ignored
 *   q_slot    int32 [batch][n_text]: the slot of each query's own token; query t sees slot s
 *             when s <= q_slot[b][t] and s < n_keys[b] (it sees nothing when q_slot < 0)
 *   scale     softmax scale (> 0), e.g. 1 / sqrt(head_dim)
 *   out       bf16 [batch][n_q_heads][n_text][head_dim]; a query that sees no key gets zeros
 * Query head hq reads key head hq / (n_q_heads / n_kv_heads). head_dim in {64, 128}. q and out
 * 16-byte aligned; cache strides as for dv_build_visual_memory. batch * n_text == 0 is a no-op.
 * Errors: DV_ERR_INVALID_ARG, DV_ERR_UNSUPPORTED_SHAPE, DV_ERR_ALIGNMENT,
 * DV_ERR_UNSUPPORTED_DEVICE, DV_ERR_CUDA. Stream-ordered and asynchronous.
 */
int dv_text_attention(const void* q, int batch, int n_q_heads, int n_kv_heads, int n_text,
                      int head_dim, const dv_kv_cache* cache, int layer, int max_keys,
                      const int* n_keys, const int* q_slot, float scale, void* out, void* stream);

/* dv_text_attention_status — synchronises the device, reads and clears the status word of the
 * attention launches on the current device: DV_OK, or DV_ERR_DEVICE_TIMEOUT when a launch gave
 * up on a wait (its output is then incomplete). */
int dv_text_attention_status(void);

/* dv_free — release the plan and everything it owns (synchronises the device first).
 * dv_free(NULL) is a no-op. */
void dv_free(dv_plan* plan);

/* dv_error_string — static description of a status code (never NULL). */
const char* dv_error_string(int status);

/*
 * Per-stage device timing of builds, for measurement. While enabled, each build records
 * CUDA events around its stages on the build's stream (at most 4096 builds are recorded).
 *   dv_timing_enable(plan, 1) starts a new record (0 stops recording).
 *   dv_timing_read(plan, ms, n_stages, n_builds) synchronises on the recorded events and
 *   writes the summed milliseconds of each stage into ms[0..n_stages-1] (stage order:
 *   0 stacked down-projection + SiLU, 1 row sums of squares of E, 2 RMS statistics,
 *   3 K/V projection + RoPE + cache store; recurrent adapter: 0 E D^T of every layer (empty
 *   when the on-chip chain runs), 1 the adapter chain through all layers, 2 RMS statistics from
 *   the chain's partial sums, 3 as above) and the number of builds into *n_builds.
 */
int dv_timing_enable(dv_plan* plan, int on);
int dv_timing_read(dv_plan* plan, double* ms, int n_stages, int* n_builds);

/* Number of kernels one build of the plan's full size (max_batch x max_n_vis tokens) launches
 * (for launch accounting). */
int dv_kernels_per_build(const dv_plan* plan);

/* Which kernel computes K/V (Sec. 3.2 Eq. 7) in a build of `tokens` tokens, for reporting:
 * DV_KV_ENGINE_WEIGHTS_AS_M (weight rows as the MMA's M, tokens as N: dv_kv_pair_kernel) or
 * DV_KV_ENGINE_TOKENS_AS_M (256-token blocks as M: dv_pair_tm_kernel); 0 for a NULL plan or
 * tokens <= 0. */
enum { DV_KV_ENGINE_WEIGHTS_AS_M = 1, DV_KV_ENGINE_TOKENS_AS_M = 2 };
int dv_kv_engine(const dv_plan* plan, long long tokens);

/*
 * dv_debug_wait_timeout — failure-detection self-test. Launches one kernel whose single
 * thread waits on a shared-memory barrier that nothing will complete, with a limit of
 * timeout_us microseconds; the wait gives up, the kernel records DV_ERR_DEVICE_TIMEOUT in
 * the plan's status word and returns normally, so the context stays usable. Read the result
 * with dv_plan_status. timeout_us must be in [1, 2000000].
 */
int dv_debug_wait_timeout(dv_plan* plan, int timeout_us, void* stream);

/*
 * dv_debug_copy_workspace — copies the intermediate results of the last build on this plan
 * into caller-owned device buffers (stream-ordered), for stage-wise testing:
 *   H     bf16 [tokens][n_planned * r_pad]  SiLU(E D_l) (recurrent: SiLU(M_{l-1} D_l)) of
 *         every planned layer, r_pad = rank rounded up to 64 (columns past rank are zero)
 *   rstd  fp32 [n_planned][tokens]           1 / sqrt(mean(M_l^2) + eps)
 *   xx    fp32 [tokens]                     sum of squares of each row of E (embedding
 *         adapter only; not written by recurrent builds)
 * n_planned is the number of layers whose mode is not DV_LAYER_DROP (n_layers when the plan
 * was made without layer modes); planned layers appear in layer order. Any of the three may
 * be NULL. tokens must not exceed the last build's token count; *r_pad_out (if not NULL)
 * receives r_pad.
 */
int dv_debug_copy_workspace(dv_plan* plan, int tokens, void* H, void* rstd, void* xx,
                            int* r_pad_out, void* stream);

/*
 * dv_debug_copy_memory — recurrent adapter only: copies bf16 M_l of every planned layer of the
 * last build, [n_planned][tokens][d], into a caller-owned device buffer (stream-ordered), for
 * stage-wise testing of the chain M_l = M_{l-1} + SiLU(M_{l-1} D_l) U_l (Sec. 3.1 Eq. 6).
 * tokens must not exceed the last build's token count. DV_ERR_INVALID_ARG for a plan with the
 * embedding adapter (it never forms M_l).
 */
int dv_debug_copy_memory(dv_plan* plan, int tokens, void* mem, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* DV_H */
