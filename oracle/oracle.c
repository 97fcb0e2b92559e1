/*
 * ORACLE — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, fp64 CPU statement of the visual-memory build of "Just MLPs: Efficient
 * Visual State Reconstruction for Multimodal Language Models" (delta-Vision), with the
 * embedding or the recurrent adapter, and of its consumer, the text queries' causal attention
 * over the visual and text keys/values (oracle_text_attention, at the end). Only the tests,
 * the smoke check and the benchmark's CPU-baseline and reference legs may load it. It shares
 * no code, header, table or helper with the CUDA path.
 *
 * What it computes, for every visual token row x = E_i (a row of the initial visual
 * embeddings, Sec. 2 Eq. 1) and every layer l, in this order:
 *   z = x D_l                          Sec. 3.1 Eq. 4: D_l in R^{d x r}; stored [r][d]
 *   h = phi(z), phi = SiLU             Sec. 3.1 Eq. 4: phi(u) = u / (1 + exp(-u))
 *   m = x + h U_l                      Sec. 3.1 Eqs. 4-5: M_l = E + Delta_l(E); U_l in
 *                                      R^{r x d}, stored [d][r]
 *   n = gamma_l * m / sqrt(mean(m^2) + eps)
 *                                      Sec. 3.2 Eq. 7 applies the frozen input norm LN_l;
 *                                      App. K names it RMSNorm (learnable gain, no centring)
 *   k = W_K,l n (+ b_K,l), v = W_V,l n (+ b_V,l)
 *                                      Sec. 3.2 Eq. 7: K^v_l = W_K,l LN_l(M_l), same for V;
 *                                      W stored [kv][d]; the bias is the backbone's, if any
 *   k <- RoPE(k, positions of token i) Sec. 3.2 keeps the original causal attention and
 *                                      Sec. 1 / App. H keep the visual positions, so the
 *                                      backbone's rotary embedding is applied to visual keys
 *                                      at their original positions; V is not rotated.
 * Recurrent variant (Sec. 3.1 Eq. 6): M_0 = E and M_l = A_l(M_{l-1}) for l = 1..L, where
 * A_l(X) = X + phi(X D_l) U_l is the same adapter as above; each layer's norm, projections
 * and rotation then act on that layer's M_l exactly as listed. The chain runs through the
 * layers in order for each token on its own (the adapter acts row by row).
 *
 * RoPE reading: rotate-half pairs (j, j + D_h/2) of each head, inverse frequency
 * theta^(-2j/D_h); the angle of pair j is p * theta^(-2j/D_h), where p is the 1-D
 * position, or for M-RoPE the (t, h, w) position of the axis that frequency j belongs to:
 * contiguous sections (j < s0 -> t, then s1 of h, then s2 of w), or the interleaved layout
 * of Qwen3-VL backbones (j = 1 mod 3 with j < 3 s1 -> h, j = 2 mod 3 with j < 3 s2 -> w,
 * every other j -> t).
 *
 * Per-head K normalisation (Qwen3-VL backbones normalise each key head before RoPE, the
 * "query normalization" the paper's default backbone applies): when enabled, each head of
 * k (after the bias) becomes g * k_h / sqrt(mean(k_h^2) + eps_k), g the layer's gain [D_h].
 *
 * Every input is a bf16 bit pattern widened exactly to double; every step runs in double.
 * Tokens are independent of each other (every step above acts on one row), so the only
 * parallelism is an OpenMP loop over the requested tokens.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int d;               /* hidden size */
  int n_layers;        /* L */
  int n_kv_heads;      /* H_kv */
  int head_dim;        /* D_h */
  int rank;            /* r */
  int rope;            /* 0: 1-D RoPE, 1: M-RoPE (t, h, w) */
  double rope_theta;
  int mrope_section[3];
  double rms_eps;
  int recurrent;       /* 0: embedding adapter (Sec. 3.1 Eq. 5), 1: recurrent (Eq. 6) */
  int k_norm;          /* 1: per-head RMSNorm of K before RoPE */
  double k_norm_eps;
} oracle_cfg;

static double bf16_to_f64(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* phi of Sec. 3.1 Eq. 4: SiLU(u) = u * sigmoid(u) = u / (1 + e^-u). */
double oracle_silu(double u) { return u / (1.0 + exp(-u)); }

/* Adapter of Sec. 3.1 Eqs. 4-5 for one token row and one layer.
 * x[d] in; Dl = D_l stored [r][d]; Ul = U_l stored [d][r]; z[r], h[r], m[d] out. */
void oracle_adapter_row(int d, int r, const double* x, const uint16_t* Dl, const uint16_t* Ul,
                        double* z, double* h, double* m) {
  for (int k = 0; k < r; ++k) {
    double s = 0.0;
    for (int j = 0; j < d; ++j) s += x[j] * bf16_to_f64(Dl[(int64_t)k * d + j]);
    z[k] = s;
    h[k] = oracle_silu(s);
  }
  for (int j = 0; j < d; ++j) {
    double s = 0.0;
    for (int k = 0; k < r; ++k) s += h[k] * bf16_to_f64(Ul[(int64_t)j * r + k]);
    m[j] = x[j] + s;
  }
}

/* RMSNorm with gain (LN_l of Sec. 3.2 Eq. 7; RMSNorm per App. K):
 * n_j = gamma_j * m_j / sqrt((1/d) sum_i m_i^2 + eps). */
void oracle_rmsnorm_row(int d, const double* m, const double* gamma, double eps, double* n) {
  double ss = 0.0;
  for (int j = 0; j < d; ++j) ss += m[j] * m[j];
  double inv = 1.0 / sqrt(ss / (double)d + eps);
  for (int j = 0; j < d; ++j) n[j] = gamma[j] * m[j] * inv;
}

/* One projection of Sec. 3.2 Eq. 7: out = W n (+ b), W stored [kv][d], b [kv] or NULL. */
void oracle_project_row(int d, int kv, const uint16_t* W, const uint16_t* b, const double* n,
                        double* out) {
  for (int c = 0; c < kv; ++c) {
    double s = 0.0;
    for (int j = 0; j < d; ++j) s += bf16_to_f64(W[(int64_t)c * d + j]) * n[j];
    out[c] = s + (b ? bf16_to_f64(b[c]) : 0.0);
  }
}

/* Axis (0 = t, 1 = h, 2 = w) of frequency j under M-RoPE layout `mrope`
 * (1: contiguous sections, 2: interleaved). */
static int mrope_axis(int mrope, const int* section, int j) {
  if (mrope == 1) {
    if (j >= section[0] + section[1]) return 2;
    if (j >= section[0]) return 1;
    return 0;
  }
  if (j % 3 == 1 && j < 3 * section[1]) return 1;
  if (j % 3 == 2 && j < 3 * section[2]) return 2;
  return 0;
}

/* Per-head RMSNorm of a key head x[head_dim] with gain g (bf16 [head_dim]):
 * x_j <- g_j * x_j / sqrt(mean(x^2) + eps). */
void oracle_head_rmsnorm(int head_dim, const uint16_t* g, double eps, double* x) {
  double ss = 0.0;
  for (int j = 0; j < head_dim; ++j) ss += x[j] * x[j];
  const double inv = 1.0 / sqrt(ss / (double)head_dim + eps);
  for (int j = 0; j < head_dim; ++j) x[j] = bf16_to_f64(g[j]) * x[j] * inv;
}

/* Rotary position embedding of one head (rotate-half pairs (j, j + D/2)).
 * pos3 holds the position of each axis: pos3[0] for 1-D RoPE (mrope = 0); (t, h, w) for
 * M-RoPE (mrope = 1 contiguous sections, 2 interleaved), where pair j takes its axis's
 * position. */
void oracle_rope_head(int head_dim, double theta, int mrope, const int* section,
                      const double* pos3, double* x) {
  int half = head_dim / 2;
  for (int j = 0; j < half; ++j) {
    double p = pos3[0];
    if (mrope) p = pos3[mrope_axis(mrope, section, j)];
    double a = p * pow(theta, -2.0 * (double)j / (double)head_dim);
    double c = cos(a), s = sin(a);
    double x1 = x[j], x2 = x[j + half];
    x[j] = x1 * c - x2 * s;
    x[j + half] = x2 * c + x1 * s;
  }
}

/* Norm, projections, rotation and output of one token's memory m at layer l (the steps of
 * Sec. 3.2 Eq. 7 and the RoPE reading above), written at output index o. */
static void memory_outputs(const oracle_cfg* c, int l, const double* m, const double* h,
                           const uint16_t* gamma, const uint16_t* Wk, const uint16_t* Wv,
                           const uint16_t* bk, const uint16_t* bv, const uint16_t* kgamma,
                           const double* p3, int64_t o,
                           double* g, double* n, double* kk, double* vv, double* k_out,
                           double* v_out, double* m_out, double* h_out, double* n_out) {
  const int d = c->d, r = c->rank, Dh = c->head_dim, kv = c->n_kv_heads * Dh;
  for (int j = 0; j < d; ++j) g[j] = bf16_to_f64(gamma[(int64_t)l * d + j]);
  oracle_rmsnorm_row(d, m, g, c->rms_eps, n);
  oracle_project_row(d, kv, Wk + (int64_t)l * kv * d, bk ? bk + (int64_t)l * kv : NULL, n, kk);
  oracle_project_row(d, kv, Wv + (int64_t)l * kv * d, bv ? bv + (int64_t)l * kv : NULL, n, vv);
  if (c->k_norm)
    for (int hh = 0; hh < c->n_kv_heads; ++hh)
      oracle_head_rmsnorm(Dh, kgamma + (int64_t)l * Dh, c->k_norm_eps, kk + hh * Dh);
  for (int hh = 0; hh < c->n_kv_heads; ++hh)
    oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, kk + hh * Dh);
  if (k_out) memcpy(k_out + o * kv, kk, sizeof(double) * kv);
  if (v_out) memcpy(v_out + o * kv, vv, sizeof(double) * kv);
  if (m_out) memcpy(m_out + o * d, m, sizeof(double) * d);
  if (n_out) memcpy(n_out + o * d, n, sizeof(double) * d);
  if (h_out) memcpy(h_out + o * r, h, sizeof(double) * r);
}

/* Recurrent variant (Sec. 3.1 Eq. 6) of oracle_build_tokens: for each token, M_0 = E and
 * M_l = A_l(M_{l-1}) through the layers in order; the memory of every requested layer goes
 * through memory_outputs. Same arguments and output layout as oracle_build_tokens. */
static int build_tokens_recurrent(const oracle_cfg* c, const uint16_t* x0, int n_vis,
                                  const int32_t* pos, const uint16_t* D, const uint16_t* U,
                                  const uint16_t* gamma, const uint16_t* Wk, const uint16_t* Wv,
                                  const uint16_t* bk, const uint16_t* bv, const uint16_t* kgamma,
                                  const int64_t* tokens,
                                  int64_t n_tokens, const int32_t* layers, int Ls,
                                  double* k_out, double* v_out, double* m_out, double* h_out,
                                  double* n_out) {
  const int d = c->d, L = c->n_layers, r = c->rank, kv = c->n_kv_heads * c->head_dim;
  const int P = c->rope ? 3 : 1;
  int last = 0;  /* deepest layer any output needs */
  for (int s = 0; s < Ls; ++s) {
    const int l = layers ? layers[s] : s;
    if (l > last) last = l;
  }
#pragma omp parallel
  {
    double* prev = malloc(sizeof(double) * d);
    double* m = malloc(sizeof(double) * d);
    double* n = malloc(sizeof(double) * d);
    double* g = malloc(sizeof(double) * d);
    double* z = malloc(sizeof(double) * r);
    double* h = malloc(sizeof(double) * r);
    double* kk = malloc(sizeof(double) * kv);
    double* vv = malloc(sizeof(double) * kv);
#pragma omp for schedule(dynamic, 1)
    for (int64_t q = 0; q < n_tokens; ++q) {
      const int64_t t = tokens[q];
      const int64_t b = t / n_vis, i = t % n_vis;
      double p3[3];
      for (int a = 0; a < P; ++a) p3[a] = (double)pos[(b * P + a) * n_vis + i];
      for (int j = 0; j < d; ++j) prev[j] = bf16_to_f64(x0[t * d + j]);  /* M_0 = E */
      for (int l = 0; l <= last && l < L; ++l) {
        /* M_l = A_l(M_{l-1}) (layer l + 1 of Eq. 6 in the paper's 1-based numbering) */
        oracle_adapter_row(d, r, prev, D + (int64_t)l * r * d, U + (int64_t)l * d * r, z, h, m);
        for (int s = 0; s < Ls; ++s)
          if ((layers ? layers[s] : s) == l)
            memory_outputs(c, l, m, h, gamma, Wk, Wv, bk, bv, kgamma, p3, q * Ls + s, g, n, kk, vv,
                           k_out, v_out, m_out, h_out, n_out);
        memcpy(prev, m, sizeof(double) * d);
      }
    }
    free(prev); free(m); free(n); free(g); free(z); free(h); free(kk); free(vv);
  }
  return 0;
}

/*
 * The whole build for a list of tokens.
 *   x0    bf16 [B][n_vis][d];   pos int32 [B][P][n_vis], P = 1 (1-D) or 3 (M-RoPE)
 *   D [L][r][d], U [L][d][r], gamma [L][d], Wk/Wv [L][kv][d], bk/bv [L][kv] or NULL,
 *   kgamma [L][D_h] per-head K-norm gain (read when cfg->k_norm)
 *   tokens: flat token ids t = b * n_vis + i;  n_tokens of them
 *   layers: the layers to evaluate (n_sel_layers of them), or NULL for all L in order
 * Outputs (each may be NULL), indexed by the position q of the token in `tokens` and the
 * position s of the layer in `layers` (Ls = number of evaluated layers):
 *   k_out, v_out [q][Ls][kv];  m_out [q][Ls][d];  h_out [q][Ls][r];  n_out [q][Ls][d]
 * Returns 0, or -1 on a bad argument.
 */
int oracle_build_tokens(const oracle_cfg* c, const uint16_t* x0, int n_vis, const int32_t* pos,
                        const uint16_t* D, const uint16_t* U, const uint16_t* gamma,
                        const uint16_t* Wk, const uint16_t* Wv, const uint16_t* bk,
                        const uint16_t* bv, const uint16_t* kgamma, const int64_t* tokens,
                        int64_t n_tokens,
                        const int32_t* layers, int n_sel_layers,
                        double* k_out, double* v_out, double* m_out, double* h_out,
                        double* n_out) {
  if (!c || !x0 || !pos || !D || !U || !gamma || !Wk || !Wv || !tokens) return -1;
  const int d = c->d, L = c->n_layers, r = c->rank, Dh = c->head_dim;
  const int kv = c->n_kv_heads * Dh;
  const int P = c->rope ? 3 : 1;
  if (d <= 0 || L <= 0 || r <= 0 || Dh <= 0 || (Dh & 1) || n_vis <= 0) return -1;
  if (c->rope < 0 || c->rope > 2 || (c->k_norm && !kgamma)) return -1;
  if (c->rope && c->mrope_section[0] + c->mrope_section[1] + c->mrope_section[2] != Dh / 2)
    return -1;
  const int Ls = layers ? n_sel_layers : L;
  if (Ls <= 0) return -1;
  for (int s = 0; layers && s < Ls; ++s)
    if (layers[s] < 0 || layers[s] >= L) return -1;
  if (c->recurrent) return build_tokens_recurrent(c, x0, n_vis, pos, D, U, gamma, Wk, Wv, bk, bv,
                                                 kgamma, tokens, n_tokens, layers, Ls, k_out,
                                                 v_out, m_out, h_out, n_out);
#pragma omp parallel
  {
    double* x = malloc(sizeof(double) * d);
    double* m = malloc(sizeof(double) * d);
    double* n = malloc(sizeof(double) * d);
    double* g = malloc(sizeof(double) * d);
    double* z = malloc(sizeof(double) * r);
    double* h = malloc(sizeof(double) * r);
    double* kk = malloc(sizeof(double) * kv);
    double* vv = malloc(sizeof(double) * kv);
#pragma omp for schedule(dynamic, 1) collapse(2)
    for (int64_t q = 0; q < n_tokens; ++q) {
      for (int ls = 0; ls < Ls; ++ls) {
        const int l = layers ? layers[ls] : ls;
        const int64_t t = tokens[q];
        const int64_t b = t / n_vis, i = t % n_vis;
        for (int j = 0; j < d; ++j) x[j] = bf16_to_f64(x0[t * d + j]);
        /* M_l = A_l(E) (Eq. 5) */
        oracle_adapter_row(d, r, x, D + (int64_t)l * r * d, U + (int64_t)l * d * r, z, h, m);
        double p3[3];
        for (int a = 0; a < P; ++a) p3[a] = (double)pos[(b * P + a) * n_vis + i];
        memory_outputs(c, l, m, h, gamma, Wk, Wv, bk, bv, kgamma, p3, q * Ls + ls, g, n, kk, vv,
                       k_out, v_out, m_out, h_out, n_out);
      }
    }
    free(x); free(m); free(n); free(g); free(z); free(h); free(kk); free(vv);
  }
  return 0;
}

/* Number of threads the OpenMP runtime will use (reported beside oracle timings). */
int oracle_num_threads(void) {
  int nt = 1;
#pragma omp parallel
  {
#pragma omp single
    nt = omp_get_num_threads();
  }
  return nt;
}

/*
 * Consumer of the visual memory (Sec. 3.2): text queries attend jointly to the visual
 * keys/values and the text context, with the original causal structure, O = Attn(Q, [K^v; K^t],
 * [V^v; V^t]). The sequence is a list of cache slots in order; query t of batch element b sits
 * at slot q_slot[b][t] and sees slot s when s <= q_slot[b][t] and s < n_keys[b]. Grouped
 * queries: query head hq reads key head hq / (n_q_heads / n_kv_heads).
 *   q    [B][Hq][Nt][D];  k, v [B][S][Hkv][D] (slots);  out [B][Hq][Nt][D]   (all fp64)
 *   o = sum_s softmax_s(scale * q . k_s) v_s over the visible slots; 0 when none is visible.
 * Returns 0, or -1 on a bad argument.
 */
int oracle_text_attention(int B, int Hq, int Hkv, int Nt, int S, int D, const double* q,
                          const double* k, const double* v, const int32_t* n_keys,
                          const int32_t* q_slot, double scale, double* out) {
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || Nt <= 0 || S <= 0 || D <= 0) return -1;
  const int G = Hq / Hkv;
#pragma omp parallel for collapse(3) schedule(dynamic, 1)
  for (int b = 0; b < B; ++b) {
    for (int hq = 0; hq < Hq; ++hq) {
      for (int t = 0; t < Nt; ++t) {
        const int h = hq / G;
        const double* qr = q + (((int64_t)b * Hq + hq) * Nt + t) * D;
        double* o = out + (((int64_t)b * Hq + hq) * Nt + t) * D;
        int last = q_slot[(int64_t)b * Nt + t];
        if (last >= n_keys[b]) last = n_keys[b] - 1;
        if (last >= S) last = S - 1;
        for (int j = 0; j < D; ++j) o[j] = 0.0;
        if (last < 0) continue;
        double mx = -INFINITY;
        for (int s = 0; s <= last; ++s) {
          const double* kr = k + (((int64_t)b * S + s) * Hkv + h) * D;
          double dot = 0.0;
          for (int j = 0; j < D; ++j) dot += qr[j] * kr[j];
          if (scale * dot > mx) mx = scale * dot;
        }
        double den = 0.0;
        for (int s = 0; s <= last; ++s) {
          const double* kr = k + (((int64_t)b * S + s) * Hkv + h) * D;
          const double* vr = v + (((int64_t)b * S + s) * Hkv + h) * D;
          double dot = 0.0;
          for (int j = 0; j < D; ++j) dot += qr[j] * kr[j];
          const double w = exp(scale * dot - mx);
          den += w;
          for (int j = 0; j < D; ++j) o[j] += w * vr[j];
        }
        for (int j = 0; j < D; ++j) o[j] /= den;
      }
    }
  }
  return 0;
}
