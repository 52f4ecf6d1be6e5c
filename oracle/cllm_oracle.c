/*
 * Oracle forward pass: a plain, slow, fp64 CPU implementation of the decoder
 * whose greedy next-token map  y_i = argmax_y p(y | y_<i, x)  (Eq. 1) the Jacobi
 * iteration (Eq. 3, Sec. 3.1) solves in parallel.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load this library.  The product path (the
 * CUDA library behind include/cllm.h) never links, loads or calls it, and this
 * file shares no code, header, table or constant with that path.
 *
 * The paper names its target models (LLaMA-2-7B and Deepseek-coder-7B,
 * Sec. 4.1) without restating their architecture.  The decoder written out here
 * is the standard pre-norm LLaMA layer, each step a plain definition:
 *
 *   h      = x / sqrt(mean(x^2) + eps) * g_attn          (RMSNorm)
 *   q,k,v  = h Wq^T, h Wk^T, h Wv^T                      (no biases)
 *   q,k    = RoPE(q, pos), RoPE(k, pos)                   (rotate-half pairs (i, i+hd/2),
 *                                                          angle pos * theta^(-2i/hd))
 *   a      = softmax(q k^T / sqrt(hd)) v over keys at positions 0..pos (causal)
 *   x      = x + a Wo^T
 *   h2     = x / sqrt(mean(x^2) + eps) * g_mlp
 *   x      = x + (silu(h2 Wg^T) * (h2 Wu^T)) Wd^T         (SwiGLU MLP)
 *   logits = (x / sqrt(mean(x^2)+eps) * g_final) Wlm^T    (untied LM head)
 *
 * The embedding is an unscaled row lookup.  Grouped-query attention maps query
 * head h to key/value head h / (n_heads / n_kv_heads).
 *
 * Jacobi decoding with a KV cache (Sec. 3.1, Alg. 3) keeps the keys and values
 * of committed tokens and recomputes only the n-token block: orc_forward(...)
 * takes the block's tokens and the position of its first row, writes the
 * block's keys/values at those positions of the cache, and attends over cache
 * positions 0..pos for the row at position pos.  "Removing the KV cache of
 * false tokens" (Alg. 3) is implicit: positions past the committed length are
 * simply overwritten by the next call.
 *
 * All arithmetic is fp64.  Weights are read in their stored precision (fp32,
 * or bf16 bit patterns) and widened exactly to double.  Dot products use eight
 * interleaved partial sums added in a fixed order, so results are deterministic
 * and independent of the thread count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORC_F32 = 0, ORC_BF16 = 1 };

typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab;
  double rms_eps, rope_theta;
  int wdtype;
  int max_pos;
  /* weights, borrowed from the caller */
  const void *tok_emb, *final_norm, *lm_head;
  const void **attn_norm, **wq, **wk, **wv, **wo, **mlp_norm, **w_gate, **w_up,
      **w_down;
  /* KV cache: [layer][pos][n_kv_heads * head_dim] */
  double *kc, *vc;
} orc_model;

/* ---- weight access: exact widening of fp32 or bf16 to double ---------------- */

static double bf16_bits_to_double(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static void load_row(const orc_model *m, const void *w, size_t row, int ncols,
                     double *dst) {
  size_t off = row * (size_t)ncols;
  if (m->wdtype == ORC_F32) {
    const float *p = (const float *)w + off;
    for (int i = 0; i < ncols; ++i) dst[i] = (double)p[i];
  } else {
    const uint16_t *p = (const uint16_t *)w + off;
    for (int i = 0; i < ncols; ++i) dst[i] = bf16_bits_to_double(p[i]);
  }
}

static double dot(const double *a, const double *b, int n) {
  double acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int k = 0;
  for (; k + 8 <= n; k += 8)
    for (int u = 0; u < 8; ++u) acc[u] += a[k + u] * b[k + u];
  for (; k < n; ++k) acc[k & 7] += a[k] * b[k];
  return ((acc[0] + acc[1]) + (acc[2] + acc[3])) +
         ((acc[4] + acc[5]) + (acc[6] + acc[7]));
}

/* Y[t][j] = sum_k W[j][k] X[t][k]  for t < T, j < out_dim (W stored [out][in]) */
static void linear(const orc_model *m, const void *w, int out_dim, int in_dim,
                   const double *x, int T, double *y) {
#pragma omp parallel
  {
    double *wrow = (double *)malloc(sizeof(double) * (size_t)in_dim);
#pragma omp for schedule(static)
    for (int j = 0; j < out_dim; ++j) {
      load_row(m, w, (size_t)j, in_dim, wrow);
      for (int t = 0; t < T; ++t)
        y[(size_t)t * out_dim + j] = dot(wrow, x + (size_t)t * in_dim, in_dim);
    }
    free(wrow);
  }
}

/* ---- layer primitives (also exported for the pin tests) --------------------- */

/* out = x / sqrt(mean(x^2) + eps) * g */
void orc_rmsnorm(const double *x, const double *g, int d, double eps,
                 double *out) {
  double ss = 0.0;
  for (int i = 0; i < d; ++i) ss += x[i] * x[i];
  double r = 1.0 / sqrt(ss / d + eps);
  for (int i = 0; i < d; ++i) out[i] = x[i] * r * g[i];
}

/* Rotate-half RoPE of one head vector in place: pairs (i, i + hd/2) are
 * rotated by the angle pos * theta^(-2i/hd). */
void orc_rope(double *v, int head_dim, int pos, double theta) {
  int half = head_dim / 2;
  for (int i = 0; i < half; ++i) {
    double ang = (double)pos * pow(theta, -2.0 * (double)i / (double)head_dim);
    double c = cos(ang), s = sin(ang);
    double a = v[i], b = v[i + half];
    v[i] = a * c - b * s;
    v[i + half] = b * c + a * s;
  }
}

double orc_silu(double z) { return z / (1.0 + exp(-z)); }

/* One query attending to n_keys keys: out = sum_p softmax_p(q.k_p / sqrt(hd)) v_p.
 * Keys and values are rows of length `stride` starting at k[0], v[0]. */
void orc_attend(const double *q, const double *k, const double *v, int n_keys,
                int head_dim, int stride, double *out) {
  double *s = (double *)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1));
  double scale = 1.0 / sqrt((double)head_dim);
  double mx = -INFINITY;
  for (int p = 0; p < n_keys; ++p) {
    double acc = 0.0;
    for (int i = 0; i < head_dim; ++i) acc += q[i] * k[(size_t)p * stride + i];
    s[p] = acc * scale;
    if (s[p] > mx) mx = s[p];
  }
  double z = 0.0;
  for (int p = 0; p < n_keys; ++p) {
    s[p] = exp(s[p] - mx);
    z += s[p];
  }
  for (int i = 0; i < head_dim; ++i) {
    double acc = 0.0;
    for (int p = 0; p < n_keys; ++p) acc += s[p] * v[(size_t)p * stride + i];
    out[i] = acc / z;
  }
  free(s);
}

/* ---- model ------------------------------------------------------------------ */

/* iarch = {n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab}
 * farch = {rms_eps, rope_theta}
 * wptrs = {tok_emb, final_norm, lm_head, then per layer:
 *          attn_norm, wq, wk, wv, wo, mlp_norm, w_gate, w_up, w_down} */
orc_model *orc_create(const int *iarch, const double *farch, int wdtype,
                      const void *const *wptrs, int max_pos) {
  orc_model *m = (orc_model *)calloc(1, sizeof(orc_model));
  if (!m) return NULL;
  m->n_layers = iarch[0];
  m->d_model = iarch[1];
  m->n_heads = iarch[2];
  m->n_kv_heads = iarch[3];
  m->head_dim = iarch[4];
  m->ffn = iarch[5];
  m->vocab = iarch[6];
  m->rms_eps = farch[0];
  m->rope_theta = farch[1];
  m->wdtype = wdtype;
  m->max_pos = max_pos;
  m->tok_emb = wptrs[0];
  m->final_norm = wptrs[1];
  m->lm_head = wptrs[2];
  int L = m->n_layers;
  const void ***lists[9] = {&m->attn_norm, &m->wq, &m->wk, &m->wv, &m->wo,
                            &m->mlp_norm, &m->w_gate, &m->w_up, &m->w_down};
  for (int j = 0; j < 9; ++j) {
    *lists[j] = (const void **)malloc(sizeof(void *) * (size_t)L);
    for (int l = 0; l < L; ++l) (*lists[j])[l] = wptrs[3 + 9 * l + j];
  }
  size_t kvd = (size_t)m->n_kv_heads * m->head_dim;
  size_t n = (size_t)L * (size_t)max_pos * kvd;
  m->kc = (double *)calloc(n, sizeof(double));
  m->vc = (double *)calloc(n, sizeof(double));
  if (!m->kc || !m->vc) {
    free(m->kc);
    free(m->vc);
    free(m);
    return NULL;
  }
  return m;
}

void orc_destroy(orc_model *m) {
  if (!m) return;
  free(m->attn_norm);
  free(m->wq);
  free(m->wk);
  free(m->wv);
  free(m->wo);
  free(m->mlp_norm);
  free(m->w_gate);
  free(m->w_up);
  free(m->w_down);
  free(m->kc);
  free(m->vc);
  free(m);
}

/* Forward of T tokens at positions start_pos .. start_pos+T-1 over the cached
 * prefix 0..start_pos-1.  Writes the rows' keys/values into the cache and, for
 * each of the n_rows row indices in logit_rows, the vocab logits into
 * logits[i][vocab].  Returns 0, or -1 on bad arguments. */
int orc_forward(orc_model *m, const int32_t *tokens, int T, int start_pos,
                const int32_t *logit_rows, int n_rows, double *logits) {
  const int d = m->d_model, H = m->n_heads, Hkv = m->n_kv_heads,
            hd = m->head_dim, F = m->ffn, V = m->vocab;
  const int dq = H * hd, dkv = Hkv * hd, grp = H / Hkv;
  if (T <= 0 || start_pos < 0 || start_pos + T > m->max_pos) return -1;
  for (int t = 0; t < T; ++t)
    if (tokens[t] < 0 || tokens[t] >= V) return -1;
  for (int i = 0; i < n_rows; ++i)
    if (logit_rows[i] < 0 || logit_rows[i] >= T) return -1;

  double *x = (double *)malloc(sizeof(double) * (size_t)T * d);
  double *h = (double *)malloc(sizeof(double) * (size_t)T * d);
  double *q = (double *)malloc(sizeof(double) * (size_t)T * dq);
  double *k = (double *)malloc(sizeof(double) * (size_t)T * dkv);
  double *v = (double *)malloc(sizeof(double) * (size_t)T * dkv);
  double *a = (double *)malloc(sizeof(double) * (size_t)T * dq);
  double *o = (double *)malloc(sizeof(double) * (size_t)T * d);
  double *g = (double *)malloc(sizeof(double) * (size_t)T * F);
  double *u = (double *)malloc(sizeof(double) * (size_t)T * F);
  double *gain = (double *)malloc(sizeof(double) * (size_t)d);

  /* embedding lookup */
  for (int t = 0; t < T; ++t) load_row(m, m->tok_emb, (size_t)tokens[t], d, x + (size_t)t * d);

  for (int l = 0; l < m->n_layers; ++l) {
    double *kl = m->kc + (size_t)l * m->max_pos * dkv;
    double *vl = m->vc + (size_t)l * m->max_pos * dkv;

    /* attention sub-layer */
    load_row(m, m->attn_norm[l], 0, d, gain);
    for (int t = 0; t < T; ++t)
      orc_rmsnorm(x + (size_t)t * d, gain, d, m->rms_eps, h + (size_t)t * d);
    linear(m, m->wq[l], dq, d, h, T, q);
    linear(m, m->wk[l], dkv, d, h, T, k);
    linear(m, m->wv[l], dkv, d, h, T, v);
    for (int t = 0; t < T; ++t) {
      int pos = start_pos + t;
      for (int hh = 0; hh < H; ++hh)
        orc_rope(q + (size_t)t * dq + (size_t)hh * hd, hd, pos, m->rope_theta);
      for (int hh = 0; hh < Hkv; ++hh)
        orc_rope(k + (size_t)t * dkv + (size_t)hh * hd, hd, pos, m->rope_theta);
      memcpy(kl + (size_t)pos * dkv, k + (size_t)t * dkv, sizeof(double) * dkv);
      memcpy(vl + (size_t)pos * dkv, v + (size_t)t * dkv, sizeof(double) * dkv);
    }
#pragma omp parallel for collapse(2) schedule(static)
    for (int t = 0; t < T; ++t)
      for (int hh = 0; hh < H; ++hh) {
        int pos = start_pos + t;
        int kvh = hh / grp;
        orc_attend(q + (size_t)t * dq + (size_t)hh * hd, kl + (size_t)kvh * hd,
                   vl + (size_t)kvh * hd, pos + 1, hd, dkv,
                   a + (size_t)t * dq + (size_t)hh * hd);
      }
    linear(m, m->wo[l], d, dq, a, T, o);
    for (size_t i = 0; i < (size_t)T * d; ++i) x[i] += o[i];

    /* SwiGLU MLP sub-layer */
    load_row(m, m->mlp_norm[l], 0, d, gain);
    for (int t = 0; t < T; ++t)
      orc_rmsnorm(x + (size_t)t * d, gain, d, m->rms_eps, h + (size_t)t * d);
    linear(m, m->w_gate[l], F, d, h, T, g);
    linear(m, m->w_up[l], F, d, h, T, u);
    for (size_t i = 0; i < (size_t)T * F; ++i) g[i] = orc_silu(g[i]) * u[i];
    linear(m, m->w_down[l], d, F, g, T, o);
    for (size_t i = 0; i < (size_t)T * d; ++i) x[i] += o[i];
  }

  if (n_rows > 0) {
    double *hr = (double *)malloc(sizeof(double) * (size_t)n_rows * d);
    load_row(m, m->final_norm, 0, d, gain);
    for (int i = 0; i < n_rows; ++i)
      orc_rmsnorm(x + (size_t)logit_rows[i] * d, gain, d, m->rms_eps,
                  hr + (size_t)i * d);
    linear(m, m->lm_head, V, d, hr, n_rows, logits);
    free(hr);
  }

  free(x);
  free(h);
  free(q);
  free(k);
  free(v);
  free(a);
  free(o);
  free(g);
  free(u);
  free(gain);
  return 0;
}

int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void orc_set_num_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}
