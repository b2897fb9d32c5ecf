/*
 * Oracle for incremental ViT encoding with temporal token reuse (Sec. III-B).
 *
 * TEST INFRASTRUCTURE ONLY: a plain, slow, step-by-step CPU restatement used to
 * check the CUDA library.  Nothing in the library's product path may call it.
 *
 * Each function follows one step of the method as the paper states it:
 *   - vision encoder: image -> patch tokens (Sec. III-A), pre-LN transformer blocks;
 *   - change score: cosine similarity against the reference (Eq. 3);
 *   - selection of the tokens to update, by threshold or top-k (Sec. III-B), made
 *     once, before the first layer, and reused by every layer (Fig. 2);
 *   - Q/K/V recomputed for the updated tokens only (Eq. 4);
 *   - the full K/V assembled by scattering the new rows into the cached ones (Eq. 5);
 *   - attention computed for the updated tokens only, which attend over all tokens;
 *     reused tokens keep their cached outputs (Sec. III-B).
 * Readings where the paper is silent are listed in the repository's design notes:
 * the score compares either the patch embeddings (before the position embedding) or
 * the first layer's keys (Eq. 3 as printed) with their reference; all updated tokens'
 * K/V of a layer are written before that layer's attention; the cached output is the
 * post-final-LN token; a cold view (no reference yet) updates every token.  Two readings
 * of what the reused tokens do after attention (mlp_tokens): either their residual
 * streams are never touched and they keep their cached outputs (0), or they take their
 * cached attention-block output, and every token goes through the residual addition,
 * the MLP of every layer and the final LN (1).
 *
 * Precision: fp32 storage, double accumulation of every dot product, LN statistic and
 * softmax sum; the Eq. 3 score in fp32.  OpenMP splits independent output elements
 * across threads; each element's arithmetic order is fixed, so results do not depend
 * on the thread count.
 */
#include "ivit_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
  const float *ln1_g, *ln1_b, *W_qkv, *b_qkv, *W_o, *b_o;
  const float *ln2_g, *ln2_b, *W_1, *b_1, *W_2, *b_2;
} orc_layer;

struct orc_state {
  orc_config cfg;
  int N, D, F, H, dh, L, SV, Kp;
  float* wbuf;
  const float *W_pe, *b_pe, *pos, *lnf_g, *lnf_b;
  orc_layer* layer;
  float* e_ref;   /* [SV][N][D] reference score vectors */
  float* e_t;     /* [SV][N][D] scratch: this frame's patch embeddings */
  float* s_t;     /* [SV][N][D] scratch: this frame's score vectors (first-layer keys) */
  long long chunk; /* incremental calls made (odd/even schedule) */
  float* cacheK;  /* [L][SV][N][D] */
  float* cacheV;  /* [L][SV][N][D] */
  float* tok_out; /* [SV][N][D] final tokens (post final LN) */
  float* cacheA;  /* [L][SV][N][D] attention-block outputs W_o O + b_o (mlp_tokens = 1) */
  uint8_t* cold;  /* [SV] */
};

static float bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

void orc_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* ------------------------------------------------------------- building blocks */

void orc_patch_embed(const orc_config* cfg, const float* W_pe, const float* b_pe,
                     const uint8_t* frame, float* e) {
  const int P = cfg->patch, D = cfg->dim, W = cfg->img_w;
  const int gw = cfg->img_w / P, N = (cfg->img_h / P) * gw, Kp = P * P * 3;
#pragma omp parallel for collapse(2) schedule(static)
  for (int i = 0; i < N; ++i) {
    for (int d = 0; d < D; ++d) {
      const int py = i / gw, px = i % gw;
      double acc = 0.0;
      for (int ky = 0; ky < P; ++ky)
        for (int kx = 0; kx < P; ++kx)
          for (int c = 0; c < 3; ++c) {
            const int k = (ky * P + kx) * 3 + c;
            const int pix = frame[((size_t)(py * P + ky) * W + (px * P + kx)) * 3 + c];
            acc += (double)W_pe[(size_t)d * Kp + k] * (double)(pix - 128);
          }
      e[(size_t)i * D + d] = (float)(acc + (double)b_pe[d]);
    }
  }
}

float orc_cosine(const float* a, const float* b, int n) {
  float dot = 0.f, na = 0.f, nb = 0.f;
  for (int i = 0; i < n; ++i) {
    dot += a[i] * b[i];
    na += a[i] * a[i];
    nb += b[i] * b[i];
  }
  return dot / fmaxf(sqrtf(na) * sqrtf(nb), 1e-12f);
}

int orc_select_threshold(const float* sims, int n, float tau, int32_t* idx) {
  int m = 0;
  for (int i = 0; i < n; ++i)
    if (sims[i] < tau) idx[m++] = i;
  return m;
}

int orc_select_topk(const float* sims, int n, int k, int32_t* idx) {
  if (k < 0) k = 0;
  if (k > n) k = n;
  int m = 0;
  for (int i = 0; i < n; ++i) {
    /* rank of token i in the order (sim ascending, index ascending) */
    int rank = 0;
    for (int j = 0; j < n; ++j)
      if (sims[j] < sims[i] || (sims[j] == sims[i] && j < i)) ++rank;
    if (rank < k) idx[m++] = i;
  }
  return m;
}

void orc_layernorm(const float* x, const float* g, const float* b, int n, float eps,
                   float* y) {
  double mean = 0.0, var = 0.0;
  for (int i = 0; i < n; ++i) mean += x[i];
  mean /= n;
  for (int i = 0; i < n; ++i) var += ((double)x[i] - mean) * ((double)x[i] - mean);
  var /= n;
  const double rstd = 1.0 / sqrt(var + (double)eps);
  for (int i = 0; i < n; ++i)
    y[i] = (float)((double)g[i] * (((double)x[i] - mean) * rstd) + (double)b[i]);
}

void orc_linear(const float* x, const float* W, const float* b, int n_in, int n_out,
                float* y) {
  for (int o = 0; o < n_out; ++o) {
    double acc = 0.0;
    for (int i = 0; i < n_in; ++i) acc += (double)W[(size_t)o * n_in + i] * (double)x[i];
    y[o] = (float)(acc + (double)b[o]);
  }
}

float orc_gelu(float x, int mode) {
  const double xd = x;
  if (mode == 1) return (float)(0.5 * xd * (1.0 + erf(xd / sqrt(2.0))));
  const double c = sqrt(2.0 / M_PI);
  return (float)(0.5 * xd * (1.0 + tanh(c * (xd + 0.044715 * xd * xd * xd))));
}

void orc_layer0_keys(const float* e, const float* pos, const float* ln_g, const float* ln_b,
                     const float* W_K, const float* b_K, int n, int D, float eps, float* k) {
#pragma omp parallel for schedule(static)
  for (int i = 0; i < n; ++i) {
    float* x = (float*)malloc(sizeof(float) * (size_t)D);
    float* xn = (float*)malloc(sizeof(float) * (size_t)D);
    for (int d = 0; d < D; ++d) x[d] = e[(size_t)i * D + d] + pos[(size_t)i * D + d];
    orc_layernorm(x, ln_g, ln_b, D, eps, xn);
    orc_linear(xn, W_K, b_K, D, D, k + (size_t)i * D);
    free(x);
    free(xn);
  }
}

static void attention_row(const float* q, const float* k, const float* v, int kv_stride,
                          int n, int dh, double* s, float* o) {
  const double scale = 1.0 / sqrt((double)dh);
  double mx = -INFINITY;
  for (int j = 0; j < n; ++j) {
    double acc = 0.0;
    for (int d = 0; d < dh; ++d) acc += (double)q[d] * (double)k[(size_t)j * kv_stride + d];
    s[j] = acc * scale;
    if (s[j] > mx) mx = s[j];
  }
  double z = 0.0;
  for (int j = 0; j < n; ++j) {
    s[j] = exp(s[j] - mx);
    z += s[j];
  }
  for (int d = 0; d < dh; ++d) {
    double acc = 0.0;
    for (int j = 0; j < n; ++j) acc += s[j] * (double)v[(size_t)j * kv_stride + d];
    o[d] = (float)(acc / z);
  }
}

void orc_attention(const float* q, int q_stride, const float* k, const float* v,
                   int kv_stride, int m, int n, int dh, float* o, int o_stride) {
  double* s = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  for (int r = 0; r < m; ++r)
    attention_row(q + (size_t)r * q_stride, k, v, kv_stride, n, dh, s,
                  o + (size_t)r * o_stride);
  free(s);
}

/* ------------------------------------------------------------------ the encoder */

/* Rows-wise linear: Y[r][o] (+)= X[r] . W[o] + b[o] for r < m. */
static void linear_rows(const float* X, const float* W, const float* b, int m, int n_in,
                        int n_out, float* Y, int accumulate) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int r = 0; r < m; ++r)
    for (int o = 0; o < n_out; ++o) {
      const float* x = X + (size_t)r * n_in;
      double acc = 0.0;
      for (int i = 0; i < n_in; ++i) acc += (double)W[(size_t)o * n_in + i] * (double)x[i];
      const float y = (float)(acc + (double)b[o]);
      if (accumulate)
        Y[(size_t)r * n_out + o] += y;
      else
        Y[(size_t)r * n_out + o] = y;
    }
}

/* Runs every transformer block on the updated tokens U (ascending, m entries) of view
 * v, reading the reused tokens' K/V from the cache, and writes their final tokens. */
static void encode_rows(orc_state* s, int v, const int32_t* U, int m) {
  if (m == 0) return;
  const int N = s->N, D = s->D, F = s->F, H = s->H, dh = s->dh, SV = s->SV;
  const float eps = s->cfg.ln_eps;
  const float* e_t = s->e_t + (size_t)v * N * D;
  float* x = (float*)malloc(sizeof(float) * (size_t)m * D);
  float* xn = (float*)malloc(sizeof(float) * (size_t)m * D);
  float* qkv = (float*)malloc(sizeof(float) * (size_t)m * 3 * D);
  float* att = (float*)malloc(sizeof(float) * (size_t)m * D);
  float* hid = (float*)malloc(sizeof(float) * (size_t)m * F);

  /* tokens entering the first block: patch embedding + position embedding */
  for (int r = 0; r < m; ++r)
    for (int d = 0; d < D; ++d)
      x[(size_t)r * D + d] = e_t[(size_t)U[r] * D + d] + s->pos[(size_t)U[r] * D + d];

  for (int l = 0; l < s->L; ++l) {
    const orc_layer* w = &s->layer[l];
    float* Kl = s->cacheK + ((size_t)l * SV + v) * N * D;
    float* Vl = s->cacheV + ((size_t)l * SV + v) * N * D;

    /* Eq. 4: Q, K, V of the updated tokens, from the pre-attention LN */
#pragma omp parallel for schedule(static)
    for (int r = 0; r < m; ++r)
      orc_layernorm(x + (size_t)r * D, w->ln1_g, w->ln1_b, D, eps, xn + (size_t)r * D);
    linear_rows(xn, w->W_qkv, w->b_qkv, m, D, 3 * D, qkv, 0);

    /* Eq. 5: scatter the new K/V rows into the cached K/V of the view */
    for (int r = 0; r < m; ++r) {
      memcpy(Kl + (size_t)U[r] * D, qkv + (size_t)r * 3 * D + D, sizeof(float) * D);
      memcpy(Vl + (size_t)U[r] * D, qkv + (size_t)r * 3 * D + 2 * D, sizeof(float) * D);
    }

    /* attention only for the updated tokens, over all N tokens of the view */
#pragma omp parallel for collapse(2) schedule(static)
    for (int r = 0; r < m; ++r)
      for (int h = 0; h < H; ++h) {
        double* sc = (double*)malloc(sizeof(double) * (size_t)N);
        attention_row(qkv + (size_t)r * 3 * D + (size_t)h * dh, Kl + (size_t)h * dh,
                      Vl + (size_t)h * dh, D, N, dh, sc, att + (size_t)r * D + (size_t)h * dh);
        free(sc);
      }

    /* output projection + residual */
    linear_rows(att, w->W_o, w->b_o, m, D, D, x, 1);

    /* MLP on the updated tokens: x += W_2 GELU(W_1 LN2(x) + b_1) + b_2 */
#pragma omp parallel for schedule(static)
    for (int r = 0; r < m; ++r)
      orc_layernorm(x + (size_t)r * D, w->ln2_g, w->ln2_b, D, eps, xn + (size_t)r * D);
    linear_rows(xn, w->W_1, w->b_1, m, D, F, hid, 0);
#pragma omp parallel for schedule(static)
    for (size_t t = 0; t < (size_t)m * F; ++t) hid[t] = orc_gelu(hid[t], s->cfg.gelu);
    linear_rows(hid, w->W_2, w->b_2, m, F, D, x, 1);
  }

  /* final LN; the result becomes the cached output of each updated token */
  for (int r = 0; r < m; ++r)
    orc_layernorm(x + (size_t)r * D, s->lnf_g, s->lnf_b, D, eps,
                  s->tok_out + ((size_t)v * N + U[r]) * D);

  free(x);
  free(xn);
  free(qkv);
  free(att);
  free(hid);
}

/* mlp_tokens = 1: runs every block on view v with attention for the updated tokens U
 * (ascending, m entries) only.  Reused tokens' keys and values come from the cache
 * (Eq. 5) and so do their attention-block outputs; after the residual addition every
 * token of the view goes through LN2 and the MLP, and every token's final LN output
 * is written. */
static void encode_rows_all(orc_state* s, int v, const int32_t* U, int m) {
  const int N = s->N, D = s->D, F = s->F, H = s->H, dh = s->dh, SV = s->SV;
  const float eps = s->cfg.ln_eps;
  const float* e_t = s->e_t + (size_t)v * N * D;
  const int mq = m > 0 ? m : 1;
  float* x = (float*)malloc(sizeof(float) * (size_t)N * D);      /* every token */
  float* xn = (float*)malloc(sizeof(float) * (size_t)N * D);
  float* qkv = (float*)malloc(sizeof(float) * (size_t)mq * 3 * D); /* updated tokens */
  float* att = (float*)malloc(sizeof(float) * (size_t)mq * D);
  float* a = (float*)malloc(sizeof(float) * (size_t)mq * D);
  float* hid = (float*)malloc(sizeof(float) * (size_t)N * F);

  /* every token enters the first block: patch embedding + position embedding */
  for (size_t t = 0; t < (size_t)N * D; ++t) x[t] = e_t[t] + s->pos[t];

  for (int l = 0; l < s->L; ++l) {
    const orc_layer* w = &s->layer[l];
    float* Kl = s->cacheK + ((size_t)l * SV + v) * N * D;
    float* Vl = s->cacheV + ((size_t)l * SV + v) * N * D;
    float* Al = s->cacheA + ((size_t)l * SV + v) * N * D;

    if (m > 0) {
      /* Eq. 4 for the updated tokens */
#pragma omp parallel for schedule(static)
      for (int r = 0; r < m; ++r)
        orc_layernorm(x + (size_t)U[r] * D, w->ln1_g, w->ln1_b, D, eps, xn + (size_t)r * D);
      linear_rows(xn, w->W_qkv, w->b_qkv, m, D, 3 * D, qkv, 0);
      /* Eq. 5 */
      for (int r = 0; r < m; ++r) {
        memcpy(Kl + (size_t)U[r] * D, qkv + (size_t)r * 3 * D + D, sizeof(float) * D);
        memcpy(Vl + (size_t)U[r] * D, qkv + (size_t)r * 3 * D + 2 * D, sizeof(float) * D);
      }
      /* attention for the updated tokens over all N tokens */
#pragma omp parallel for collapse(2) schedule(static)
      for (int r = 0; r < m; ++r)
        for (int h = 0; h < H; ++h) {
          double* sc = (double*)malloc(sizeof(double) * (size_t)N);
          attention_row(qkv + (size_t)r * 3 * D + (size_t)h * dh, Kl + (size_t)h * dh,
                        Vl + (size_t)h * dh, D, N, dh, sc, att + (size_t)r * D + (size_t)h * dh);
          free(sc);
        }
      /* their attention-block outputs replace the cached ones */
      linear_rows(att, w->W_o, w->b_o, m, D, D, a, 0);
      for (int r = 0; r < m; ++r) memcpy(Al + (size_t)U[r] * D, a + (size_t)r * D, sizeof(float) * D);
    }

    /* residual addition for every token (reused tokens: the cached output) */
    for (size_t t = 0; t < (size_t)N * D; ++t) x[t] += Al[t];

    /* MLP for every token */
#pragma omp parallel for schedule(static)
    for (int i = 0; i < N; ++i)
      orc_layernorm(x + (size_t)i * D, w->ln2_g, w->ln2_b, D, eps, xn + (size_t)i * D);
    linear_rows(xn, w->W_1, w->b_1, N, D, F, hid, 0);
#pragma omp parallel for schedule(static)
    for (size_t t = 0; t < (size_t)N * F; ++t) hid[t] = orc_gelu(hid[t], s->cfg.gelu);
    linear_rows(hid, w->W_2, w->b_2, N, F, D, x, 1);
  }

  for (int i = 0; i < N; ++i)
    orc_layernorm(x + (size_t)i * D, s->lnf_g, s->lnf_b, D, eps, s->tok_out + ((size_t)v * N + i) * D);

  free(x);
  free(xn);
  free(qkv);
  free(att);
  free(a);
  free(hid);
}

static void encode_view(orc_state* s, int v, const int32_t* U, int m) {
  if (s->cfg.mlp_tokens == 1)
    encode_rows_all(s, v, U, m);
  else
    encode_rows(s, v, U, m);
}

orc_state* orc_create(const orc_config* cfg, const uint16_t* wb) {
  if (!cfg || !wb) return NULL;
  if (cfg->patch <= 0 || cfg->img_h % cfg->patch || cfg->img_w % cfg->patch) return NULL;
  if (cfg->dim <= 0 || cfg->heads <= 0 || cfg->dim % cfg->heads || cfg->depth <= 0 ||
      cfg->mlp_dim <= 0 || cfg->n_streams <= 0 || cfg->n_views <= 0)
    return NULL;
  if (cfg->mlp_tokens != 0 && cfg->mlp_tokens != 1) return NULL;
  orc_state* s = (orc_state*)calloc(1, sizeof(orc_state));
  s->cfg = *cfg;
  s->N = (cfg->img_h / cfg->patch) * (cfg->img_w / cfg->patch);
  s->D = cfg->dim;
  s->F = cfg->mlp_dim;
  s->H = cfg->heads;
  s->dh = cfg->dim / cfg->heads;
  s->L = cfg->depth;
  s->SV = cfg->n_streams * cfg->n_views;
  s->Kp = cfg->patch * cfg->patch * 3;
  const size_t D = s->D, F = s->F, N = s->N;
  const size_t per_layer = 2 * D + 3 * D * D + 3 * D + D * D + D + 2 * D + F * D + F + D * F + D;
  const size_t total = D * s->Kp + D + N * D + per_layer * s->L + 2 * D;
  s->wbuf = (float*)malloc(sizeof(float) * total);
  for (size_t i = 0; i < total; ++i) s->wbuf[i] = bf16_to_f32(wb[i]);
  const float* p = s->wbuf;
  s->W_pe = p; p += D * s->Kp;
  s->b_pe = p; p += D;
  s->pos = p; p += N * D;
  s->layer = (orc_layer*)calloc((size_t)s->L, sizeof(orc_layer));
  for (int l = 0; l < s->L; ++l) {
    orc_layer* w = &s->layer[l];
    w->ln1_g = p; p += D;
    w->ln1_b = p; p += D;
    w->W_qkv = p; p += 3 * D * D;
    w->b_qkv = p; p += 3 * D;
    w->W_o = p; p += D * D;
    w->b_o = p; p += D;
    w->ln2_g = p; p += D;
    w->ln2_b = p; p += D;
    w->W_1 = p; p += F * D;
    w->b_1 = p; p += F;
    w->W_2 = p; p += D * F;
    w->b_2 = p; p += D;
  }
  s->lnf_g = p; p += D;
  s->lnf_b = p; p += D;
  const size_t view = (size_t)s->SV * N * D;
  s->e_ref = (float*)calloc(view, sizeof(float));
  s->e_t = (float*)calloc(view, sizeof(float));
  s->s_t = (float*)calloc(view, sizeof(float));
  s->tok_out = (float*)calloc(view, sizeof(float));
  s->cacheK = (float*)calloc(view * s->L, sizeof(float));
  s->cacheV = (float*)calloc(view * s->L, sizeof(float));
  s->cacheA = cfg->mlp_tokens == 1 ? (float*)calloc(view * s->L, sizeof(float)) : NULL;
  s->cold = (uint8_t*)malloc((size_t)s->SV);
  if (!s->e_ref || !s->e_t || !s->s_t || !s->tok_out || !s->cacheK || !s->cacheV || !s->cold ||
      (cfg->mlp_tokens == 1 && !s->cacheA)) {
    orc_destroy(s);
    return NULL;
  }
  memset(s->cold, 1, (size_t)s->SV);
  return s;
}

void orc_destroy(orc_state* s) {
  if (!s) return;
  free(s->wbuf);
  free(s->layer);
  free(s->e_ref);
  free(s->e_t);
  free(s->s_t);
  free(s->tok_out);
  free(s->cacheK);
  free(s->cacheV);
  free(s->cacheA);
  free(s->cold);
  free(s);
}

/* Patch embeddings of every view, and the score vectors Eq. 3 compares: the
 * embeddings themselves, or the first layer's keys of every token. */
static void embed_all(orc_state* s, const uint8_t* frames) {
  const size_t frame_bytes = (size_t)s->cfg.img_h * s->cfg.img_w * 3;
  const size_t D = s->D;
  for (int v = 0; v < s->SV; ++v) {
    float* e = s->e_t + (size_t)v * s->N * D;
    orc_patch_embed(&s->cfg, s->W_pe, s->b_pe, frames + (size_t)v * frame_bytes, e);
    if (s->cfg.score_source == 1)
      orc_layer0_keys(e, s->pos, s->layer[0].ln1_g, s->layer[0].ln1_b, s->layer[0].W_qkv + D * D,
                      s->layer[0].b_qkv + D, s->N, s->D, s->cfg.ln_eps, s->s_t + (size_t)v * s->N * D);
  }
}

static const float* score_vectors(const orc_state* s) {
  return s->cfg.score_source == 1 ? s->s_t : s->e_t;
}

static void copy_out(const orc_state* s, float* tokens_out) {
  if (tokens_out)
    memcpy(tokens_out, s->tok_out, sizeof(float) * (size_t)s->SV * s->N * s->D);
}

int orc_encode_full(orc_state* s, const uint8_t* frames, float* tokens_out) {
  if (!s || !frames) return -1;
  const int N = s->N, D = s->D;
  embed_all(s, frames);
  int32_t* U = (int32_t*)malloc(sizeof(int32_t) * (size_t)N);
  for (int i = 0; i < N; ++i) U[i] = i;
  for (int v = 0; v < s->SV; ++v) {
    memcpy(s->e_ref + (size_t)v * N * D, score_vectors(s) + (size_t)v * N * D,
           sizeof(float) * (size_t)N * D);
    encode_view(s, v, U, N);
    s->cold[v] = 0;
  }
  free(U);
  copy_out(s, tokens_out);
  return 0;
}

int orc_encode_incremental(orc_state* s, const uint8_t* frames, float* tokens_out,
                           int32_t* counts_out, int32_t* idx_out, float* sims_out) {
  if (!s || !frames) return -1;
  const int N = s->N, D = s->D;
  /* odd/even schedule: odd chunks (1st, 3rd, ... call) encode every token in full */
  if (s->cfg.schedule == 1 && (s->chunk++ % 2) == 0) {
    orc_encode_full(s, frames, tokens_out);
    for (int v = 0; v < s->SV; ++v) {
      if (counts_out) counts_out[v] = N;
      if (idx_out)
        for (int i = 0; i < N; ++i) idx_out[(size_t)v * N + i] = i;
      if (sims_out)
        for (int i = 0; i < N; ++i) sims_out[(size_t)v * N + i] = -2.f;
    }
    return 0;
  }
  embed_all(s, frames);
  int32_t* U = (int32_t*)malloc(sizeof(int32_t) * (size_t)N);
  float* sims = (float*)malloc(sizeof(float) * (size_t)N);
  for (int v = 0; v < s->SV; ++v) {
    const float* et = score_vectors(s) + (size_t)v * N * D;
    float* er = s->e_ref + (size_t)v * N * D;
    int m;
    if (s->cold[v]) {
      for (int i = 0; i < N; ++i) {
        U[i] = i;
        sims[i] = -2.f;
      }
      m = N;
    } else {
      /* Eq. 3 against the reference embedding of each token */
      for (int i = 0; i < N; ++i) sims[i] = orc_cosine(et + (size_t)i * D, er + (size_t)i * D, D);
      m = s->cfg.select_mode == 1 ? orc_select_topk(sims, N, s->cfg.topk, U)
                                  : orc_select_threshold(sims, N, s->cfg.threshold, U);
    }
    /* reference update */
    if (s->cold[v] || s->cfg.ref_mode == 0) {
      memcpy(er, et, sizeof(float) * (size_t)N * D);
    } else {
      for (int r = 0; r < m; ++r)
        memcpy(er + (size_t)U[r] * D, et + (size_t)U[r] * D, sizeof(float) * D);
    }
    encode_view(s, v, U, m);
    s->cold[v] = 0;
    if (counts_out) counts_out[v] = m;
    if (idx_out)
      for (int i = 0; i < N; ++i) idx_out[(size_t)v * N + i] = i < m ? U[i] : -1;
    if (sims_out) memcpy(sims_out + (size_t)v * N, sims, sizeof(float) * (size_t)N);
  }
  free(U);
  free(sims);
  copy_out(s, tokens_out);
  return 0;
}

int orc_reset(orc_state* s, int stream) {
  if (!s) return -1;
  if (stream < -1 || stream >= s->cfg.n_streams) return -1;
  for (int v = 0; v < s->SV; ++v)
    if (stream == -1 || v / s->cfg.n_views == stream) s->cold[v] = 1;
  return 0;
}

int orc_get_cache(const orc_state* s, int which, int layer, float* out) {
  if (!s || !out) return -1;
  const size_t view = (size_t)s->SV * s->N * s->D;
  const float* src;
  if (which == 0 || which == 1) {
    if (layer < 0 || layer >= s->L) return -1;
    src = (which == 0 ? s->cacheK : s->cacheV) + (size_t)layer * view;
  } else if (which == 2) {
    src = s->tok_out;
  } else if (which == 3) {
    src = s->e_ref;
  } else if (which == 4 && s->cacheA) {
    if (layer < 0 || layer >= s->L) return -1;
    src = s->cacheA + (size_t)layer * view;
  } else {
    return -1;
  }
  memcpy(out, src, sizeof(float) * view);
  return 0;
}

/* Eq. 9: the final action state from the two anchor velocities. */
void orc_action_combine(const float* x0, const float* v0, const float* v7, const float* alpha,
                        const float* beta, const float* b, int batch, int dim, float* xT) {
  for (int s = 0; s < batch; ++s)
    for (int i = 0; i < dim; ++i) {
      const size_t k = (size_t)s * dim + i;
      const double y = (double)x0[k] + (double)alpha[s] * v0[k] + (double)beta[s] * v7[k] +
                       (b ? (double)b[k] : 0.0);
      xT[k] = (float)y;
    }
}

/* Euler integration of the velocity sequence (the sum Eq. 9 compresses). */
void orc_euler(const float* x0, const float* v, int steps, float dt, int batch, int dim, float* xT) {
  const size_t n = (size_t)batch * dim;
  for (size_t k = 0; k < n; ++k) {
    double y = x0[k];
    for (int t = 0; t < steps; ++t) y += (double)dt * v[(size_t)t * n + k];
    xT[k] = (float)y;
  }
}
