/*
 * Oracle for incremental ViT encoding (temporal token reuse, Sec. III-B, Eq. 3-5).
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow CPU restatement of the method,
 * used to check the CUDA library.  Only the test suite, the smoke check and the
 * bench's CPU-baseline leg and reference arm (both time it on the host cores) load
 * it; the library never calls it and shares no code, header or constant with it.
 *
 * Storage is fp32; every dot product, layer-norm statistic and softmax sum is
 * accumulated in double.  The change score (Eq. 3) is computed in fp32, the
 * precision the GPU path takes that decision in.
 *
 * Weight buffer: bf16 bit patterns in the order
 *   W_pe[D][P*P*3] (column k = (ky*P+kx)*3+c), b_pe[D], pos[N][D],
 *   per layer: ln1_g[D] ln1_b[D] W_qkv[3D][D] b_qkv[3D] W_o[D][D] b_o[D]
 *              ln2_g[D] ln2_b[D] W_1[F][D] b_1[F] W_2[D][F] b_2[D],
 *   lnf_g[D], lnf_b[D].
 * Frames: uint8 [S*V][H][W][3].
 */
#ifndef IVIT_ORACLE_H
#define IVIT_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct orc_config {
  int32_t img_h, img_w, patch, dim, depth, heads, mlp_dim;
  int32_t n_streams, n_views;
  float ln_eps;
  int32_t gelu;        /* 0: tanh approximation, 1: erf */
  int32_t select_mode; /* 0: sim < threshold, 1: top-k lowest sims */
  float threshold;
  int32_t topk;
  int32_t ref_mode;    /* 0: reference = previous frame, 1: reference = last refresh */
  int32_t score_source; /* 0: patch embeddings (before the position embedding),
                           1: first-layer keys (Eq. 3) */
  int32_t schedule;     /* 0: every incremental call is incremental,
                           1: odd/even chunks (odd calls encode in full, Sec. III-B) */
  int32_t mlp_tokens;   /* 0: the blocks run on the updated tokens only (reused tokens keep
                           their cached outputs); 1: attention runs on the updated tokens,
                           reused tokens take their cached attention outputs, and every
                           token goes through the residual addition and the MLP of every
                           layer (Sec. III-B, the passage after Eq. 5) */
} orc_config;

typedef struct orc_state orc_state;

orc_state* orc_create(const orc_config* cfg, const uint16_t* weights_bf16);
void orc_destroy(orc_state* s);
void orc_set_threads(int n);

/* Full forward of every token of every view; seeds every cache (odd chunk, Sec. III-B).
 * tokens_out: float [S*V][N][D] or NULL. */
int orc_encode_full(orc_state* s, const uint8_t* frames, float* tokens_out);

/* Incremental step (even chunk, Sec. III-B).  counts_out [S*V], idx_out [S*V][N]
 * (ascending, first counts_out[v] entries valid, the rest -1), sims_out [S*V][N]
 * (Eq. 3 scores; a cold view has no reference and reports -2 for every token).
 * Any output pointer may be NULL. */
int orc_encode_incremental(orc_state* s, const uint8_t* frames, float* tokens_out,
                           int32_t* counts_out, int32_t* idx_out, float* sims_out);

/* Marks the views of camera stream `stream` (or all, if -1) cold: their next
 * incremental step recomputes every token. */
int orc_reset(orc_state* s, int stream);

/* Cache read-out for tests.  which: 0 = K, 1 = V (layer `layer`), 2 = final tokens,
 * 3 = reference score vectors (patch embeddings or first-layer keys, per
 * score_source), 4 = attention-block outputs W_o O + b_o of layer `layer` (mlp_tokens
 * = 1 only).  out: float [S*V][N][D]. */
int orc_get_cache(const orc_state* s, int which, int layer, float* out);

/* ---- building blocks (each a step of the method, exported for pinning) ---- */

/* Patch embedding of one view: e[i][d] = sum_k W_pe[d][k] (p_i[k] - 128) + b_pe[d]. */
void orc_patch_embed(const orc_config* cfg, const float* W_pe, const float* b_pe,
                     const uint8_t* frame, float* e);
/* Eq. 3: cos(a, b) = <a,b> / max(|a| |b|, 1e-12), in fp32. */
float orc_cosine(const float* a, const float* b, int n);
/* Selection: ascending index list of tokens with sims[i] < tau.  Returns the count. */
int orc_select_threshold(const float* sims, int n, float tau, int32_t* idx);
/* Selection: the k lowest sims, ties broken by lower token index, listed ascending. */
int orc_select_topk(const float* sims, int n, int k, int32_t* idx);
/* y = g (x - mean) / sqrt(var + eps) + b over n features (biased variance). */
void orc_layernorm(const float* x, const float* g, const float* b, int n, float eps,
                   float* y);
/* y[o] = sum_i W[o][i] x[i] + b[o]. */
void orc_linear(const float* x, const float* W, const float* b, int n_in, int n_out,
                float* y);
float orc_gelu(float x, int mode);
/* Eq. 3 key vectors of the first layer for n tokens: k[i] = W_K LN1(e[i] + pos[i]) + b_K,
 * as the paper defines them (no rounding of the LN output; fp32 storage, double
 * accumulation).  W_K [D][D]. */
void orc_layer0_keys(const float* e, const float* pos, const float* ln_g, const float* ln_b,
                     const float* W_K, const float* b_K, int n, int D, float eps, float* k);
/* One head: o[r] = softmax_j(<q[r], k[j]> / sqrt(dh)) v[j]; q [m][q_stride],
 * k, v [n][kv_stride], o [m][o_stride]; head width dh. */
void orc_attention(const float* q, int q_stride, const float* k, const float* v,
                   int kv_stride, int m, int n, int dh, float* o, int o_stride);

/* ---- the 2-step action combine (Sec. III-C, Eq. 9), for B samples of A action values ---- */

/* x_T[s][i] = x_0[s][i] + alpha[s] v_0[s][i] + beta[s] v_7[s][i] + b[s][i] (b may be NULL:
 * zero).  The anchor velocities v_0, v_7 and the coefficients come from the caller. */
void orc_action_combine(const float* x0, const float* v0, const float* v7, const float* alpha,
                        const float* beta, const float* b, int batch, int dim, float* xT);
/* Euler integration the combine approximates (the equation before Eq. 9):
 * x_T = x_0 + sum_t dt v_t over T steps; v [T][B][A]. */
void orc_euler(const float* x0, const float* v, int steps, float dt, int batch, int dim, float* xT);

#ifdef __cplusplus
}
#endif
#endif
