/*
 * ivit -- incremental ViT encoding of streaming camera frames on one GB300 (sm_103a).
 *
 * The library implements temporal token reuse (Sec. III-B of "Reducing Temporal
 * Redundancy for Efficient Vision-Language-Action Inference"): a frame is encoded
 * in full once (the paper's "odd chunk"); every later frame re-encodes only the
 * tokens whose patch embedding changed (Eq. 3 score, threshold or top-k selection),
 * with their queries attending over all tokens and the other tokens' per-layer K/V
 * read from a resident cache (Eq. 4-5); reused tokens keep their cached outputs.
 *
 * Conventions for every entry point:
 *  - Return value: IVIT_OK (0) or a negative IVIT_ERR_* code.  Nothing throws or
 *    aborts across the ABI; ivit_last_error() describes the last failure.
 *  - Device pointers ("_dev") are caller-owned CUDA global memory on the device the
 *    handle was created on; host pointers ("_host") are caller-owned host memory.
 *    The library never frees caller memory.  All work is enqueued on the caller's
 *    cudaStream_t (passed as void*, NULL = legacy default stream) and is
 *    asynchronous: outputs are valid once that stream has reached the call.
 *  - A handle owns the weights (copied at create), every per-view cache and all
 *    workspaces.  One handle may be used from one host thread at a time; calls on
 *    one handle must be ordered on one stream (or explicitly synchronised).
 *  - Shapes: S = n_streams camera streams, V = n_views views each, SV = S*V
 *    independent views (each with its own caches), N = (img_h/patch)*(img_w/patch)
 *    tokens per view, D = dim, L = depth, F = mlp_dim.
 */
#ifndef IVIT_H
#define IVIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define IVIT_OK 0
#define IVIT_ERR_ARG (-1)      /* null handle/pointer, bad enum, out-of-range index */
#define IVIT_ERR_SHAPE (-2)    /* configuration the kernels do not support */
#define IVIT_ERR_OOM (-3)      /* device allocation failed */
#define IVIT_ERR_CUDA (-4)     /* a CUDA runtime/driver call failed */
#define IVIT_ERR_DEVICE (-5)   /* a kernel reported an error (bounded wait expired) */

#define IVIT_GELU_TANH 0       /* 0.5x(1+tanh(sqrt(2/pi)(x+0.044715x^3))) (SigLIP) */
#define IVIT_GELU_ERF 1        /* 0.5x(1+erf(x/sqrt 2)) (ViT) */
#define IVIT_SEL_THRESHOLD 0   /* update token i iff sim(i) < threshold (strict) */
#define IVIT_SEL_TOPK 1        /* update the topk lowest sims, ties by lower index */
#define IVIT_REF_PREV_FRAME 0  /* reference = previous frame's embeddings (all tokens) */
#define IVIT_REF_LAST_REFRESH 1 /* reference of token i updated only when i is updated */
#define IVIT_SCORE_EMBED 0     /* Eq. 3 on patch embeddings (before position embedding) */
#define IVIT_SCORE_KEY0 1      /* Eq. 3 as printed: first-layer keys W_K LN1(e+pos) + b_K */
#define IVIT_SCHED_INCREMENTAL 0 /* every ivit_encode_incremental call is incremental */
#define IVIT_SCHED_ODD_EVEN 1  /* odd calls encode in full, even calls incrementally */
#define IVIT_MLP_UPDATED 0     /* every block runs on the updated tokens only */
#define IVIT_MLP_ALL 1         /* attention on the updated tokens, residual + MLP on all */

/* Encoder + selection configuration.
 * Supported by the kernels: patch >= 1 dividing img_h and img_w; N <= 1024;
 * dim % 64 == 0, dim <= 2048, heads dividing dim with head_dim = dim/heads a multiple of 8,
 * at most 128; mlp_dim % 8 == 0; SV <= 4096. */
typedef struct ivit_config {
  int32_t img_h, img_w;  /* frame size in pixels */
  int32_t patch;         /* patch edge P; patch k-vector is P*P*3 (HWC order) */
  int32_t dim;           /* D */
  int32_t depth;         /* L transformer blocks (pre-LN) */
  int32_t heads;         /* H */
  int32_t mlp_dim;       /* F */
  int32_t n_streams;     /* S */
  int32_t n_views;       /* V */
  float ln_eps;          /* layer-norm epsilon (1e-6) */
  int32_t gelu;          /* IVIT_GELU_* */
  int32_t select_mode;   /* IVIT_SEL_* */
  float threshold;       /* IVIT_SEL_THRESHOLD: refresh where sim < threshold */
  int32_t topk;          /* IVIT_SEL_TOPK: tokens refreshed per view, clamped to [0, N] */
  int32_t ref_mode;      /* IVIT_REF_* */
  int32_t score_source;  /* IVIT_SCORE_*: what Eq. 3's cosine compares (Sec. III-B) */
  int32_t schedule;      /* IVIT_SCHED_*: odd/even chunking of Sec. III-B, or none */
  int32_t mlp_tokens;    /* IVIT_MLP_*: which tokens go through the residual addition and
                            the MLP after attention (Sec. III-B, the passage after Eq. 5).
                            IVIT_MLP_ALL keeps every token's attention-block output
                            W_o O + b_o per layer (fp32 [L][SV][N][D]); reused tokens take
                            theirs from that cache, every token runs LN2 + MLP and the
                            final LN, and every output token is recomputed. */
} ivit_config;

typedef struct ivit_handle ivit_handle;

/* Number of bf16 elements of the weight buffer for `cfg`, 0 if cfg is invalid.
 * Layout (row-major tensors, back to back):
 *   W_pe[D][P*P*3] (column k = (ky*P+kx)*3+c, applied to pixel-128), b_pe[D], pos[N][D],
 *   per layer: ln1_g[D] ln1_b[D] W_qkv[3D][D] b_qkv[3D] W_o[D][D] b_o[D]
 *              ln2_g[D] ln2_b[D] W_1[F][D] b_1[F] W_2[D][F] b_2[D],
 *   lnf_g[D] lnf_b[D].
 * W_qkv rows: query block, key block, value block; head h owns rows h*dh..h*dh+dh-1
 * of each block (Eq. 4: Q = W_Q T, K = W_K T, V = W_V T). */
size_t ivit_weights_size(const ivit_config* cfg);

/* Creates a handle on the current CUDA device: validates cfg, copies the weights
 * (bf16 bit patterns, host memory, ivit_weights_size(cfg) elements) to the device,
 * allocates every cache and workspace, and marks every view cold.
 * On failure *out is NULL and the code says why. */
int ivit_create(const ivit_config* cfg, const uint16_t* weights_bf16_host,
                ivit_handle** out);

/* Full encode of one frame per view (the paper's full forward that seeds the
 * reference, Sec. III-B).  frames_dev: uint8 [SV][img_h][img_w][3], any byte address
 * (an odd address makes the patchify kernel use byte loads).
 * tokens_out_dev: bf16 [SV][N][D] final tokens (after the final LN), or NULL.
 * Re-seeds every cache and reference and marks every view warm. */
int ivit_encode_full(ivit_handle* h, const uint8_t* frames_dev, uint16_t* tokens_out_dev,
                     void* stream);

/* Incremental encode (Sec. III-B, Eq. 3-5): scores every token's patch embedding, or
 * its first-layer key (score_source), against its reference (cosine, fp32), selects
 * the tokens to update per view, runs
 * every block on those tokens only (their queries attend over all N tokens of the
 * view, the others' K/V come from the cache), and returns all tokens: updated ones
 * recomputed, the rest from the final-token cache.  A cold view updates every token.
 * tokens_out_dev: bf16 [SV][N][D] or NULL.  changed_count_dev: int32 [SV] number of
 * updated tokens per view, or NULL.  No host synchronisation happens inside.  With
 * schedule = IVIT_SCHED_ODD_EVEN the 1st, 3rd, ... call encodes in full (count N).
 * With mlp_tokens = IVIT_MLP_ALL the blocks after attention run on every token (see
 * ivit_config). */
int ivit_encode_incremental(ivit_handle* h, const uint8_t* frames_dev,
                            uint16_t* tokens_out_dev, int32_t* changed_count_dev,
                            void* stream);

/* Copies the ascending updated-token list of view `sv` from the last encode call:
 * idx_dev int32 [N] (first *count entries valid), count_dev int32 [1] (either may be
 * NULL).  Enqueued on `stream`.  IVIT_ERR_ARG if sv is outside [0, SV). */
int ivit_get_changed(ivit_handle* h, int sv, int32_t* idx_dev, int32_t* count_dev,
                     void* stream);

/* Copies per-view state for inspection: which = 0 key cache of `layer`, 1 value cache
 * of `layer`, 2 final-token cache (all bf16 [SV][N][D]), 3 reference score vectors
 * (patch embeddings or first-layer keys, fp32 [SV][N][D]), 4 attention-block outputs of
 * `layer` (fp32 [SV][N][D], mlp_tokens = IVIT_MLP_ALL only).  dst_dev must hold that
 * many bytes.  IVIT_ERR_ARG for a NULL destination, an unknown `which` (4 without that
 * reading) or, for 0, 1 and 4, a layer outside [0, L). */
int ivit_get_cache(ivit_handle* h, int which, int layer, void* dst_dev, void* stream);

/* Marks the views of camera stream `stream_index` (all streams if -1) cold: the next
 * incremental call recomputes every token of those views.  Host-side only.
 * IVIT_ERR_ARG if stream_index is outside [-1, n_streams). */
int ivit_reset(ivit_handle* h, int stream_index);

/* Kernel timeline.  With enable != 0 every later call records, for each of its kernel
 * launches, the global time at which each CTA started its work (after the wait on the
 * previous kernel) and finished; the captured CUDA graphs are rebuilt with the
 * recording in them, so the calls still run as replayed graphs (enable = 0 rebuilds
 * them without it).  Allocates 8 MB of device memory on first use.
 * ivit_timeline_read synchronises `stream` and reads the last call: per kernel family
 * (index 0 tensor-core GEMMs, 1 attention, 2 layer norms, 3 patchify / score /
 * selection / gather) the sum over its launches of (last CTA end - first CTA start)
 * in ms and the number of launches (arrays of 4, either may be NULL), the algorithmic
 * bytes of the GEMM launches (weights + input rows + outputs + bias, with this call's
 * updated-row count), and the span from the first start to the last end in ms.  Only
 * the first 1024 CTAs of a launch record.  IVIT_ERR_ARG when timeline mode is off. */
int ivit_timeline(ivit_handle* h, int enable);
int ivit_timeline_read(ivit_handle* h, void* stream, double* family_ms, int64_t* family_launches,
                       double* gemm_bytes_total, double* span_ms);

/* Reads and clears the device error word (0 = none; nonzero = a kernel's bounded
 * wait expired, the kernel skipped its work and returned).  Synchronises `stream`. */
int ivit_device_status(ivit_handle* h, void* stream);

/* Execution paths (chosen at create; the environment variable IVIT_PATH=kernels,
 * IVIT_PATH=persistent or IVIT_PATH=stream selects one): one kernel per operation,
 * chained with programmatic dependent launch and replayed as a CUDA graph (every
 * incremental call, and the full encodes for dim > 384); every transformer block of a
 * call in one persistent cooperative kernel with grid barriers (the full encodes for
 * dim <= 384, where per-operation launches dominate); or, on request only
 * (IVIT_PATH=stream), the incremental calls without cold views in one cooperative
 * weight-streaming kernel that keeps each SM's share of the next weights in flight
 * through a shared-memory ring.  All give the same result within the bf16 rounding. */

/* Number of the library's kernel launches made by the last encode call. */
int64_t ivit_last_launch_count(const ivit_handle* h);

/* Releases the handle and every device buffer, CUDA graph and stream it owns (weights,
 * caches, workspaces).  The device memory is freed with cudaFree, which waits for work
 * in flight on the device; the caller must not use `h` from another thread meanwhile or
 * afterwards.  NULL does nothing. */
void ivit_destroy(ivit_handle* h);

/* Token selection that allocates nothing.  The paper has no counterpart: this entry
 * point exists for callers that cannot call cudaMalloc when they need the lists --
 * code enqueuing work while a stream is captured into a CUDA graph (allocation is not
 * permitted there), plugins whose host framework forbids allocation inside its enqueue
 * callback, and real-time loops that allocate only at start-up.
 *
 * It computes what the selection step of ivit_encode_incremental computes (cosine of
 * each token against its reference in fp32, then threshold or top-k), from embeddings
 * the caller holds: e_cur_dev and e_ref_dev fp32 [n_views][n_tok][dim], 16-byte
 * aligned (they are read with 128-bit loads).  Outputs, all caller-owned device memory,
 * 4-byte aligned: idx_out_dev int32 [n_views][n_tok] (ascending updated indices, then
 * -1), counts_out_dev int32 [n_views].  A NULL or misaligned pointer returns
 * IVIT_ERR_ARG before any device work.  Enqueued on `stream`; no handle.
 *
 * Its scratch (one fp32 score per token) is a file-scope device array of
 * IVIT_NOALLOC_MAX_TOKENS floats (256 KiB) that every GPU loading the library holds
 * until the process exits.  n_views * n_tok above that maximum returns IVIT_ERR_SHAPE
 * (message via ivit_last_error(NULL)); no cudaMalloc, cudaFree or allocating library
 * routine is ever called.  The first call on a device, with that device current, looks
 * up the array's device address (cudaGetSymbolAddress) and caches it: make that first
 * call before any stream capture.  cudaDeviceReset invalidates the cached address:
 * do not call this entry point on a device after resetting it in the same process.
 * All calls share the array; each call writes every
 * score it reads, so nothing carries over, but calls that overlap on the GPU (two
 * streams, or two threads) race on it and must be serialised by the caller. */
#define IVIT_NOALLOC_MAX_TOKENS 65536
int ivit_select_noalloc(const float* e_cur_dev, const float* e_ref_dev, int32_t n_views,
                        int32_t n_tok, int32_t dim, int32_t select_mode, float threshold,
                        int32_t topk, int32_t* idx_out_dev, int32_t* counts_out_dev,
                        void* stream);

/* The 2-step action combine of the flow-matching head (Sec. III-C, Eq. 9):
 *   xT[s][i] = x0[s][i] + alpha[s] v0[s][i] + beta[s] v7[s][i] + b[s][i]
 * for `batch` samples of `dim` action values (row-major [batch][dim], fp32, device
 * memory; alpha, beta fp32 [batch]; b may be NULL, read as zero).  v0 and v7 are the
 * solver's anchor velocities (first and eighth step) and (alpha, beta, b) the adaptor's
 * prediction, all computed by the caller: this library holds neither network.  Needs no
 * handle; enqueued on `stream`, no allocation.  IVIT_ERR_ARG for negative sizes, a
 * NULL required pointer or a pointer that is not 4-byte aligned (checked before any
 * device work); batch * dim == 0 does nothing.  128-bit accesses are used when dim is a
 * multiple of 4 and the arrays are 16-byte aligned, scalar ones otherwise. */
int ivit_action_combine(const float* x0_dev, const float* v0_dev, const float* v7_dev,
                        const float* alpha_dev, const float* beta_dev, const float* b_dev,
                        int32_t batch, int32_t dim, float* xT_dev, void* stream);

/* Message of the last failure on `h` (or of the last failed create if h is NULL). */
const char* ivit_last_error(const ivit_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* IVIT_H */
