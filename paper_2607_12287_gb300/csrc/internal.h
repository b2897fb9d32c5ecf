// Kernel launch interfaces shared by the engine and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ivit {

using bf16 = __nv_bfloat16;

// Programmatic dependent launch for every kernel of the library (on by default; the
// IVIT_NO_PDL environment variable turns it off at handle creation).
extern bool g_use_pdl;

// Stamp block (timeline mode) the next launch of this host thread passes to its kernel:
// [kStampCtas][2] global times, or null.  Set by the engine before each launch.
extern thread_local unsigned long long* g_stamp;

// cudaLaunchKernelEx with optional cluster width and the PDL attribute.
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                      unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (g_use_pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// ------------------------------------------------------------------ GEMM (tcgen05)
// Y[r][f] = sum_k X[r][k] * W[f][k] for r < M rows, f < Nout features, then an
// epilogue.  W is the weight matrix in Linear layout [Nout][K] (bf16, K-major), X the
// packed activation rows [M][K] (bf16, K-major).
enum EpiKind : int {
  kEpiF32Bias = 0,  // out_f32[r][f] = y + bias[f]
  kEpiQKV = 1,      // f <  D: out_bf16[r][f] = y + b (queries, packed rows)
                    // f < 2D: cache_k[rowtok[r]][f-D], else cache_v[rowtok[r]][f-2D]  (Eq. 5)
  kEpiResid = 2,    // out_f32[r][f] += y + bias[f]  (residual stream, fp32)
  kEpiGelu = 3,     // out_bf16[r][f] = gelu(y + bias[f])
  kEpiScatterF32 = 4,  // out_f32[rowtok[r]][f] = y + bias[f]  (per-token output cache)
};

struct GemmEpilogue {
  int kind = kEpiF32Bias;
  const float* bias = nullptr;   // [Nout]
  float* out_f32 = nullptr;      // kEpiF32Bias / kEpiResid, row stride ld_out
  bf16* out_bf16 = nullptr;      // kEpiGelu / kEpiQKV (queries), row stride ld_out
  bf16* cache_k = nullptr;       // kEpiQKV: this layer's key cache [SV*N][D]
  bf16* cache_v = nullptr;       // kEpiQKV: this layer's value cache [SV*N][D]
  const int* rowtok = nullptr;   // kEpiQKV: packed row -> token index v*N + i
  int dim = 0;                   // kEpiQKV: D
  int gelu_mode = 0;             // kEpiGelu: 0 tanh form, 1 erf form
  int ld_out = 0;
};

struct GemmArgs {
  int n_out = 0;                 // Nout
  int k = 0;                     // K
  const int* d_rows = nullptr;   // device row count M (nullptr: use m_static)
  int m_static = 0;
  int* err = nullptr;            // device error word
  // Split-K exchange scratch (global memory, stays in L2): slot [cluster][rank][BN_MAX][128]
  // floats for every CTA of the launch.  Required when the launch's clusters have more
  // than one CTA.
  float* partials = nullptr;
  // With clusters of more than one CTA and defer set, the split-K partial tiles are left
  // in the scratch, slot (tile * csize + rank) with tile = feature tile + n_ft * row tile,
  // and the kernel neither reduces them nor runs the epilogue: the next kernel sums them
  // (layernorm_sum, for the residual epilogue).  The scratch then holds
  // n_ft * ceil(M / BN_MAX) * csize slots.
  int defer = 0;
  // With defer set and vsplit > 0, K is split over vsplit consecutive CTAs launched as
  // clusters of one (no cluster barrier is needed to leave the partials): the split
  // count is then free of the GPC packing that limits cluster sizes.
  int vsplit = 0;
  unsigned long long* stamp = nullptr;  // timeline stamps of this launch (or null)
  GemmEpilogue epi;
};

// A residual update x += bias + sum_s partial_s still split over the scratch slots of a
// deferred GEMM (see GemmArgs::defer).
struct PendingSum {
  const float* partials = nullptr;  // the GEMM's scratch
  const float* bias = nullptr;      // [dim]
  int csize = 0;                    // splits (CTAs per cluster), 2..16
  int bn = 0;                       // rows per row tile (the GEMM's BN_MAX)
  int n_ft = 0;                     // feature tiles of 128
};

// Returns the dynamic shared memory size (bytes) of the GEMM variant.
size_t gemm_smem_bytes(int bn_max);
// One-time attribute setup (dynamic smem opt-in, clusters of up to 16).
cudaError_t gemm_setup(int bn_max);
// Clusters of `csize` CTAs of the variant that can be resident at once (0 if none).
int gemm_max_clusters(int bn_max, int csize);
// Launches n_clusters clusters of csize CTAs.  The CTAs of a cluster split K and reduce
// their partial tiles through distributed shared memory; clusters walk the output tiles.
cudaError_t launch_gemm(int bn_max, const CUtensorMap& tm_w, const CUtensorMap& tm_x,
                        const GemmArgs& a, int n_clusters, int csize, cudaStream_t s);

// ------------------------------------------------------- persistent encoder (small M)
struct LayerParams {
  const float *bqkv, *bo, *b1, *b2, *ln1g, *ln1b, *ln2g, *ln2b;
};

struct PersistentArgs {
  int N, D, F, H, dh, L, SV, M_max;
  float eps;
  int gelu;
  const int* cu_rows;             // [SV+1], cu_rows[SV] = updated rows M
  const int* rowtok;              // [M] packed row -> token v*N + i
  const CUtensorMap* wmaps;       // [L][4] weight maps (qkv, out, up, down), device memory
  const CUtensorMap* xmaps;       // [3] activation maps (xn, o, h), device memory
  const CUtensorMap* kvmaps;      // [L][2] key/value cache maps, box [N rows][dh], device memory
  const LayerParams* layers;      // [L], device memory
  const float *lnfg, *lnfb;
  float* x;                       // fp32 residual stream [M_max][D]
  bf16 *xn, *q, *o, *h, *cacheK, *cacheV, *tok_out;
  float* part;                    // K-split partial tiles
  unsigned* gbar;                 // [count, generation, abort], zero at launch
  int* err;
  unsigned long long* trace;      // optional: [0] count, then phase-exit times of CTA 0
};

size_t persistent_smem_bytes(int n_tok, int head_dim);
size_t persistent_part_floats(int max_items);
cudaError_t persistent_setup(size_t smem);
int persistent_max_ctas(size_t smem);
// Cooperative launch (all CTAs resident); fails if the grid cannot be resident.
cudaError_t launch_persistent(const PersistentArgs& a, int grid, size_t smem, cudaStream_t s);

// ------------------------------------------------ weight-streaming encoder (small M)
struct StreamArgs {
  int N, D, F, H, dh, L, SV, M_max;
  float eps;
  int gelu;
  int ring_stages;                // weight ring depth (16 KB stages), >= the k-blocks of a task
  int region_bytes;               // activation operand / attention region of shared memory
  int att_groups;                 // query groups per (view, head)
  int splits[4];                  // K splits of the QKV, out-proj, MLP-up and MLP-down GEMMs
  int qkv_tiles;                  // 128-feature tiles of the QKV GEMM
  int n_barriers;                 // grid barriers per launch (7 L)
  const int* cu_rows;             // [SV+1], cu_rows[SV] = updated rows M
  const int* rowtok;              // [M] packed row -> token v*N + i
  const CUtensorMap* wmaps;       // [L][4] weights (qkv, out, up, down), box 64 x 128, 128B swizzle
  const CUtensorMap* bmaps;       // [3] LN output xn, attention output o, MLP hidden h; box 64 x 32
  const CUtensorMap* kvmaps;      // [L][2] key / value caches, box dh x N, no swizzle
  const LayerParams* layers;      // [L], device memory
  const float *lnfg, *lnfb;
  float* x;                       // fp32 residual stream [M_max][D] (packed rows)
  bf16 *xn, *q, *o, *h, *cacheK, *cacheV, *tok_out;
  float* part;                    // split partials [splits][M_max][n_out] of the current GEMM
  unsigned* sync;                 // [0] barrier count, [2] abort, [4 + ...] tile counters of the
                                  // QKV and MLP-up GEMMs [L][tiles][passes]; zeroed per launch
  int* err;
  // Optional timeline (IVIT_TRACE): [n_barriers][G] barrier arrival times,
  // [n_barriers] barrier exit times of CTA 0, [G][8][8] per-CTA accumulators.
  unsigned long long* trace;
};

// k-blocks (64 wide) of one task of a GEMM with K = k split `splits` ways.
int stream_task_kblocks(int k, int splits);
// Bytes of the activation operand / attention region (1 KB multiple).
size_t stream_region_bytes(int max_task_kblocks, int n_tok, int head_dim);
// Dynamic shared memory of one CTA with `ring_stages` 16 KB weight stages.
size_t stream_smem_bytes(int ring_stages, size_t region);
// Most weight stages that fit beside the region within `smem_limit` bytes (<= 16).
int stream_ring_stages_for(size_t smem_limit, size_t region);
// Largest model width a row stage holds in registers.
int stream_max_dim();
// Updated rows per pass of a GEMM task.
int stream_rows_per_pass();
cudaError_t stream_setup(size_t smem);
int stream_max_ctas(size_t smem);
// Cooperative launch (all CTAs resident); fails if the grid cannot be resident.
cudaError_t launch_stream(const StreamArgs& a, int grid, size_t smem, cudaStream_t s);

// ------------------------------------------------------------------- other kernels
struct ColdMask {
  uint32_t bits[128];  // bit v set: view v is cold (updates every token); up to 4096 views
};

cudaError_t launch_patchify(const uint8_t* frames, bf16* patches, int sv, int img_h, int img_w,
                            int patch, int kpad, cudaStream_t s);

cudaError_t launch_score(const float* e_t, float* e_ref, float* sims, int rows, int dim,
                         int copy_ref, cudaStream_t s);

cudaError_t launch_select(const float* sims, int n_tok, int sv, int mode, float tau, int topk,
                          const ColdMask& cold, int* idx, int* counts, int* cu_rows, int* rowtok,
                          int* done_ctr, int* user_counts, cudaStream_t s);

// Row-count bands of an incremental call's CUDA graph: the launch plans of band b are
// made for at most ub[b] updated rows; the graph's switch node runs the body of the
// smallest band that holds the call's row count.
struct RowBands {
  unsigned long long handle = 0;  // cudaGraphConditionalHandle of the switch node (0: none)
  int n = 0;
  int ub[4] = {0, 0, 0, 0};
};

// x[r] = e_t[tok] + pos[tok % N] for the packed rows; refreshes e_ref[tok] from
// ref_src[tok] for refreshed tokens (last-refresh reference or cold view).  With
// bands.handle set, thread 0 of CTA 0 also selects the band of the row count.
cudaError_t launch_gather(const int* cu_rows_total, const int* rowtok, const float* e_t,
                          const float* pos, float* x, const float* ref_src, float* e_ref, int n_tok,
                          int dim, int ref_last_refresh, const ColdMask& cold, int max_rows, int grid,
                          cudaStream_t s, const RowBands& bands = RowBands());

// y[r] = LN(x[r]) (bf16) for r < *rows; when dst_rowtok is set, row r is written to
// row dst_rowtok[r] of y instead (final-token cache scatter).
cudaError_t launch_layernorm(const int* rows, const float* x, const float* gamma, const float* beta,
                             bf16* y, const int* dst_rowtok, int dim, float eps, int max_rows,
                             int grid, cudaStream_t s);
// The same, reading row src_rowtok[r] of x when src_rowtok is set, and when `add` is set
// first adding row src_rowtok[r] (or r) of `add` to x in place: x += add; y = LN(x).
cudaError_t launch_layernorm_ex(const int* rows, float* x, const float* add, const int* src_rowtok,
                                const float* gamma, const float* beta, bf16* y, const int* dst_rowtok, int dim,
                                float eps, int max_rows, int grid, cudaStream_t s);

// x[r] += bias + sum_s partial_s[r] (splits in order, as the GEMM's own reduction sums
// them), written back to x, then y = LN(x[r]) (row dst_rowtok[r] of y when set), for
// r < *rows.  dim a multiple of 4, at most 4096.
cudaError_t launch_layernorm_sum(const int* rows, float* x, const PendingSum& ps, const float* gamma,
                                 const float* beta, bf16* y, const int* dst_rowtok, int dim, float eps,
                                 int max_rows, int grid, cudaStream_t s);

// One-time function attributes of the attention kernel (dynamic shared memory opt-in).
cudaError_t attention_setup();

// O[r] = softmax(Q[r] K_v^T / sqrt(dh)) V_v per head, for the packed query rows r of
// each view v (cu_rows), over the N cached keys/values of that view.
// Keys per CTA of the attention kernel for N tokens per view (the key-split width).
int attention_keys_per_split(int n_tok);
// tm_k / tm_v: this layer's key / value cache, bf16 [SV*N][D], box [kps rows][dh], no
// swizzle.  rowtok lists the updated tokens (packed row -> v*N + i): their keys are
// re-read after the wait on the QKV kernel, every other key is loaded before it.
// query_blocks: clusters per (view, head) along the queries (each loops over blocks of
// 32 queries with its key tile resident); any value is correct, it sets parallelism.
cudaError_t launch_attention(const CUtensorMap& tm_k, const CUtensorMap& tm_v, const bf16* q,
                             const bf16* cache_k, const bf16* cache_v, const int* cu_rows,
                             const int* rowtok, bf16* o, int sv, int n_tok, int dim, int heads,
                             int query_blocks, cudaStream_t s);

// ----------------------------------------------------------- attention (tcgen05)
struct AttnTcArgs {
  const bf16* cache_k = nullptr;  // this layer's key cache, bf16 [SV*N][D] (token-major)
  const bf16* cache_v = nullptr;  // this layer's value cache, same layout
  const int* cu_rows = nullptr;   // [SV+1] packed-row offsets of the views' updated rows
  const int* rowtok = nullptr;    // packed row -> token v*N + i
  bf16* o = nullptr;              // [rows][D] attention output, packed rows
  int* err = nullptr;             // device error word
  int n_tok = 0, dim = 0, dh = 0, heads = 0, sv = 0;
  int qtiles = 0;                 // query tiles of 128 rows per (view, head): ceil(N / 128)
  int key_splits = 1;             // CTAs per cluster splitting the keys (1..8, N/splits <= 256)
  int prefetch = 0;               // 1: cached K/V loaded before the wait, then the updated
                                  //    rows re-read (incremental calls)
  unsigned long long* stamp = nullptr;  // timeline stamps of this launch (or null)
};

// One-time function attributes of the tensor-core attention kernel.
cudaError_t attention_tc_setup();

// Rows of the K/V TMA box the tensor-core attention kernel expects (the tensor maps of
// the caches use box 64 columns x this many rows).
int attention_tc_kv_box_rows();

// Dynamic shared memory of one tensor-core attention CTA for N keys split key_splits ways.
size_t attention_tc_smem(int n_tok, int dh, int key_splits);

// O[r] = softmax(Q[r] K_v^T / sqrt(dh)) V_v per head on the tensor cores, for the packed
// query rows r of each view v, over the N cached keys/values of that view.  tm_q: the
// packed queries bf16 [rows][D] with box 64 columns x 32 rows; tm_k / tm_v: this
// layer's caches bf16 [SV*N][D] with box 64 columns x attention_tc_kv_box_rows(); all
// three with 128-byte swizzle.  Grid: clusters of
// key_splits CTAs (128 threads each), at most max_ctas CTAs, walking the (query tile,
// view, head) items.
cudaError_t launch_attention_tc(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                                const AttnTcArgs& a, int max_ctas, cudaStream_t s);

}  // namespace ivit
