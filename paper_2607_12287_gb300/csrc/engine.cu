// Engine behind the C ABI of include/ivit.h: weight upload, per-view caches,
// workspaces, TMA descriptors and the per-frame launch chain of temporal token reuse
// (Sec. III-B): embed -> score (Eq. 3) -> select/compact -> gather -> per layer
// {LN1, QKV + K/V cache scatter (Eq. 4-5), attention of updated queries over all
// tokens, out-proj + residual, LN2, MLP up + GELU, MLP down + residual} -> final LN
// scattered into the final-token cache -> output copy.
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdlib>
#include <cstdio>
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/ivit.h"
#include "internal.h"
#include "ptx.cuh"

using ivit::bf16;

namespace {

struct LayerW {
  bf16 *wqkv, *wo, *w1, *w2;
  float *bqkv, *bo, *b1, *b2, *ln1g, *ln1b, *ln2g, *ln2b;
  CUtensorMap tm_qkv, tm_o, tm_1, tm_2;
  CUtensorMap tm_ck, tm_cv;  // this layer's key / value cache, SIMT attention key-split tiles
  CUtensorMap tm_ak, tm_av;  // the same caches, 64 x 128 boxes, 128-byte swizzle (tcgen05)
};

// Kernel families of the timeline.
enum Family : int { kFamGemm = 0, kFamAttn = 1, kFamLN = 2, kFamOther = 3, kFamilies = 4 };

struct TimelineSlot {
  int family = kFamOther;
  int n_out = 0, k = 0, kind = 0;  // GEMM shape and epilogue
  int m_static = -1;               // GEMM rows when fixed, -1 when read from the device
};

// Launch shape of one GEMM: row-tile variant, CTAs per cluster (the K split), clusters.
struct GemmPlan {
  int bn = 64, csize = 1, n_clusters = 1;
  bool defer = false;  // residual GEMMs: leave the split partials to the next layer norm
  bool vsplit = false; // deferred: K split over CTAs launched without clusters
};

enum GemmSlot { kGemmEmbed = 0, kGemmQKV, kGemmO, kGemmUp, kGemmDown, kGemmSlots };

thread_local std::string g_create_error;

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// bf16 2-D tensor [rows][inner] with the given row stride; box = box_inner x box_rows,
// 128-byte swizzle (box_inner * 2 == 128) or dense rows, out-of-bounds elements read as 0.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t stride_bytes,
              uint32_t box_inner, uint32_t box_rows, bool swizzle = true) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Bump allocator over one device allocation; every sub-buffer 256-byte aligned.
struct Arena {
  size_t size = 0;
  char* base = nullptr;
  size_t take(size_t bytes) {
    const size_t off = size;
    size += (bytes + 255) & ~static_cast<size_t>(255);
    return off;
  }
  template <class T>
  T* at(size_t off) const {
    return reinterpret_cast<T*>(base + off);
  }
};

inline float bf16_bits_to_float(uint16_t b) {
  uint32_t u = static_cast<uint32_t>(b) << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

}  // namespace

namespace ivit {
void set_create_error(const char* msg) { g_create_error = msg ? msg : ""; }
}  // namespace ivit

struct ivit_handle {
  ivit_config cfg{};
  int N = 0, D = 0, F = 0, H = 0, L = 0, SV = 0, Kp = 0, KPAD = 0, M_max = 0;
  int device = 0, num_sms = 0;
  int row_grid = 0;
  GemmPlan plan_full[kGemmSlots], plan_inc[kGemmSlots];
  // Row-count bands of the incremental graph (band 0 = plan_inc): launch plans and
  // attention key splits made for at most band_ub[b] updated rows; a switch node picks
  // the band of each call's device-resident row count.
  int n_bands = 1;
  int band_ub[4] = {0, 0, 0, 0};
  GemmPlan plan_band[4][kGemmSlots];
  int attn_splits_band[4] = {1, 1, 1, 1};
  bool capture_bands = false;  // set while the incremental graph is captured with bands
  int known_band = -1;         // set while it is captured for a row count known in advance
  ivit::RowBands bands;        // the switch node's handle and the bands' row bounds
  cudaStream_t cap_stream2 = nullptr;  // captures the band bodies

  void* wmem = nullptr;  // weights (device)
  void* smem = nullptr;  // state + workspaces (device)
  bf16* w_pe = nullptr;
  float *b_pe = nullptr, *pos = nullptr, *lnfg = nullptr, *lnfb = nullptr;
  std::vector<LayerW> layers;
  CUtensorMap tm_pe, tm_patches, tm_xn, tm_o, tm_h;
  CUtensorMap tm_qa;     // packed queries, 64 x 32 boxes, 128-byte swizzle (tcgen05 attention)
  bool attn_tc = true;   // tensor-core attention (IVIT_ATTN=simt selects the SIMT kernel)
  int attn_splits_full = 1, attn_splits_inc = 1;  // key splits (CTAs per item) of that kernel

  bf16* patches = nullptr;
  float *e_t = nullptr, *e_ref = nullptr, *sims = nullptr, *x = nullptr;
  float* key_t = nullptr;          // first-layer keys of every token (score_source KEY0)
  float* acache = nullptr;         // [L][M_max][D] attention-block outputs (mlp_tokens ALL)
  float* gemm_partials = nullptr;  // split-K exchange slots of the GEMMs (global scratch)
  int* rowtok_all = nullptr;       // identity row -> token map, all SV*N rows
  int* m_all = nullptr;            // device copy of SV*N
  CUtensorMap tm_wk0;              // layer 0's key projection (rows D..2D-1 of W_qkv)
  long long chunk = 0;             // ivit_encode_incremental calls (odd/even schedule)
  int *idx = nullptr, *counts = nullptr, *cu_rows = nullptr, *rowtok = nullptr, *done_ctr = nullptr;
  int* err = nullptr;
  bf16 *xn = nullptr, *q = nullptr, *o = nullptr, *hbuf = nullptr, *cacheK = nullptr,
       *cacheV = nullptr, *tok_out = nullptr;

  std::vector<uint8_t> cold;
  int64_t launches = 0;

  // Persistent encoder (all blocks in one cooperative launch) for small encoders: it runs
  // the full encodes; incremental calls run it only when forced (persistent_inc), since
  // the kernel chain is faster for a few updated rows (its tensor-core attention against
  // the persistent kernel's SIMT attention phase).
  bool persistent = false;
  bool persistent_inc = false;
  size_t pt_smem = 0;
  int pt_grid = 0;
  void* pt_mem = nullptr;  // device: tensor maps, layer parameters, partials, barrier words
  ivit::PersistentArgs pt_args{};

  // Weight-streaming kernel (every block of an incremental call in one cooperative
  // launch, weights streamed through a shared-memory ring) for small updated-row counts.
  bool stream_ok = false;
  size_t sk_smem = 0;
  int sk_grid = 0;
  void* sk_mem = nullptr;  // device: tensor maps, layer parameters, partials, sync words
  size_t sk_sync_bytes = 0;
  ivit::StreamArgs sk_args{};

  // CUDA graphs of the full and the steady-state incremental chain.  Inputs and outputs
  // are staged through handle-owned buffers (copies outside the graph), so the graph's
  // kernel parameters never change.
  bool use_graphs = true;
  cudaStream_t cap_stream = nullptr;
  cudaGraphExec_t graph_full = nullptr, graph_inc = nullptr;
  int64_t graph_full_launches = 0, graph_inc_launches = 0;
  uint8_t* frames_buf = nullptr;
  int* counts_buf = nullptr;

  // Timeline mode (ivit_timeline): every launch of a call writes per-CTA start/end
  // stamps into its slot of `stamps`; `slots_*` record each slot's kernel family and,
  // for GEMMs, the shape that gives its algorithmic bytes.
  bool timeline = false;
  unsigned long long* stamps = nullptr;
  int stamp_cap = 0, stamp_used = 0;
  std::vector<TimelineSlot> slots_cur, slots_full, slots_inc, slots_last;

  std::string error;

  int fail(int code, const std::string& msg) {
    error = msg;
    return code;
  }
  int cuda_fail(const char* what, cudaError_t e) {
    error = std::string(what) + ": " + cudaGetErrorString(e);
    return e == cudaErrorMemoryAllocation ? IVIT_ERR_OOM : IVIT_ERR_CUDA;
  }
};

#define IVIT_CK(h, call)                                 \
  do {                                                   \
    cudaError_t e_ = (call);                             \
    if (e_ != cudaSuccess) return (h)->cuda_fail(#call, e_); \
  } while (0)

namespace {

const char* validate(const ivit_config* c) {
  if (!c) return "null config";
  if (c->patch <= 0 || c->img_h <= 0 || c->img_w <= 0) return "patch and image size must be positive";
  if (c->img_h % c->patch || c->img_w % c->patch) return "patch must divide img_h and img_w";
  const long long n = static_cast<long long>(c->img_h / c->patch) * (c->img_w / c->patch);
  if (n > 1024) return "at most 1024 tokens per view";
  if (c->dim <= 0 || c->dim % 64 || c->dim > 2048) return "dim must be a multiple of 64 in [64, 2048]";
  if (c->heads <= 0 || c->dim % c->heads) return "heads must divide dim";
  const int dh = c->dim / c->heads;
  if (dh % 8 || dh > 128) return "head_dim must be a multiple of 8 and at most 128";
  if (c->depth <= 0) return "depth must be positive";
  if (c->mlp_dim <= 0 || c->mlp_dim % 8) return "mlp_dim must be a positive multiple of 8";
  if (c->n_streams <= 0 || c->n_views <= 0) return "n_streams and n_views must be positive";
  if (static_cast<long long>(c->n_streams) * c->n_views > 4096) return "at most 4096 views";
  if (!(c->ln_eps > 0.f)) return "ln_eps must be positive";
  if (c->gelu != IVIT_GELU_TANH && c->gelu != IVIT_GELU_ERF) return "bad gelu";
  if (c->select_mode != IVIT_SEL_THRESHOLD && c->select_mode != IVIT_SEL_TOPK) return "bad select_mode";
  if (c->ref_mode != IVIT_REF_PREV_FRAME && c->ref_mode != IVIT_REF_LAST_REFRESH) return "bad ref_mode";
  if (c->select_mode == IVIT_SEL_TOPK && c->topk < 0) return "topk must be >= 0";
  if (!std::isfinite(c->threshold)) return "threshold must be finite";
  if (c->score_source != IVIT_SCORE_EMBED && c->score_source != IVIT_SCORE_KEY0) return "bad score_source";
  if (c->schedule != IVIT_SCHED_INCREMENTAL && c->schedule != IVIT_SCHED_ODD_EVEN) return "bad schedule";
  if (c->mlp_tokens != IVIT_MLP_UPDATED && c->mlp_tokens != IVIT_MLP_ALL) return "bad mlp_tokens";
  return nullptr;
}

size_t weights_count(const ivit_config* c) {
  const size_t D = c->dim, F = c->mlp_dim, N = static_cast<size_t>(c->img_h / c->patch) * (c->img_w / c->patch);
  const size_t Kp = static_cast<size_t>(c->patch) * c->patch * 3;
  const size_t per_layer = 2 * D + 3 * D * D + 3 * D + D * D + D + 2 * D + F * D + F + D * F + D;
  return D * Kp + D + N * D + per_layer * c->depth + 2 * D;
}

// Launch shape of a GEMM with a K split over clusters of c CTAs.  Cost model (fitted
// to measurements of this kernel on GB300 with small row counts): a launch pays a fixed
// ~4 us plus ~0.35 us per 16 KB weight stage a CTA streams, once per round of tiles
// over the clusters that fit on the GPU.  Cluster sizes above 9 lose SMs to GPC packing.
GemmPlan plan_gemm(int num_sms, int bn, int n_out, int k, int m_expected) {
  GemmPlan best;
  best.bn = bn;
  const int n_ft = (n_out + 127) / 128, n_tt = (m_expected + bn - 1) / bn, n_kb = (k + 63) / 64;
  const int tiles = std::max(1, n_ft * n_tt);
  double best_cost = 1e30;
  for (int c = 1; c <= std::min(16, n_kb); ++c) {
    const int fit = ivit::gemm_max_clusters(bn, c);
    if (fit <= 0) continue;
    const int ncl = std::max(1, std::min({tiles, fit, num_sms / c}));
    const int rounds = (tiles + ncl - 1) / ncl;
    const double cost = rounds * (4.0 + 0.35 * ((n_kb + c - 1) / c));
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best.csize = c;
      best.n_clusters = ncl;
    }
  }
  return best;
}

// Prepares the persistent encoder when its shared memory fits (attention keeps a whole
// view's keys and values of one head resident, so N * head_dim is bounded).
int setup_persistent(ivit_handle* h) {
  // IVIT_PATH=kernels / IVIT_PATH=persistent (every call) override the choice made from
  // the shape.  Default: the full encodes of small encoders (dim <= 384), whose
  // per-layer kernels are launch-bound at every row of every view.
  const char* path = std::getenv("IVIT_PATH");
  if (path && std::strcmp(path, "kernels") == 0) return IVIT_OK;
  if (h->cfg.mlp_tokens == IVIT_MLP_ALL) return IVIT_OK;  // the kernel chain runs that reading
  const bool forced = path && std::strcmp(path, "persistent") == 0;
  if (!forced && h->D > 384) return IVIT_OK;
  const int dh = h->D / h->H;
  const size_t smem = ivit::persistent_smem_bytes(h->N, dh);
  if (smem > 227 * 1024 || h->D > 2048 || h->N > 256) return IVIT_OK;
  IVIT_CK(h, ivit::persistent_setup(smem));
  const int grid = std::min(h->num_sms, ivit::persistent_max_ctas(smem));
  if (grid < 1) return IVIT_OK;
  const int L = h->L;
  // partial slots: at most one item per CTA with K split, else one per tile
  const int n_tt = (h->M_max + 63) / 64;
  const int max_tiles = std::max({(3 * h->D + 127) / 128, (h->F + 127) / 128}) * n_tt;
  const int max_items = std::max(grid, max_tiles);
  Arena pa;
  const size_t o_w = pa.take(sizeof(CUtensorMap) * 4 * L), o_x = pa.take(sizeof(CUtensorMap) * 3);
  const size_t o_kv = pa.take(sizeof(CUtensorMap) * 2 * L);
  const size_t o_lp = pa.take(sizeof(ivit::LayerParams) * L);
  const size_t o_part = pa.take(ivit::persistent_part_floats(max_items) * sizeof(float));
  const size_t o_bar = pa.take(4 * sizeof(unsigned));
  IVIT_CK(h, cudaMalloc(&h->pt_mem, pa.size));
  IVIT_CK(h, cudaMemset(h->pt_mem, 0, pa.size));
  pa.base = static_cast<char*>(h->pt_mem);
  std::vector<CUtensorMap> wm(4 * L);
  std::vector<ivit::LayerParams> lp(L);
  for (int l = 0; l < L; ++l) {
    const LayerW& w = h->layers[l];
    wm[4 * l + 0] = w.tm_qkv;
    wm[4 * l + 1] = w.tm_o;
    wm[4 * l + 2] = w.tm_1;
    wm[4 * l + 3] = w.tm_2;
    lp[l] = ivit::LayerParams{w.bqkv, w.bo, w.b1, w.b2, w.ln1g, w.ln1b, w.ln2g, w.ln2b};
  }
  const CUtensorMap xm[3] = {h->tm_xn, h->tm_o, h->tm_h};
  std::vector<CUtensorMap> kvm(2 * L);
  for (int l = 0; l < L; ++l) {
    const size_t off = static_cast<size_t>(l) * h->M_max * h->D;
    if (!make_map(&kvm[2 * l], h->cacheK + off, h->D, h->M_max, h->D * 2, dh, h->N, false) ||
        !make_map(&kvm[2 * l + 1], h->cacheV + off, h->D, h->M_max, h->D * 2, dh, h->N, false))
      return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for a cache tile");
  }
  IVIT_CK(h, cudaMemcpy(pa.base + o_kv, kvm.data(), sizeof(CUtensorMap) * 2 * L, cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(pa.base + o_w, wm.data(), sizeof(CUtensorMap) * 4 * L, cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(pa.base + o_x, xm, sizeof(xm), cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(pa.base + o_lp, lp.data(), sizeof(ivit::LayerParams) * L, cudaMemcpyHostToDevice));
  ivit::PersistentArgs& a = h->pt_args;
  a.N = h->N;
  a.D = h->D;
  a.F = h->F;
  a.H = h->H;
  a.dh = dh;
  a.L = L;
  a.SV = h->SV;
  a.M_max = h->M_max;
  a.eps = h->cfg.ln_eps;
  a.gelu = h->cfg.gelu;
  a.cu_rows = h->cu_rows;
  a.rowtok = h->rowtok;
  a.wmaps = pa.at<CUtensorMap>(o_w);
  a.xmaps = pa.at<CUtensorMap>(o_x);
  a.kvmaps = pa.at<CUtensorMap>(o_kv);
  a.layers = pa.at<ivit::LayerParams>(o_lp);
  a.lnfg = h->lnfg;
  a.lnfb = h->lnfb;
  a.x = h->x;
  a.xn = h->xn;
  a.q = h->q;
  a.o = h->o;
  a.h = h->hbuf;
  a.cacheK = h->cacheK;
  a.cacheV = h->cacheV;
  a.tok_out = h->tok_out;
  a.part = pa.at<float>(o_part);
  a.gbar = pa.at<unsigned>(o_bar);
  a.err = h->err;
  a.trace = nullptr;
  if (std::getenv("IVIT_TRACE")) {
    IVIT_CK(h, cudaMalloc(&a.trace, 4096 * sizeof(unsigned long long)));
    IVIT_CK(h, cudaMemset(a.trace, 0, 4096 * sizeof(unsigned long long)));
  }
  h->pt_smem = smem;
  h->pt_grid = grid;
  h->persistent = true;
  h->persistent_inc = forced;
  return IVIT_OK;
}

// Prepares the weight-streaming kernel (IVIT_PATH=stream: every incremental call without
// a cold view runs it).  It is not the default: on the So400m camera stream it measured
// 1.5 ms per frame against the kernel chain's 1.0 ms (seven grid barriers per layer and
// the dependent latencies inside each stage cost more than the chain's launch handoffs).
int setup_stream(ivit_handle* h) {
  const ivit_config& c = h->cfg;
  const char* path = std::getenv("IVIT_PATH");
  if (!path || std::strcmp(path, "stream") != 0) return IVIT_OK;
  if (c.mlp_tokens == IVIT_MLP_ALL) return IVIT_OK;  // the kernel chain runs that reading
  const int N = h->N, D = h->D, F = h->F, H = h->H, L = h->L, SV = h->SV, dh = D / H;
  if (D > ivit::stream_max_dim() || N > 256) return IVIT_OK;
  int optin = 0;
  IVIT_CK(h, cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device));
  const int grid = h->num_sms;
  // K splits: enough tasks (tile x split) to give about one to every CTA
  const int n_out[4] = {3 * D, D, F, D}, kdim[4] = {D, D, D, F};
  int splits[4], max_kb = 0;
  size_t part_floats = 0;
  for (int g = 0; g < 4; ++g) {
    const int tiles = (n_out[g] + 127) / 128, nkb = (kdim[g] + 63) / 64;
    splits[g] = std::max(1, std::min(nkb, grid / tiles));
    max_kb = std::max(max_kb, ivit::stream_task_kblocks(kdim[g], splits[g]));
    part_floats = std::max(part_floats, static_cast<size_t>(splits[g]) * h->M_max * n_out[g]);
  }
  const size_t region = ivit::stream_region_bytes(max_kb, N, dh);
  const int rs = ivit::stream_ring_stages_for(static_cast<size_t>(optin), region);
  if (rs < std::max(4, max_kb)) return IVIT_OK;
  const size_t smem = ivit::stream_smem_bytes(rs, region);
  IVIT_CK(h, ivit::stream_setup(smem));
  if (ivit::stream_max_ctas(smem) < grid) return IVIT_OK;
  const int rpp = ivit::stream_rows_per_pass();
  const int passes_max = (h->M_max + rpp - 1) / rpp;
  const int qkv_tiles = (3 * D + 127) / 128, up_tiles = (F + 127) / 128;
  const size_t sync_words = 4 + static_cast<size_t>(L) * (qkv_tiles + up_tiles) * passes_max;
  Arena ka;
  const size_t o_w = ka.take(sizeof(CUtensorMap) * 4 * L), o_b = ka.take(sizeof(CUtensorMap) * 3);
  const size_t o_kv = ka.take(sizeof(CUtensorMap) * 2 * L), o_lp = ka.take(sizeof(ivit::LayerParams) * L);
  const size_t o_part = ka.take(part_floats * sizeof(float)), o_sync = ka.take(sync_words * sizeof(unsigned));
  IVIT_CK(h, cudaMalloc(&h->sk_mem, ka.size));
  IVIT_CK(h, cudaMemset(h->sk_mem, 0, ka.size));
  ka.base = static_cast<char*>(h->sk_mem);
  std::vector<CUtensorMap> wm(4 * L), kvm(2 * L);
  std::vector<ivit::LayerParams> lp(L);
  for (int l = 0; l < L; ++l) {
    const LayerW& w = h->layers[l];
    const size_t off = static_cast<size_t>(l) * h->M_max * D;
    wm[4 * l + 0] = w.tm_qkv;
    wm[4 * l + 1] = w.tm_o;
    wm[4 * l + 2] = w.tm_1;
    wm[4 * l + 3] = w.tm_2;
    if (!make_map(&kvm[2 * l], h->cacheK + off, D, h->M_max, D * 2, dh, N, false) ||
        !make_map(&kvm[2 * l + 1], h->cacheV + off, D, h->M_max, D * 2, dh, N, false))
      return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for the weight-streaming kernel");
    lp[l] = ivit::LayerParams{w.bqkv, w.bo, w.b1, w.b2, w.ln1g, w.ln1b, w.ln2g, w.ln2b};
  }
  const CUtensorMap bm[3] = {h->tm_xn, h->tm_o, h->tm_h};
  IVIT_CK(h, cudaMemcpy(ka.base + o_w, wm.data(), sizeof(CUtensorMap) * 4 * L, cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(ka.base + o_b, bm, sizeof(bm), cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(ka.base + o_kv, kvm.data(), sizeof(CUtensorMap) * 2 * L, cudaMemcpyHostToDevice));
  IVIT_CK(h, cudaMemcpy(ka.base + o_lp, lp.data(), sizeof(ivit::LayerParams) * L, cudaMemcpyHostToDevice));
  ivit::StreamArgs& a = h->sk_args;
  a.N = N;
  a.D = D;
  a.F = F;
  a.H = H;
  a.dh = dh;
  a.L = L;
  a.SV = SV;
  a.M_max = h->M_max;
  a.eps = c.ln_eps;
  a.gelu = c.gelu;
  a.ring_stages = rs;
  a.region_bytes = static_cast<int>(region);
  a.att_groups = std::max(1, std::min(16, grid / std::max(1, SV * H)));
  for (int g = 0; g < 4; ++g) a.splits[g] = splits[g];
  a.qkv_tiles = qkv_tiles;
  a.n_barriers = 7 * L;
  a.cu_rows = h->cu_rows;
  a.rowtok = h->rowtok;
  a.wmaps = ka.at<CUtensorMap>(o_w);
  a.bmaps = ka.at<CUtensorMap>(o_b);
  a.kvmaps = ka.at<CUtensorMap>(o_kv);
  a.layers = ka.at<ivit::LayerParams>(o_lp);
  a.lnfg = h->lnfg;
  a.lnfb = h->lnfb;
  a.x = h->x;
  a.xn = h->xn;
  a.q = h->q;
  a.o = h->o;
  a.h = h->hbuf;
  a.cacheK = h->cacheK;
  a.cacheV = h->cacheV;
  a.tok_out = h->tok_out;
  a.part = ka.at<float>(o_part);
  a.sync = ka.at<unsigned>(o_sync);
  a.err = h->err;
  a.trace = nullptr;
  if (std::getenv("IVIT_TRACE")) {
    const size_t n = static_cast<size_t>(a.n_barriers) * (grid + 1) + 64 * static_cast<size_t>(grid);
    IVIT_CK(h, cudaMalloc(&a.trace, n * sizeof(unsigned long long)));
    IVIT_CK(h, cudaMemset(a.trace, 0, n * sizeof(unsigned long long)));
  }
  h->sk_sync_bytes = sync_words * sizeof(unsigned);
  h->sk_smem = smem;
  h->sk_grid = grid;
  h->stream_ok = true;
  if (std::getenv("IVIT_DEBUG"))
    std::fprintf(stderr, "ivit stream kernel: grid %d, smem %zu, ring %d stages, region %zu, groups %d, "
                 "splits %d %d %d %d\n", grid, smem, rs, region, a.att_groups, splits[0], splits[1], splits[2],
                 splits[3]);
  return IVIT_OK;
}

int setup(ivit_handle* h, const uint16_t* wb) {
  const ivit_config& c = h->cfg;
  h->N = (c.img_h / c.patch) * (c.img_w / c.patch);
  h->D = c.dim;
  h->F = c.mlp_dim;
  h->H = c.heads;
  h->L = c.depth;
  h->SV = c.n_streams * c.n_views;
  h->Kp = c.patch * c.patch * 3;
  h->KPAD = (h->Kp + 63) / 64 * 64;
  h->M_max = h->SV * h->N;
  h->cold.assign(h->SV, 1);
  const size_t D = h->D, F = h->F, N = h->N, L = h->L, M = h->M_max;

  IVIT_CK(h, cudaGetDevice(&h->device));
  IVIT_CK(h, cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
  IVIT_CK(h, ivit::gemm_setup(64));
  IVIT_CK(h, ivit::gemm_setup(256));
  IVIT_CK(h, ivit::attention_setup());
  IVIT_CK(h, ivit::attention_tc_setup());
  if (const char* at = std::getenv("IVIT_ATTN")) h->attn_tc = std::string(at) != "simt";
  {
    // Row bands: the first holds a tenth of the tokens (rounded up to 16, at least 64),
    // each next one twice the previous, the last all of them; at most four.
    int ub = std::max(64, (static_cast<int>(M / 10) + 15) / 16 * 16);
    h->n_bands = 0;
    while (h->n_bands < 4) {
      const bool last = ub >= static_cast<int>(M) || h->n_bands == 3;
      h->band_ub[h->n_bands++] = last ? static_cast<int>(M) : ub;
      if (last) break;
      ub *= 2;
    }
    if (std::getenv("IVIT_NO_BANDS")) h->n_bands = 1;
  }
  {
    // Key splits of the tensor-core attention: as many as fill the SMs once for the
    // expected items (query tiles x heads x views: all tokens when full, a tenth when
    // incremental), at least 64 keys per CTA, one (online softmax over key groups) when
    // the items alone fill the GPU; more while one CTA's shared memory exceeds the limit.
    int optin = 0;
    IVIT_CK(h, cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device));
    const int dh = h->D / h->H;
    auto splits = [&](int m_exp) {
      const int ns_cap = std::max(1, std::min(8, (h->N + 63) / 64));  // at least 64 keys per CTA
      const int items = h->SV * h->H * ((m_exp + 127) / 128);
      int ns = std::max(1, std::min(ns_cap, h->num_sms / std::max(1, items)));
      if (const char* e = std::getenv("IVIT_ATTN_SPLITS")) ns = std::max(1, std::min(8, std::atoi(e)));
      while (ns < 8 && ivit::attention_tc_smem(h->N, dh, ns) > static_cast<size_t>(optin)) ++ns;
      return ns;
    };
    h->attn_splits_full = splits(h->N);
    h->attn_splits_inc = splits(std::max(1, h->N / 10));
    h->attn_splits_band[0] = h->attn_splits_inc;
    for (int b = 1; b < h->n_bands; ++b) h->attn_splits_band[b] = splits(std::max(1, h->band_ub[b] / h->SV));
    if (ivit::attention_tc_smem(h->N, dh, h->attn_splits_full) > static_cast<size_t>(optin) ||
        ivit::attention_tc_smem(h->N, dh, h->attn_splits_inc) > static_cast<size_t>(optin))
      h->attn_tc = false;  // not reachable for N <= 1024, dh <= 128
  }
  if (std::getenv("IVIT_NO_PDL")) ivit::g_use_pdl = false;
  if (std::getenv("IVIT_NO_GRAPH")) h->use_graphs = false;
  IVIT_CK(h, cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking));
  IVIT_CK(h, cudaStreamCreateWithFlags(&h->cap_stream2, cudaStreamNonBlocking));
  h->row_grid = h->num_sms * 4;
  {
    // Full encodes know M = SV*N.  Incremental calls are planned for a tenth of the
    // tokens updated (any count still runs correctly, with more or fewer tile rounds).
    const int m_inc = std::max(1, static_cast<int>(M / 10));
    // (64-row tiles for full encodes of up to 256 rows: on a 256-row So400m view they
    // measured 1.78 ms per full encode against 1.92-2.01 ms with one 256-row tile split
    // over clusters, whose split partials are four times larger)
    const int bn_full = M <= 256 ? 64 : 256, bn_inc = M <= 1024 ? 64 : 256;
    const int shapes[kGemmSlots][2] = {{static_cast<int>(D), h->KPAD}, {3 * static_cast<int>(D), static_cast<int>(D)},
                                       {static_cast<int>(D), static_cast<int>(D)}, {static_cast<int>(F), static_cast<int>(D)},
                                       {static_cast<int>(D), static_cast<int>(F)}};
    for (int g = 0; g < kGemmSlots; ++g) {
      h->plan_full[g] = plan_gemm(h->num_sms, bn_full, shapes[g][0], shapes[g][1], static_cast<int>(M));
      h->plan_inc[g] = g == kGemmEmbed ? h->plan_full[g]
                                       : plan_gemm(h->num_sms, bn_inc, shapes[g][0], shapes[g][1], m_inc);
      h->plan_band[0][g] = h->plan_inc[g];
      // (the band of all rows runs the full encode's plans: it attends like one too)
      for (int b = 1; b < h->n_bands; ++b)
        h->plan_band[b][g] = g == kGemmEmbed || h->band_ub[b] >= static_cast<int>(M)
                                 ? h->plan_full[g]
                                 : plan_gemm(h->num_sms, h->band_ub[b] <= 256 ? 64 : 256, shapes[g][0], shapes[g][1],
                                             h->band_ub[b]);
    }
    // Residual GEMMs with a K split leave their partials to the layer norm that follows
    // (one slot per tile and split, sized for the most rows the plan can see), while that
    // scratch stays under 64 MB.  Needing no cluster barrier, such a GEMM then splits K
    // over plain CTAs, with the split re-chosen by the same cost model without the
    // cluster packing limit (at most 16 splits, the layer norm's limit).
    auto replan_free = [&](GemmPlan& pl, int n_out, int k, int m_expected) {
      const int n_ft = (n_out + 127) / 128, n_tt = (m_expected + pl.bn - 1) / pl.bn, n_kb = (k + 63) / 64;
      const int tiles = std::max(1, n_ft * n_tt);
      double best_cost = 1e30;
      GemmPlan best = pl;
      for (int c = 2; c <= std::min(16, n_kb); ++c) {
        const int rounds = (tiles * c + h->num_sms - 1) / h->num_sms;
        const double cost = rounds * (4.0 + 0.35 * ((n_kb + c - 1) / c));
        if (cost < best_cost - 1e-9) {
          best_cost = cost;
          best.csize = c;
          best.n_clusters = tiles;
        }
      }
      if (best_cost < 1e29 && !std::getenv("IVIT_NO_VSPLIT")) {
        pl = best;
        pl.vsplit = true;
      }
    };
    auto set_defer = [&](GemmPlan& pl, int n_out, int m_bound) {
      const size_t slots = static_cast<size_t>((n_out + 127) / 128) * ((m_bound + pl.bn - 1) / pl.bn) * pl.csize;
      pl.defer = pl.csize > 1 && !std::getenv("IVIT_NO_DEFER") && slots * pl.bn * 128 * 4 <= (64ull << 20) &&
                 h->D % 4 == 0 && h->D <= 4096;
    };
    // a deferred plan re-planned without clusters, kept if its scratch still fits
    auto refine = [&](GemmPlan& pl, int g, int m_expected, int m_bound) {
      if (!pl.defer) return;
      const GemmPlan orig = pl;
      replan_free(pl, shapes[g][0], shapes[g][1], m_expected);
      set_defer(pl, static_cast<int>(D), m_bound);
      if (!pl.defer) pl = orig;
    };
    for (int g : {static_cast<int>(kGemmO), static_cast<int>(kGemmDown)}) {
      set_defer(h->plan_full[g], static_cast<int>(D), static_cast<int>(M));
      set_defer(h->plan_inc[g], static_cast<int>(D), static_cast<int>(M));
      refine(h->plan_full[g], g, static_cast<int>(M), static_cast<int>(M));
      refine(h->plan_inc[g], g, std::max(1, static_cast<int>(M / 10)), static_cast<int>(M));
      h->plan_band[0][g] = h->plan_inc[g];
      for (int b = 1; b < h->n_bands; ++b) {
        set_defer(h->plan_band[b][g], static_cast<int>(D), h->band_ub[b]);
        refine(h->plan_band[b][g], g, h->band_ub[b], h->band_ub[b]);
      }
    }
    if (std::getenv("IVIT_DEBUG")) {
      static const char* names[kGemmSlots] = {"embed", "qkv", "out", "up", "down"};
      for (int g = 0; g < kGemmSlots; ++g)
        std::fprintf(stderr, "ivit gemm %-5s full bn=%d %s=%d x %d (fit %d) | inc bn=%d %s=%d x %d (fit %d)\n",
                     names[g], h->plan_full[g].bn, h->plan_full[g].vsplit ? "split" : "cluster", h->plan_full[g].csize,
                     h->plan_full[g].n_clusters, ivit::gemm_max_clusters(h->plan_full[g].bn, h->plan_full[g].csize),
                     h->plan_inc[g].bn, h->plan_inc[g].vsplit ? "split" : "cluster", h->plan_inc[g].csize,
                     h->plan_inc[g].n_clusters, ivit::gemm_max_clusters(h->plan_inc[g].bn, h->plan_inc[g].csize));
      for (int b = 1; b < h->n_bands; ++b)
        std::fprintf(stderr, "ivit band %d (<= %d rows): attention splits %d\n", b, h->band_ub[b], h->attn_splits_band[b]);
    }
  }

  // ---- weights: bf16 matrices (W_pe padded to KPAD columns), fp32 vectors
  Arena wa;
  const size_t o_pe = wa.take(D * h->KPAD * 2), o_bpe = wa.take(D * 4), o_pos = wa.take(N * D * 4);
  struct LOff { size_t qkv, o, w1, w2, bqkv, bo, b1, b2, g1, be1, g2, be2; };
  std::vector<LOff> lo(L);
  for (size_t l = 0; l < L; ++l) {
    lo[l].qkv = wa.take(3 * D * D * 2);
    lo[l].o = wa.take(D * D * 2);
    lo[l].w1 = wa.take(F * D * 2);
    lo[l].w2 = wa.take(D * F * 2);
    lo[l].bqkv = wa.take(3 * D * 4);
    lo[l].bo = wa.take(D * 4);
    lo[l].b1 = wa.take(F * 4);
    lo[l].b2 = wa.take(D * 4);
    lo[l].g1 = wa.take(D * 4);
    lo[l].be1 = wa.take(D * 4);
    lo[l].g2 = wa.take(D * 4);
    lo[l].be2 = wa.take(D * 4);
  }
  const size_t o_gf = wa.take(D * 4), o_bf = wa.take(D * 4);

  std::vector<char> host(wa.size, 0);
  auto put_bf16 = [&](size_t off, const uint16_t* src, size_t rows, size_t cols, size_t ld) {
    for (size_t r = 0; r < rows; ++r) std::memcpy(&host[off + r * ld * 2], src + r * cols, cols * 2);
  };
  auto put_f32 = [&](size_t off, const uint16_t* src, size_t n) {
    float* dst = reinterpret_cast<float*>(&host[off]);
    for (size_t i = 0; i < n; ++i) dst[i] = bf16_bits_to_float(src[i]);
  };
  const uint16_t* p = wb;
  put_bf16(o_pe, p, D, h->Kp, h->KPAD); p += D * h->Kp;
  put_f32(o_bpe, p, D); p += D;
  put_f32(o_pos, p, N * D); p += N * D;
  for (size_t l = 0; l < L; ++l) {
    put_f32(lo[l].g1, p, D); p += D;
    put_f32(lo[l].be1, p, D); p += D;
    put_bf16(lo[l].qkv, p, 3 * D, D, D); p += 3 * D * D;
    put_f32(lo[l].bqkv, p, 3 * D); p += 3 * D;
    put_bf16(lo[l].o, p, D, D, D); p += D * D;
    put_f32(lo[l].bo, p, D); p += D;
    put_f32(lo[l].g2, p, D); p += D;
    put_f32(lo[l].be2, p, D); p += D;
    put_bf16(lo[l].w1, p, F, D, D); p += F * D;
    put_f32(lo[l].b1, p, F); p += F;
    put_bf16(lo[l].w2, p, D, F, F); p += D * F;
    put_f32(lo[l].b2, p, D); p += D;
  }
  put_f32(o_gf, p, D); p += D;
  put_f32(o_bf, p, D); p += D;

  IVIT_CK(h, cudaMalloc(&h->wmem, wa.size));
  IVIT_CK(h, cudaMemcpy(h->wmem, host.data(), wa.size, cudaMemcpyHostToDevice));
  wa.base = static_cast<char*>(h->wmem);
  h->w_pe = wa.at<bf16>(o_pe);
  h->b_pe = wa.at<float>(o_bpe);
  h->pos = wa.at<float>(o_pos);
  h->lnfg = wa.at<float>(o_gf);
  h->lnfb = wa.at<float>(o_bf);
  h->layers.resize(L);
  for (size_t l = 0; l < L; ++l) {
    LayerW& w = h->layers[l];
    w.wqkv = wa.at<bf16>(lo[l].qkv);
    w.wo = wa.at<bf16>(lo[l].o);
    w.w1 = wa.at<bf16>(lo[l].w1);
    w.w2 = wa.at<bf16>(lo[l].w2);
    w.bqkv = wa.at<float>(lo[l].bqkv);
    w.bo = wa.at<float>(lo[l].bo);
    w.b1 = wa.at<float>(lo[l].b1);
    w.b2 = wa.at<float>(lo[l].b2);
    w.ln1g = wa.at<float>(lo[l].g1);
    w.ln1b = wa.at<float>(lo[l].be1);
    w.ln2g = wa.at<float>(lo[l].g2);
    w.ln2b = wa.at<float>(lo[l].be2);
    if (!make_map(&w.tm_qkv, w.wqkv, D, 3 * D, D * 2, 64, 128) ||
        !make_map(&w.tm_o, w.wo, D, D, D * 2, 64, 128) ||
        !make_map(&w.tm_1, w.w1, D, F, D * 2, 64, 128) ||
        !make_map(&w.tm_2, w.w2, F, D, F * 2, 64, 128))
      return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for a weight matrix");
  }
  if (!make_map(&h->tm_pe, h->w_pe, h->KPAD, D, h->KPAD * 2, 64, 128))
    return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for W_pe");

  // ---- state and workspaces
  Arena sa;
  const size_t o_patch = sa.take(M * h->KPAD * 2), o_et = sa.take(M * D * 4), o_er = sa.take(M * D * 4);
  const size_t o_sims = sa.take(M * 4), o_idx = sa.take(M * 4), o_cnt = sa.take(h->SV * 4);
  const size_t o_cu = sa.take((h->SV + 1) * 4), o_rt = sa.take(M * 4), o_done = sa.take(4);
  const size_t o_x = sa.take(M * D * 4), o_xn = sa.take(M * D * 2), o_q = sa.take(M * D * 2);
  const size_t o_o = sa.take(M * D * 2), o_h = sa.take(M * F * 2);
  const size_t o_ck = sa.take(L * M * D * 2), o_cv = sa.take(L * M * D * 2), o_tok = sa.take(M * D * 2);
  const size_t o_err = sa.take(4);
  const size_t o_key = c.score_source == IVIT_SCORE_KEY0 ? sa.take(M * D * 4) : 0;
  const size_t o_acache = c.mlp_tokens == IVIT_MLP_ALL ? sa.take(L * M * D * 4) : 0;
  // slots for every plan: clusters x CTAs per cluster x row tile x 128 features, fp32
  size_t part_floats = 0;
  for (int g = 0; g < kGemmSlots; ++g)
  {
    auto need = [&](const GemmPlan& pl, int m_bound) {
      if (!pl.defer) return static_cast<size_t>(pl.n_clusters) * pl.csize * pl.bn * 128;
      return static_cast<size_t>((D + 127) / 128) * ((m_bound + pl.bn - 1) / pl.bn) * pl.csize * pl.bn * 128;
    };
    part_floats = std::max(part_floats, need(h->plan_full[g], static_cast<int>(M)));
    part_floats = std::max(part_floats, need(h->plan_inc[g], static_cast<int>(M)));
    for (int b = 0; b < h->n_bands; ++b)
      part_floats = std::max(part_floats, need(h->plan_band[b][g], b == 0 ? static_cast<int>(M) : h->band_ub[b]));
  }
  const size_t o_gpart = sa.take(part_floats * 4);
  const size_t o_rta = sa.take(M * 4), o_mall = sa.take(4);
  const size_t o_fb = sa.take(static_cast<size_t>(h->SV) * c.img_h * c.img_w * 3);
  const size_t o_cb = sa.take(h->SV * 4);
  IVIT_CK(h, cudaMalloc(&h->smem, sa.size));
  IVIT_CK(h, cudaMemset(h->smem, 0, sa.size));
  sa.base = static_cast<char*>(h->smem);
  h->patches = sa.at<bf16>(o_patch);
  h->e_t = sa.at<float>(o_et);
  h->e_ref = sa.at<float>(o_er);
  h->sims = sa.at<float>(o_sims);
  h->idx = sa.at<int>(o_idx);
  h->counts = sa.at<int>(o_cnt);
  h->cu_rows = sa.at<int>(o_cu);
  h->rowtok = sa.at<int>(o_rt);
  h->done_ctr = sa.at<int>(o_done);
  h->x = sa.at<float>(o_x);
  h->xn = sa.at<bf16>(o_xn);
  h->q = sa.at<bf16>(o_q);
  h->o = sa.at<bf16>(o_o);
  h->hbuf = sa.at<bf16>(o_h);
  h->cacheK = sa.at<bf16>(o_ck);
  h->cacheV = sa.at<bf16>(o_cv);
  h->tok_out = sa.at<bf16>(o_tok);
  h->err = sa.at<int>(o_err);
  if (c.score_source == IVIT_SCORE_KEY0) h->key_t = sa.at<float>(o_key);
  if (c.mlp_tokens == IVIT_MLP_ALL) h->acache = sa.at<float>(o_acache);
  h->gemm_partials = sa.at<float>(o_gpart);
  h->rowtok_all = sa.at<int>(o_rta);
  h->m_all = sa.at<int>(o_mall);
  {
    std::vector<int> ident(M);
    for (size_t i = 0; i < M; ++i) ident[i] = static_cast<int>(i);
    const int m_host = static_cast<int>(M);
    IVIT_CK(h, cudaMemcpy(h->rowtok_all, ident.data(), M * sizeof(int), cudaMemcpyHostToDevice));
    IVIT_CK(h, cudaMemcpy(h->m_all, &m_host, sizeof(int), cudaMemcpyHostToDevice));
  }
  if (!make_map(&h->tm_wk0, h->layers[0].wqkv + D * D, D, D, D * 2, 64, 128))
    return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for the first-layer key projection");
  h->frames_buf = sa.at<uint8_t>(o_fb);
  h->counts_buf = sa.at<int>(o_cb);
  const int kps = ivit::attention_keys_per_split(h->N);
  for (size_t l = 0; l < L; ++l) {
    const size_t off = l * M * D;
    if (!make_map(&h->layers[l].tm_ck, h->cacheK + off, D, M, D * 2, D / h->H, kps, false) ||
        !make_map(&h->layers[l].tm_cv, h->cacheV + off, D, M, D * 2, D / h->H, kps, false) ||
        !make_map(&h->layers[l].tm_ak, h->cacheK + off, D, M, D * 2, 64, ivit::attention_tc_kv_box_rows()) ||
        !make_map(&h->layers[l].tm_av, h->cacheV + off, D, M, D * 2, 64, ivit::attention_tc_kv_box_rows()))
      return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for a cache tile");
  }
  if (!make_map(&h->tm_patches, h->patches, h->KPAD, M, h->KPAD * 2, 64, 32) ||
      !make_map(&h->tm_xn, h->xn, D, M, D * 2, 64, 32) ||
      !make_map(&h->tm_o, h->o, D, M, D * 2, 64, 32) ||
      !make_map(&h->tm_qa, h->q, D, M, D * 2, 64, 32) ||
      !make_map(&h->tm_h, h->hbuf, F, M, F * 2, 64, 32))
    return h->fail(IVIT_ERR_CUDA, "cuTensorMapEncodeTiled failed for an activation buffer");
  if (int r = setup_persistent(h)) return r;
  if (int r = setup_stream(h)) return r;
  IVIT_CK(h, cudaDeviceSynchronize());
  return IVIT_OK;
}

void release(ivit_handle* h) {
  if (h->sk_args.trace) cudaFree(h->sk_args.trace);
  h->sk_args.trace = nullptr;
  if (h->sk_mem) cudaFree(h->sk_mem);
  h->sk_mem = nullptr;
  if (h->pt_args.trace) cudaFree(h->pt_args.trace);
  h->pt_args.trace = nullptr;
  if (h->pt_mem) cudaFree(h->pt_mem);
  h->pt_mem = nullptr;
  if (h->graph_full) cudaGraphExecDestroy(h->graph_full);
  if (h->graph_inc) cudaGraphExecDestroy(h->graph_inc);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  if (h->cap_stream2) cudaStreamDestroy(h->cap_stream2);
  h->cap_stream2 = nullptr;
  h->graph_full = h->graph_inc = nullptr;
  h->cap_stream = nullptr;
  if (h->wmem) cudaFree(h->wmem);
  if (h->smem) cudaFree(h->smem);
  if (h->stamps) cudaFree(h->stamps);
  h->stamps = nullptr;
  h->wmem = h->smem = nullptr;
}

// Algorithmic bytes of one GEMM launch at M rows (weights, input rows, output rows, bias).
double gemm_bytes(int n_out, int k, int kind, long long M) {
  const double out_b = kind == ivit::kEpiF32Bias ? 4.0 : kind == ivit::kEpiResid ? 8.0 : 2.0;
  return 2.0 * n_out * k + 2.0 * M * k + out_b * M * n_out + 4.0 * n_out;
}

// Before each launch: the stamp slot of the launch in timeline mode (else none).
void next_launch(ivit_handle* h, int family, const ivit::GemmArgs* ga = nullptr, int other_kind = 0) {
  ivit::g_stamp = nullptr;
  if (!h->timeline || !h->stamps || h->stamp_used >= h->stamp_cap) return;
  ivit::g_stamp = h->stamps + static_cast<size_t>(h->stamp_used++) * 2 * ivit::kStampCtas;
  TimelineSlot sl;
  sl.family = family;
  sl.kind = other_kind;
  if (ga) {
    sl.n_out = ga->n_out;
    sl.k = ga->k;
    sl.kind = ga->epi.kind;
    sl.m_static = ga->d_rows ? -1 : ga->m_static;
  }
  h->slots_cur.push_back(sl);
}

int gemm(ivit_handle* h, const GemmPlan& plan, const CUtensorMap& tw, const CUtensorMap& tx,
         ivit::GemmArgs a, cudaStream_t s) {
  a.err = h->err;
  a.partials = h->gemm_partials;
  next_launch(h, kFamGemm, &a);
  IVIT_CK(h, ivit::launch_gemm(plan.bn, tw, tx, a, plan.n_clusters, plan.csize, s));
  ++h->launches;
  return IVIT_OK;
}

// Debug aid (IVIT_TRACE): mean time of each phase kind of the last persistent launch.
void print_trace(ivit_handle* h, cudaStream_t s) {
  std::vector<unsigned long long> t(4096);
  if (cudaStreamSynchronize(s) != cudaSuccess) return;
  cudaMemcpy(t.data(), h->pt_args.trace, t.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost);
  const int n = static_cast<int>(t[0]);
  static const char* names[9] = {"qkv gemm", "qkv reduce", "attention", "out gemm", "out red+LN2",
                                 "up gemm", "up reduce", "down gemm", "down red+LN"};
  double acc[9] = {0};
  int cnt[9] = {0};
  for (int i = 2; i < n; ++i) {  // entry 1 = start, entry 2 = after the first LN phase
    const int k = (i - 2) % 9;
    acc[k] += 1e-3 * static_cast<double>(t[1 + i] - t[i]);
    ++cnt[k];
  }
  std::fprintf(stderr, "ivit trace: %d phases, total %.1f us, first LN %.1f us\n", n - 1,
               1e-3 * static_cast<double>(t[n] - t[1]), 1e-3 * static_cast<double>(t[2] - t[1]));
  for (int k = 0; k < 9; ++k)
    if (cnt[k]) std::fprintf(stderr, "  %-12s %6.2f us x %d\n", names[k], acc[k] / cnt[k], cnt[k]);
}

// Debug aid (IVIT_TRACE): stage durations of the last weight-streaming launch (critical
// path: the last CTA's arrival at each grid barrier after the previous barrier's exit),
// barrier latencies, and per-task phase times.
void print_stream_trace(ivit_handle* h, cudaStream_t s) {
  const int L = h->L, G = h->sk_grid, NB = h->sk_args.n_barriers;
  std::vector<unsigned long long> t(static_cast<size_t>(NB) * (G + 1) + 64 * static_cast<size_t>(G));
  if (cudaStreamSynchronize(s) != cudaSuccess) return;
  cudaMemcpy(t.data(), h->sk_args.trace, t.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost);
  static const char* names[7] = {"qkv", "attention", "out", "ln2", "up", "down", "ln1"};
  double dur[7] = {0}, lat[7] = {0}, mean_arr[7] = {0};
  int cnt[7] = {0};
  for (int k = 1; k < NB; ++k) {
    unsigned long long mx = 0;
    double sum = 0;
    for (int c = 0; c < G; ++c) {
      mx = std::max(mx, t[static_cast<size_t>(k) * G + c]);
      sum += static_cast<double>(t[static_cast<size_t>(k) * G + c]);
    }
    const double prev_exit = static_cast<double>(t[static_cast<size_t>(NB) * G + k - 1]);
    const double exit_k = static_cast<double>(t[static_cast<size_t>(NB) * G + k]);
    const int j = (k - 1) % 7;
    dur[j] += 1e-3 * (static_cast<double>(mx) - prev_exit);
    lat[j] += 1e-3 * (exit_k - static_cast<double>(mx));
    mean_arr[j] += 1e-3 * (sum / G - prev_exit);
    ++cnt[j];
  }
  std::fprintf(stderr, "ivit stream trace: %d barriers, first exit %.1f us after CTA 0 arrived, last exit %.1f us\n",
               NB, 1e-3 * static_cast<double>(t[static_cast<size_t>(NB) * G] - t[0]),
               1e-3 * static_cast<double>(t[static_cast<size_t>(NB) * G + NB - 1] - t[0]));
  for (int j = 0; j < 7; ++j)
    if (cnt[j])
      std::fprintf(stderr, "  %-9s stage %6.2f us (mean arrival %6.2f) barrier %5.2f us\n", names[j], dur[j] / cnt[j],
                   mean_arr[j] / cnt[j], lat[j] / cnt[j]);
  static const char* kinds[6] = {"qkv", "out", "up", "down", "attn", "rows"};
  static const char* slots[6][7] = {{"w-wait", "B", "mma", "acc-wait", "epilogue", "fixup", ""},
                                    {"w-wait", "B", "mma", "acc-wait", "epilogue", "fixup", ""},
                                    {"w-wait", "B", "mma", "acc-wait", "epilogue", "fixup", ""},
                                    {"w-wait", "B", "mma", "acc-wait", "epilogue", "fixup", ""},
                                    {"kv+patch", "compute", "scores", "softmax+pv", "", "", ""},
                                    {"row", "", "", "", "", "", ""}};
  const size_t base = static_cast<size_t>(NB) * (G + 1);
  for (int g = 0; g < 6; ++g) {
    double n = 0;
    for (int c = 0; c < G; ++c) n += static_cast<double>(t[base + (c * 8 + g) * 8 + 7]);
    if (n == 0) continue;
    std::fprintf(stderr, "  %-5s x%6.0f/call:", kinds[g], n);
    for (int k = 0; k < 7; ++k) {
      if (!slots[g][k][0]) continue;
      double sum = 0;
      for (int c = 0; c < G; ++c) sum += 1e-3 * static_cast<double>(t[base + (c * 8 + g) * 8 + k]);
      std::fprintf(stderr, " %s %.2f", slots[g][k], sum / n);
    }
    std::fprintf(stderr, "\n");
  }
  (void)L;
  cudaMemset(h->sk_args.trace, 0, t.size() * sizeof(unsigned long long));
}

// Attention of the updated queries over all tokens of their view for one layer.
int attention(ivit_handle* h, const LayerW& w, const bf16* ck, const bf16* cv, bool full, cudaStream_t s,
              int key_splits = 0) {
  const int N = h->N, D = h->D, SV = h->SV;
  if (h->attn_tc) {
    ivit::AttnTcArgs at;
    at.cache_k = ck;
    at.cache_v = cv;
    at.cu_rows = h->cu_rows;
    at.rowtok = h->rowtok;
    at.o = h->o;
    at.err = h->err;
    at.n_tok = N;
    at.dim = D;
    at.dh = D / h->H;
    at.heads = h->H;
    at.sv = SV;
    at.qtiles = (N + 127) / 128;
    at.prefetch = full ? 0 : 1;
    at.key_splits = key_splits > 0 ? key_splits : (full ? h->attn_splits_full : h->attn_splits_inc);
    next_launch(h, kFamAttn);
    at.stamp = ivit::g_stamp;
    IVIT_CK(h, ivit::launch_attention_tc(h->tm_qa, w.tm_ak, w.tm_av, at, h->num_sms, s));
  } else {
    next_launch(h, kFamAttn);
    IVIT_CK(h, ivit::launch_attention(w.tm_ck, w.tm_cv, h->q, ck, cv, h->cu_rows, h->rowtok, h->o, SV, N, D, h->H,
                                      full ? (N + 31) / 32 : std::max(1, (N / 10 + 31) / 32), s));
  }
  ++h->launches;
  return IVIT_OK;
}

// The blocks under the MLP-on-all-tokens reading (Sec. III-B, after Eq. 5): x holds
// every token's residual stream (row = token v*N + i).  Per layer, the updated tokens
// (packed rows, rowtok) run LN1, QKV with the K/V scatter (Eq. 5), attention over all
// tokens and the output projection, whose result replaces their rows of the layer's
// attention-output cache; then every token adds its cached attention output to its
// stream (fused into LN2) and runs the MLP; the final LN writes every output token.
int run_layers_mlp_all(ivit_handle* h, const GemmPlan* plan, bool full, cudaStream_t s) {
  const ivit_config& c = h->cfg;
  const int N = h->N, D = h->D, F = h->F, SV = h->SV, M = h->M_max;
  const int* total = h->cu_rows + SV;
  for (int l = 0; l < h->L; ++l) {
    const LayerW& w = h->layers[l];
    bf16* ck = h->cacheK + static_cast<size_t>(l) * M * D;
    bf16* cv = h->cacheV + static_cast<size_t>(l) * M * D;
    float* al = h->acache + static_cast<size_t>(l) * M * D;
    next_launch(h, kFamLN);
    IVIT_CK(h, ivit::launch_layernorm_ex(total, h->x, nullptr, h->rowtok, w.ln1g, w.ln1b, h->xn, nullptr, D,
                                         c.ln_eps, M, h->row_grid, s));
    ++h->launches;
    {
      ivit::GemmArgs a;
      a.n_out = 3 * D;
      a.k = D;
      a.d_rows = total;
      a.epi.kind = ivit::kEpiQKV;
      a.epi.bias = w.bqkv;
      a.epi.out_bf16 = h->q;
      a.epi.ld_out = D;
      a.epi.cache_k = ck;
      a.epi.cache_v = cv;
      a.epi.rowtok = h->rowtok;
      a.epi.dim = D;
      if (int r = gemm(h, plan[kGemmQKV], w.tm_qkv, h->tm_xn, a, s)) return r;
    }
    if (int r = attention(h, w, ck, cv, full, s)) return r;
    {
      ivit::GemmArgs a;
      a.n_out = D;
      a.k = D;
      a.d_rows = total;
      a.epi.kind = ivit::kEpiScatterF32;
      a.epi.bias = w.bo;
      a.epi.out_f32 = al;
      a.epi.ld_out = D;
      a.epi.rowtok = h->rowtok;
      if (int r = gemm(h, plan[kGemmO], w.tm_o, h->tm_o, a, s)) return r;
    }
    next_launch(h, kFamLN);
    IVIT_CK(h, ivit::launch_layernorm_ex(h->m_all, h->x, al, nullptr, w.ln2g, w.ln2b, h->xn, nullptr, D, c.ln_eps,
                                         M, h->row_grid, s));
    ++h->launches;
    {
      ivit::GemmArgs a;
      a.n_out = F;
      a.k = D;
      a.m_static = M;
      a.epi.kind = ivit::kEpiGelu;
      a.epi.bias = w.b1;
      a.epi.out_bf16 = h->hbuf;
      a.epi.ld_out = F;
      a.epi.gelu_mode = c.gelu;
      if (int r = gemm(h, h->plan_full[kGemmUp], w.tm_1, h->tm_xn, a, s)) return r;
    }
    {
      ivit::GemmArgs a;
      a.n_out = D;
      a.k = F;
      a.m_static = M;
      a.epi.kind = ivit::kEpiResid;
      a.epi.bias = w.b2;
      a.epi.out_f32 = h->x;
      a.epi.ld_out = D;
      if (int r = gemm(h, h->plan_full[kGemmDown], w.tm_2, h->tm_h, a, s)) return r;
    }
  }
  next_launch(h, kFamLN);
  IVIT_CK(h, ivit::launch_layernorm(h->m_all, h->x, h->lnfg, h->lnfb, h->tok_out, nullptr, D, c.ln_eps, M,
                                    h->row_grid, s));
  ++h->launches;
  (void)N;
  return IVIT_OK;
}

// Per layer {LN1, QKV + K/V cache scatter (Eq. 4-5), attention, out-proj + residual,
// LN2, MLP up + GELU, MLP down + residual}, then the final LN scattered into the
// final-token cache, with the given launch plans and attention key splits.
int run_layers(ivit_handle* h, const GemmPlan* plan, int attn_splits, bool full, cudaStream_t s) {
  const ivit_config& c = h->cfg;
  const int D = h->D, F = h->F, SV = h->SV, M = h->M_max;
  const int* total = h->cu_rows + SV;
  // A residual update still split over the GEMM scratch (deferred out-projection or
  // MLP-down GEMM): the next layer norm adds it to x.
  ivit::PendingSum pend;
  auto layernorm = [&](const float* g, const float* b, bf16* y, const int* dst) -> int {
    next_launch(h, kFamLN);
    if (pend.partials) {
      IVIT_CK(h, ivit::launch_layernorm_sum(total, h->x, pend, g, b, y, dst, D, c.ln_eps, M, h->row_grid, s));
      pend = ivit::PendingSum();
    } else {
      IVIT_CK(h, ivit::launch_layernorm(total, h->x, g, b, y, dst, D, c.ln_eps, M, h->row_grid, s));
    }
    ++h->launches;
    return IVIT_OK;
  };
  auto residual = [&](const GemmPlan& pl, const float* bias, const CUtensorMap& tw, const CUtensorMap& tx,
                      int k) -> int {
    ivit::GemmArgs a;
    a.n_out = D;
    a.k = k;
    a.d_rows = total;
    a.epi.kind = ivit::kEpiResid;
    a.epi.bias = bias;
    a.epi.out_f32 = h->x;
    a.epi.ld_out = D;
    a.defer = pl.defer ? 1 : 0;
    a.vsplit = pl.defer && pl.vsplit ? pl.csize : 0;
    if (int r = gemm(h, pl, tw, tx, a, s)) return r;
    if (pl.defer) {
      pend.partials = h->gemm_partials;
      pend.bias = bias;
      pend.csize = pl.csize;
      pend.bn = pl.bn;
      pend.n_ft = (D + 127) / 128;
    }
    return IVIT_OK;
  };
  for (int l = 0; l < h->L; ++l) {
    const LayerW& w = h->layers[l];
    bf16* ck = h->cacheK + static_cast<size_t>(l) * M * D;
    bf16* cv = h->cacheV + static_cast<size_t>(l) * M * D;
    if (int r = layernorm(w.ln1g, w.ln1b, h->xn, nullptr)) return r;
    {
      ivit::GemmArgs a;
      a.n_out = 3 * D;
      a.k = D;
      a.d_rows = total;
      a.epi.kind = ivit::kEpiQKV;
      a.epi.bias = w.bqkv;
      a.epi.out_bf16 = h->q;
      a.epi.ld_out = D;
      a.epi.cache_k = ck;
      a.epi.cache_v = cv;
      a.epi.rowtok = h->rowtok;
      a.epi.dim = D;
      if (int r = gemm(h, plan[kGemmQKV], w.tm_qkv, h->tm_xn, a, s)) return r;
    }
    if (int r = attention(h, w, ck, cv, full, s, attn_splits)) return r;
    if (int r = residual(plan[kGemmO], w.bo, w.tm_o, h->tm_o, D)) return r;
    if (int r = layernorm(w.ln2g, w.ln2b, h->xn, nullptr)) return r;
    {
      ivit::GemmArgs a;
      a.n_out = F;
      a.k = D;
      a.d_rows = total;
      a.epi.kind = ivit::kEpiGelu;
      a.epi.bias = w.b1;
      a.epi.out_bf16 = h->hbuf;
      a.epi.ld_out = F;
      a.epi.gelu_mode = c.gelu;
      if (int r = gemm(h, plan[kGemmUp], w.tm_1, h->tm_xn, a, s)) return r;
    }
    if (int r = residual(plan[kGemmDown], w.b2, w.tm_2, h->tm_h, F)) return r;
  }
  return layernorm(h->lnfg, h->lnfb, h->tok_out, h->rowtok);
}

// Under capture of an incremental graph with row bands: a switch node after the
// gather (which sets its value from the row count) with one body per band, each the
// layer chain with that band's launch plans, captured on a second stream.  The
// launches of one body count for the call.
int capture_band_bodies(ivit_handle* h, cudaStream_t s) {
  cudaStreamCaptureStatus st;
  cudaGraph_t graph = nullptr;
  const cudaGraphNode_t* deps = nullptr;
  size_t ndeps = 0;
  IVIT_CK(h, cudaStreamGetCaptureInfo(s, &st, nullptr, &graph, &deps, nullptr, &ndeps));
  cudaGraphNodeParams np = {};
  np.type = cudaGraphNodeTypeConditional;
  np.conditional.handle = static_cast<cudaGraphConditionalHandle>(h->bands.handle);
  np.conditional.type = cudaGraphCondTypeSwitch;
  np.conditional.size = static_cast<unsigned>(h->n_bands);
  cudaGraphNode_t node;
  IVIT_CK(h, cudaGraphAddNode(&node, graph, deps, nullptr, ndeps, &np));
  IVIT_CK(h, cudaStreamUpdateCaptureDependencies(s, &node, nullptr, 1, cudaStreamSetCaptureDependencies));
  const int64_t pre = h->launches;
  for (int b = 0; b < h->n_bands; ++b) {
    h->launches = pre;
    IVIT_CK(h, cudaStreamBeginCaptureToGraph(h->cap_stream2, np.conditional.phGraph_out[b], nullptr, nullptr, 0,
                                             cudaStreamCaptureModeThreadLocal));
    // (the band of every row attends like a full encode: no cached-K/V prefetch to patch)
    const int r = run_layers(h, h->plan_band[b], h->attn_splits_band[b], h->band_ub[b] >= h->M_max, h->cap_stream2);
    cudaGraph_t body = nullptr;
    const cudaError_t e = cudaStreamEndCapture(h->cap_stream2, &body);
    if (r) return r;
    if (e != cudaSuccess) return h->cuda_fail("cudaStreamEndCapture (band body)", e);
  }
  return IVIT_OK;
}

// Enqueues the whole chain for one frame per view on `s` (eagerly or under capture).
int run_core(ivit_handle* h, const uint8_t* frames, int32_t* user_counts, bool full, cudaStream_t s) {
  const ivit_config& c = h->cfg;
  const int N = h->N, D = h->D, SV = h->SV, M = h->M_max;
  ivit::ColdMask cm;
  std::memset(&cm, 0, sizeof cm);
  for (int v = 0; v < SV; ++v)
    if (full || h->cold[v]) cm.bits[v >> 5] |= 1u << (v & 31);
  const GemmPlan* plan = full ? h->plan_full : h->plan_inc;
  const int* total = h->cu_rows + SV;
  h->launches = 0;
  h->slots_cur.clear();
  h->stamp_used = 0;
  if (h->timeline && h->stamps)  // CTAs that leave early write nothing: clear the last call's stamps
    IVIT_CK(h, cudaMemsetAsync(h->stamps, 0, static_cast<size_t>(h->stamp_cap) * 2 * ivit::kStampCtas *
                                                 sizeof(unsigned long long), s));

  next_launch(h, kFamOther, nullptr, 0);  // patchify
  IVIT_CK(h, ivit::launch_patchify(frames, h->patches, SV, c.img_h, c.img_w, c.patch, h->KPAD, s));
  ++h->launches;
  {
    ivit::GemmArgs a;
    a.n_out = D;
    a.k = h->KPAD;
    a.m_static = M;
    a.epi.kind = ivit::kEpiF32Bias;
    a.epi.bias = h->b_pe;
    a.epi.out_f32 = h->e_t;
    a.epi.ld_out = D;
    if (int r = gemm(h, plan[kGemmEmbed], h->tm_pe, h->tm_patches, a, s)) return r;
  }
  const float* score_vec = h->e_t;
  if (c.score_source == IVIT_SCORE_KEY0) {
    // Eq. 3 on first-layer keys of every token: W_K LN1(e + pos) + b_K (x, xn are free
    // until the updated rows are gathered below)
    next_launch(h, kFamOther, nullptr, 3);  // gather
    IVIT_CK(h, ivit::launch_gather(h->m_all, h->rowtok_all, h->e_t, h->pos, h->x, nullptr, h->e_ref, N, D, 0,
                                   cm, M, h->row_grid, s));
    next_launch(h, kFamLN);
    IVIT_CK(h, ivit::launch_layernorm(h->m_all, h->x, h->layers[0].ln1g, h->layers[0].ln1b, h->xn, nullptr, D,
                                      c.ln_eps, M, h->row_grid, s));
    h->launches += 2;
    ivit::GemmArgs a;
    a.n_out = D;
    a.k = D;
    a.m_static = M;
    a.epi.kind = ivit::kEpiF32Bias;
    a.epi.bias = h->layers[0].bqkv + D;
    a.epi.out_f32 = h->key_t;
    a.epi.ld_out = D;
    // a D x D projection of every row: the full encode's out-projection launch shape
    if (int r = gemm(h, h->plan_full[kGemmO], h->tm_wk0, h->tm_xn, a, s)) return r;
    score_vec = h->key_t;
  }
  if (!full) {
    next_launch(h, kFamOther, nullptr, 1);  // score
    IVIT_CK(h, ivit::launch_score(score_vec, h->e_ref, h->sims, M, D, c.ref_mode == IVIT_REF_PREV_FRAME, s));
    ++h->launches;
  }
  next_launch(h, kFamOther, nullptr, 2);  // select
  IVIT_CK(h, ivit::launch_select(h->sims, N, SV, full ? IVIT_SEL_THRESHOLD : c.select_mode, c.threshold,
                                 c.topk, cm, h->idx, h->counts, h->cu_rows, h->rowtok, h->done_ctr,
                                 user_counts, s));
  ++h->launches;
  if (c.mlp_tokens == IVIT_MLP_ALL) {
    // every token's residual stream (token-indexed), then the references of the updated
    // tokens (last-refresh mode, cold views) without touching x
    next_launch(h, kFamOther, nullptr, 3);  // gather
    IVIT_CK(h, ivit::launch_gather(h->m_all, h->rowtok_all, h->e_t, h->pos, h->x, nullptr, h->e_ref, N, D, 0,
                                   cm, M, h->row_grid, s));
    next_launch(h, kFamOther, nullptr, 3);  // gather
    IVIT_CK(h, ivit::launch_gather(total, h->rowtok, h->e_t, h->pos, nullptr, score_vec, h->e_ref, N, D,
                                   c.ref_mode == IVIT_REF_LAST_REFRESH, cm, M, h->row_grid, s));
    h->launches += 2;
    return run_layers_mlp_all(h, plan, full, s);
  }
  ivit::RowBands bands;  // (no switch node: handle 0)
  if (h->capture_bands) {
    cudaStreamCaptureStatus st;
    cudaGraph_t graph = nullptr;
    IVIT_CK(h, cudaStreamGetCaptureInfo(s, &st, nullptr, &graph));
    cudaGraphConditionalHandle ch;
    IVIT_CK(h, cudaGraphConditionalHandleCreate(&ch, graph, 0, cudaGraphCondAssignDefault));
    bands.handle = static_cast<unsigned long long>(ch);
    bands.n = h->n_bands;
    for (int b = 0; b < h->n_bands; ++b) bands.ub[b] = h->band_ub[b];
    h->bands = bands;
  }
  next_launch(h, kFamOther, nullptr, 3);  // gather
  IVIT_CK(h, ivit::launch_gather(total, h->rowtok, h->e_t, h->pos, h->x, score_vec, h->e_ref, N, D,
                                 c.ref_mode == IVIT_REF_LAST_REFRESH, cm, M, h->row_grid, s, bands));
  ++h->launches;

  bool any_cold = false;
  for (int v = 0; v < SV; ++v) any_cold = any_cold || (cm.bits[v >> 5] >> (v & 31)) & 1u;
  if (h->stream_ok && !full && !any_cold) {
    IVIT_CK(h, cudaMemsetAsync(h->sk_args.sync, 0, h->sk_sync_bytes, s));
    IVIT_CK(h, ivit::launch_stream(h->sk_args, h->sk_grid, h->sk_smem, s));
    ++h->launches;
    if (h->sk_args.trace) {
      cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
      cudaStreamIsCapturing(s, &cs);
      if (cs == cudaStreamCaptureStatusNone) print_stream_trace(h, s);
    }
    return IVIT_OK;
  }
  if (h->persistent && (full || h->persistent_inc)) {
    IVIT_CK(h, cudaMemsetAsync(h->pt_args.gbar, 0, 4 * sizeof(unsigned), s));
    IVIT_CK(h, ivit::launch_persistent(h->pt_args, h->pt_grid, h->pt_smem, s));
    ++h->launches;
    if (h->pt_args.trace && !h->timeline) {
      cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
      cudaStreamIsCapturing(s, &cs);
      if (cs == cudaStreamCaptureStatusNone) print_trace(h, s);
    }
    return IVIT_OK;
  }
  if (h->capture_bands) return capture_band_bodies(h, s);
  if (!full && h->known_band >= 0)  // top-k: the row count is fixed, so is its band
    return run_layers(h, h->plan_band[h->known_band], h->attn_splits_band[h->known_band],
                      h->band_ub[h->known_band] >= h->M_max, s);
  return run_layers(h, plan, full ? h->attn_splits_full : h->attn_splits_inc, full, s);
}

int capture_once(ivit_handle* h, bool full, cudaGraphExec_t* exec, int64_t* launches);

// The incremental graph of the kernel chain is captured with a switch over the row
// bands when there are several; if that capture fails the plain graph (band 0's plans
// for every row count) is captured instead.
int capture(ivit_handle* h, bool full, cudaGraphExec_t* exec, int64_t* launches) {
  const bool chain = h->cfg.mlp_tokens == IVIT_MLP_UPDATED && !h->stream_ok && !h->persistent_inc;
  if (!full && chain && h->n_bands > 1 && h->cfg.select_mode == IVIT_SEL_TOPK) {
    // top-k (no cold view in a captured call): exactly k rows per view, so the band is
    // known when the graph is captured and no switch is needed
    const long long m = std::min<long long>(static_cast<long long>(h->cfg.topk), h->N) * h->SV;
    int b = 0;
    while (b + 1 < h->n_bands && m > h->band_ub[b]) ++b;
    h->known_band = b;
    const int r = capture_once(h, full, exec, launches);
    h->known_band = -1;
    return r;
  }
  // threshold selection: the row count is known only on the device; the switch pays its
  // fixed cost (no programmatic overlap across the node) when a tenth of the tokens
  // already exceeds 32 rows, so that row counts commonly cross bands
  if (!full && chain && h->n_bands > 1 && h->M_max / 10 > 32) {
    h->capture_bands = true;
    const int r = capture_once(h, full, exec, launches);
    h->capture_bands = false;
    if (r == IVIT_OK) return IVIT_OK;
    if (std::getenv("IVIT_DEBUG")) std::fprintf(stderr, "ivit: row-band graph failed (%s)\n", h->error.c_str());
    cudaGetLastError();
    h->n_bands = 1;
  }
  return capture_once(h, full, exec, launches);
}

int capture_once(ivit_handle* h, bool full, cudaGraphExec_t* exec, int64_t* launches) {
  IVIT_CK(h, cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
  const int r = run_core(h, h->frames_buf, h->counts_buf, full, h->cap_stream);
  cudaGraph_t g = nullptr;
  const cudaError_t e = cudaStreamEndCapture(h->cap_stream, &g);
  if (r != IVIT_OK) {
    if (g) cudaGraphDestroy(g);
    return r;
  }
  if (e != cudaSuccess) return h->cuda_fail("cudaStreamEndCapture", e);
  const cudaError_t ei = cudaGraphInstantiate(exec, g, 0);
  cudaGraphDestroy(g);
  if (ei != cudaSuccess) return h->cuda_fail("cudaGraphInstantiate", ei);
  *launches = h->launches;
  (full ? h->slots_full : h->slots_inc) = h->slots_cur;
  return IVIT_OK;
}

int run(ivit_handle* h, const uint8_t* frames, uint16_t* out, int32_t* user_counts, bool full,
        cudaStream_t s) {
  const int SV = h->SV;
  const size_t tok_bytes = static_cast<size_t>(h->M_max) * h->D * 2;
  bool any_cold = false;
  for (int v = 0; v < SV; ++v) any_cold = any_cold || h->cold[v];
  if (h->use_graphs && (full || !any_cold)) {
    cudaGraphExec_t* exec = full ? &h->graph_full : &h->graph_inc;
    int64_t* nl = full ? &h->graph_full_launches : &h->graph_inc_launches;
    if (!*exec) {
      const int r = capture(h, full, exec, nl);
      ivit::g_stamp = nullptr;
      if (r) return r;
    }
    h->slots_last = full ? h->slots_full : h->slots_inc;
    const size_t fbytes = static_cast<size_t>(SV) * h->cfg.img_h * h->cfg.img_w * 3;
    IVIT_CK(h, cudaMemcpyAsync(h->frames_buf, frames, fbytes, cudaMemcpyDeviceToDevice, s));
    IVIT_CK(h, cudaGraphLaunch(*exec, s));
    if (out) IVIT_CK(h, cudaMemcpyAsync(out, h->tok_out, tok_bytes, cudaMemcpyDeviceToDevice, s));
    if (user_counts)
      IVIT_CK(h, cudaMemcpyAsync(user_counts, h->counts_buf, SV * sizeof(int), cudaMemcpyDeviceToDevice, s));
    h->launches = *nl;
  } else {
    const int r = run_core(h, frames, user_counts, full, s);
    ivit::g_stamp = nullptr;
    if (r) return r;
    h->slots_last = h->slots_cur;
    if (out) IVIT_CK(h, cudaMemcpyAsync(out, h->tok_out, tok_bytes, cudaMemcpyDeviceToDevice, s));
  }
  for (int v = 0; v < SV; ++v) h->cold[v] = 0;

  return IVIT_OK;
}

}  // namespace

extern "C" {

size_t ivit_weights_size(const ivit_config* cfg) {
  if (validate(cfg)) return 0;
  return weights_count(cfg);
}

int ivit_create(const ivit_config* cfg, const uint16_t* weights_bf16_host, ivit_handle** out) {
  if (!out) {
    g_create_error = "null output pointer";
    return IVIT_ERR_ARG;
  }
  *out = nullptr;
  if (const char* why = validate(cfg)) {
    g_create_error = why;
    return cfg ? IVIT_ERR_SHAPE : IVIT_ERR_ARG;
  }
  if (!weights_bf16_host) {
    g_create_error = "null weights";
    return IVIT_ERR_ARG;
  }
  ivit_handle* h = new (std::nothrow) ivit_handle();
  if (!h) {
    g_create_error = "host allocation failed";
    return IVIT_ERR_OOM;
  }
  h->cfg = *cfg;
  const int r = setup(h, weights_bf16_host);
  if (r != IVIT_OK) {
    g_create_error = h->error;
    release(h);
    delete h;
    return r;
  }
  *out = h;
  return IVIT_OK;
}

int ivit_encode_full(ivit_handle* h, const uint8_t* frames_dev, uint16_t* tokens_out_dev, void* stream) {
  if (!h) return IVIT_ERR_ARG;
  if (!frames_dev) return h->fail(IVIT_ERR_ARG, "null frames");
  return run(h, frames_dev, tokens_out_dev, nullptr, true, static_cast<cudaStream_t>(stream));
}

int ivit_encode_incremental(ivit_handle* h, const uint8_t* frames_dev, uint16_t* tokens_out_dev,
                            int32_t* changed_count_dev, void* stream) {
  if (!h) return IVIT_ERR_ARG;
  if (!frames_dev) return h->fail(IVIT_ERR_ARG, "null frames");
  // odd/even chunks (Sec. III-B): the 1st, 3rd, ... call is a full forward
  const bool full = h->cfg.schedule == IVIT_SCHED_ODD_EVEN && (h->chunk++ % 2) == 0;
  return run(h, frames_dev, tokens_out_dev, changed_count_dev, full, static_cast<cudaStream_t>(stream));
}

int ivit_get_changed(ivit_handle* h, int sv, int32_t* idx_dev, int32_t* count_dev, void* stream) {
  if (!h) return IVIT_ERR_ARG;
  if (sv < 0 || sv >= h->SV) return h->fail(IVIT_ERR_ARG, "view index out of range");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (idx_dev)
    IVIT_CK(h, cudaMemcpyAsync(idx_dev, h->idx + static_cast<size_t>(sv) * h->N, h->N * sizeof(int),
                               cudaMemcpyDeviceToDevice, s));
  if (count_dev)
    IVIT_CK(h, cudaMemcpyAsync(count_dev, h->counts + sv, sizeof(int), cudaMemcpyDeviceToDevice, s));
  return IVIT_OK;
}

int ivit_get_cache(ivit_handle* h, int which, int layer, void* dst_dev, void* stream) {
  if (!h) return IVIT_ERR_ARG;
  if (!dst_dev) return h->fail(IVIT_ERR_ARG, "null destination");
  const size_t elems = static_cast<size_t>(h->M_max) * h->D;
  const void* src = nullptr;
  size_t bytes = elems * 2;
  if (which == 0 || which == 1) {
    if (layer < 0 || layer >= h->L) return h->fail(IVIT_ERR_ARG, "layer out of range");
    src = (which == 0 ? h->cacheK : h->cacheV) + static_cast<size_t>(layer) * elems;
  } else if (which == 2) {
    src = h->tok_out;
  } else if (which == 3) {
    src = h->e_ref;
    bytes = elems * 4;
  } else if (which == 4 && h->acache) {
    if (layer < 0 || layer >= h->L) return h->fail(IVIT_ERR_ARG, "layer out of range");
    src = h->acache + static_cast<size_t>(layer) * elems;
    bytes = elems * 4;
  } else {
    return h->fail(IVIT_ERR_ARG, "bad cache selector");
  }
  IVIT_CK(h, cudaMemcpyAsync(dst_dev, src, bytes, cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream)));
  return IVIT_OK;
}

int ivit_reset(ivit_handle* h, int stream_index) {
  if (!h) return IVIT_ERR_ARG;
  if (stream_index < -1 || stream_index >= h->cfg.n_streams)
    return h->fail(IVIT_ERR_ARG, "stream index out of range");
  for (int v = 0; v < h->SV; ++v)
    if (stream_index == -1 || v / h->cfg.n_views == stream_index) h->cold[v] = 1;
  return IVIT_OK;
}

int ivit_timeline(ivit_handle* h, int enable) {
  if (!h) return IVIT_ERR_ARG;
  const bool on = enable != 0;
  if (on && !h->stamps) {
    h->stamp_cap = 512;
    IVIT_CK(h, cudaMalloc(&h->stamps, static_cast<size_t>(h->stamp_cap) * 2 * ivit::kStampCtas *
                                          sizeof(unsigned long long)));
    IVIT_CK(h, cudaMemset(h->stamps, 0, static_cast<size_t>(h->stamp_cap) * 2 * ivit::kStampCtas *
                                            sizeof(unsigned long long)));
  }
  if (on != h->timeline) {
    // the graphs are captured again, with or without the stamps
    IVIT_CK(h, cudaDeviceSynchronize());
    if (h->graph_full) cudaGraphExecDestroy(h->graph_full);
    if (h->graph_inc) cudaGraphExecDestroy(h->graph_inc);
    h->graph_full = h->graph_inc = nullptr;
    h->timeline = on;
  }
  return IVIT_OK;
}

int ivit_timeline_read(ivit_handle* h, void* stream, double* family_ms, int64_t* family_launches,
                       double* gemm_bytes_total, double* span_ms) {
  if (!h) return IVIT_ERR_ARG;
  if (!h->timeline || !h->stamps) return h->fail(IVIT_ERR_ARG, "timeline mode is off");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t n = h->slots_last.size();
  std::vector<unsigned long long> t(n * 2 * ivit::kStampCtas);
  int rows = 0;
  IVIT_CK(h, cudaMemcpyAsync(&rows, h->cu_rows + h->SV, sizeof(int), cudaMemcpyDeviceToHost, s));
  if (n) IVIT_CK(h, cudaMemcpyAsync(t.data(), h->stamps, t.size() * sizeof(unsigned long long),
                                    cudaMemcpyDeviceToHost, s));
  IVIT_CK(h, cudaStreamSynchronize(s));
  double ms[kFamilies] = {0}, bytes = 0;
  int64_t cnt[kFamilies] = {0};
  unsigned long long first = ~0ull, last = 0;
  for (size_t i = 0; i < n; ++i) {
    unsigned long long b = ~0ull, e = 0;
    for (int c = 0; c < ivit::kStampCtas; ++c) {
      const unsigned long long sb = t[(i * ivit::kStampCtas + c) * 2], se = t[(i * ivit::kStampCtas + c) * 2 + 1];
      if (sb) b = std::min(b, sb);
      if (se) e = std::max(e, se);
    }
    const TimelineSlot& sl = h->slots_last[i];
    if (b == ~0ull) continue;  // not run (another row band's body of the graph)
    ++cnt[sl.family];
    if (e > b) {
      ms[sl.family] += 1e-6 * static_cast<double>(e - b);
      first = std::min(first, b);
      last = std::max(last, e);
    }
    if (sl.family == kFamGemm) bytes += gemm_bytes(sl.n_out, sl.k, sl.kind, sl.m_static >= 0 ? sl.m_static : rows);
  }
  if (std::getenv("IVIT_DEBUG")) {  // mean launch time per family and GEMM epilogue kind
    double kms[kFamilies][8] = {};
    int kn[kFamilies][8] = {};
    for (size_t i = 0; i < n; ++i) {
      unsigned long long b = ~0ull, e = 0;
      for (int c = 0; c < ivit::kStampCtas; ++c) {
        const unsigned long long sb = t[(i * ivit::kStampCtas + c) * 2], se = t[(i * ivit::kStampCtas + c) * 2 + 1];
        if (sb) b = std::min(b, sb);
        if (se) e = std::max(e, se);
      }
      const TimelineSlot& sl = h->slots_last[i];
      const int k = std::min(7, std::max(0, sl.kind));
      if (e > b && b != ~0ull) {
        kms[sl.family][k] += 1e-3 * static_cast<double>(e - b);
        ++kn[sl.family][k];
      }
    }
    static const char* fam[kFamilies] = {"gemm", "attention", "layernorm", "other"};
    for (int f = 0; f < kFamilies; ++f)
      for (int k = 0; k < 8; ++k)
        if (kn[f][k])
          std::fprintf(stderr, "ivit timeline: %s%s%d: %d launches, %.2f us each\n", fam[f], f == kFamGemm ? " epilogue " : " ",
                       k, kn[f][k], kms[f][k] / kn[f][k]);
  }
  for (int f = 0; f < kFamilies; ++f) {
    if (family_ms) family_ms[f] = ms[f];
    if (family_launches) family_launches[f] = cnt[f];
  }
  if (gemm_bytes_total) *gemm_bytes_total = bytes;
  if (span_ms) *span_ms = last > first ? 1e-6 * static_cast<double>(last - first) : 0.0;
  return IVIT_OK;
}

int ivit_device_status(ivit_handle* h, void* stream) {
  if (!h) return IVIT_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int word = 0;
  IVIT_CK(h, cudaMemcpyAsync(&word, h->err, sizeof(int), cudaMemcpyDeviceToHost, s));
  IVIT_CK(h, cudaMemsetAsync(h->err, 0, sizeof(int), s));
  IVIT_CK(h, cudaStreamSynchronize(s));
  return word;
}

int64_t ivit_last_launch_count(const ivit_handle* h) { return h ? h->launches : 0; }

void ivit_destroy(ivit_handle* h) {
  if (!h) return;
  release(h);
  delete h;
}

const char* ivit_last_error(const ivit_handle* h) {
  return h ? h->error.c_str() : g_create_error.c_str();
}

}  // extern "C"
