// Attention of the updated queries of every view over all N keys of that view, on the
// tensor cores (Sec. III-B: attention is computed only for the updated tokens; Eq. 5:
// the keys and values of reused tokens come from the per-layer cache):
//
//   O = softmax(Q K^T / sqrt(dh)) V          per (view, head).
//
// Work item = (query tile of up to 128 packed updated rows of view v, head h).  Each
// item is handled by a thread-block cluster of `ns` CTAs that split the view's keys:
// CTA rank s takes keys [s*kpc, (s+1)*kpc), kpc = ceil(N / ns), in groups of up to 256
// keys with an online softmax across the groups.  The clusters
// walk the items with a stride; items past a view's row count (device-resident, written
// by the selection kernel) are skipped, so one launch shape serves every row count and
// the launch can sit in a CUDA graph.  Shared memory and TMEM are sized by kpc, so that
// with 64 keys per CTA an attention CTA fits on an SM beside a GEMM CTA and starts (and
// prefetches) while the QKV GEMM is still running.
//
// Per item and CTA, 128 threads (thread i <-> query row i <-> TMEM lane i) or, for key
// groups of 128 keys and more, 256: threads i and i + 128 share row i, each taking every
// other 32-key chunk of S (their partial row maxima and sums meet in shared memory) and
// every other 16-column chunk of the output, so that two warps per TMEM lane quadrant
// hide each other's latencies:
//   Q tile [128 rows][dh] by TMA (128-byte swizzle, 64-column slices; the padding columns
//   dh..round16(dh) are zeroed in shared memory); K, V of the CTA's keys by TMA into
//   [kpc keys][64 columns] slices;
//   per key group (its K/V tile fetched as soon as the previous group's one is consumed):
//   S = Q K^T   tcgen05.mma M = 128, N = the group's keys, K = round16(dh), fp32 in TMEM;
//   softmax     each thread reads its row of S from TMEM; running max m, P = 2^((S - m) c)
//               (c = log2(e) / sqrt(dh)) rounded to bf16 into shared memory as the next
//               MMA's A operand (K-major, 128-byte swizzle), l = the running sum of those
//               values;
//   O_g = P V   V is the B operand in MN-major form (its rows are the keys = the MMA's
//               K, its columns the head's dims = the MMA's N): one MMA for dims 0..63
//               and one for the rest, each inside one 64-column swizzle atom; the thread
//               folds O_g into its running output (registers), rescaled when m grows;
//   merge       every CTA stores the partial (m, l, O_s) of each row into the shared
//               memory of the row's owner CTA (distributed shared memory stores); after
//               a cluster barrier the owner combines them in rank order (deterministic):
//               M = max m_s,  O = sum_s 2^((m_s - M) c) O_s / sum_s 2^((m_s - M) c) l_s.
// Incremental calls fetch the cached K/V of the item's view before waiting on the QKV
// kernel (programmatic dependent launch: reused tokens' keys are final) and afterwards
// copy only the rows of this call's updated tokens into the swizzled tiles.
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
namespace {

constexpr int AQ = 128;            // queries per item (MMA M)
constexpr int AKMAX = 256;         // max keys per CTA (MMA N of S)
constexpr int KROWS = 64;          // rows of one K/V TMA box
constexpr int SLICE_Q = AQ * 128;  // [128 rows][128 B]: 16 KB (a Q slice or a 64-key P slice)
constexpr int QBOX = 32;           // rows of one query TMA box
constexpr int MAX_SPLITS = 8;

// Shared-memory and TMEM layout of one CTA for kpc keys and head width dhp (padded to
// 16), identical on host and device.
struct AttnLayout {
  int nt;        // threads per CTA (128 or 256)
  int nsl;       // 64-column slices per row
  int kgrp;      // keys per group: the CTA's keys, at most AKMAX (more run in several groups)
  int kpad;      // keys per group rounded up to 64 (K/V slice rows)
  int kslice;    // bytes of one K or V slice
  int rp, pst;   // merge: row slots per owner, row stride of a partial output (floats)
  int off_q, off_p, off_k, off_v, off_part, off_red, off_bar, bytes;
  int tm_o, tm_cols;
};

// Threads per CTA for kpc keys per CTA: two per query row once a key group holds 128 keys.
__host__ __device__ inline int attn_threads(int kpc) { return kpc >= 128 ? 2 * AQ : AQ; }

__host__ __device__ inline AttnLayout attn_layout(int kpc, int dhp, int ns) {
  AttnLayout L;
  L.nt = attn_threads(kpc);
  L.nsl = dhp > 64 ? 2 : 1;
  L.kgrp = kpc < AKMAX ? kpc : AKMAX;
  L.kpad = (L.kgrp + 63) / 64 * 64;
  L.kslice = L.kpad * 128;
  L.rp = (AQ + ns - 1) / ns;
  L.pst = dhp + 4;
  L.off_q = 0;
  L.off_p = L.off_q + L.nsl * SLICE_Q;
  L.off_k = L.off_p + (L.kpad / 64) * SLICE_Q;
  L.off_v = L.off_k + L.nsl * L.kslice;
  L.off_part = L.off_v + L.nsl * L.kslice;
  const int part = ns > 1 ? ns * L.rp * (L.pst + 2) * 4 : 0;  // O_s, m, l of every slot
  L.off_red = L.off_part + (part + 1023) / 1024 * 1024;
  L.off_bar = L.off_red + (L.nt > AQ ? 2 * AQ * 4 : 0);  // row max / sum exchange [2][AQ]
  L.bytes = L.off_bar + 64 + 1024;  // barriers + TMEM slot, alignment slack
  L.tm_o = L.kpad;
  int need = L.kpad + dhp, cols = 32;
  while (cols < need) cols *= 2;
  L.tm_cols = cols;
  return L;
}

// Byte offset of 16-byte chunk `chunk` (0..7) of row `row` in a slice of 128-byte rows
// written by TMA with 128-byte swizzle (slice base 1024-byte aligned).
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

struct Item {
  int v, h, r0, nq;
};

// Item s = (query tile, view, head) with the query tile slowest, so that the first
// tiles of every (view, head) are spread over the grid first.
__device__ __forceinline__ bool item_at(int s, const AttnTcArgs& a, Item& it) {
  const int vh = a.sv * a.heads;
  const int qt = s / vh, rem = s - qt * vh;
  it.v = rem / a.heads;
  it.h = rem - it.v * a.heads;
  const int rb = a.cu_rows[it.v], m = a.cu_rows[it.v + 1] - rb;
  it.r0 = rb + qt * AQ;
  it.nq = min(AQ, m - qt * AQ);
  return it.nq > 0;
}

// 2^x (the softmax's exponentials on logits pre-scaled by log2(e) / sqrt(dh)).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Running maximum of the valid entries (index < lim) of a 32-column chunk of S, in four
// independent accumulators.
__device__ __forceinline__ void chunk_max(const uint32_t (&r)[32], int lim, float (&mx)[4]) {
  if (lim >= 32) {
#pragma unroll
    for (int u = 0; u < 32; ++u) mx[u & 3] = fmaxf(mx[u & 3], __uint_as_float(r[u]));
  } else {
#pragma unroll
    for (int u = 0; u < 32; ++u)
      if (u < lim) mx[u & 3] = fmaxf(mx[u & 3], __uint_as_float(r[u]));
  }
}

// P = 2^(S c - mo) of a 32-column chunk (0 past lim), rounded to bf16 and stored as the
// row's 16-byte chunks kc0.. of the P operand (those below gns); lsum gets the rounded
// values.
__device__ __forceinline__ void chunk_exp(const uint32_t (&r)[32], int lim, float sc, float mo, uint8_t* sp,
                                          int row, int kc0, int gns, float (&lsum)[4]) {
  uint32_t pk[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) {
    const int j = 2 * u;
    const float p0 = j < lim ? ex2(fmaf(__uint_as_float(r[j]), sc, -mo)) : 0.f;
    const float p1 = j + 1 < lim ? ex2(fmaf(__uint_as_float(r[j + 1]), sc, -mo)) : 0.f;
    const __nv_bfloat162 b = __floats2bfloat162_rn(p0, p1);
    const float2 f = __bfloat1622float2(b);
    lsum[u & 3] += f.x + f.y;  // the normaliser sums the values the MMA multiplies
    pk[u] = *reinterpret_cast<const uint32_t*>(&b);
  }
#pragma unroll
  for (int q4 = 0; q4 < 4; ++q4) {
    const int kc = kc0 + q4;  // 16-byte chunk (8 keys) of this row of P
    if (kc * 8 < gns)
      *reinterpret_cast<uint4*>(sp + (kc >> 3) * SLICE_Q + swz(row, kc & 7)) =
          make_uint4(pk[4 * q4], pk[4 * q4 + 1], pk[4 * q4 + 2], pk[4 * q4 + 3]);
  }
}

template <int DHP, int NT>
__global__ void __launch_bounds__(NT, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                        const __grid_constant__ CUtensorMap tm_v, const AttnTcArgs a) {
  constexpr int NH = NT / AQ;                       // threads per query row
  constexpr int OCH = (DHP / 16 + NH - 1) / NH;     // 16-column output chunks per thread
  extern __shared__ uint8_t at_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(at_raw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  const int tid = threadIdx.x, warp = tid >> 5;
  const int row = tid & (AQ - 1), hf = tid / AQ;  // query row (TMEM lane) and column half
  const int N = a.n_tok, D = a.dim, dh = a.dh;
  const int n_items = a.sv * a.heads * a.qtiles;
  const int ns = static_cast<int>(cluster_nctarank()), rank = static_cast<int>(cluster_ctarank());
  const int cl = blockIdx.x / ns, ncl = gridDim.x / ns;
  const int kpc = (N + ns - 1) / ns;
  const int k0 = rank * kpc, nk = max(0, min(kpc, N - k0));  // this CTA's keys
  const AttnLayout L = attn_layout(kpc, DHP, ns);
  const int G = L.kgrp;                                      // keys per group
  const int ngroups = (nk + G - 1) / G;
  const int NSL = L.nsl;
  const uint32_t sb = smem_u32(sm);
  const uint32_t bq = sb + L.off_bar, bk = bq + 8, bv = bq + 16, bs = bq + 24, bo = bq + 32;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + L.off_bar + 40);
  // merge slots of the rows this CTA owns: O_s [ns][rp][pst], then m [ns][rp], l [ns][rp]
  float* po = reinterpret_cast<float*>(sm + L.off_part);
  float* pm = po + ns * L.rp * L.pst;
  float* pl = pm + ns * L.rp;
  float* red = reinterpret_cast<float*>(sm + L.off_red);  // [NH][AQ] partial row max / sum

  // The row offsets come from the selection kernel, at least two launches back (every
  // kernel of the library triggers its dependents only after its own wait).  Every CTA
  // of a cluster walks the same items, so a cluster leaves as a whole.
  int s = cl;
  Item it;
  while (s < n_items && !item_at(s, a, it)) s += ncl;
  if (s >= n_items) return;

  if (tid == 0) {
    mbar_init(bq, 1);
    mbar_init(bk, 1);
    mbar_init(bv, 1);
    mbar_init(bs, 1);
    mbar_init(bo, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), static_cast<uint32_t>(L.tm_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
  const uint32_t tm_s = tmem, tm_o = tmem + static_cast<uint32_t>(L.tm_o);
  const uint64_t pol_q = l2_policy_evict_first(), pol_kv = l2_policy_evict_last();

  // K or V of key group g of this CTA's keys of item (v, h): boxes of 64 keys x 64 dims
  // per slice.
  auto load_kv = [&](uint32_t bar, int off, const CUtensorMap* map, int v, int h, int g) {
    const int gk0 = k0 + g * G, gn = min(G, nk - g * G);
    const int nbox = (gn + KROWS - 1) / KROWS;
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(nbox * NSL * KROWS * 128));
    for (int sl = 0; sl < NSL; ++sl)
      for (int b = 0; b < nbox; ++b)
        tma_load_2d(sb + off + sl * L.kslice + b * KROWS * 128, map, h * dh + sl * 64, v * N + gk0 + b * KROWS,
                    bar, pol_kv);
  };

  // Incremental calls whose keys fit one group fetch the cached K/V before the wait.
  const bool pre = a.prefetch && ngroups == 1;
  if (pre && tid == 0) {
    load_kv(bk, L.off_k, &tm_k, it.v, it.h, 0);
    load_kv(bv, L.off_v, &tm_v, it.v, it.h, 0);
  }
  pdl_wait();  // queries and this call's K/V rows (QKV kernel) are visible from here
  pdl_launch_dependents();
  stamp_begin(a.stamp);

  uint32_t ph_q = 0, ph_g = 0;  // completed phases: bq once per item, the others once per group
  bool ok = true;
  const float sc = rsqrtf(static_cast<float>(dh)) * 1.4426950408889634f;  // log2(e) / sqrt(dh)
  bool first = true;
  while (true) {
    const bool patch = first && pre;
    first = false;
    if (tid == 0) {
      // only the 32-row boxes that hold the item's queries (rows past them are never stored)
      const int nqb = (it.nq + QBOX - 1) / QBOX;
      mbar_arrive_expect_tx(bq, static_cast<uint32_t>(NSL * nqb * QBOX * 128));
      for (int sl = 0; sl < NSL; ++sl)
        for (int b = 0; b < nqb; ++b)
          tma_load_2d(sb + L.off_q + sl * SLICE_Q + b * QBOX * 128, &tm_q, it.h * dh + sl * 64, it.r0 + b * QBOX, bq,
                      pol_q);
      if (!patch && ngroups > 0) {
        load_kv(bk, L.off_k, &tm_k, it.v, it.h, 0);
        load_kv(bv, L.off_v, &tm_v, it.v, it.h, 0);
      }
    }
    if (patch) {
      // the prefetched tiles hold the cache as it was before the QKV kernel: overwrite
      // the rows of the tokens it updated that fall in this CTA's key range
      if (!mbar_wait(bk, ph_g & 1) || !mbar_wait(bv, ph_g & 1)) ok = false;
      const int rb = a.cu_rows[it.v], m = a.cu_rows[it.v + 1] - rb;
      const int dh8 = dh >> 3;
      for (int e = tid; e < m * dh8; e += blockDim.x) {
        const int r = e / dh8, c = e - r * dh8;
        const int j = a.rowtok[rb + r] - it.v * N - k0;
        if (j < 0 || j >= nk) continue;
        const size_t g = (static_cast<size_t>(it.v) * N + k0 + j) * D + it.h * dh + c * 8;
        const uint32_t off = (c >> 3) * L.kslice + swz(j, c & 7);
        *reinterpret_cast<uint4*>(sm + L.off_k + off) = __ldcg(reinterpret_cast<const uint4*>(a.cache_k + g));
        *reinterpret_cast<uint4*>(sm + L.off_v + off) = __ldcg(reinterpret_cast<const uint4*>(a.cache_v + g));
      }
    }
    if (!mbar_wait(bq, ph_q & 1)) ok = false;
    ++ph_q;
    if (DHP != dh && tid < AQ) {  // columns dh..dh+7 of the Q tile hold the next head: zero them
      const int c = dh >> 3;
      *reinterpret_cast<uint4*>(sm + L.off_q + (c >> 3) * SLICE_Q + swz(tid, c & 7)) = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();

    // Online softmax over the key groups (running max m, running sum l, output in
    // registers rescaled by 2^((m_old - m_new) c) when the max grows).
    const bool wrow = (warp & 3) * 32 < it.nq;  // warp-uniform: padding warps skip the math
    float m_run = -INFINITY, l_run = 0.f;       // l_run: this thread's columns only
    float o_run[OCH * 16];                      // chunks hf, hf + NH, ... of the output row
#pragma unroll
    for (int d = 0; d < OCH * 16; ++d) o_run[d] = 0.f;
    for (int g = 0; g < ngroups; ++g) {
      const int gn = min(G, nk - g * G), gns = (gn + 15) & ~15;
      // ---- S = Q K^T
      if (tid == 0) {
        tc_fence_after();
        if (!mbar_wait(bk, ph_g & 1)) ok = false;
        tc_fence_after();
        if (ok) {
          const uint32_t id = idesc_bf16_f32(AQ, gns);
#pragma unroll
          for (int t = 0; t < DHP / 16; ++t) {
            const uint32_t qo = sb + L.off_q + (t >> 2) * SLICE_Q + (t & 3) * 32;
            const uint32_t ko = sb + L.off_k + (t >> 2) * L.kslice + (t & 3) * 32;
            umma_bf16(tm_s, sdesc_kmajor_sw128(qo), sdesc_kmajor_sw128(ko), id, t > 0);
          }
        }
        umma_commit(bs);
      }
      __syncwarp();
      if (!mbar_wait(bs, ph_g & 1)) ok = false;
      tc_fence_after();
      if (tid == 0 && g + 1 < ngroups) load_kv(bk, L.off_k, &tm_k, it.v, it.h, g + 1);  // K tile consumed

      // ---- softmax of the group, P to shared memory.  This thread's 32-column chunks of
      // S are cb = 32 hf, 32 (hf + NH), ...; two TMEM loads are in flight at a time.
      float alpha = 1.f;
      float mpart = -INFINITY;
      if (wrow) {
        float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        for (int cb = 32 * hf; cb < gns; cb += 64 * NH) {
          const int cb1 = cb + 32 * NH;
          uint32_t r0[32], r1[32];
          tmem_ld32_async(trow + cb, r0);
          if (cb1 < gns) tmem_ld32_async(trow + cb1, r1);
          tmem_ld_wait_regs(r0);
          chunk_max(r0, gn - cb, mx);
          if (cb1 < gns) {
            tmem_ld_wait_regs(r1);
            chunk_max(r1, gn - cb1, mx);
          }
        }
        mpart = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
      }
      if (NH > 1) {  // the row's maximum over both halves' columns
        red[hf * AQ + row] = mpart;
        __syncthreads();
        mpart = fmaxf(mpart, red[(hf ^ 1) * AQ + row]);
      }
      if (wrow) {
        const float m_new = fmaxf(m_run, mpart);
        alpha = ex2((m_run - m_new) * sc);  // 0 on the first group (m_run = -inf)
        const float mo = m_new * sc;
        float lsum[4] = {0.f, 0.f, 0.f, 0.f};
        if constexpr (NH > 1) {
          uint32_t ra[32], rb[32];
          int cb = 32 * hf;
          if (cb < gns) {
            tmem_ld32_async(trow + cb, ra);
            tmem_ld_wait_regs(ra);
          }
          while (cb < gns) {  // chunk cb is in ra; the next one loads while it is used
            const int cn = cb + 32 * NH;
            if (cn < gns) tmem_ld32_async(trow + cn, rb);
            chunk_exp(ra, gn - cb, sc, mo, sm + L.off_p, row, cb >> 3, gns, lsum);
            if (cn >= gns) break;
            tmem_ld_wait_regs(rb);
            const int cn2 = cn + 32 * NH;
            if (cn2 < gns) tmem_ld32_async(trow + cn2, ra);
            chunk_exp(rb, gn - cn, sc, mo, sm + L.off_p, row, cn >> 3, gns, lsum);
            if (cn2 >= gns) break;
            tmem_ld_wait_regs(ra);
            cb = cn2;
          }
        } else {  // one thread per row holds the whole output row: one chunk at a time
          for (int cb = 0; cb < gns; cb += 32) {
            uint32_t r[32];
            tmem_ld32_async(trow + cb, r);
            tmem_ld_wait_regs(r);
            chunk_exp(r, gn - cb, sc, mo, sm + L.off_p, row, cb >> 3, gns, lsum);
          }
        }
        l_run = l_run * alpha + ((lsum[0] + lsum[1]) + (lsum[2] + lsum[3]));
        m_run = m_new;
      }
      fence_proxy_async_shared();
      tc_fence_before();
      __syncthreads();

      // ---- O_g = P V, folded into the running output
      if (tid == 0) {
        tc_fence_after();
        if (!mbar_wait(bv, ph_g & 1)) ok = false;
        tc_fence_after();
        if (ok) {
          const uint32_t id0 = idesc_bf16_f32_bmn(AQ, DHP > 64 ? 64 : DHP);
          const uint32_t id1 = idesc_bf16_f32_bmn(AQ, DHP > 64 ? DHP - 64 : 16);
          for (int t = 0; t < gns / 16; ++t) {
            const uint64_t ad = sdesc_kmajor_sw128(sb + L.off_p + (t >> 2) * SLICE_Q + (t & 3) * 32);
            umma_bf16(tm_o, ad, sdesc_sw128(sb + L.off_v + t * 2048, 1024, 1024), id0, t > 0);
            if (DHP > 64)
              umma_bf16(tm_o + 64, ad, sdesc_sw128(sb + L.off_v + L.kslice + t * 2048, 1024, 1024), id1, t > 0);
          }
        }
        umma_commit(bo);
      }
      __syncwarp();
      if (!mbar_wait(bo, ph_g & 1)) ok = false;
      tc_fence_after();
      ++ph_g;
      if (tid == 0 && g + 1 < ngroups) load_kv(bv, L.off_v, &tm_v, it.v, it.h, g + 1);  // V tile consumed
      if (wrow) {  // warp-uniform: tcgen05.ld is a warp-collective instruction
        // two chunks' loads in flight per wait (one for the widest heads with two threads
        // per row, whose registers are otherwise spent)
        constexpr int OB = (DHP >= 112 && NH > 1) ? 1 : 2;
#pragma unroll
        for (int q = 0; q < OCH; q += OB) {
          uint32_t ov[OB][16];
#pragma unroll
          for (int t = 0; t < OB; ++t)
            if (q + t < OCH && (hf + (q + t) * NH) * 16 < DHP)
              tmem_ld16_async(trow + L.tm_o + (hf + (q + t) * NH) * 16, ov[t]);
          tmem_ld_wait();
#pragma unroll
          for (int t = 0; t < OB; ++t) {
            tmem_regs_after_wait16(ov[t]);
            if (q + t < OCH && (hf + (q + t) * NH) * 16 < DHP) {
#pragma unroll
              for (int u = 0; u < 16; ++u)
                o_run[(q + t) * 16 + u] = o_run[(q + t) * 16 + u] * alpha + __uint_as_float(ov[t][u]);
            }
          }
        }
      }
    }

    // next item of this cluster (the same for every rank)
    int s_next = s + ncl;
    Item nxt;
    while (s_next < n_items && !item_at(s_next, a, nxt)) s_next += ncl;

    if (NH > 1) {  // the row's sum over both halves' columns (the same order on both)
      red[hf * AQ + row] = l_run;
      __syncthreads();
      const float lo_ = red[row], hi_ = red[AQ + row];
      l_run = lo_ + hi_;
    }
    if (ns == 1) {
      if (wrow && row < it.nq) {
        const float inv = 1.f / l_run;
        bf16* orow = a.o + static_cast<size_t>(it.r0 + row) * D + it.h * dh;
#pragma unroll
        for (int q = 0; q < OCH; ++q) {
#pragma unroll
          for (int h8 = 0; h8 < 16; h8 += 8) {
            const int c = (hf + q * NH) * 16 + h8;
            if (c < dh) {
              uint4 u;
              uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const __nv_bfloat162 b = __floats2bfloat162_rn(o_run[q * 16 + h8 + 2 * e] * inv,
                                                               o_run[q * 16 + h8 + 2 * e + 1] * inv);
                w[e] = *reinterpret_cast<const uint32_t*>(&b);
              }
              *reinterpret_cast<uint4*>(orow + c) = u;
            }
          }
        }
      }
    } else {
      // push this CTA's partial (m, l, O_s) of row i to slot [rank][i - owner * rpi] of
      // the owner CTA i / rpi; a CTA without keys pushes m = -inf, l = 0, O = 0
      const int rpi = (it.nq + ns - 1) / ns;  // rows per owner in this item (<= rp)
      if (row < it.nq) {
        const int owner = row / rpi, slot = row - owner * rpi;
        const uint32_t obase =
            mapa_shared(smem_u32(po + (rank * L.rp + slot) * L.pst), static_cast<uint32_t>(owner));
#pragma unroll
        for (int q = 0; q < OCH; ++q) {
          const int c0 = (hf + q * NH) * 16;
          if (c0 < DHP) {
#pragma unroll
            for (int c = 0; c < 16; c += 4)
              st_dsmem_f32x4(obase + 4 * (c0 + c), make_float4(o_run[q * 16 + c], o_run[q * 16 + c + 1],
                                                               o_run[q * 16 + c + 2], o_run[q * 16 + c + 3]));
          }
        }
        if (hf == 0) {
          st_dsmem_f32(mapa_shared(smem_u32(pm + rank * L.rp + slot), static_cast<uint32_t>(owner)), m_run);
          st_dsmem_f32(mapa_shared(smem_u32(pl + rank * L.rp + slot), static_cast<uint32_t>(owner)), l_run);
        }
      }
      cluster_sync();  // every rank's partials of this CTA's rows are in its shared memory
      const int lo = rank * rpi, nmine = max(0, min(it.nq, lo + rpi) - lo);
      constexpr int C8 = DHP / 8;
      for (int e = tid; e < nmine * C8; e += blockDim.x) {
        const int sl = e / C8, c = e - sl * C8;
        if (c * 8 >= dh) continue;
        float M = -INFINITY;
#pragma unroll
        for (int q = 0; q < MAX_SPLITS; ++q)
          if (q < ns) M = fmaxf(M, pm[q * L.rp + sl]);
        float Lsum = 0.f, acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < MAX_SPLITS; ++q) {
          if (q < ns) {
            const float w = ex2((pm[q * L.rp + sl] - M) * sc);  // m = -inf (no keys): w = 0
            Lsum += w * pl[q * L.rp + sl];
            const float4 x0 = *reinterpret_cast<const float4*>(po + (q * L.rp + sl) * L.pst + c * 8);
            const float4 x1 = *reinterpret_cast<const float4*>(po + (q * L.rp + sl) * L.pst + c * 8 + 4);
            acc[0] += w * x0.x;
            acc[1] += w * x0.y;
            acc[2] += w * x0.z;
            acc[3] += w * x0.w;
            acc[4] += w * x1.x;
            acc[5] += w * x1.y;
            acc[6] += w * x1.z;
            acc[7] += w * x1.w;
          }
        }
        const float inv = 1.f / Lsum;
        uint4 u;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const __nv_bfloat162 b = __floats2bfloat162_rn(acc[2 * q] * inv, acc[2 * q + 1] * inv);
          w[q] = *reinterpret_cast<const uint32_t*>(&b);
        }
        *reinterpret_cast<uint4*>(a.o + static_cast<size_t>(it.r0 + lo + sl) * D + it.h * dh + c * 8) = u;
      }
      if (s_next < n_items) cluster_sync();  // slots are read before the next item's pushes
    }
    tc_fence_before();
    __syncthreads();  // Q, P and TMEM are reused by the next item

    if (s_next >= n_items) break;
    s = s_next;
    it = nxt;
  }

  if (!ok) atomicExch(a.err, kErrWaitTmaFull);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, static_cast<uint32_t>(L.tm_cols));
  stamp_end(a.stamp);
}

template <int DHP>
cudaError_t launch_dhp(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                       const AttnTcArgs& a, int grid, int smem, int nt, cudaStream_t s) {
  if (nt > AQ)
    return launch_ex(attention_tc_kernel<DHP, 2 * AQ>, dim3(grid), dim3(nt), static_cast<size_t>(smem), s,
                     static_cast<unsigned>(a.key_splits), tm_q, tm_k, tm_v, a);
  return launch_ex(attention_tc_kernel<DHP, AQ>, dim3(grid), dim3(nt), static_cast<size_t>(smem), s,
                   static_cast<unsigned>(a.key_splits), tm_q, tm_k, tm_v, a);
}

// The device's opt-in limit of dynamic shared memory per block (0 when unknown).
int smem_optin() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
  return v;
}

}  // namespace

int attention_tc_kv_box_rows() { return KROWS; }

size_t attention_tc_smem(int n_tok, int dh, int key_splits) {
  const int kpc = (n_tok + key_splits - 1) / key_splits;
  return static_cast<size_t>(attn_layout(kpc, (dh + 15) & ~15, key_splits).bytes);
}

cudaError_t attention_tc_setup() {
  const int max_bytes = smem_optin();
  if (max_bytes <= 0) return cudaErrorInvalidDevice;
  cudaError_t e = cudaSuccess;
  auto set = [&](auto kern) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, max_bytes);
  };
  set(attention_tc_kernel<16, AQ>);
  set(attention_tc_kernel<16, 2 * AQ>);
  set(attention_tc_kernel<32, AQ>);
  set(attention_tc_kernel<32, 2 * AQ>);
  set(attention_tc_kernel<48, AQ>);
  set(attention_tc_kernel<48, 2 * AQ>);
  set(attention_tc_kernel<64, AQ>);
  set(attention_tc_kernel<64, 2 * AQ>);
  set(attention_tc_kernel<80, AQ>);
  set(attention_tc_kernel<80, 2 * AQ>);
  set(attention_tc_kernel<96, AQ>);
  set(attention_tc_kernel<96, 2 * AQ>);
  set(attention_tc_kernel<112, AQ>);
  set(attention_tc_kernel<112, 2 * AQ>);
  set(attention_tc_kernel<128, AQ>);
  set(attention_tc_kernel<128, 2 * AQ>);
  return e;
}

cudaError_t launch_attention_tc(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                                const AttnTcArgs& a, int max_ctas, cudaStream_t s) {
  const int ns = a.key_splits;
  if (ns < 1 || ns > MAX_SPLITS) return cudaErrorInvalidValue;
  const int items = a.sv * a.heads * a.qtiles;
  const int clusters = max(1, min(items, max_ctas / ns));
  const int grid = clusters * ns;
  const int smem = static_cast<int>(attention_tc_smem(a.n_tok, a.dh, ns));
  if (smem > smem_optin()) return cudaErrorInvalidValue;
  const int nt = attn_threads((a.n_tok + ns - 1) / ns);
  switch ((a.dh + 15) & ~15) {
    case 16: return launch_dhp<16>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 32: return launch_dhp<32>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 48: return launch_dhp<48>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 64: return launch_dhp<64>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 80: return launch_dhp<80>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 96: return launch_dhp<96>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 112: return launch_dhp<112>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    case 128: return launch_dhp<128>(tm_q, tm_k, tm_v, a, grid, smem, nt, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace ivit
