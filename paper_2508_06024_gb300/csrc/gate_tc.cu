// Gate of the layer path on the sm_103a tensor cores (Eq. 4-7 gate, Top-k
// and the fused routing reservations); the SIMT gates and the dispatch are in
// gate.cu.
#include <stdlib.h>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include "common.cuh"
#include "gate_common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace ec2moe {

__device__ unsigned int g_gate_error;  // bit 0: a bounded wait of the tensor-core gate timed out

namespace gatek {
namespace {

// ---------------------------------------------------------------------------
// Gate on the tensor cores (bf16 activations, O = E + K <= 80 gate rows).
//
// The logits are the contraction X_tile W^T with W the fp32 gate rows.  Each
// fp32 weight is split exactly into three bf16 terms, w = w0 + w1 + w2 (w0 =
// bf16(w), w1 = bf16(w - w0), w2 = bf16(w - w0 - w1); every difference is
// exact in fp32, and the remainder is below 2^-24 |w|).  A bf16 activation
// times a bf16 term is exact in fp32, so X W^T = X w0^T + X w1^T + X w2^T keeps
// the fp32 weights to fp32 accuracy.  The three terms are stacked as the rows
// of one B operand [w0; w1; w2] (N = 3 * O_pad, O_pad = O rounded up to 16),
// so one tcgen05.mma per 16 columns of d_model produces all three partial
// products side by side in TMEM; the epilogue adds them in fp32.
//
// One CTA owns 128-token tiles; d_model streams through shared memory 64
// columns per stage:
//   warp 0       TMA: the X box (128 x 64 bf16, 128-byte swizzle) and the
//                stacked split rows of the stage -- either straight from a
//                prepared [3 * O_pad, d] bf16 matrix (PREP: made by
//                gate_split_kernel), or as raw fp32 rows (O x 64, unswizzled)
//                that warps 6..13 split into the swizzled layout;
//   warp 1       4 MMAs (M = 128, N = 3 O_pad, K = 16) per stage into one of
//                two TMEM accumulators; every GC_SEG stages (256 columns of
//                d_model) the accumulator is handed over and the next segment
//                starts from zero in the other one;
//   warps 2..5   add each segment into fp32 registers (one token row per
//                thread; warp w reads TMEM lanes 32 (w % 4) .. +31), so every
//                dot product is a sum of short partial sums; at the end of the
//                tile add the bias and take the token's softmax / Top-k
//                decision (decide_token_thread);
//   warps 2..13  on the layer path, reserve the tile's rows per expert.
// With d_model of 2048 or more (32 or more stages per tile) a tile belongs to
// a cluster of GC_CS CTAs on as many SMs instead: CTA c of the cluster runs
// the stages [c nk / GC_CS, (c + 1) nk / GC_CS) and owns the decisions of
// rows [c 128 / GC_CS, (c + 1) 128 / GC_CS).  Each drain thread sends its
// row's partial logits to the row's owner (st.async into the owner's shared
// memory, counted on the owner's receive barrier), and the owner adds the
// cluster's partials in CTA order before the bias and the decision; every CTA
// reserves the rows it decided.  One tile per cluster: such grids are one
// cluster per tile, run in waves when they exceed the SMs.  A tile's stages
// (the stream of X, the MMAs and the accumulator drains) are then spread over
// twice the SMs.
// Every mbarrier wait is bounded; on a timeout the error word is set, copies
// and MMAs in flight are drained and the CTA finishes its tiles without
// waiting (the decisions then see garbage logits but still name valid experts).
constexpr int GC_BM = 128;
constexpr int GC_BK = 64;
constexpr int GC_SEG = 4;
constexpr int GC_MAX_O = 80;
constexpr int GC_MAX_STAGES = 10;
constexpr int GC_THREADS = 448;
constexpr int GC_WORKERS = 384;     // warps 2..13
constexpr int GC_ACC_STRIDE = 256;  // TMEM columns between the two accumulators (3 * O_pad <= 240 each)
constexpr int GC_CS = 2;            // CTAs per tile (cluster) when d_model is split
constexpr int GC_SPLIT_MIN_NK = 32; // stages per tile from which d_model is split

struct GcLayout {
  int n_pad, O, k, E, stages, cs;
  int stage_bytes, w3_off, raw_off;
  int log_stride;  // logits row of a token: O logits + 16 group scratch words, odd (conflict-free rows)
  int rstride;     // floats per received partial-logit row: n_pad + 4 (16-byte rows, shifted banks)
  int log_off, idx_off, tab_off, base_off, bias_off, recv_off, bar_off, total;
  __host__ __device__ GcLayout(int O_, int k_, int E_, int stages_, bool prep, int cs_)
      : O(O_), k(k_), E(E_), stages(stages_), cs(cs_) {
    n_pad = (O + 15) / 16 * 16;
    w3_off = GC_BM * GC_BK * 2;
    raw_off = w3_off + 3 * n_pad * 128;
    stage_bytes = raw_off + (prep ? 0 : n_pad * 256);  // a multiple of 1024
    log_stride = (O + 16) | 1;
    rstride = n_pad + 4;
    log_off = stages * stage_bytes;
    idx_off = log_off + GC_BM * log_stride * 4;
    tab_off = idx_off + GC_BM * k * 4;
    base_off = tab_off + (GC_BM * k / 32) * E * 4;
    bias_off = base_off + 4 * E;
    // received partials: [source CTA][owned row][rstride] (cs > 1)
    recv_off = (bias_off + 4 * O + 15) / 16 * 16;
    bar_off = (recv_off + (cs > 1 ? GC_BM * rstride * 4 : 0) + 7) / 8 * 8;
    total = bar_off + (3 * stages + 6) * 8 + 16;
  }
};

struct GcParams {
  KParams kp;
  int n_pad;
  int stages;
  int cs;  // CTAs per tile (cluster size); 1 = one CTA per tile, persistent over tiles
  long long timeout;
};

// One token's decision by one thread, from its logits row L[0..E) (local),
// L[E..E+K) (global) and a scratch row G[0..K) -- the arithmetic of
// decide_token_warp with sequential sums: per-group log-sum-exp over the
// allowed members (Eq. 5), top-group pruning when top_groups > 0 (only the
// top_groups live groups by m stay), log-sum-exp of the global logits over the
// live (kept) groups (Eq. 6), key = (m_g - lse_g) + l_i (K = 1: l_i), weight
// exp((m_g - LSE_m) + (l_i - lse_g)) (Eq. 7); Top-k by insertion into a sorted list (larger key
// first, ties to the lower index).  Slots left empty by non-finite keys take
// the lowest allowed experts not chosen yet.  The mask words are in
// registers, so the loads of one pass are independent of each other.
struct MaskRegs {
  uint32_t w0, w1, w2, w3;
  __device__ __forceinline__ bool has(int e) const {
    const uint32_t w = e < 64 ? (e < 32 ? w0 : w1) : (e < 96 ? w2 : w3);
    return (w >> (e & 31)) & 1u;
  }
};

// Insert (key, e, lw) into a list sorted by key (descending); e arrives in
// ascending order, so an equal key stays behind the earlier expert.
template <int KS>
__device__ __forceinline__ void topk_insert(float* tk, float* tl, int* ti, float key, int e, float lw) {
#pragma unroll
  for (int q = KS - 1; q >= 0; --q) {
    if (key > tk[q]) {
      if (q > 0 && key > tk[q - 1]) {
        tk[q] = tk[q - 1];
        tl[q] = tl[q - 1];
        ti[q] = ti[q - 1];
      } else {
        tk[q] = key;
        tl[q] = lw;
        ti[q] = e;
      }
    }
  }
}

// KS >= k slots are kept (KS in {1, 2, 4, 8}).
template <int KS>
__device__ void decide_token_thread(int E, int K, int k, int renorm, int top_groups, const MaskRegs m, const float* L,
                                    float* G, int32_t* topk_idx, float* topk_w, int tok, int* s_idx) {
  const bool grouped = K > 1;
  const int ng = grouped ? K : 1;
  const int gsize = E / ng;
  float tk[KS], tl[KS];
  int ti[KS];
#pragma unroll
  for (int j = 0; j < KS; ++j) {
    tk[j] = -CUDART_INF_F;
    tl[j] = 0.0f;
    ti[j] = -1;
  }
  float lse_m = 0.0f;
  if (!grouped) {
    // one group: the keys are the logits themselves, so Top-k rides on the max pass
    float mx = -CUDART_INF_F;
#pragma unroll 1
    for (int e = 0; e < E; ++e) {
      if (!m.has(e)) continue;
      const float le = L[e];
      mx = fmaxf(mx, le);
      if (le > tk[KS - 1]) topk_insert<KS>(tk, tl, ti, le, e, le);
    }
    float sum = 0.0f;
#pragma unroll 1
    for (int e = 0; e < E; ++e)
      if (m.has(e)) sum += expf(L[e] - mx);
    G[0] = mx + logf(sum);
#pragma unroll
    for (int j = 0; j < KS; ++j) tl[j] -= G[0];
  } else {
    float mxm = -CUDART_INF_F;
#pragma unroll 1
    for (int g = 0; g < ng; ++g) {
      const int lo = g * gsize, hi = lo + gsize;
      float mx = -CUDART_INF_F;
#pragma unroll 4
      for (int e = lo; e < hi; ++e)
        if (m.has(e)) mx = fmaxf(mx, L[e]);
      float sum = 0.0f;
#pragma unroll 4
      for (int e = lo; e < hi; ++e)
        if (m.has(e)) sum += expf(L[e] - mx);
      G[g] = mx > -CUDART_INF_F ? mx + logf(sum) : -CUDART_INF_F;
    }
    // top-group pruning: only the top_groups live groups by m (ties to the
    // lower group index) keep their experts and their share of p_group
    if (top_groups > 0 && top_groups < ng) {
      uint32_t keep = 0;
#pragma unroll 1
      for (int g = 0; g < ng; ++g) {
        if (G[g] == -CUDART_INF_F) continue;
        const float mg = L[E + g];
        int rank = 0;
#pragma unroll 1
        for (int j = 0; j < ng; ++j) {
          const float mj = L[E + j];
          if (j != g && G[j] > -CUDART_INF_F && (mj > mg || (mj == mg && j < g))) ++rank;
        }
        if (rank < top_groups) keep |= 1u << g;
      }
#pragma unroll 1
      for (int g = 0; g < ng; ++g)
        if (!((keep >> g) & 1u)) G[g] = -CUDART_INF_F;
    }
#pragma unroll 1
    for (int g = 0; g < ng; ++g)
      if (G[g] > -CUDART_INF_F) mxm = fmaxf(mxm, L[E + g]);
    float summ = 0.0f;
#pragma unroll 1
    for (int g = 0; g < K; ++g)
      if (G[g] > -CUDART_INF_F) summ += expf(L[E + g] - mxm);
    lse_m = mxm + logf(summ);
#pragma unroll 1
    for (int g = 0; g < ng; ++g) {
      const float lg = G[g];
      if (lg == -CUDART_INF_F) continue;  // no allowed member, or pruned
      const float mk = L[E + g];
      const int lo = g * gsize, hi = lo + gsize;
#pragma unroll 2
      for (int e = lo; e < hi; ++e) {
        const float le = L[e];
        const float key = (mk - lg) + le;
        if (m.has(e) && key > tk[KS - 1]) topk_insert<KS>(tk, tl, ti, key, e, (mk - lse_m) + (le - lg));
      }
    }
  }
  // non-finite keys: fill empty slots with the lowest allowed experts not chosen
  int next = 0;
#pragma unroll
  for (int s = 0; s < KS; ++s) {
    if (s < k && ti[s] < 0) {
#pragma unroll 1
      for (; next < E; ++next) {
        if (!m.has(next)) continue;
        bool used = false;
#pragma unroll
        for (int q = 0; q < KS; ++q) used |= (ti[q] == next);
        if (!used) break;
      }
      const int e = next < E ? next : 0;
      ++next;
      const int g = e / gsize;
      ti[s] = e;
      tl[s] = grouped ? (L[E + g] - lse_m) + (L[e] - G[g]) : L[e] - G[0];
    }
  }
  float gw[KS];
  float wsum = 0.0f;
#pragma unroll
  for (int s = 0; s < KS; ++s) {
    gw[s] = s < k ? expf(tl[s]) : 0.0f;
    wsum += gw[s];
  }
#pragma unroll
  for (int s = 0; s < KS; ++s)
    if (s < k) {
      topk_idx[(size_t)tok * k + s] = ti[s];
      topk_w[(size_t)tok * k + s] = renorm ? gw[s] / wsum : gw[s];
      if (s_idx) s_idx[s] = ti[s];
    }
}

// The same decision for K = 1 from the logits in registers (x[o] for o < E,
// bias included), fully unrolled so the mask tests are compile-time bit
// selects and the exponentials are independent: key = l_i, weight
// exp(l_i - lse) with lse the log-sum-exp of the allowed logits.
template <int NB, int KS>
__device__ __forceinline__ void decide_k1_regs(const float (&x)[NB][16], int E, int k, int renorm, const MaskRegs m,
                                               int32_t* topk_idx, float* topk_w, int tok, int* s_idx) {
  float tk[KS], tl[KS];
  int ti[KS];
#pragma unroll
  for (int j = 0; j < KS; ++j) {
    tk[j] = -CUDART_INF_F;
    tl[j] = 0.0f;
    ti[j] = -1;
  }
  float mx = -CUDART_INF_F;
#pragma unroll
  for (int b = 0; b < NB; ++b)
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int e = b * 16 + j;
      if (e < E && m.has(e)) {
        mx = fmaxf(mx, x[b][j]);
        if (x[b][j] > tk[KS - 1]) topk_insert<KS>(tk, tl, ti, x[b][j], e, x[b][j]);
      }
    }
  float sum = 0.0f;
#pragma unroll
  for (int b = 0; b < NB; ++b)
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int e = b * 16 + j;
      if (e < E && m.has(e)) sum += expf(x[b][j] - mx);
    }
  const float lse = mx + logf(sum);
  // non-finite logits: fill empty slots with the lowest allowed experts not chosen
#pragma unroll
  for (int s = 0; s < KS; ++s) {
    if (s < k && ti[s] < 0) {
      int pick = -1;
      float lp = 0.0f;
#pragma unroll
      for (int b = NB - 1; b >= 0; --b)
#pragma unroll
        for (int j = 15; j >= 0; --j) {
          const int e = b * 16 + j;
          bool used = false;
#pragma unroll
          for (int q = 0; q < KS; ++q) used |= (ti[q] == e);
          if (e < E && m.has(e) && !used) {
            pick = e;
            lp = x[b][j];
          }
        }
      ti[s] = pick < 0 ? 0 : pick;
      tl[s] = lp;
    }
  }
  float gw[KS];
  float wsum = 0.0f;
#pragma unroll
  for (int s = 0; s < KS; ++s) {
    gw[s] = s < k ? expf(tl[s] - lse) : 0.0f;
    wsum += gw[s];
  }
#pragma unroll
  for (int s = 0; s < KS; ++s)
    if (s < k) {
      topk_idx[(size_t)tok * k + s] = ti[s];
      topk_w[(size_t)tok * k + s] = renorm ? gw[s] / wsum : gw[s];
      if (s_idx) s_idx[s] = ti[s];
    }
}

// Rows [row_lo, row_lo + n_rows) of the tile reserved per expert (the layer
// path), with the worker warps only: entry i of the range (token row_lo + i /
// k of the tile, slot i % k) gets route_rel = the expert's reserved base + the
// number of earlier entries of the range with the same expert.  sIdx holds the
// range's decisions.  32-entry chunks are ranked with a warp match, chunk
// counts are turned into per-expert prefixes, and one atomicAdd per expert
// reserves the range's rows.
__device__ void route_tile_workers(const KParams& p, int tile, int row_lo, int n_rows, const int* sIdx, int* sTab,
                                   int* s_base, int wt) {
  const int wi = wt >> 5, lane = wt & 31;
  const int nt = n_rows * p.k;
  const long long e0 = ((long long)tile * GC_BM + row_lo) * p.k;
  const long long n = (long long)p.T * p.k;
  const long long rem = n - e0;
  const int live = rem <= 0 ? 0 : (int)(rem < nt ? rem : nt);
  const int nch = (live + 31) / 32;
  constexpr int NW = GC_WORKERS / 32;
  constexpr int MAXC = (GC_BM * MAX_TOPK / 32 + NW - 1) / NW;
  for (int i = wt; i < nch * p.E; i += GC_WORKERS) sTab[i] = 0;
  asm volatile("bar.sync 1, %0;" ::"r"(GC_WORKERS) : "memory");
  int rank[MAXC], ex[MAXC];
#pragma unroll
  for (int ci = 0; ci < MAXC; ++ci) {
    const int c = wi + ci * NW;
    const int i = c * 32 + lane;
    int e = -1;
    if (c < nch && i < live) {
      e = sIdx[i];
      if (e < 0 || e >= p.E) e = -1;
    }
    ex[ci] = e;
    rank[ci] = 0;
    if (c < nch) {
      const unsigned m = __match_any_sync(0xffffffffu, e);
      rank[ci] = __popc(m & ((1u << lane) - 1u));
      if (e >= 0 && lane == __ffs(m) - 1) sTab[c * p.E + e] = __popc(m);
    }
  }
  asm volatile("bar.sync 1, %0;" ::"r"(GC_WORKERS) : "memory");
  if (wt < p.E) {
    int run = 0;
    for (int c = 0; c < nch; ++c) {
      const int t = sTab[c * p.E + wt];
      sTab[c * p.E + wt] = run;
      run += t;
    }
    s_base[wt] = run ? atomicAdd(&p.route_counts[wt], run) : 0;
  }
  asm volatile("bar.sync 1, %0;" ::"r"(GC_WORKERS) : "memory");
#pragma unroll
  for (int ci = 0; ci < MAXC; ++ci) {
    const int c = wi + ci * NW;
    const int e = ex[ci];
    if (c < nch && e >= 0) p.route_rel[e0 + c * 32 + lane] = s_base[e] + sTab[c * p.E + e] + rank[ci];
  }
}

// The three bf16 terms of one fp32 pair, packed as bf16x2 words.
__device__ __forceinline__ void split3_pair(float lo, float hi, uint32_t& t0, uint32_t& t1, uint32_t& t2) {
  t0 = pack_bf16x2(lo, hi);
  const float lo1 = lo - bf16_lo(t0), hi1 = hi - bf16_hi(t0);
  t1 = pack_bf16x2(lo1, hi1);
  const float lo2 = lo1 - bf16_lo(t1), hi2 = hi1 - bf16_hi(t1);
  t2 = pack_bf16x2(lo2, hi2);
}

// Prepared split rows for the layer path: Wsplit[j * O_pad + o][c] = term j
// of W[o][c] (local rows, then global rows; rows O..O_pad-1 zero), bf16
// [3 * O_pad, d].  Block 0 also clears the expert row counters the gate's
// routing reserves from.  Thread = 8 consecutive columns of one gate row.
__global__ void __launch_bounds__(256) gate_split_kernel(const float* W_local, const float* W_global, int E, int K,
                                                         int d, int n_pad, __nv_bfloat16* Wsplit,
                                                         int32_t* route_counts) {
  pdl_trigger();
  const int O = E + (K == 1 ? 0 : K);
  if (blockIdx.x == 0 && route_counts)
    for (int e = threadIdx.x; e < E; e += blockDim.x) route_counts[e] = 0;
  const int per_row = d / 8;
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)n_pad * per_row) return;
  const int o = (int)(i / per_row);
  const int c = (int)(i % per_row) * 8;
  float v[8];
  if (o < O) {
    const float* src = o < E ? W_local + (size_t)o * d : W_global + (size_t)(o - E) * d;
    load8(src + c, v);
  } else {
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = 0.0f;
  }
  uint32_t t[3][4];
#pragma unroll
  for (int u = 0; u < 4; ++u) split3_pair(v[2 * u], v[2 * u + 1], t[0][u], t[1][u], t[2][u]);
#pragma unroll
  for (int j = 0; j < 3; ++j)
    *reinterpret_cast<U4*>(Wsplit + ((size_t)j * n_pad + o) * d + c) = U4{t[j][0], t[j][1], t[j][2], t[j][3]};
}

template <int NB, bool PREP>
__global__ void __launch_bounds__(GC_THREADS, 1)
    gate_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                   const __grid_constant__ CUtensorMap tmWg, const __grid_constant__ GcParams gp) {
  using namespace tc;
  const KParams& p = gp.kp;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nglob = (p.K == 1) ? 0 : p.K;
  const int O = p.E + nglob;
  const int cs = gp.cs;
  const GcLayout L(O, p.k, p.E, gp.stages, PREP, cs);
  const int S = gp.stages;
  float* sLog = reinterpret_cast<float*>(smem + L.log_off);
  int* sIdx = reinterpret_cast<int*>(smem + L.idx_off);
  int* sTab = reinterpret_cast<int*>(smem + L.tab_off);
  int* s_base = reinterpret_cast<int*>(smem + L.base_off);
  float* s_bias = reinterpret_cast<float*>(smem + L.bias_off);
  float* s_recv = reinterpret_cast<float*>(smem + L.recv_off);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bar_off);
  uint64_t* conv = full + S;
  uint64_t* empty = conv + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* recvb = drain + 1;  // partial logits from the other CTAs of the cluster (cs > 1)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(recvb + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_tiles = (p.T + GC_BM - 1) / GC_BM;
  const int nk = (p.d + GC_BK - 1) / GC_BK;
  const long long budget = gp.timeout;
  const int n_pad = gp.n_pad;
  // cs > 1: cluster `tile` of cs CTAs (one tile per cluster); this CTA runs
  // stages [kb_lo, kb_lo + cnt) and decides rows [rank * rows_own, ...)
  const int rank = cs > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int tile_first = cs > 1 ? static_cast<int>(cluster_id_x()) : static_cast<int>(blockIdx.x);
  const int tile_step = cs > 1 ? static_cast<int>(cluster_count_x()) : static_cast<int>(gridDim.x);
  const int kb_lo = rank * nk / cs;
  const int cnt = (rank + 1) * nk / cs - kb_lo;
  const int rows_own = GC_BM / cs;
  pdl_trigger();

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&conv[s]), 8);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4);
    }
    mbar_init(smem_u32(drain), 1);
    mbar_init(smem_u32(recvb), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // the owned rows' partials of the other cs - 1 CTAs (one tile per cluster)
    if (cs > 1) mbar_expect_tx(smem_u32(recvb), static_cast<uint32_t>((cs - 1) * rows_own * n_pad * 4));
  }
  for (int o = threadIdx.x - 64; o >= 0 && o < O; o += GC_THREADS - 64)
    s_bias[o] = o < p.E ? p.b_local[o] : p.b_global[o - p.E];
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
    if (!PREP && nglob) tma_prefetch_desc(&tmWg);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  // every receive barrier of the cluster is initialised before any partial is sent
  if (cs > 1) cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // Activations do not depend on the previous kernel, the prepared split
    // rows (PREP) do: the X boxes of the first stages go out before the
    // dependency wait, their split rows after it.
    if (lane == 0) {
      const uint32_t xbytes = GC_BM * GC_BK * 2;
      const uint32_t wbytes = PREP ? 3 * n_pad * GC_BK * 2 : O * GC_BK * 4;
      const int my_tiles = tile_first < n_tiles ? (n_tiles - 1 - tile_first) / tile_step + 1 : 0;
      const int total = my_tiles * cnt;
      const int pre = PREP ? (total < S ? total : S) : 0;
      auto load_w = [&](int c, uint8_t* st, uint32_t fb) {
        const int kc = kb_lo + c % cnt;
        if (PREP) {
          tma_load_2d(smem_u32(st + L.w3_off), &tmW, kc * GC_BK, 0, fb);
        } else {
          tma_load_2d(smem_u32(st + L.raw_off), &tmW, kc * GC_BK, 0, fb);
          if (nglob) tma_load_2d(smem_u32(st + L.raw_off + p.E * GC_BK * 4), &tmWg, kc * GC_BK, 0, fb);
        }
      };
      for (int c = 0; c < pre; ++c) {
        const uint32_t fb = smem_u32(&full[c]);
        mbar_expect_tx(fb, xbytes + wbytes);
        tma_load_2d(smem_u32(smem + c * L.stage_bytes), &tmX, (kb_lo + c % cnt) * GC_BK,
                    (tile_first + (c / cnt) * tile_step) * GC_BM, fb);
      }
      pdl_wait();
      for (int c = 0; c < pre; ++c) load_w(c, smem + c * L.stage_bytes, smem_u32(&full[c]));
      int stage = pre % S;
      uint32_t phase = (pre == S) ? 1u : 0u;
      uint32_t issued = pre ? ((1u << pre) - 1u) : 0u, issued_phase = 0;
      bool ok = true;
      for (int c = pre; c < total; ++c) {
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, budget, abort_flag, &g_gate_error)) {
          ok = false;
          break;
        }
        uint8_t* st = smem + stage * L.stage_bytes;
        const uint32_t fb = smem_u32(&full[stage]);
        mbar_expect_tx(fb, xbytes + wbytes);
        tma_load_2d(smem_u32(st), &tmX, (kb_lo + c % cnt) * GC_BK, (tile_first + (c / cnt) * tile_step) * GC_BM,
                    fb);
        load_w(c, st, fb);
        issued |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == S) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok || *abort_flag) {
        for (int s = 0; s < S; ++s)
          if (issued & (1u << s)) mbar_drain(smem_u32(&full[s]), (issued_phase >> s) & 1u, DRAIN_CYCLES);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(GC_BM, 3 * n_pad);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t uses0 = 0, uses1 = 0;
      bool ok = true, any = false;
      for (int tile = tile_first; tile < n_tiles && ok; tile += tile_step) {
        for (int seg = 0; seg < cnt && ok; seg += GC_SEG) {
          const uint32_t uses = acc ? uses1 : uses0;
          if (!mbar_wait(smem_u32(&tempty[acc]), (uses & 1u) ^ 1u, budget, abort_flag, &g_gate_error)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * GC_ACC_STRIDE;
          const int seg_end = seg + GC_SEG < cnt ? seg + GC_SEG : cnt;
          for (int kc = seg; kc < seg_end; ++kc) {
            if ((!PREP && !mbar_wait(smem_u32(&conv[stage]), phase, budget, abort_flag, &g_gate_error)) ||
                !mbar_wait(smem_u32(&full[stage]), phase, budget, abort_flag, &g_gate_error)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint8_t* st = smem + stage * L.stage_bytes;
            const uint64_t da = sdesc_sw128(smem_u32(st));
            const uint64_t db = sdesc_sw128(smem_u32(st + L.w3_off));
#pragma unroll
            for (int kk = 0; kk < GC_BK / 16; ++kk)
              umma_bf16(d_tmem, da + 2 * kk, db + 2 * kk, idesc, (kc != seg || kk != 0) ? 1u : 0u);
            any = true;
            umma_commit(smem_u32(&empty[stage]));
            if (++stage == S) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          umma_commit(smem_u32(&tfull[acc]));
          if (acc) ++uses1;
          else ++uses0;
          acc ^= 1;
        }
      }
      if ((!ok || *abort_flag) && any) {
        umma_commit(smem_u32(drain));
        mbar_drain(smem_u32(drain), 0, DRAIN_CYCLES);
      }
    }
  } else {
    // ------------------------------------------------------------ worker warps
    pdl_wait();  // the routing counters are cleared by the previous kernel (PREP)
    const int wt = threadIdx.x - 64;
    const bool is_drain = warp < 6;
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t t_lane = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    const MaskRegs mregs{p.mask_bits[0], p.mask_bits[1], p.mask_bits[2], p.mask_bits[3]};
    int stage = 0;
    uint32_t phase = 0;
    int acc_sel = 0;
    uint32_t uses0 = 0, uses1 = 0;
    bool ok = true;
    for (int tile = tile_first; tile < n_tiles; tile += tile_step) {
      if (is_drain) {
        float acc[NB][16];
#pragma unroll
        for (int b = 0; b < NB; ++b)
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[b][j] = 0.0f;
        for (int seg = 0; seg < cnt; seg += GC_SEG) {
          const uint32_t uses = acc_sel ? uses1 : uses0;
          if (ok) ok = mbar_wait(smem_u32(&tfull[acc_sel]), uses & 1u, budget, abort_flag, &g_gate_error);
          if (ok) {
            tc_fence_after();
            const uint32_t t_acc = t_lane + acc_sel * GC_ACC_STRIDE;
#pragma unroll
            for (int b = 0; b < NB; ++b) {
              uint32_t v0[16], v1[16], v2[16];
              tmem_ld16_nw(t_acc + b * 16, v0);
              tmem_ld16_nw(t_acc + n_pad + b * 16, v1);
              tmem_ld16_nw(t_acc + 2 * n_pad + b * 16, v2);
              tmem_wait();
#pragma unroll
              for (int j = 0; j < 16; ++j)
                acc[b][j] += (__uint_as_float(v0[j]) + __uint_as_float(v1[j])) + __uint_as_float(v2[j]);
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&tempty[acc_sel]));
          if (acc_sel) ++uses1;
          else ++uses0;
          acc_sel ^= 1;
        }
        bool decide_here = true;
        if (cs > 1) {
          // this row's partial logits go to the CTA that owns its decision;
          // the owner adds the cluster's partials in CTA order
          const int owner = row / rows_own;
          const int lrow = row - owner * rows_own;
          if (owner != rank) {
            decide_here = false;
            if (ok) {
              const uint32_t dst = map_to_rank(smem_u32(s_recv + (rank * rows_own + lrow) * L.rstride), owner);
              const uint32_t rb = map_to_rank(smem_u32(recvb), owner);
#pragma unroll
              for (int b = 0; b < NB; ++b)
                if (b * 16 < n_pad)
#pragma unroll
                  for (int j = 0; j < 16; j += 4)
                    st_async_v4(dst + (b * 16 + j) * 4, acc[b][j], acc[b][j + 1], acc[b][j + 2], acc[b][j + 3], rb);
            }
          } else {
            if (ok) ok = mbar_wait_cluster(smem_u32(recvb), 0, budget, abort_flag, &g_gate_error);
            if (ok) {
#pragma unroll
              for (int b = 0; b < NB; ++b)
                if (b * 16 < n_pad)
#pragma unroll
                  for (int j = 0; j < 16; ++j) {
                    float t = rank == 0 ? acc[b][j] : s_recv[lrow * L.rstride + b * 16 + j];
                    for (int c = 1; c < cs; ++c)
                      t += c == rank ? acc[b][j] : s_recv[(c * rows_own + lrow) * L.rstride + b * 16 + j];
                    acc[b][j] = t;
                  }
            }
          }
        }
        if (decide_here) {
#pragma unroll
          for (int b = 0; b < NB; ++b)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int o = b * 16 + j;
              if (o < O) acc[b][j] += s_bias[o];
            }
          const int tok = tile * GC_BM + row;
          int* sx = p.route_counts ? sIdx + row * p.k : nullptr;
          if (!nglob) {
            if (tok < p.T) {
              if (p.k == 1) decide_k1_regs<NB, 1>(acc, p.E, p.k, p.renorm, mregs, p.topk_idx, p.topk_w, tok, sx);
              else if (p.k == 2) decide_k1_regs<NB, 2>(acc, p.E, p.k, p.renorm, mregs, p.topk_idx, p.topk_w, tok, sx);
              else if (p.k <= 4) decide_k1_regs<NB, 4>(acc, p.E, p.k, p.renorm, mregs, p.topk_idx, p.topk_w, tok, sx);
              else decide_k1_regs<NB, 8>(acc, p.E, p.k, p.renorm, mregs, p.topk_idx, p.topk_w, tok, sx);
            }
          } else {
            float* Lrow = sLog + row * L.log_stride;
#pragma unroll
            for (int b = 0; b < NB; ++b)
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const int o = b * 16 + j;
                if (o < O) Lrow[o] = acc[b][j];
              }
            if (tok < p.T) {
              if (p.k == 1) decide_token_thread<1>(p.E, p.K, p.k, p.renorm, p.top_groups, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
              else if (p.k == 2) decide_token_thread<2>(p.E, p.K, p.k, p.renorm, p.top_groups, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
              else if (p.k <= 4) decide_token_thread<4>(p.E, p.K, p.k, p.renorm, p.top_groups, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
              else decide_token_thread<8>(p.E, p.K, p.k, p.renorm, p.top_groups, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
            }
          }
        }  // decide_here
      } else if (!PREP) {
        // split the raw fp32 gate rows of each stage into three bf16 terms,
        // written in the swizzled K-major layout of the B operand
        const int ct = threadIdx.x - 192;
        for (int kc = 0; kc < cnt; ++kc) {
          if (ok) ok = mbar_wait(smem_u32(&full[stage]), phase, budget, abort_flag, &g_gate_error);
          if (ok) {
            uint8_t* st = smem + stage * L.stage_bytes;
            const float* raw = reinterpret_cast<const float*>(st + L.raw_off);
            for (int i = ct; i < n_pad * 8; i += 256) {
              const int r = i >> 3, ch = i & 7;
              float v[8];
              if (r < O) {
                const float4 a = *reinterpret_cast<const float4*>(raw + r * GC_BK + ch * 8);
                const float4 b = *reinterpret_cast<const float4*>(raw + r * GC_BK + ch * 8 + 4);
                v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
              } else {
#pragma unroll
                for (int u = 0; u < 8; ++u) v[u] = 0.0f;
              }
              uint32_t t0[4], t1[4], t2[4];
#pragma unroll
              for (int u = 0; u < 4; ++u) split3_pair(v[2 * u], v[2 * u + 1], t0[u], t1[u], t2[u]);
              const int off = L.w3_off + r * 128 + ((ch ^ (r & 7)) << 4);
              *reinterpret_cast<U4*>(st + off) = U4{t0[0], t0[1], t0[2], t0[3]};
              *reinterpret_cast<U4*>(st + off + n_pad * 128) = U4{t1[0], t1[1], t1[2], t1[3]};
              *reinterpret_cast<U4*>(st + off + 2 * n_pad * 128) = U4{t2[0], t2[1], t2[2], t2[3]};
            }
            // the tensor core reads these through the async proxy
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&conv[stage]));
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (p.route_counts) {
        asm volatile("bar.sync 1, %0;" ::"r"(GC_WORKERS) : "memory");
        route_tile_workers(p, tile, rank * rows_own, rows_own, sIdx + rank * rows_own * p.k, sTab, s_base, wt);
      }
    }
    tc_fence_before();
  }

  tc_fence_before();
  __syncthreads();
  // no CTA of the cluster leaves while partials to or from it are in flight
  if (cs > 1) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
  }
}

// Stages that fit next to the logits, routing tables and received partials.
int gc_stages(int O, int k, int E, bool prep, int cs) {
  for (int s = GC_MAX_STAGES; s >= 2; --s)
    if (GcLayout(O, k, E, s, prep, cs).total + 1024 <= 232448) return s;
  return 0;
}

// CTAs per tile: d_model is split over a cluster of GC_CS when a tile has at
// least GC_SPLIT_MIN_NK stages and the received partials still leave four
// pipeline stages (counted for the larger, self-splitting layout), whatever
// the token count and whether the rows come prepared, so every call of one
// layer shape sums its logits in the same order.
// EC2MOE_GATE_SPLIT_MIN_STAGES=n in the environment moves the threshold
// (A/B comparisons; the split computes the same logits up to summation order).
int gc_cluster_size(int O, int k, int E, int d) {
  static const int min_nk = [] {
    const char* v = getenv("EC2MOE_GATE_SPLIT_MIN_STAGES");
    return v && atoi(v) > 0 ? atoi(v) : GC_SPLIT_MIN_NK;
  }();
  if ((d + GC_BK - 1) / GC_BK < min_nk) return 1;
  return gc_stages(O, k, E, false, GC_CS) >= 4 ? GC_CS : 1;
}

// CTAs the gate kernel launches (cs > 1: a cluster per tile, run in waves
// when they exceed the SMs; cs = 1: persistent, at most one per SM).
int gc_blocks(int T, int cs) {
  const int n_tiles = (T + GC_BM - 1) / GC_BM;
  if (cs > 1) return n_tiles * cs;
  return n_tiles < sm_count() ? n_tiles : sm_count();
}

template <int NB, bool PREP>
cudaError_t launch_gate_tc_nb(const KParams& p, int stages, int cs, cudaStream_t s, const CUtensorMap& mX,
                              const CUtensorMap& mW, const CUtensorMap& mWg) {
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  GcParams gp;
  gp.kp = p;
  gp.n_pad = (O + 15) / 16 * 16;
  gp.stages = stages;
  gp.cs = cs;
  gp.timeout = default_timeout_cycles();
  const int smem = GcLayout(O, p.k, p.E, stages, PREP, cs).total + 1024;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(gate_tc_kernel<NB, PREP>), smem);
  if (e != cudaSuccess) return e;
  const int blocks = gc_blocks(p.T, cs);
  if (cs == 1)
    return launch_kernel(gate_tc_kernel<NB, PREP>, dim3(blocks), dim3(GC_THREADS), (size_t)smem, s, mX, mW, mWg, gp);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(blocks);
  cfg.blockDim = dim3(GC_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = next_launch_pdl() ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, gate_tc_kernel<NB, PREP>, mX, mW, mWg, gp);
}

template <bool PREP>
cudaError_t launch_gate_tc(const KParams& p, int stages, int cs, cudaStream_t s, const CUtensorMap& mX,
                           const CUtensorMap& mW, const CUtensorMap& mWg) {
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  // NB = accumulator blocks of 16 gate rows a drain thread keeps; 3 and 4
  // run as 5 (the extra blocks read allocated TMEM columns past the gate rows
  // and are never used), which keeps the number of kernel variants small.
  switch ((O + 15) / 16) {
    case 1: return launch_gate_tc_nb<1, PREP>(p, stages, cs, s, mX, mW, mWg);
    case 2: return launch_gate_tc_nb<2, PREP>(p, stages, cs, s, mX, mW, mWg);
    default: return launch_gate_tc_nb<5, PREP>(p, stages, cs, s, mX, mW, mWg);
  }
}

}  // namespace

cudaError_t launch_gate_tensor(const GateArgs& a, KParams p, int O, bool bf16, cudaStream_t s, bool* routed, int* held_sms,
                               bool* handled) {
  *handled = false;
  cudaError_t e = cudaSuccess;
  // Tensor-core gate (bf16 activations, up to 80 gate rows).  With a
  // workspace for the prepared split rows (layer path) a small kernel first
  // splits the gate rows and clears the routing counters; without one the
  // gate kernel splits them itself.
  static const bool simt_only = [] {
    const char* v = getenv("EC2MOE_GATE_SIMT");
    return v && atoi(v) > 0;
  }();
  const bool w_aligned = (reinterpret_cast<uintptr_t>(a.W_local) % 16 == 0) &&
                         (a.K == 1 || reinterpret_cast<uintptr_t>(a.W_global) % 16 == 0);
  if (bf16 && !simt_only && O <= GC_MAX_O && a.d % 8 == 0 && a.T > 0 && w_aligned) {
    const bool prep = a.w_split != nullptr;
    const int n_pad = (O + 15) / 16 * 16;
    const int cs = gc_cluster_size(O, a.k, a.E, a.d);
    const int stages = gc_stages(O, a.k, a.E, prep, cs);
    CUtensorMap mX, mW, mWg;
    bool maps = stages >= 2 && make_tensor_map_bf16(&mX, a.X, a.T, a.d, GC_BM);
    if (prep) {
      maps = maps && make_tensor_map_bf16(&mW, a.w_split, 3LL * n_pad, a.d, 3 * n_pad);
      mWg = mW;
    } else {
      maps = maps && make_tensor_map_f32(&mW, a.W_local, a.E, a.d, a.E);
      if (maps && a.K > 1) maps = make_tensor_map_f32(&mWg, a.W_global, a.K, a.d, a.K);
      else mWg = mW;
    }
    if (maps) {
      *handled = true;
      const bool route = a.route_counts && a.route_rel;
      if (route) {
        p.route_counts = a.route_counts;
        p.route_rel = a.route_rel;
        if (!prep) {
          e = cudaMemsetAsync(a.route_counts, 0, sizeof(int32_t) * a.E, s);
          if (e != cudaSuccess) return e;
        }
        if (routed) *routed = true;
      }
      if (prep) {
        KernelScope ks("gate_prep", s);
        const long long items = (long long)n_pad * (a.d / 8);
        e = launch_kernel(gate_split_kernel, dim3((unsigned)((items + 255) / 256)), dim3(256), 0, s, a.W_local,
                          a.W_global, a.E, a.K, a.d, n_pad, static_cast<__nv_bfloat16*>(a.w_split),
                          route ? a.route_counts : nullptr);
        if (e != cudaSuccess) return e;
      }
      KernelScope ks("gate_topk", s);
      if (held_sms) {  // one CTA per SM (the kernel's shared memory allows no second)
        const int b = gc_blocks(a.T, cs);
        *held_sms = b < sm_count() ? b : sm_count();
      }
      e = prep ? launch_gate_tc<true>(p, stages, cs, s, mX, mW, mWg)
               : launch_gate_tc<false>(p, stages, cs, s, mX, mW, mWg);
      if (e != cudaSuccess) return e;
      return cudaGetLastError();
    }
  }
  return cudaSuccess;
}

}  // namespace gatek

using namespace gatek;

size_t gate_split_bytes(int E, int K, int d, bool bf16) {
  const int O = E + (K == 1 ? 0 : K);
  if (!bf16 || O > GC_MAX_O || d % 8 != 0) return 0;
  return (size_t)3 * ((O + 15) / 16 * 16) * d * 2;
}

cudaError_t read_gate_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_gate_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_gate_error, &zero, sizeof(unsigned int));
}

}  // namespace ec2moe
