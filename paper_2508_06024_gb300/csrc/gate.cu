// Steps 1-3a of the layer: local expert filter (Eq. 4), lightweight group gate
// (Eq. 5 per-group softmax, Eq. 6 global group softmax, Eq. 7 fusion
// g_i = p_group^(k) * p_local,i^(k)) and Top-k routing.
//
// One warp owns TPW tokens at a time.  The gate weights [E + K, d] (fp32) are
// staged in shared memory when they fit, else read through L1.  Each lane
// accumulates 8-element column slices of the d_model axis for TPW tokens x OB
// gate rows, so one 16-byte shared-memory load of a weight slice feeds 4*TPW
// FMAs; the 32 lane partials are then summed with xor shuffles.
//
// Decision arithmetic (fp32): masked experts get score -inf.  Inside a group
// the order is the order of the local logits l_i; across groups the score is
// (m_k - lse_k) + l_i = log p_group^(k) + log p_local,i + const, with lse_k the
// log-sum-exp of the allowed logits of group k.  With K = 1 the score is l_i
// itself.  Top-k takes the largest score, ties to the lower index, k times.
// The combine weight is g_i = exp((m_k - LSE_m) + (l_i - lse_k)) where LSE_m is
// the log-sum-exp of m over groups with at least one allowed expert.
//
// Top-group pruning (top_groups = G > 0): before the scores, each token keeps
// only the G live groups with the largest global logit m_k (the order of
// p_group; ties to the lower group index); the other groups are treated as if
// they had no allowed expert, so their experts are not candidates and LSE_m
// runs over the kept groups (p_group renormalised over them).
#include <stdlib.h>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include "common.cuh"
#include "internal.h"
#include "gate_common.cuh"

namespace ec2moe {

using namespace gatek;

namespace {

constexpr int WARPS = 4;
constexpr int TPW = 4;      // tokens per warp pass
constexpr int OB = 8;       // gate rows per accumulation block
constexpr int MAXO = 144;   // E + K <= 128 + 16


__device__ __forceinline__ bool allowed_bit(const KParams& p, int e) { return (p.mask_bits[e >> 5] >> (e & 31)) & 1u; }

// (key, idx) ordering for Top-k: larger key first, ties to the lower index.
__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) { return ka > kb || (ka == kb && ia < ib); }

// When no allowed expert has a finite score left (NaN or infinite logits), the
// slot takes the lowest allowed expert not yet chosen, with its (non-finite)
// weight, so every index handed to the routing stays a valid expert.  The
// result is warp-uniform; the host guarantees k <= popcount(mask).
__device__ __forceinline__ int fallback_expert(const bool* al, const bool* taken, const float* lw, int lane,
                                               float* bw) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const unsigned m = __ballot_sync(0xffffffffu, al[i] && !taken[i]);
    if (m) {
      const int src = __ffs(m) - 1;
      *bw = __shfl_sync(0xffffffffu, lw[i], src);
      return src + 32 * i;
    }
  }
  *bw = 0.0f;
  return 0;
}

template <typename TX, bool W_SMEM>
__global__ void __launch_bounds__(WARPS * 32) gate_topk_kernel(const KParams p) {
  extern __shared__ float smem_f[];
  const int nglob = (p.K == 1) ? 0 : p.K;  // global gate rows (none when K == 1)
  const int O = p.E + nglob;
  float* sW = smem_f;                                   // [O, d] when W_SMEM
  float* sLog = smem_f + (W_SMEM ? O * p.d : 0);        // [WARPS][TPW][MAXO]
  float* sGrp = sLog + WARPS * TPW * MAXO;              // [WARPS][TPW][2 * 16]: lse_k, then live flag
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  pdl_trigger();
  pdl_wait();

  if (W_SMEM) {
    const int n4 = O * p.d / 4;
    for (int i = threadIdx.x; i < n4; i += blockDim.x) {
      const int row = (i * 4) / p.d;
      const int col = (i * 4) % p.d;
      const float* src = row < p.E ? p.W_local + (size_t)row * p.d : p.W_global + (size_t)(row - p.E) * p.d;
      reinterpret_cast<float4*>(sW)[i] = *reinterpret_cast<const float4*>(src + col);
    }
    __syncthreads();
  }
  auto wrow = [&](int o) -> const float* {
    if (W_SMEM) return sW + (size_t)o * p.d;
    return o < p.E ? p.W_local + (size_t)o * p.d : p.W_global + (size_t)(o - p.E) * p.d;
  };

  const TX* X = reinterpret_cast<const TX*>(p.X);
  float* lg = sLog + (warp * TPW) * MAXO;
  float* gs = sGrp + (warp * TPW) * 32;
  const int gsize = p.E / p.K;
  const int n_pass = (p.T + TPW - 1) / TPW;

  for (int pass = blockIdx.x * WARPS + warp; pass < n_pass; pass += gridDim.x * WARPS) {
    const int t0 = pass * TPW;
    // ---- logits: lg[t][o] = <x_t, W_o> + b_o
    for (int ob = 0; ob < O; ob += OB) {
      float acc[TPW][OB];
#pragma unroll
      for (int t = 0; t < TPW; ++t)
#pragma unroll
        for (int o = 0; o < OB; ++o) acc[t][o] = 0.0f;
      for (int c = lane * 8; c < p.d; c += 256) {
        float xv[TPW][8];
#pragma unroll
        for (int t = 0; t < TPW; ++t) {
          if (t0 + t < p.T) {
            load8(X + (size_t)(t0 + t) * p.d + c, xv[t]);
          } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) xv[t][j] = 0.0f;
          }
        }
#pragma unroll
        for (int o = 0; o < OB; ++o) {
          if (ob + o < O) {
            float wv[8];
            load8(wrow(ob + o) + c, wv);
#pragma unroll
            for (int t = 0; t < TPW; ++t)
#pragma unroll
              for (int j = 0; j < 8; ++j) acc[t][o] = fmaf(xv[t][j], wv[j], acc[t][o]);
          }
        }
      }
#pragma unroll
      for (int t = 0; t < TPW; ++t)
#pragma unroll
        for (int o = 0; o < OB; ++o) {
          float v = acc[t][o];
#pragma unroll
          for (int sh = 16; sh > 0; sh >>= 1) v += __shfl_xor_sync(0xffffffffu, v, sh);
          acc[t][o] = v;
        }
      if (lane == 0) {
#pragma unroll
        for (int t = 0; t < TPW; ++t)
#pragma unroll
          for (int o = 0; o < OB; ++o) {
            const int oo = ob + o;
            if (oo < O) lg[t * MAXO + oo] = acc[t][o] + (oo < p.E ? p.b_local[oo] : p.b_global[oo - p.E]);
          }
      }
    }
    __syncwarp();

    for (int t = 0; t < TPW; ++t) {
      const int tok = t0 + t;
      if (tok >= p.T) break;
      const float* L = lg + t * MAXO;
      float* G = gs + t * 32;
      // ---- per-group log-sum-exp over allowed members (Eq. 5), lane j owns group j
      if (lane < p.K) {
        const int lo = lane * gsize;
        float mx = -CUDART_INF_F;
        for (int e = lo; e < lo + gsize; ++e)
          if (allowed_bit(p, e)) mx = fmaxf(mx, L[e]);
        float sum = 0.0f;
        for (int e = lo; e < lo + gsize; ++e)
          if (allowed_bit(p, e)) sum += expf(L[e] - mx);
        const bool live = mx > -CUDART_INF_F;
        G[lane] = live ? mx + logf(sum) : -CUDART_INF_F;
        G[16 + lane] = live ? 1.0f : 0.0f;
      }
      __syncwarp();
      // ---- top-group pruning: only the top_groups live groups by m stay live
      if (nglob && p.top_groups > 0 && p.top_groups < p.K) {
        bool keep = false;
        if (lane < p.K && G[16 + lane] != 0.0f) {
          const float mg = L[p.E + lane];
          int rank = 0;
          for (int j = 0; j < p.K; ++j) {
            const float mj = L[p.E + j];
            if (j != lane && G[16 + j] != 0.0f && (mj > mg || (mj == mg && j < lane))) ++rank;
          }
          keep = rank < p.top_groups;
        }
        __syncwarp();
        if (lane < p.K) G[16 + lane] = keep ? 1.0f : 0.0f;
        __syncwarp();
      }
      // ---- log-sum-exp of the global logits over live groups (Eq. 6)
      float lse_m = 0.0f;
      if (nglob) {
        float mx = -CUDART_INF_F;
        for (int j = 0; j < p.K; ++j)
          if (G[16 + j] != 0.0f) mx = fmaxf(mx, L[p.E + j]);
        float sum = 0.0f;
        for (int j = 0; j < p.K; ++j)
          if (G[16 + j] != 0.0f) sum += expf(L[p.E + j] - mx);
        lse_m = mx + logf(sum);
      }
      // ---- scores and weights for the experts this lane owns (e = lane + 32 i)
      float key[4], lw[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = lane + 32 * i;
        key[i] = -CUDART_INF_F;
        lw[i] = 0.0f;
        if (e < p.E && allowed_bit(p, e)) {
          const int grp = e / gsize;
          const float le = L[e];
          if (nglob) {
            if (G[16 + grp] != 0.0f) {  // a kept group
              const float mk = L[p.E + grp];
              key[i] = (mk - G[grp]) + le;
              lw[i] = (mk - lse_m) + (le - G[grp]);
            }
          } else {
            key[i] = le;
            lw[i] = le - G[0];
          }
        }
      }
      // ---- Top-k by k rounds of a warp argmax
      int sel_idx[MAX_TOPK];
      float sel_w[MAX_TOPK];
      float wsum = 0.0f;
      bool al[4], taken[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        al[i] = lane + 32 * i < p.E && allowed_bit(p, lane + 32 * i);
        taken[i] = false;
      }
      for (int s = 0; s < p.k; ++s) {
        float bk = -CUDART_INF_F;
        int bi = 0x7fffffff;
        float bw = 0.0f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int e = lane + 32 * i;
          if (e < p.E && key[i] > -CUDART_INF_F && better(key[i], e, bk, bi)) {
            bk = key[i];
            bi = e;
            bw = lw[i];
          }
        }
#pragma unroll
        for (int sh = 16; sh > 0; sh >>= 1) {
          const float ok = __shfl_xor_sync(0xffffffffu, bk, sh);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, sh);
          const float ow = __shfl_xor_sync(0xffffffffu, bw, sh);
          if (better(ok, oi, bk, bi)) {
            bk = ok;
            bi = oi;
            bw = ow;
          }
        }
        if (bi == 0x7fffffff) bi = fallback_expert(al, taken, lw, lane, &bw);  // non-finite logits
        // remove the winner from its owner's candidates
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (lane + 32 * i == bi) {
            key[i] = -CUDART_INF_F;
            taken[i] = true;
          }
        const float g = expf(bw);
        sel_idx[s] = bi;
        sel_w[s] = g;
        wsum += g;
      }
      if (lane == 0) {
        const float inv = p.renorm ? 1.0f / wsum : 1.0f;
        for (int s = 0; s < p.k; ++s) {
          p.topk_idx[(size_t)tok * p.k + s] = sel_idx[s];
          p.topk_w[(size_t)tok * p.k + s] = p.renorm ? sel_w[s] * inv : sel_w[s];
        }
      }
      __syncwarp();
    }
    __syncwarp();
  }
}

// Warp-cooperative decision for one token from its logits L[0..E) (local) and
// L[E..E+K) (global) in shared memory.  Lane l owns experts l, l+32, l+64, l+96.
// Same arithmetic as gate_topk_kernel: key = l_i (K = 1) or (m_k - lse_k) + l_i,
// Top-k by k rounds of a warp argmax with ties to the lower index, weight
// g_i = exp((m_k - LSE_m) + (l_i - lse_k)).
__device__ void decide_token_warp(const KParams& p, const float* L, int tok, int lane, int* s_idx,
                                  bool write_out = true) {
  const int nglob = (p.K == 1) ? 0 : p.K;
  const int gsize = p.E / p.K;
  float lv[4];
  bool al[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = lane + 32 * i;
    al[i] = e < p.E && allowed_bit(p, e);
    lv[i] = al[i] ? L[e] : -CUDART_INF_F;
  }
  float key[4], lw[4];
  if (!nglob) {
    // one group: warp max and warp sum of the allowed logits
    float mx = fmaxf(fmaxf(lv[0], lv[1]), fmaxf(lv[2], lv[3]));
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, sh));
    float sum = 0.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (al[i]) sum += expf(lv[i] - mx);
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sh);
    const float lse = mx + logf(sum);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      key[i] = lv[i];
      lw[i] = lv[i] - lse;
    }
  } else {
    // lane g < K: log-sum-exp of group g's allowed logits; then the group softmax
    float lse_mine = -CUDART_INF_F;
    if (lane < p.K) {
      const int lo = lane * gsize;
      float mx = -CUDART_INF_F;
      for (int e = lo; e < lo + gsize; ++e)
        if (allowed_bit(p, e)) mx = fmaxf(mx, L[e]);
      float sum = 0.0f;
      for (int e = lo; e < lo + gsize; ++e)
        if (allowed_bit(p, e)) sum += expf(L[e] - mx);
      if (mx > -CUDART_INF_F) lse_mine = mx + logf(sum);
    }
    // groups that stay: the live ones, or with top-group pruning the
    // top_groups live ones by m (ties to the lower group index)
    unsigned kept = __ballot_sync(0xffffffffu, lane < p.K && lse_mine > -CUDART_INF_F);
    if (p.top_groups > 0 && p.top_groups < p.K) {
      bool keep = false;
      if ((kept >> lane) & 1u) {
        const float mg = L[p.E + lane];
        int rank = 0;
        for (int j = 0; j < p.K; ++j)
          if (j != lane && ((kept >> j) & 1u)) {
            const float mj = L[p.E + j];
            rank += (mj > mg || (mj == mg && j < lane)) ? 1 : 0;
          }
        keep = rank < p.top_groups;
      }
      kept = __ballot_sync(0xffffffffu, keep);
      if (!keep) lse_mine = -CUDART_INF_F;
    }
    const float mk_mine = ((kept >> lane) & 1u) ? L[p.E + lane] : -CUDART_INF_F;
    float mxm = mk_mine;
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) mxm = fmaxf(mxm, __shfl_xor_sync(0xffffffffu, mxm, sh));
    float summ = (mk_mine > -CUDART_INF_F) ? expf(mk_mine - mxm) : 0.0f;
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) summ += __shfl_xor_sync(0xffffffffu, summ, sh);
    const float lse_m = mxm + logf(summ);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = lane + 32 * i;
      const int g = (e < p.E ? e : 0) / gsize;
      const float lse_g = __shfl_sync(0xffffffffu, lse_mine, g);
      const float mk = L[p.E + (g < p.K ? g : 0)];
      key[i] = (al[i] && ((kept >> g) & 1u)) ? (mk - lse_g) + lv[i] : -CUDART_INF_F;
      lw[i] = (mk - lse_m) + (lv[i] - lse_g);
    }
  }
  float wsum = 0.0f, w_mine = 0.0f;
  int id_mine = 0;
  bool taken[4] = {false, false, false, false};
  for (int s = 0; s < p.k; ++s) {
    float bk = -CUDART_INF_F, bw = 0.0f;
    int bi = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = lane + 32 * i;
      if (key[i] > -CUDART_INF_F && better(key[i], e, bk, bi)) {
        bk = key[i];
        bi = e;
        bw = lw[i];
      }
    }
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) {
      const float ok = __shfl_xor_sync(0xffffffffu, bk, sh);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, sh);
      const float ow = __shfl_xor_sync(0xffffffffu, bw, sh);
      if (better(ok, oi, bk, bi)) {
        bk = ok;
        bi = oi;
        bw = ow;
      }
    }
    if (bi == 0x7fffffff) bi = fallback_expert(al, taken, lw, lane, &bw);  // non-finite logits
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (lane + 32 * i == bi) {
        key[i] = -CUDART_INF_F;
        taken[i] = true;
      }
    const float g = expf(bw);
    wsum += g;
    if (lane == s) {
      id_mine = bi;
      w_mine = g;
    }
  }
  if (lane < p.k) {
    if (write_out) {
      p.topk_idx[(size_t)tok * p.k + lane] = id_mine;
      p.topk_w[(size_t)tok * p.k + lane] = p.renorm ? w_mine / wsum : w_mine;
    }
    if (s_idx) s_idx[lane] = id_mine;
  }
}

// Gate with every gate row resident in shared memory.  A block of 256 threads
// owns BT = TPT * 256 / S tokens at a time; thread (s, q) holds the slice
// [s*SW, (s+1)*SW) of d_model of TPT tokens in registers (all loads issued
// before the first FMA) and accumulates their dot products with up to NB gate
// rows, so every 16-byte weight load from shared memory (a broadcast shared by
// the threads of a slice) feeds 4*TPT FMAs.  Slice partials go to shared
// memory in an [n][slice][token] layout padded so both the writes and the
// fixed-order sums over slices are free of bank conflicts; one warp per token
// then takes the softmax / Top-k decision.
constexpr int SL_THREADS = 256;
constexpr int SL_RED_PAD = 16;

// Raw 16-byte vectors of one 8-element activation chunk (bf16: one, fp32: two).
template <typename TX>
struct Chunk8 {
  static constexpr int NV = sizeof(TX) == 2 ? 1 : 2;
  U4 v[NV];
  __device__ __forceinline__ void load(const TX* p) {
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = reinterpret_cast<const U4*>(p)[i];
  }
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = U4{0u, 0u, 0u, 0u};
  }
  __device__ __forceinline__ void to_float(float* f) const {
    if (NV == 1) {
      f[0] = bf16_lo(v[0].x); f[1] = bf16_hi(v[0].x); f[2] = bf16_lo(v[0].y); f[3] = bf16_hi(v[0].y);
      f[4] = bf16_lo(v[0].z); f[5] = bf16_hi(v[0].z); f[6] = bf16_lo(v[0].w); f[7] = bf16_hi(v[0].w);
    } else {
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        f[4 * i + 0] = __uint_as_float(v[i].x); f[4 * i + 1] = __uint_as_float(v[i].y);
        f[4 * i + 2] = __uint_as_float(v[i].z); f[4 * i + 3] = __uint_as_float(v[i].w);
      }
    }
  }
};

// ---- routing fused into the gate (layer path)
// For each tile of BT tokens (nt = BT * k consecutive (token, slot) entries),
// every expert present in the tile reserves a contiguous run of its rows with
// one atomicAdd on route_counts[e] (zero at launch), and each entry's row
// relative to its expert's first row -- the reserved base plus the entry's
// stable rank among the tile's entries of that expert -- goes to route_rel.
// After the kernel route_counts holds the per-expert histogram; the consumer
// adds the exclusive prefix of the counts to place rows.  Rows of one expert
// are grouped by tile in the order the tiles reserved them; that order does
// not change any output, since every GEMM row depends only on its own input.
__device__ void route_tile(const KParams& p, int tile, int BT, const int* sIdx, int* s_base) {
  const int nt = BT * p.k;
  const long long e0 = (long long)tile * nt;
  const long long n = (long long)p.T * p.k;
  const int live = (int)((n - e0) < nt ? (n - e0) : nt);
  for (int e = threadIdx.x; e < p.E; e += SL_THREADS) {
    int c = 0;
    for (int j = 0; j < live; ++j) c += (sIdx[j] == e) ? 1 : 0;
    s_base[e] = c ? atomicAdd(&p.route_counts[e], c) : 0;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < live; i += SL_THREADS) {
    const int e = sIdx[i];
    int rank = 0;
    for (int j = 0; j < i; ++j) rank += (sIdx[j] == e) ? 1 : 0;
    p.route_rel[e0 + i] = s_base[e] + rank;
  }
  __syncthreads();
}

template <typename TX, int XC, int TPT, int NB>
__global__ void __launch_bounds__(SL_THREADS) gate_slices_kernel(const KParams p, int S) {
  extern __shared__ float smem_f[];
  const int nglob = (p.K == 1) ? 0 : p.K;
  const int O = p.E + nglob;
  const int JQ = SL_THREADS / S;       // token groups per tile
  const int BT = JQ * TPT;             // tokens per tile
  const int SW = p.d / S;
  const int nch = SW / 8;
  const int RS = S * BT + SL_RED_PAD;  // row stride of the partials
  float* sW = smem_f;                   // [O][d]
  float* sRed = sW + (size_t)O * p.d;   // [NB][RS]
  float* sLog = sRed + NB * RS;         // [BT][O]
  int* sIdx = reinterpret_cast<int*>(sLog + BT * O);  // [BT * k] this tile's expert ids
  __shared__ int s_base[128];
  const int jq = threadIdx.x % JQ;
  const int sl = threadIdx.x / JQ;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_trigger();

  {  // stage the gate rows, eight 16-byte loads in flight per thread
    const int n4 = O * p.d / 4;
    float4* dst = reinterpret_cast<float4*>(sW);
    const int e4 = p.E * p.d / 4;
    for (int base = threadIdx.x; base < n4; base += SL_THREADS * 8) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + u * SL_THREADS;
        if (i < n4)
          v[u] = i < e4 ? reinterpret_cast<const float4*>(p.W_local)[i]
                        : reinterpret_cast<const float4*>(p.W_global)[i - e4];
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + u * SL_THREADS;
        if (i < n4) dst[i] = v[u];
      }
    }
  }
  pdl_wait();
  __syncthreads();

  const TX* X = reinterpret_cast<const TX*>(p.X);
  const int n_tiles = (p.T + BT - 1) / BT;
  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    Chunk8<TX> xs[TPT][XC];
#pragma unroll
    for (int t = 0; t < TPT; ++t) {
      const int tok = tile * BT + jq * TPT + t;
#pragma unroll
      for (int c = 0; c < XC; ++c) {
        if (c < nch && tok < p.T) xs[t][c].load(X + (size_t)tok * p.d + sl * SW + c * 8);
        else xs[t][c].zero();
      }
    }
    for (int ob = 0; ob < O; ob += NB) {
      float acc[TPT][NB];
#pragma unroll
      for (int t = 0; t < TPT; ++t)
#pragma unroll
        for (int n = 0; n < NB; ++n) acc[t][n] = 0.0f;
#pragma unroll
      for (int c = 0; c < XC; ++c) {
        if (c < nch) {
          float xf[TPT][8];
#pragma unroll
          for (int t = 0; t < TPT; ++t) xs[t][c].to_float(xf[t]);
          const float* wcol = sW + sl * SW + c * 8;
#pragma unroll
          for (int n = 0; n < NB; ++n) {
            if (ob + n < O) {
              float wv[8];
              load8(wcol + (size_t)(ob + n) * p.d, wv);
#pragma unroll
              for (int t = 0; t < TPT; ++t)
#pragma unroll
                for (int q = 0; q < 8; ++q) acc[t][n] = fmaf(xf[t][q], wv[q], acc[t][n]);
            }
          }
        }
      }
#pragma unroll
      for (int n = 0; n < NB; ++n) {
        float* dst = sRed + n * RS + sl * BT + jq * TPT;
        if (TPT == 2) *reinterpret_cast<float2*>(dst) = make_float2(acc[0][n], acc[TPT - 1][n]);
        else dst[0] = acc[0][n];
      }
      __syncthreads();
      for (int i = threadIdx.x; i < BT * NB; i += SL_THREADS) {
        const int n = i / BT, jj = i % BT;
        const int o = ob + n;
        if (o < O) {
          float sum = 0.0f;
          for (int q = 0; q < S; ++q) sum += sRed[n * RS + q * BT + jj];
          sLog[jj * O + o] = sum + (o < p.E ? p.b_local[o] : p.b_global[o - p.E]);
        }
      }
      __syncthreads();
    }
    for (int jj = warp; jj < BT; jj += SL_THREADS / 32) {
      const int tok = tile * BT + jj;
      if (tok < p.T) decide_token_warp(p, sLog + jj * O, tok, lane, p.route_counts ? sIdx + jj * p.k : nullptr);
    }
    __syncthreads();
    if (p.route_counts) route_tile(p, tile, BT, sIdx, s_base);
  }
}

// Gate for gate matrices that do not fit in shared memory (many experts and a
// wide d_model): a register-tiled fp32 product of a 64-token tile with all
// O = E + K gate rows, d_model streamed through shared memory 32 columns at a
// time (the next chunk is loaded into registers while the current one is
// used).  Thread (q, g) owns tokens 4q .. 4q+3 and gate rows OPT*g .. +OPT-1.
// Each dot product is summed in 256-column partials that are then added,
// keeping the fp32 rounding close to that of a short sum.  One warp per token
// then takes the softmax / Top-k decision; the layer path also reserves the
// tile's rows per expert.
constexpr int GT_BM = 64;
constexpr int GT_KC = 32;
constexpr int GT_PARTIAL = 256;

template <typename TX, int OPT>
__global__ void __launch_bounds__(SL_THREADS) gate_tiled_kernel(const KParams p) {
  constexpr int OP = 16 * OPT;
  constexpr int NW4 = (OP * 8 + SL_THREADS - 1) / SL_THREADS;  // 16-byte weight loads per thread per chunk
  __shared__ __align__(16) float sX[GT_KC][GT_BM + 4];  // k-major activations
  __shared__ __align__(16) float sW[GT_KC][OP + 4];     // k-major gate rows
  __shared__ int s_base[128];
  extern __shared__ float smem_f[];
  const int nglob = (p.K == 1) ? 0 : p.K;
  const int O = p.E + nglob;
  float* sLog = smem_f;                                  // [GT_BM][O]
  int* sIdx = reinterpret_cast<int*>(sLog + GT_BM * O);  // [GT_BM * k]
  const int tq = threadIdx.x >> 4;  // token quad
  const int og = threadIdx.x & 15;  // gate-row group
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_trigger();
  pdl_wait();
  const TX* X = reinterpret_cast<const TX*>(p.X);
  const int n_tiles = (p.T + GT_BM - 1) / GT_BM;
  const int nk = p.d / GT_KC;
  // staging assignment: X chunk = 64 tokens x 32 columns (8 per thread);
  // W chunk = OP rows x 32 columns (OP * 8 float4, NW4 per thread)
  const int xr = threadIdx.x >> 2, xc = (threadIdx.x & 3) * 8;
  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int t0 = tile * GT_BM;
    float acc[4][OPT], part[4][OPT];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < OPT; ++j) acc[i][j] = part[i][j] = 0.0f;
    float xv[8];
    float4 wv[NW4];
    auto load_chunk = [&](int kc) {
      const int tok = t0 + xr;
      if (tok < p.T) load8(X + (size_t)tok * p.d + kc * GT_KC + xc, xv);
      else
#pragma unroll
        for (int q = 0; q < 8; ++q) xv[q] = 0.0f;
#pragma unroll
      for (int u = 0; u < NW4; ++u) {
        const int i = threadIdx.x + u * SL_THREADS;  // float4 index in the [OP][8] chunk
        const int o = i >> 3, c = (i & 7) * 4;
        wv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i < OP * 8 && o < O) {
          const float* src = o < p.E ? p.W_local + (size_t)o * p.d : p.W_global + (size_t)(o - p.E) * p.d;
          wv[u] = *reinterpret_cast<const float4*>(src + kc * GT_KC + c);
        }
      }
    };
    load_chunk(0);
    for (int kc = 0; kc < nk; ++kc) {
      __syncthreads();
#pragma unroll
      for (int q = 0; q < 8; ++q) sX[xc + q][xr] = xv[q];
#pragma unroll
      for (int u = 0; u < NW4; ++u) {
        const int i = threadIdx.x + u * SL_THREADS;
        if (i < OP * 8) {
          const int o = i >> 3, c = (i & 7) * 4;
          sW[c + 0][o] = wv[u].x;
          sW[c + 1][o] = wv[u].y;
          sW[c + 2][o] = wv[u].z;
          sW[c + 3][o] = wv[u].w;
        }
      }
      __syncthreads();
      if (kc + 1 < nk) load_chunk(kc + 1);  // in flight during this chunk's FMAs
#pragma unroll 8
      for (int k = 0; k < GT_KC; ++k) {
        const float4 x4 = *reinterpret_cast<const float4*>(&sX[k][tq * 4]);
        float w[OPT];
#pragma unroll
        for (int j = 0; j < OPT; ++j) w[j] = sW[k][og * OPT + j];
#pragma unroll
        for (int j = 0; j < OPT; ++j) {
          part[0][j] = fmaf(x4.x, w[j], part[0][j]);
          part[1][j] = fmaf(x4.y, w[j], part[1][j]);
          part[2][j] = fmaf(x4.z, w[j], part[2][j]);
          part[3][j] = fmaf(x4.w, w[j], part[3][j]);
        }
      }
      if (((kc + 1) * GT_KC) % GT_PARTIAL == 0 || kc + 1 == nk) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < OPT; ++j) {
            acc[i][j] += part[i][j];
            part[i][j] = 0.0f;
          }
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < OPT; ++j) {
        const int o = og * OPT + j;
        if (o < O) sLog[(tq * 4 + i) * O + o] = acc[i][j] + (o < p.E ? p.b_local[o] : p.b_global[o - p.E]);
      }
    __syncthreads();
    for (int jj = warp; jj < GT_BM; jj += SL_THREADS / 32) {
      const int tok = t0 + jj;
      if (tok < p.T) decide_token_warp(p, sLog + jj * O, tok, lane, p.route_counts ? sIdx + jj * p.k : nullptr);
    }
    __syncthreads();
    if (p.route_counts) route_tile(p, tile, GT_BM, sIdx, s_base);
  }
}

// ---- small batches (T <= 256): the d_model axis split across CTAs
// One or two 128-token tiles leave a per-tile kernel with one or two CTAs
// walking all of d_model.  Here CTA (c, b) takes the GP_DC columns of chunk c
// for the GP_TB tokens of tile b: it stages the gate-row slice (fp32) and the
// activation slice (as fp32) in shared memory and writes the fp32 partial
// logits of its chunk; a second kernel adds the chunks in chunk order, adds
// the bias, and takes the same warp decision and in-kernel routing as the
// other gates.  Partials: [n_chunks][T][O].
constexpr int GP_TB = 64;
constexpr int GP_DC = 128;
constexpr int GP_PITCH = GP_DC + 4;  // floats; rows 16-byte aligned, float4 reads of 8 rows on distinct banks
constexpr int GP_OB = 8;
constexpr int GP_THREADS = 256;
constexpr int GD_BT = 8;             // tokens per CTA of the decision kernel (one warp each)

size_t gp_smem(int O) { return (size_t)(O + GP_TB) * GP_PITCH * sizeof(float); }

template <typename TX>
__global__ void __launch_bounds__(GP_THREADS) gate_partial_kernel(const KParams p, float* __restrict__ part) {
  extern __shared__ float4 gp_smem_v[];
  float* sW = reinterpret_cast<float*>(gp_smem_v);  // [O][GP_PITCH]
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  float* sX = sW + (size_t)O * GP_PITCH;            // [GP_TB][GP_PITCH]
  const int c0 = blockIdx.x * GP_DC;
  const int t0 = blockIdx.y * GP_TB;
  pdl_trigger();
  // gate-row slice: constant weights, staged before waiting on the previous kernel
  for (int i = threadIdx.x; i < O * (GP_DC / 4); i += GP_THREADS) {
    const int o = i / (GP_DC / 4), c = (i % (GP_DC / 4)) * 4;
    float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    if (c0 + c < p.d) {
      const float* row = o < p.E ? p.W_local + (size_t)o * p.d : p.W_global + (size_t)(o - p.E) * p.d;
      v = *reinterpret_cast<const float4*>(row + c0 + c);
    }
    *reinterpret_cast<float4*>(sW + o * GP_PITCH + c) = v;
  }
  pdl_wait();
  if (p.route_counts && blockIdx.x == 0 && blockIdx.y == 0)
    for (int e = threadIdx.x; e < p.E; e += GP_THREADS) p.route_counts[e] = 0;
  const TX* X = reinterpret_cast<const TX*>(p.X);
  for (int i = threadIdx.x; i < GP_TB * (GP_DC / 8); i += GP_THREADS) {
    const int t = i / (GP_DC / 8), c = (i % (GP_DC / 8)) * 8;
    float f[8];
    Chunk8<TX> x;
    if (t0 + t < p.T && c0 + c < p.d) x.load(X + (size_t)(t0 + t) * p.d + c0 + c);
    else x.zero();
    x.to_float(f);
    *reinterpret_cast<float4*>(sX + t * GP_PITCH + c) = make_float4(f[0], f[1], f[2], f[3]);
    *reinterpret_cast<float4*>(sX + t * GP_PITCH + c + 4) = make_float4(f[4], f[5], f[6], f[7]);
  }
  __syncthreads();
  // item = (token t, block of GP_OB gate rows); lanes run over tokens so the
  // gate-row reads are warp broadcasts
  const int nob = (O + GP_OB - 1) / GP_OB;
  for (int item = threadIdx.x; item < GP_TB * nob; item += GP_THREADS) {
    const int t = item % GP_TB, ob = item / GP_TB;
    const int tok = t0 + t;
    if (tok >= p.T) continue;
    float acc[GP_OB];
#pragma unroll
    for (int j = 0; j < GP_OB; ++j) acc[j] = 0.0f;
    const float* xr = sX + t * GP_PITCH;
#pragma unroll 4
    for (int c = 0; c < GP_DC; c += 4) {
      const float4 xv = *reinterpret_cast<const float4*>(xr + c);
#pragma unroll
      for (int j = 0; j < GP_OB; ++j) {
        const int o = ob * GP_OB + j < O ? ob * GP_OB + j : O - 1;  // clamped read, result unused
        const float4 wv = *reinterpret_cast<const float4*>(sW + o * GP_PITCH + c);
        acc[j] = fmaf(xv.x, wv.x, acc[j]);
        acc[j] = fmaf(xv.y, wv.y, acc[j]);
        acc[j] = fmaf(xv.z, wv.z, acc[j]);
        acc[j] = fmaf(xv.w, wv.w, acc[j]);
      }
    }
    float* dst = part + ((size_t)blockIdx.x * p.T + tok) * O;
#pragma unroll
    for (int j = 0; j < GP_OB; ++j)
      if (ob * GP_OB + j < O) dst[ob * GP_OB + j] = acc[j];
  }
}

// Decision kernel: GD_BT tokens per CTA (one warp each).  The chunk sums are
// split four ways (group g adds chunks g, g + 4, ... in order; then the four
// group sums are added in group order), so each thread keeps eight loads in
// flight and the result does not depend on the launch.
// With the prefetch (p.pf_w1, one tile of tokens) every CTA takes the same
// decisions, CTA 0 alone writes them, and CTA u then prefetches into L2 the
// first p.pf_row_bytes of each row of weight tile u of the up projection (the
// first tile the swapped-operand GEMM's CTA u streams), so the HBM otherwise
// idle during the codec kernels that follow fills L2 with weights.
constexpr int GD_SPLIT = 4;
__global__ void __launch_bounds__(SL_THREADS) gate_decide_kernel(const KParams p, const float* __restrict__ part,
                                                                 int n_chunks) {
  extern __shared__ float4 gd_smem_v[];
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  const int pairs = GD_BT * O;
  float* sLog = reinterpret_cast<float*>(gd_smem_v);                  // [GD_BT][O]
  float* sGrp = sLog + pairs;                                          // [GD_SPLIT][GD_BT * O]
  int* sIdx = reinterpret_cast<int*>(sGrp + GD_SPLIT * pairs);        // [GD_BT * k]
  __shared__ int s_base[128];
  __shared__ int s_active[129];  // prefetch: chosen experts in id order, then their count
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool pf = p.pf_w1 != nullptr;
  const int tile = pf ? 0 : blockIdx.x;
  const bool writer = !pf || blockIdx.x == 0;
  pdl_trigger();
  pdl_wait();
  const size_t plane = (size_t)p.T * O;
  for (int i = threadIdx.x; i < GD_SPLIT * pairs; i += SL_THREADS) {
    const int g = i / pairs, pr = i % pairs;
    const int tok = tile * GD_BT + pr / O;
    float sum = 0.0f;
    if (tok < p.T) {
      const float* src = part + (size_t)tok * O + pr % O;
      for (int c0 = g; c0 < n_chunks; c0 += 8 * GD_SPLIT) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int c = c0 + u * GD_SPLIT;
          v[u] = c < n_chunks ? src[(size_t)c * plane] : 0.0f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) sum += v[u];  // chunk order within the group
      }
    }
    sGrp[i] = sum;
  }
  __syncthreads();
  for (int pr = threadIdx.x; pr < pairs; pr += SL_THREADS) {
    const int o = pr % O;
    float sum = sGrp[pr];
#pragma unroll
    for (int g = 1; g < GD_SPLIT; ++g) sum += sGrp[g * pairs + pr];
    sLog[pr] = sum + (o < p.E ? p.b_local[o] : p.b_global[o - p.E]);
  }
  __syncthreads();
  for (int jj = warp; jj < GD_BT; jj += SL_THREADS / 32) {
    const int tok = tile * GD_BT + jj;
    if (tok < p.T)
      decide_token_warp(p, sLog + jj * O, tok, lane, (p.route_counts || pf) ? sIdx + jj * p.k : nullptr, writer);
  }
  __syncthreads();
  if (writer && p.route_counts) route_tile(p, tile, GD_BT, sIdx, s_base);
  if (!pf) return;
  // the chosen experts in id order (the swapped GEMM's active groups)
  if (warp == 0) {
    const int n_ent = p.T * p.k;
    int count = 0;
    for (int e0 = 0; e0 < p.E; e0 += 32) {
      const int e = e0 + lane;
      bool hit = false;
      for (int i = 0; i < n_ent; ++i) hit |= (sIdx[i] == e);
      const unsigned m = __ballot_sync(0xffffffffu, hit && e < p.E);
      if (hit && e < p.E) s_active[count + __popc(m & ((1u << lane) - 1u))] = e;
      count += __popc(m);
    }
    if (lane == 0) s_active[128] = count;
  }
  __syncthreads();
  const int tiles_per_expert = p.pf_dff / p.pf_tile_rows;
  const int a = blockIdx.x / tiles_per_expert;
  if (a >= s_active[128]) return;
  const int e = s_active[a];
  const int nb = blockIdx.x % tiles_per_expert;
  const int n_mats = p.pf_w3 ? 2 : 1;
  if (threadIdx.x < n_mats * p.pf_tile_rows) {
    const int m = threadIdx.x / p.pf_tile_rows;
    const long long row = (long long)e * p.pf_dff + (long long)nb * p.pf_tile_rows + threadIdx.x % p.pf_tile_rows;
    const char* base = static_cast<const char*>(m ? p.pf_w3 : p.pf_w1);
    const char* src = base + row * (long long)p.d * 2;
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(p.pf_row_bytes) : "memory");
  }
}

constexpr int GP_MAX_T = 256;
constexpr int GP_MIN_D = 1024;

}  // namespace

int gate_prefetch_max_tokens() { return GD_BT; }

size_t gate_partial_bytes(int T, int d, int E, int K) {
  const int O = E + (K == 1 ? 0 : K);
  if (T < 1 || T > GP_MAX_T || d < GP_MIN_D || d % 8 != 0 || O > MAXO) return 0;
  return (size_t)((d + GP_DC - 1) / GP_DC) * T * O * sizeof(float);
}

namespace {

template <typename TX>
cudaError_t launch_gate_partial(const GateArgs& a, const KParams& p, int O, cudaStream_t s) {
  const int n_chunks = (a.d + GP_DC - 1) / GP_DC;
  const int smem_a = static_cast<int>(gp_smem(O));
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(gate_partial_kernel<TX>), smem_a);
  if (e != cudaSuccess) return e;
  {
    KernelScope ks("gate_topk", s);
    e = launch_kernel(gate_partial_kernel<TX>, dim3(n_chunks, (a.T + GP_TB - 1) / GP_TB), dim3(GP_THREADS),
                      (size_t)smem_a, s, p, a.gate_partial);
    if (e != cudaSuccess) return e;
  }
  const int smem_b = (GD_BT * O * (1 + GD_SPLIT) + GD_BT * a.k) * 4;
  e = ensure_smem_attr(reinterpret_cast<const void*>(gate_decide_kernel), smem_b);
  if (e != cudaSuccess) return e;
  KernelScope ks("gate_decide", s);
  // with the prefetch: one CTA per swapped-GEMM CTA, all on the one tile
  const int blocks = p.pf_w1 ? a.pf_units : (a.T + GD_BT - 1) / GD_BT;
  e = launch_kernel(gate_decide_kernel, dim3(blocks), dim3(SL_THREADS), (size_t)smem_b, s, p,
                    static_cast<const float*>(a.gate_partial), n_chunks);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gate(const GateArgs& a, bool bf16, cudaStream_t s, bool* routed, int* held_sms) {
  if (routed) *routed = false;
  // The SIMT gates launch at least one CTA per SM once the batch fills the
  // GPU; counted as holding every SM.
  if (held_sms) *held_sms = sm_count();
  KParams p;
  p.X = a.X;
  p.W_local = a.W_local;
  p.b_local = a.b_local;
  p.W_global = a.W_global;
  p.b_global = a.b_global;
  for (int i = 0; i < 4; ++i) p.mask_bits[i] = a.mask_bits[i];
  p.T = a.T;
  p.d = a.d;
  p.E = a.E;
  p.K = a.K;
  p.k = a.k;
  p.renorm = a.renorm;
  p.top_groups = a.top_groups;
  p.topk_idx = a.topk_idx;
  p.topk_w = a.topk_w;
  p.route_counts = nullptr;
  p.route_rel = nullptr;
  p.pf_w1 = nullptr;
  p.pf_w3 = nullptr;
  p.pf_dff = p.pf_tile_rows = p.pf_row_bytes = 0;
  const int O = a.E + (a.K == 1 ? 0 : a.K);
  cudaError_t e;
  if (a.gate_partial && gate_partial_bytes(a.T, a.d, a.E, a.K) &&
      reinterpret_cast<uintptr_t>(a.gate_partial) % 16 == 0 && reinterpret_cast<uintptr_t>(a.W_local) % 16 == 0 &&
      (a.K == 1 || reinterpret_cast<uintptr_t>(a.W_global) % 16 == 0)) {
    if (a.route_counts && a.route_rel) {
      p.route_counts = a.route_counts;
      p.route_rel = a.route_rel;
      if (routed) *routed = true;
    }
    // the weight prefetch needs one tile of tokens, whole 16-byte pieces
    // and tiles that divide d_ff
    if (a.pf_w1 && a.T <= GD_BT && a.pf_units > 0 && a.pf_tile_rows > 0 && a.pf_tile_rows <= 128 &&
        a.pf_dff % a.pf_tile_rows == 0 && a.pf_row_bytes >= 16 && a.pf_row_bytes % 16 == 0 &&
        a.pf_row_bytes <= a.d * 2 && reinterpret_cast<uintptr_t>(a.pf_w1) % 16 == 0 &&
        reinterpret_cast<uintptr_t>(a.pf_w3) % 16 == 0 && a.d % 8 == 0) {
      p.pf_w1 = a.pf_w1;
      p.pf_w3 = a.pf_w3;
      p.pf_dff = a.pf_dff;
      p.pf_tile_rows = a.pf_tile_rows;
      p.pf_row_bytes = a.pf_row_bytes;
    }
    if (held_sms) *held_sms = (a.T + GD_BT - 1) / GD_BT;
    return bf16 ? launch_gate_partial<__nv_bfloat16>(a, p, O, s) : launch_gate_partial<float>(a, p, O, s);
  }
  {
    bool handled = false;
    e = launch_gate_tensor(a, p, O, bf16, s, routed, held_sms, &handled);
    if (handled || e != cudaSuccess) return e;
  }
  // Slice kernel when every gate row fits in shared memory next to the
  // partials: S slices of d_model per token (SW = d / S <= 128, a multiple of
  // 8), two tokens per thread while the slice is at most 64 wide, preferring
  // enough token tiles to give every SM two.
  {
    int S = 0, TPT = 2;
    for (int cand : {8, 16, 32}) {
      if (a.d % (8 * cand) != 0 || a.d / cand > 128) continue;
      S = cand;
      TPT = (a.d / cand <= 64) ? 2 : 1;
      const long long bt = (long long)(SL_THREADS / cand) * TPT;
      if ((a.T + bt - 1) / bt >= 2LL * sm_count()) break;
    }
    const int NB = O <= 16 ? 16 : 32;
    const int BT = S ? (SL_THREADS / S) * TPT : 0;
    const size_t smem = (size_t)O * a.d * 4 + (size_t)NB * (S * BT + SL_RED_PAD) * 4 + (size_t)BT * O * 4 +
                        (size_t)BT * a.k * 4;
    if (S && smem <= 160 * 1024) {
      const long long tiles = (a.T + BT - 1) / BT;
      if (a.route_counts && a.route_rel) {
        p.route_counts = a.route_counts;
        p.route_rel = a.route_rel;
        e = cudaMemsetAsync(a.route_counts, 0, sizeof(int32_t) * a.E, s);
        if (e != cudaSuccess) return e;
        if (routed) *routed = true;
      }
      const int per_sm = smem <= 72 * 1024 ? 3 : (smem <= 110 * 1024 ? 2 : 1);
      long long blocks = tiles < (long long)sm_count() * per_sm ? tiles : (long long)sm_count() * per_sm;
      if (blocks < 1) blocks = 1;
      const int nch = a.d / S / 8;
      KernelScope ks("gate_topk", s);
#define EC2MOE_SLICES(TX, XC, TP, NBV)                                                                       \
  do {                                                                                                      \
    e = ensure_smem_attr(reinterpret_cast<const void*>(gate_slices_kernel<TX, XC, TP, NBV>), (int)smem);     \
    if (e != cudaSuccess) return e;                                                                         \
    e = launch_kernel(gate_slices_kernel<TX, XC, TP, NBV>, dim3((int)blocks), dim3(SL_THREADS), smem, s, p, S); \
    if (e != cudaSuccess) return e;                                                                         \
  } while (0)
#define EC2MOE_SLICES_NB(TX, XC, TP) \
  do {                               \
    if (NB == 16) EC2MOE_SLICES(TX, XC, TP, 16); else EC2MOE_SLICES(TX, XC, TP, 32); \
  } while (0)
      if (bf16) {
        if (nch <= 4) EC2MOE_SLICES_NB(__nv_bfloat16, 4, 2);
        else if (nch <= 8) EC2MOE_SLICES_NB(__nv_bfloat16, 8, 2);
        else EC2MOE_SLICES_NB(__nv_bfloat16, 16, 1);
      } else {
        if (nch <= 4) EC2MOE_SLICES_NB(float, 4, 2);
        else if (nch <= 8) EC2MOE_SLICES_NB(float, 8, 2);
        else EC2MOE_SLICES_NB(float, 16, 1);
      }
#undef EC2MOE_SLICES_NB
#undef EC2MOE_SLICES
      return cudaGetLastError();
    }
  }
  // Register-tiled kernel when the gate rows do not fit in shared memory.
  if (a.d % GT_KC == 0 && O <= 144) {
    const int opt = O <= 80 ? 5 : 9;
    const size_t smem = (size_t)GT_BM * O * 4 + (size_t)GT_BM * a.k * 4;
    const long long tiles = (a.T + GT_BM - 1) / GT_BM;
    long long blocks = tiles < (long long)sm_count() * 2 ? tiles : (long long)sm_count() * 2;
    if (blocks < 1) blocks = 1;
    if (a.route_counts && a.route_rel) {
      p.route_counts = a.route_counts;
      p.route_rel = a.route_rel;
      e = cudaMemsetAsync(a.route_counts, 0, sizeof(int32_t) * a.E, s);
      if (e != cudaSuccess) return e;
      if (routed) *routed = true;
    }
    KernelScope ks("gate_topk", s);
#define EC2MOE_TILED(TX, OPTV)                                                                               \
  do {                                                                                                      \
    e = ensure_smem_attr(reinterpret_cast<const void*>(gate_tiled_kernel<TX, OPTV>), (int)smem);            \
    if (e != cudaSuccess) return e;                                                                         \
    e = launch_kernel(gate_tiled_kernel<TX, OPTV>, dim3((int)blocks), dim3(SL_THREADS), smem, s, p);        \
    if (e != cudaSuccess) return e;                                                                         \
  } while (0)
    if (bf16) {
      if (opt == 5) EC2MOE_TILED(__nv_bfloat16, 5); else EC2MOE_TILED(__nv_bfloat16, 9);
    } else {
      if (opt == 5) EC2MOE_TILED(float, 5); else EC2MOE_TILED(float, 9);
    }
#undef EC2MOE_TILED
    return cudaGetLastError();
  }
  const size_t base = (size_t)(WARPS * TPW * MAXO + WARPS * TPW * 32) * sizeof(float);
  const size_t wbytes = (size_t)O * a.d * sizeof(float);
  const bool w_smem = base + wbytes <= 200 * 1024;
  const size_t smem = base + (w_smem ? wbytes : 0);
  const int n_pass = (a.T + TPW - 1) / TPW;
  int blocks = (n_pass + WARPS - 1) / WARPS;
  // With the weights staged in shared memory, one persistent block per SM keeps
  // the staging traffic at one copy per SM.
  const int cap = w_smem ? sm_count() : sm_count() * 4;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  KernelScope ks("gate_topk", s);
#define EC2MOE_GATE_LAUNCH(TX, WS)                                                                          \
  do {                                                                                                      \
    e = ensure_smem_attr(reinterpret_cast<const void*>(gate_topk_kernel<TX, WS>), (int)smem);            \
    if (e != cudaSuccess) return e;                                                                         \
    e = launch_kernel(gate_topk_kernel<TX, WS>, dim3(blocks), dim3(WARPS * 32), smem, s, p);                 \
    if (e != cudaSuccess) return e;                                                                         \
  } while (0)
  if (bf16) {
    if (w_smem) EC2MOE_GATE_LAUNCH(__nv_bfloat16, true); else EC2MOE_GATE_LAUNCH(__nv_bfloat16, false);
  } else {
    if (w_smem) EC2MOE_GATE_LAUNCH(float, true); else EC2MOE_GATE_LAUNCH(float, false);
  }
#undef EC2MOE_GATE_LAUNCH
  return cudaGetLastError();
}

}  // namespace ec2moe
