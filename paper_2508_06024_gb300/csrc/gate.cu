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
#include <stdlib.h>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace ec2moe {

__device__ unsigned int g_gate_error;  // bit 0: a bounded wait of the tensor-core gate timed out

namespace {

constexpr int WARPS = 4;
constexpr int TPW = 4;      // tokens per warp pass
constexpr int OB = 8;       // gate rows per accumulation block
constexpr int MAXO = 144;   // E + K <= 128 + 16
constexpr int MAX_TOPK = 8;

struct KParams {
  const void* X;
  const float* W_local;
  const float* b_local;
  const float* W_global;
  const float* b_global;
  uint32_t mask_bits[4];
  int T, d, E, K, k, renorm;
  int32_t* topk_idx;
  float* topk_w;
  int32_t* route_counts;  // fused routing: per-expert row counters (zero at launch); nullptr = gate only
  int32_t* route_rel;     // fused routing: [T*k] row of each entry relative to its expert's first row
};

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
            const float mk = L[p.E + grp];
            key[i] = (mk - G[grp]) + le;
            lw[i] = (mk - lse_m) + (le - G[grp]);
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
__device__ void decide_token_warp(const KParams& p, const float* L, int tok, int lane, int* s_idx) {
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
    const float mk_mine = (lane < p.K && lse_mine > -CUDART_INF_F) ? L[p.E + lane] : -CUDART_INF_F;
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
      key[i] = al[i] ? (mk - lse_g) + lv[i] : -CUDART_INF_F;
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
    p.topk_idx[(size_t)tok * p.k + lane] = id_mine;
    p.topk_w[(size_t)tok * p.k + lane] = p.renorm ? w_mine / wsum : w_mine;
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

struct GcLayout {
  int n_pad, O, k, E, stages;
  int stage_bytes, w3_off, raw_off;
  int log_stride;  // logits row of a token: O logits + 16 group scratch words, odd (conflict-free rows)
  int log_off, idx_off, tab_off, base_off, bias_off, bar_off, total;
  __host__ __device__ GcLayout(int O_, int k_, int E_, int stages_, bool prep)
      : O(O_), k(k_), E(E_), stages(stages_) {
    n_pad = (O + 15) / 16 * 16;
    w3_off = GC_BM * GC_BK * 2;
    raw_off = w3_off + 3 * n_pad * 128;
    stage_bytes = raw_off + (prep ? 0 : n_pad * 256);  // a multiple of 1024
    log_stride = (O + 16) | 1;
    log_off = stages * stage_bytes;
    idx_off = log_off + GC_BM * log_stride * 4;
    tab_off = idx_off + GC_BM * k * 4;
    base_off = tab_off + (GC_BM * k / 32) * E * 4;
    bias_off = base_off + 4 * E;
    bar_off = (bias_off + 4 * O + 7) / 8 * 8;
    total = bar_off + (3 * stages + 5) * 8 + 16;
  }
};

struct GcParams {
  KParams kp;
  int n_pad;
  int stages;
  long long timeout;
};

// One token's decision by one thread, from its logits row L[0..E) (local),
// L[E..E+K) (global) and a scratch row G[0..K) -- the arithmetic of
// decide_token_warp with sequential sums: per-group log-sum-exp over the
// allowed members (Eq. 5), log-sum-exp of the global logits over live groups
// (Eq. 6), key = (m_g - lse_g) + l_i (K = 1: l_i), weight exp((m_g - LSE_m) +
// (l_i - lse_g)) (Eq. 7); Top-k by insertion into a sorted list (larger key
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
__device__ void decide_token_thread(int E, int K, int k, int renorm, const MaskRegs m, const float* L, float* G,
                                    int32_t* topk_idx, float* topk_w, int tok, int* s_idx) {
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
      const float lse = mx > -CUDART_INF_F ? mx + logf(sum) : -CUDART_INF_F;
      G[g] = lse;
      if (lse > -CUDART_INF_F) mxm = fmaxf(mxm, L[E + g]);
    }
    float summ = 0.0f;
#pragma unroll 1
    for (int g = 0; g < K; ++g)
      if (G[g] > -CUDART_INF_F) summ += expf(L[E + g] - mxm);
    lse_m = mxm + logf(summ);
#pragma unroll 1
    for (int g = 0; g < ng; ++g) {
      const float lg = G[g];
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

// Rows of the tile reserved per expert (the layer path), with the worker warps
// only: entry i of the tile (token i / k, slot i % k) gets route_rel = the
// expert's reserved base + the number of earlier entries of the tile with the
// same expert.  32-entry chunks are ranked with a warp match, chunk counts are
// turned into per-expert prefixes, and one atomicAdd per expert reserves the
// tile's rows.
__device__ void route_tile_workers(const KParams& p, int tile, const int* sIdx, int* sTab, int* s_base, int wt) {
  const int wi = wt >> 5, lane = wt & 31;
  const int nt = GC_BM * p.k;
  const long long e0 = (long long)tile * nt;
  const long long n = (long long)p.T * p.k;
  const int live = (int)((n - e0) < nt ? (n - e0) : nt);
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
  const GcLayout L(O, p.k, p.E, gp.stages, PREP);
  const int S = gp.stages;
  float* sLog = reinterpret_cast<float*>(smem + L.log_off);
  int* sIdx = reinterpret_cast<int*>(smem + L.idx_off);
  int* sTab = reinterpret_cast<int*>(smem + L.tab_off);
  int* s_base = reinterpret_cast<int*>(smem + L.base_off);
  float* s_bias = reinterpret_cast<float*>(smem + L.bias_off);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bar_off);
  uint64_t* conv = full + S;
  uint64_t* empty = conv + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_tiles = (p.T + GC_BM - 1) / GC_BM;
  const int nk = (p.d + GC_BK - 1) / GC_BK;
  const long long budget = gp.timeout;
  const int n_pad = gp.n_pad;
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
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
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
      const int my_tiles = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
      const int total = my_tiles * nk;
      const int pre = PREP ? (total < S ? total : S) : 0;
      auto load_w = [&](int c, uint8_t* st, uint32_t fb) {
        const int kc = c % nk;
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
        tma_load_2d(smem_u32(smem + c * L.stage_bytes), &tmX, (c % nk) * GC_BK,
                    (blockIdx.x + (c / nk) * gridDim.x) * GC_BM, fb);
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
        tma_load_2d(smem_u32(st), &tmX, (c % nk) * GC_BK, (blockIdx.x + (c / nk) * gridDim.x) * GC_BM, fb);
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
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        for (int seg = 0; seg < nk && ok; seg += GC_SEG) {
          const uint32_t uses = acc ? uses1 : uses0;
          if (!mbar_wait(smem_u32(&tempty[acc]), (uses & 1u) ^ 1u, budget, abort_flag, &g_gate_error)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * GC_ACC_STRIDE;
          const int seg_end = seg + GC_SEG < nk ? seg + GC_SEG : nk;
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
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
      if (is_drain) {
        float acc[NB][16];
#pragma unroll
        for (int b = 0; b < NB; ++b)
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[b][j] = 0.0f;
        for (int seg = 0; seg < nk; seg += GC_SEG) {
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
            if (p.k == 1) decide_token_thread<1>(p.E, p.K, p.k, p.renorm, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
            else if (p.k == 2) decide_token_thread<2>(p.E, p.K, p.k, p.renorm, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
            else if (p.k <= 4) decide_token_thread<4>(p.E, p.K, p.k, p.renorm, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
            else decide_token_thread<8>(p.E, p.K, p.k, p.renorm, mregs, Lrow, Lrow + O, p.topk_idx, p.topk_w, tok, sx);
          }
        }
      } else if (!PREP) {
        // split the raw fp32 gate rows of each stage into three bf16 terms,
        // written in the swizzled K-major layout of the B operand
        const int ct = threadIdx.x - 192;
        for (int kc = 0; kc < nk; ++kc) {
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
        route_tile_workers(p, tile, sIdx, sTab, s_base, wt);
      }
    }
    tc_fence_before();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
  }
}

// Stages that fit next to the logits and routing tables.
int gc_stages(int O, int k, int E, bool prep) {
  for (int s = GC_MAX_STAGES; s >= 2; --s)
    if (GcLayout(O, k, E, s, prep).total + 1024 <= 232448) return s;
  return 0;
}

template <int NB, bool PREP>
cudaError_t launch_gate_tc_nb(const KParams& p, int stages, cudaStream_t s, const CUtensorMap& mX,
                              const CUtensorMap& mW, const CUtensorMap& mWg) {
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  GcParams gp;
  gp.kp = p;
  gp.n_pad = (O + 15) / 16 * 16;
  gp.stages = stages;
  gp.timeout = default_timeout_cycles();
  const int smem = GcLayout(O, p.k, p.E, stages, PREP).total + 1024;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(gate_tc_kernel<NB, PREP>), smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = (p.T + GC_BM - 1) / GC_BM;
  const int blocks = n_tiles < sm_count() ? n_tiles : sm_count();
  return launch_kernel(gate_tc_kernel<NB, PREP>, dim3(blocks), dim3(GC_THREADS), (size_t)smem, s, mX, mW, mWg, gp);
}

template <bool PREP>
cudaError_t launch_gate_tc(const KParams& p, int stages, cudaStream_t s, const CUtensorMap& mX,
                           const CUtensorMap& mW, const CUtensorMap& mWg) {
  const int O = p.E + (p.K == 1 ? 0 : p.K);
  switch ((O + 15) / 16) {
    case 1: return launch_gate_tc_nb<1, PREP>(p, stages, s, mX, mW, mWg);
    case 2: return launch_gate_tc_nb<2, PREP>(p, stages, s, mX, mW, mWg);
    case 3: return launch_gate_tc_nb<3, PREP>(p, stages, s, mX, mW, mWg);
    case 4: return launch_gate_tc_nb<4, PREP>(p, stages, s, mX, mW, mWg);
    default: return launch_gate_tc_nb<5, PREP>(p, stages, s, mX, mW, mWg);
  }
}

}  // namespace

cudaError_t launch_gate(const GateArgs& a, bool bf16, cudaStream_t s, bool* routed) {
  if (routed) *routed = false;
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
  p.topk_idx = a.topk_idx;
  p.topk_w = a.topk_w;
  p.route_counts = nullptr;
  p.route_rel = nullptr;
  const int O = a.E + (a.K == 1 ? 0 : a.K);
  cudaError_t e;
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
    const int stages = gc_stages(O, a.k, a.E, prep);
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
      e = prep ? launch_gate_tc<true>(p, stages, s, mX, mW, mWg) : launch_gate_tc<false>(p, stages, s, mX, mW, mWg);
      if (e != cudaSuccess) return e;
      return cudaGetLastError();
    }
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
