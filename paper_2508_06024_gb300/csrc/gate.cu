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
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include "common.cuh"
#include "internal.h"

namespace ec2moe {
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
};

__device__ __forceinline__ bool allowed_bit(const KParams& p, int e) { return (p.mask_bits[e >> 5] >> (e & 31)) & 1u; }

// (key, idx) ordering for Top-k: larger key first, ties to the lower index.
__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) { return ka > kb || (ka == kb && ia < ib); }

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
        // remove the winner from its owner's candidates
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (lane + 32 * i == bi) key[i] = -CUDART_INF_F;
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

}  // namespace

cudaError_t launch_gate(const GateArgs& a, bool bf16, cudaStream_t s) {
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
  const int O = a.E + (a.K == 1 ? 0 : a.K);
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
  cudaError_t e;
  KernelScope ks("gate_topk", s);
#define EC2MOE_GATE_LAUNCH(TX, WS)                                                                          \
  do {                                                                                                      \
    e = cudaFuncSetAttribute(gate_topk_kernel<TX, WS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
    if (e != cudaSuccess) return e;                                                                         \
    gate_topk_kernel<TX, WS><<<blocks, WARPS * 32, smem, s>>>(p);                                           \
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
