// Grouped fp32 GEMM on the CUDA cores, for layers stored in fp32.
//
// The tensor cores have no fp32 x fp32 mode that keeps full fp32 products
// (kind::tf32 rounds the operands to 10 mantissa bits, about 1e-3 relative),
// so an fp32 layer that must agree with the oracle to 1e-4 runs here.  Same
// group semantics and epilogues as the tensor-core path: C_g = A_g B_g^T with
// A_g [M_g, K], B_g [N, K] rows of a weight stored [out, in].
//
// 64 x 64 output tile per 256-thread block, K staged 16 at a time in shared
// memory, 4 x 4 outputs per thread.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace ec2moe {
// bit 1: a group range (offsets) or a scatter destination (perm) outside the
// rows of the call was skipped
__device__ unsigned int g_simt_error;

namespace {

constexpr int TM = 64, TN = 64, TK = 16;
constexpr int MAX_GROUPS = 136;

struct SParams {
  const float* A;
  const float* B;
  const float* B2;
  const int32_t* offsets;
  int G, M, a_shared;
  long long a_row_base, out_row_base;
  int N, K, b_group_rows;
  float* out;
  long long ldo;
  const int32_t* perm;
  const float* scale;
  int rep_k;
  long long self_row_base;
  int n_tiles_n;
  long long a_rows, b_rows;
  long long row_limit;  // rows of the call: group ranges and scatter destinations lie in [0, row_limit)
};

template <int EPI>
__global__ void __launch_bounds__(256) simt_gemm_kernel(const SParams p) {
  pdl_trigger();
  pdl_wait();
  __shared__ int tile_prefix[MAX_GROUPS + 1];
  __shared__ int row0[MAX_GROUPS];
  __shared__ float sA[TK][TM + 4];
  __shared__ float sB[TK][TN + 4];
  __shared__ float sB2[(EPI == EPI_SWIGLU) ? TK : 1][TN + 4];
  if (threadIdx.x == 0) {
    int acc = 0;
    tile_prefix[0] = 0;
    for (int g = 0; g < p.G; ++g) {
      int r0, mg;
      if (p.offsets) {
        r0 = p.offsets[g];
        mg = p.offsets[g + 1] - r0;
        if (r0 < 0 || mg < 0 || static_cast<long long>(r0) + mg > p.row_limit) {
          // not a range of this call's rows: the group is skipped
          atomicOr(&g_simt_error, 2u);
          r0 = 0;
          mg = 0;
        }
      } else {
        r0 = g * p.M;
        mg = p.M;
      }
      row0[g] = r0;
      acc += (mg + TM - 1) / TM;
      tile_prefix[g + 1] = acc;
    }
  }
  __syncthreads();
  const int n_tiles = tile_prefix[p.G] * p.n_tiles_n;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    int g = 0;
    while (tile >= tile_prefix[g + 1] * p.n_tiles_n) ++g;
    const int mt = tile_prefix[g + 1] - tile_prefix[g];
    const int rem = tile - tile_prefix[g] * p.n_tiles_n;
    const int m_blk = rem % mt, n_blk = rem / mt;
    const int mg = p.offsets ? (p.offsets[g + 1] - p.offsets[g]) : p.M;
    const long long a_row0 = p.a_row_base + (p.offsets ? row0[g] : (p.a_shared ? 0 : row0[g])) + (long long)m_blk * TM;
    const long long b_row0 = (long long)g * p.b_group_rows + (long long)n_blk * TN;
    float acc[4][4] = {}, acc2[4][4] = {};
    for (int k0 = 0; k0 < p.K; k0 += TK) {
      // 64 x 16 tiles of A and B: 1024 elements each, 4 per thread.
      for (int i = threadIdx.x; i < TM * TK; i += 256) {
        const int r = i / TK, c = i % TK;
        const long long ar = a_row0 + r;
        const int kc = k0 + c;
        sA[c][r] = (m_blk * TM + r < mg && ar < p.a_rows && kc < p.K) ? p.A[ar * p.K + kc] : 0.0f;
        const long long br = b_row0 + r;
        const bool bok = (n_blk * TN + r < p.N) && br < p.b_rows && kc < p.K;
        sB[c][r] = bok ? p.B[br * p.K + kc] : 0.0f;
        if (EPI == EPI_SWIGLU) sB2[c][r] = bok ? p.B2[br * p.K + kc] : 0.0f;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < TK; ++kk) {
        float a[4], b[4], b2[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          a[i] = sA[kk][ty * 4 + i];
          b[i] = sB[kk][tx * 4 + i];
          if (EPI == EPI_SWIGLU) b2[i] = sB2[kk][tx * 4 + i];
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
            if (EPI == EPI_SWIGLU) acc2[i][j] = fmaf(a[i], b2[j], acc2[i][j]);
          }
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int local = m_blk * TM + ty * 4 + i;
      if (local >= mg) continue;
      const long long out_row = p.out_row_base + row0[g] + local;
      long long dest = out_row;
      float sc = 1.0f;
      if (EPI == EPI_SCATTER) {
        dest = p.perm ? p.perm[out_row] : out_row;
        if (dest < 0 || dest >= p.row_limit) {
          atomicOr(&g_simt_error, 2u);
          continue;
        }
        if (p.scale) sc = p.scale[dest];
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int col = n_blk * TN + tx * 4 + j;
        if (col >= p.N) continue;
        float v = acc[i][j];
        if (EPI == EPI_GELU) v = gelu_erf(v);
        if (EPI == EPI_SWIGLU) v = silu(v) * acc2[i][j];
        if (EPI == EPI_SCATTER) v *= sc;
        if (EPI == EPI_REPLICATE) {
          for (int r = 0; r < p.rep_k; ++r) p.out[(long long)p.perm[out_row * p.rep_k + r] * p.ldo + col] = v;
          if (p.self_row_base >= 0) p.out[(p.self_row_base + out_row) * p.ldo + col] = v;
        } else {
          p.out[dest * p.ldo + col] = v;
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_gemm_simt(const GemmArgs& a, int epi, cudaStream_t s) {
  if (a.G < 1 || a.G > MAX_GROUPS) return cudaErrorInvalidValue;
  SParams p;
  p.A = static_cast<const float*>(a.A);
  p.B = static_cast<const float*>(a.B);
  p.B2 = static_cast<const float*>(a.B2);
  p.offsets = a.offsets;
  p.row_limit = a.max_rows > 0 ? a.max_rows : (1LL << 62);
  p.G = a.G;
  p.M = a.M;
  p.a_shared = a.a_shared;
  p.a_row_base = a.a_row_base;
  p.out_row_base = a.out_row_base;
  p.N = a.N;
  p.K = a.K;
  p.b_group_rows = a.b_group_rows;
  p.out = static_cast<float*>(a.out);
  p.ldo = a.ldo;
  p.perm = a.perm;
  p.scale = a.scale;
  p.rep_k = a.rep_k;
  p.self_row_base = a.self_row_base;
  p.n_tiles_n = (a.N + TN - 1) / TN;
  p.a_rows = a.a_rows;
  p.b_rows = a.b_rows;
  const long long tiles = (a.max_rows / TM + a.G) * p.n_tiles_n;
  const long long cap = (long long)sm_count() * 8;
  const int grid = static_cast<int>(tiles < cap ? (tiles > 0 ? tiles : 1) : cap);
  KernelScope ks(a.name ? a.name : "gemm_simt", s);
  cudaError_t e = cudaSuccess;
  switch (epi) {
    case EPI_STORE: e = launch_kernel(simt_gemm_kernel<EPI_STORE>, dim3(grid), dim3(256), 0, s, p); break;
    case EPI_GELU: e = launch_kernel(simt_gemm_kernel<EPI_GELU>, dim3(grid), dim3(256), 0, s, p); break;
    case EPI_SWIGLU: e = launch_kernel(simt_gemm_kernel<EPI_SWIGLU>, dim3(grid), dim3(256), 0, s, p); break;
    case EPI_SCATTER: e = launch_kernel(simt_gemm_kernel<EPI_SCATTER>, dim3(grid), dim3(256), 0, s, p); break;
    case EPI_REPLICATE: e = launch_kernel(simt_gemm_kernel<EPI_REPLICATE>, dim3(grid), dim3(256), 0, s, p); break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t read_simt_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_simt_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_simt_error, &zero, sizeof(unsigned int));
}

}  // namespace ec2moe
