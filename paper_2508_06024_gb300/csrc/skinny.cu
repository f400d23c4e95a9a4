// Grouped bf16 GEMM for groups of at most 16 rows (decode-sized expert
// batches, Eq. 1 steps 4-5): C_g = A_g B_g^T where every group holds only a
// few token rows, so the work is streaming the weight rows once.
//
// The tensor-core kernel spends one 128-row MMA per 16 columns of K whatever
// the number of real rows; with one or two rows per expert it would be bound
// by MMA issue rather than by the weights.  Here a block owns one group and
// SK_WARPS * SK_CPW output columns; d_model (K) streams in chunks of SK_KC:
// the block stages the group's few activation rows for the chunk in shared
// memory, and every lane loads 16-byte pieces of its warp's weight rows (read
// from HBM exactly once) and accumulates fp32 dot products for every row of
// the group; a warp butterfly then sums the lanes.  The epilogues are those of
// the tensor-core kernel: plain store, GELU, SwiGLU (W1 and W3 rows of the same
// output column), or gate scale + scatter to the token's slot (Eq. 1 combine).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace ec2moe {

// bit 1: a group range (offsets) or a scatter destination (perm) outside the
// rows of the call was skipped
__device__ unsigned int g_skinny_error;

namespace {

constexpr int SK_WARPS = 8;
constexpr int SK_THREADS = 32 * SK_WARPS;
constexpr int SK_CPW = 2;     // output columns per warp
constexpr int SK_KC = 1024;   // K columns per staged chunk (four 16-byte pieces per lane)

struct SkParams {
  const __nv_bfloat16* A;
  const __nv_bfloat16* B;
  const __nv_bfloat16* B2;
  const int32_t* offsets;
  int G, M, a_shared;
  long long a_row_base, out_row_base;
  int N, K, b_group_rows;
  __nv_bfloat16* out;
  long long ldo;
  const int32_t* perm;
  const float* scale;
  int n_blocks;  // column blocks per group
  long long row_limit;  // rows of the call: group ranges and scatter destinations lie in [0, row_limit)
};

__device__ __forceinline__ void dot8(const U4& w, const float* a, float& acc) {
  acc = fmaf(bf16_lo(w.x), a[0], acc);
  acc = fmaf(bf16_hi(w.x), a[1], acc);
  acc = fmaf(bf16_lo(w.y), a[2], acc);
  acc = fmaf(bf16_hi(w.y), a[3], acc);
  acc = fmaf(bf16_lo(w.z), a[4], acc);
  acc = fmaf(bf16_hi(w.z), a[5], acc);
  acc = fmaf(bf16_lo(w.w), a[6], acc);
  acc = fmaf(bf16_hi(w.w), a[7], acc);
}

// One unit of work: group g, output columns n0 .. n0 + SK_CPW - 1 of a warp.
struct SkUnit {
  int u, g, r0, mg;
};

// The block's next unit at or after u that has rows (u >= units: none).
__device__ __forceinline__ SkUnit next_unit(const SkParams& p, int u, int units) {
  for (; u < units; u += gridDim.x) {
    const int g = u / p.n_blocks;
    int r0, mg;
    if (p.offsets) {
      r0 = p.offsets[g];
      mg = p.offsets[g + 1] - r0;
      if (r0 < 0 || mg < 0 || static_cast<long long>(r0) + mg > p.row_limit) {
        // not a range of this call's rows: the group is skipped
        atomicOr(&g_skinny_error, 2u);
        mg = 0;
      }
    } else {
      r0 = g * p.M;
      mg = p.M;
    }
    if (mg > 0) return SkUnit{u, g, r0, mg};
  }
  return SkUnit{units, 0, 0, 0};
}

// R >= the rows of every group (2, 4, 8 or 16).  Each block walks its units
// (grid-stride, skipping groups without rows) as one stream of K chunks; the
// weight pieces of the next chunk -- of this unit or of the next one -- are
// loaded into registers before the current chunk's activations are staged and
// used, so the weight stream does not stop on the staging, the FMAs or the
// change of unit.
template <int EPI, int R>
__global__ void __launch_bounds__(SK_THREADS) skinny_kernel(const SkParams p) {
  constexpr bool GLU = EPI == EPI_SWIGLU;
  constexpr int NJ = SK_KC / 256;  // 16-byte pieces per lane and weight row in a chunk
  __shared__ __align__(16) __nv_bfloat16 sA[R][SK_KC];
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int units = p.G * p.n_blocks;
  auto rows_of = [&](const SkUnit& un, const __nv_bfloat16* (&wr)[SK_CPW], const __nv_bfloat16* (&wr2)[SK_CPW],
                     bool (&lv)[SK_CPW]) {
    const int n0 = ((un.u % p.n_blocks) * SK_WARPS + warp) * SK_CPW;
#pragma unroll
    for (int cc = 0; cc < SK_CPW; ++cc) {
      lv[cc] = n0 + cc < p.N;
      const long long br = (long long)un.g * p.b_group_rows + (lv[cc] ? n0 + cc : 0);
      wr[cc] = p.B + br * p.K;
      wr2[cc] = GLU ? p.B2 + br * p.K : nullptr;
    }
  };
  auto load_w = [&](int kc, const __nv_bfloat16* const (&wr)[SK_CPW], const __nv_bfloat16* const (&wr2)[SK_CPW],
                    const bool (&lv)[SK_CPW], U4 (&dst)[NJ][SK_CPW], U4 (&dst2)[GLU ? NJ : 1][SK_CPW]) {
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
      const int c = kc + j * 256 + lane * 8;
#pragma unroll
      for (int cc = 0; cc < SK_CPW; ++cc) {
        const bool ok = c < p.K && lv[cc];
        dst[j][cc] = ok ? *reinterpret_cast<const U4*>(wr[cc] + c) : U4{0u, 0u, 0u, 0u};
        if (GLU) dst2[j][cc] = ok ? *reinterpret_cast<const U4*>(wr2[cc] + c) : U4{0u, 0u, 0u, 0u};
      }
    }
  };

  SkUnit cur = next_unit(p, blockIdx.x, units);
  if (cur.u >= units) return;
  const __nv_bfloat16* wrow[SK_CPW];
  const __nv_bfloat16* wrow2[SK_CPW];
  bool live[SK_CPW];
  rows_of(cur, wrow, wrow2, live);
  U4 w[NJ][SK_CPW], w2[GLU ? NJ : 1][SK_CPW];
  load_w(0, wrow, wrow2, live, w, w2);
  while (true) {
    int mg = cur.mg > R ? R : cur.mg;  // the host guarantees mg <= R
    const long long a_row = p.a_row_base + (p.offsets ? cur.r0 : (p.a_shared ? 0 : cur.r0));
    float acc[SK_CPW][R];
    float acc2[GLU ? SK_CPW : 1][GLU ? R : 1];
#pragma unroll
    for (int cc = 0; cc < SK_CPW; ++cc)
#pragma unroll
      for (int r = 0; r < R; ++r) {
        acc[cc][r] = 0.0f;
        if (GLU) acc2[cc][r] = 0.0f;
      }
    SkUnit nxt{units, 0, 0, 0};
    const __nv_bfloat16* nrow[SK_CPW];
    const __nv_bfloat16* nrow2[SK_CPW];
    bool nlive[SK_CPW];
    for (int kc = 0; kc < p.K; kc += SK_KC) {
      const int kw = p.K - kc < SK_KC ? p.K - kc : SK_KC;
      U4 wn[NJ][SK_CPW], wn2[GLU ? NJ : 1][SK_CPW];
      const bool last = kc + SK_KC >= p.K;
      if (!last) {
        load_w(kc + SK_KC, wrow, wrow2, live, wn, wn2);  // in flight during this chunk
      } else {
        nxt = next_unit(p, cur.u + gridDim.x, units);
        if (nxt.u < units) {
          rows_of(nxt, nrow, nrow2, nlive);
          load_w(0, nrow, nrow2, nlive, wn, wn2);  // the next unit's first chunk
        }
      }
      __syncthreads();
      const int vec = kw / 8;
      for (int i = threadIdx.x; i < mg * vec; i += SK_THREADS) {
        const int r = i / vec, c = (i % vec) * 8;
        *reinterpret_cast<U4*>(&sA[r][c]) = *reinterpret_cast<const U4*>(p.A + (a_row + r) * p.K + kc + c);
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        const int c = j * 256 + lane * 8;
        if (c < kw) {
#pragma unroll
          for (int r = 0; r < R; ++r) {
            if (r < mg) {
              float a[8];
              load8(&sA[r][c], a);
#pragma unroll
              for (int cc = 0; cc < SK_CPW; ++cc) {
                dot8(w[j][cc], a, acc[cc][r]);
                if (GLU) dot8(w2[j][cc], a, acc2[cc][r]);
              }
            }
          }
        }
      }
#pragma unroll
      for (int j = 0; j < NJ; ++j)
#pragma unroll
        for (int cc = 0; cc < SK_CPW; ++cc) {
          w[j][cc] = wn[j][cc];
          if (GLU) w2[j][cc] = wn2[j][cc];
        }
    }
    // lane sums, then lane cc * R + r stores (column n0 + cc, row r)
    const int n0 = ((cur.u % p.n_blocks) * SK_WARPS + warp) * SK_CPW;
#pragma unroll
    for (int cc = 0; cc < SK_CPW; ++cc)
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (r >= mg) break;  // uniform across the warp
        float v = acc[cc][r];
        float v2 = GLU ? acc2[cc][r] : 0.0f;
#pragma unroll
        for (int sh = 16; sh > 0; sh >>= 1) {
          v += __shfl_xor_sync(0xffffffffu, v, sh);
          if (GLU) v2 += __shfl_xor_sync(0xffffffffu, v2, sh);
        }
        if (lane == cc * R + r && live[cc]) {
          const long long out_row = p.out_row_base + cur.r0 + r;
          long long dest = out_row;
          float y;
          if (EPI == EPI_SWIGLU) y = silu_bf16out(v) * v2;
          else if (EPI == EPI_GELU) y = gelu_bf16out(v);
          else y = v;
          bool ok = true;
          if (EPI == EPI_SCATTER) {
            dest = p.perm ? p.perm[out_row] : out_row;
            ok = dest >= 0 && dest < p.row_limit;
            if (!ok) atomicOr(&g_skinny_error, 2u);
            else if (p.scale) y *= p.scale[dest];
          }
          if (ok) p.out[dest * p.ldo + n0 + cc] = __float2bfloat16_rn(y);
        }
      }
    if (nxt.u >= units) break;
    cur = nxt;
#pragma unroll
    for (int cc = 0; cc < SK_CPW; ++cc) {
      wrow[cc] = nrow[cc];
      wrow2[cc] = nrow2[cc];
      live[cc] = nlive[cc];
    }
  }
}

template <int R>
cudaError_t launch_r(const SkParams& p, int epi, int grid, cudaStream_t s) {
  switch (epi) {
    case EPI_GELU: return launch_kernel(skinny_kernel<EPI_GELU, R>, dim3(grid), dim3(SK_THREADS), 0, s, p);
    case EPI_SWIGLU: return launch_kernel(skinny_kernel<EPI_SWIGLU, R>, dim3(grid), dim3(SK_THREADS), 0, s, p);
    case EPI_SCATTER: return launch_kernel(skinny_kernel<EPI_SCATTER, R>, dim3(grid), dim3(SK_THREADS), 0, s, p);
    default: return launch_kernel(skinny_kernel<EPI_STORE, R>, dim3(grid), dim3(SK_THREADS), 0, s, p);
  }
}

}  // namespace

// Used where it beats the tensor-core kernel on decode steps (measured on the
// d = 4096, d_ff = 14336 SwiGLU shape): down projections (store / scatter)
// with at most four rows per group, up projections with at most two.  There
// the tensor-core kernel's 128-row MMAs do almost no useful work and few
// tiles exist; with more rows it streams the weights faster.
bool gemm_skinny_supported(const GemmArgs& a, int epi) {
  if (epi == EPI_PARTIAL) return false;
  const int limit = (epi == EPI_GELU || epi == EPI_SWIGLU) ? 2 : 4;
  return a.group_rows_bound > 0 && a.group_rows_bound <= limit && a.K % 8 == 0 && epi != EPI_REPLICATE &&
         (reinterpret_cast<uintptr_t>(a.A) % 16 == 0) && (reinterpret_cast<uintptr_t>(a.B) % 16 == 0) &&
         (epi != EPI_SWIGLU || reinterpret_cast<uintptr_t>(a.B2) % 16 == 0);
}

cudaError_t launch_gemm_skinny(const GemmArgs& a, int epi, cudaStream_t s) {
  if (!gemm_skinny_supported(a, epi)) return cudaErrorInvalidValue;
  SkParams p;
  p.A = static_cast<const __nv_bfloat16*>(a.A);
  p.B = static_cast<const __nv_bfloat16*>(a.B);
  p.B2 = static_cast<const __nv_bfloat16*>(a.B2);
  p.offsets = a.offsets;
  p.G = a.G;
  p.M = a.M;
  p.a_shared = a.a_shared;
  p.a_row_base = a.a_row_base;
  p.out_row_base = a.out_row_base;
  p.N = a.N;
  p.K = a.K;
  p.b_group_rows = a.b_group_rows;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ldo = a.ldo;
  p.perm = a.perm;
  p.scale = a.scale;
  p.n_blocks = (a.N + SK_WARPS * SK_CPW - 1) / (SK_WARPS * SK_CPW);
  p.row_limit = a.max_rows > 0 ? a.max_rows : (1LL << 62);
  const long long units = (long long)a.G * p.n_blocks;
  const long long cap = (long long)sm_count() * 8;
  const int grid = (int)(units < cap ? units : cap);
  KernelScope ks(a.name ? a.name : "gemm_skinny", s);
  const long long rb = a.group_rows_bound;
  cudaError_t e = rb <= 2 ? launch_r<2>(p, epi, grid, s)
                          : (rb <= 4 ? launch_r<4>(p, epi, grid, s)
                                     : (rb <= 8 ? launch_r<8>(p, epi, grid, s) : launch_r<16>(p, epi, grid, s)));
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t read_skinny_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_skinny_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_skinny_error, &zero, sizeof(unsigned int));
}

}  // namespace ec2moe
