// Step 3b and step 5b of the layer: per-expert histogram, exclusive scan and
// stable expert-major permutation of the (token, slot) pairs chosen by Top-k;
// the row gather into expert order; and the fixed-order combine of Eq. 1.
//
// Routing runs as two kernels over blocks of CHUNK consecutive (token, slot)
// entries:
//   count    shared-memory atomic histogram per block -> blk_counts[b][e]
//   scatter  each block derives its expert bases from the column sums of
//            blk_counts, ranks its entries stably inside the block
//            (warp match + popc, then a prefix over the block's warps) and
//            writes perm / inv_perm; block 0 also writes counts and offsets.
// Rows of one expert therefore keep increasing (t, s) order, which makes the
// permutation (and everything downstream) deterministic.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>

#include "ec2moe.h"
#include "common.cuh"
#include "internal.h"

namespace ec2moe {
namespace {

// Histogram cells of ec2moe_route_noalloc: one int32 per (block of 1024
// entries, expert), EC2MOE_ROUTE_NOALLOC_MAX_CELLS of them (64 KiB).  Every GPU
// that loads the library keeps this array until the process exits.  All calls
// on a device share it; the count kernel writes every cell the scatter kernel
// later reads, so nothing in it has to start at zero, but two calls whose
// kernels overlap on the GPU race on it.
static __device__ __align__(256) int32_t g_route_noalloc_cells[EC2MOE_ROUTE_NOALLOC_MAX_CELLS];

// Bit 0: a routing kernel met an expert id outside [0, E) in the caller's
// topk_idx, or a gather met a permutation entry outside [0, rows).  Such
// entries are skipped (no shared or global access through them) and
// ec2moe_last_device_error reports EC2MOE_ERR_INVALID_ARG.
__device__ unsigned int g_route_error;

constexpr int CHUNK = 1024;  // entries per block (one per thread)
constexpr int MAXE = 128;

__device__ __forceinline__ bool valid_expert(int e, int E) {
  if (static_cast<unsigned>(e) < static_cast<unsigned>(E)) return true;
  atomicOr(&g_route_error, 1u);
  return false;
}

__global__ void __launch_bounds__(CHUNK) route_count_kernel(const int32_t* __restrict__ idx, long long n, int E,
                                                            int32_t* __restrict__ blk_counts) {
  pdl_trigger();
  pdl_wait();
  __shared__ int hist[MAXE];
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[e] = 0;
  __syncthreads();
  const long long i = (long long)blockIdx.x * CHUNK + threadIdx.x;
  if (i < n) {
    const int e = idx[i];
    if (valid_expert(e, E)) atomicAdd(&hist[e], 1);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) blk_counts[(long long)blockIdx.x * E + e] = hist[e];
}

__global__ void __launch_bounds__(CHUNK) route_scatter_kernel(const int32_t* __restrict__ idx, long long n, int E,
                                                              const int32_t* __restrict__ blk_counts, int nblk,
                                                              int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                                                              int32_t* __restrict__ perm, int32_t* __restrict__ inv_perm) {
  pdl_trigger();
  pdl_wait();
  __shared__ int s_pre[MAXE];           // entries of expert e in earlier blocks
  __shared__ int s_base[MAXE];          // offsets[e] + s_pre[e]
  __shared__ int s_tot[MAXE];
  __shared__ int s_wcnt[CHUNK / 32][MAXE];  // per-warp counts, then per-warp exclusive prefix
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < (CHUNK / 32) * MAXE; i += blockDim.x) (&s_wcnt[0][0])[i] = 0;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int pre = 0, tot = 0;
    for (int b = 0; b < nblk; ++b) {
      const int c = blk_counts[(long long)b * E + e];
      if (b < (int)blockIdx.x) pre += c;
      tot += c;
    }
    s_pre[e] = pre;
    s_tot[e] = tot;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int e = 0; e < E; ++e) {
      const int c = s_tot[e];
      s_base[e] = acc + s_pre[e];
      if (blockIdx.x == 0) {
        counts[e] = c;
        offsets[e] = acc;
      }
      acc += c;
    }
    if (blockIdx.x == 0) offsets[E] = acc;
  }
  const long long i = (long long)blockIdx.x * CHUNK + threadIdx.x;
  int e = i < n ? idx[i] : -1;
  const bool live = i < n && valid_expert(e, E);
  if (i < n && !live && inv_perm) inv_perm[i] = -1;
  const unsigned act = __ballot_sync(0xffffffffu, live);
  int rank_w = 0;
  if (live) {
    const unsigned same = __match_any_sync(act, e);
    rank_w = __popc(same & ((1u << lane) - 1u));
    if (rank_w == 0) s_wcnt[warp][e] = __popc(same);
  }
  __syncthreads();
  for (int ee = threadIdx.x; ee < E; ee += blockDim.x) {
    int acc = 0;
    for (int w = 0; w < CHUNK / 32; ++w) {
      const int c = s_wcnt[w][ee];
      s_wcnt[w][ee] = acc;
      acc += c;
    }
  }
  __syncthreads();
  if (live) {
    const int pos = s_base[e] + s_wcnt[warp][e] + rank_w;
    perm[pos] = static_cast<int32_t>(i);
    if (inv_perm) inv_perm[i] = pos;
  }
}

// Whole routing in one block for up to SMALL_MAX entries: histogram
// (warp-aggregated shared atomics), exclusive scan, then the entries in
// 1024-entry rounds in order, each ranked inside the round (warp match +
// prefix over warps) on top of per-expert running bases.  Same results as the
// two-kernel path.
constexpr int SMALL_MAX = 16384;

__global__ void __launch_bounds__(CHUNK) route_small_kernel(const int32_t* __restrict__ idx, int n, int E,
                                                            int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                                                            int32_t* __restrict__ perm, int32_t* __restrict__ inv_perm) {
  pdl_trigger();
  pdl_wait();
  __shared__ int hist[MAXE];
  __shared__ int base[MAXE];
  __shared__ int tot[MAXE];
  __shared__ int wcnt[CHUNK / 32][MAXE];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[e] = 0;
  __syncthreads();
  for (int i0 = 0; i0 < n; i0 += CHUNK) {
    const int i = i0 + threadIdx.x;
    const int e = i < n ? idx[i] : -1;
    const bool live = i < n && valid_expert(e, E);
    const unsigned act = __ballot_sync(0xffffffffu, live);
    if (live) {
      const unsigned same = __match_any_sync(act, e);
      if ((same & ((1u << lane) - 1u)) == 0) atomicAdd(&hist[e], __popc(same));
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int e = 0; e < E; ++e) {
      base[e] = acc;
      counts[e] = hist[e];
      offsets[e] = acc;
      acc += hist[e];
    }
    offsets[E] = acc;
  }
  for (int i0 = 0; i0 < n; i0 += CHUNK) {
    for (int c = threadIdx.x; c < (CHUNK / 32) * MAXE; c += blockDim.x) (&wcnt[0][0])[c] = 0;
    __syncthreads();
    const int i = i0 + threadIdx.x;
    int e = i < n ? idx[i] : -1;
    const bool live = i < n && static_cast<unsigned>(e) < static_cast<unsigned>(E);
    if (i < n && !live && inv_perm) inv_perm[i] = -1;
    const unsigned act = __ballot_sync(0xffffffffu, live);
    int rank_w = 0;
    if (live) {
      const unsigned same = __match_any_sync(act, e);
      rank_w = __popc(same & ((1u << lane) - 1u));
      if (rank_w == 0) wcnt[warp][e] = __popc(same);
    }
    __syncthreads();
    for (int ee = threadIdx.x; ee < E; ee += blockDim.x) {
      int acc = 0;
      for (int w = 0; w < CHUNK / 32; ++w) {
        const int c = wcnt[w][ee];
        wcnt[w][ee] = acc;
        acc += c;
      }
      tot[ee] = acc;
    }
    __syncthreads();
    if (live) {
      const int pos = base[e] + wcnt[warp][e] + rank_w;
      perm[pos] = i;
      if (inv_perm) inv_perm[i] = pos;
    }
    __syncthreads();
    for (int ee = threadIdx.x; ee < E; ee += blockDim.x) base[ee] += tot[ee];
  }
}

// dst[p] = src[perm[p] / k]; one warp per row, 16-byte lanes.
__global__ void gather_rows_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                   const int32_t* __restrict__ perm, long long rows, int k, int row_bytes) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const long long warps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long r = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += warps) {
    const int32_t p = perm[r];
    if (static_cast<unsigned long long>(p) >= static_cast<unsigned long long>(rows)) {
      if (lane == 0) atomicOr(&g_route_error, 1u);
      continue;
    }
    const long long t = p / k;
    const U4* s = reinterpret_cast<const U4*>(src + t * row_bytes);
    U4* d = reinterpret_cast<U4*>(dst + r * row_bytes);
    for (int c = lane; c < row_bytes / 16; c += 32) d[c] = s[c];
  }
}

// Rows into expert order from relative positions (routing fused into the
// gate): pos = offsets[e] + rel[i], dst[pos] = src[i / k], perm[pos] = i.
// Each block derives the offsets from the counts; block 0 publishes them.
__global__ void gather_rel_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                  const int32_t* __restrict__ idx, const int32_t* __restrict__ counts,
                                  const int32_t* __restrict__ rel, int32_t* __restrict__ perm,
                                  int32_t* __restrict__ offsets, int E, long long n, int k, int row_bytes) {
  pdl_trigger();
  pdl_wait();
  __shared__ int s_off[MAXE + 1];
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32)
    warp_exclusive_scan<(MAXE + 31) / 32>(E, lane, [&](int e) { return counts[e]; }, s_off,
                                          blockIdx.x == 0 ? offsets : nullptr);
  __syncthreads();
  const long long warps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long i = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < n; i += warps) {
    const int e = idx[i];
    if (static_cast<unsigned>(e) >= static_cast<unsigned>(E)) {
      if (lane == 0) atomicOr(&g_route_error, 1u);
      continue;
    }
    const int pos = s_off[e] + rel[i];
    if (lane == 0) perm[pos] = static_cast<int32_t>(i);
    const U4* sr = reinterpret_cast<const U4*>(src + (i / k) * row_bytes);
    U4* dr = reinterpret_cast<U4*>(dst + (long long)pos * row_bytes);
    for (int c = lane; c < row_bytes / 16; c += 32) dr[c] = sr[c];
  }
}

// Eight consecutive elements held as loaded (bf16: 16 bytes, fp32: 32 bytes).
template <typename TE>
struct Raw8;
template <>
struct Raw8<__nv_bfloat16> {
  U4 q;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { q = *reinterpret_cast<const U4*>(p); }
  __device__ __forceinline__ void add_to(float* acc) const {
    acc[0] += bf16_lo(q.x); acc[1] += bf16_hi(q.x); acc[2] += bf16_lo(q.y); acc[3] += bf16_hi(q.y);
    acc[4] += bf16_lo(q.z); acc[5] += bf16_hi(q.z); acc[6] += bf16_lo(q.w); acc[7] += bf16_hi(q.w);
  }
};
template <>
struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = *reinterpret_cast<const float4*>(p);
    b = *reinterpret_cast<const float4*>(p + 4);
  }
  __device__ __forceinline__ void add_to(float* acc) const {
    acc[0] += a.x; acc[1] += a.y; acc[2] += a.z; acc[3] += a.w;
    acc[4] += b.x; acc[5] += b.y; acc[6] += b.z; acc[7] += b.w;
  }
};
constexpr int CB_MAX_K = 8;       // Top-k limit of the ABI
constexpr int CB_MAX_SHARED = 4;  // shared-expert limit of the ABI
static_assert(CB_MAX_K == EC2MOE_MAX_TOPK && CB_MAX_SHARED == EC2MOE_MAX_SHARED, "combine limits follow the ABI");

// y[t] = sum_s slot[t*k+s] + sum_j shared[j*T+t] in that order, fp32 sum.
// All k + n_shared <= R rows of an 8-column chunk are loaded before the first
// add, so a thread keeps them in flight together; R is the smallest of 2, 4,
// 8, 12 that holds them, so the register count (and occupancy) follows the
// rows a token actually has.
template <typename TE, int R>
__global__ void combine_kernel(const TE* __restrict__ slot, const TE* __restrict__ shared, int n_shared,
                               TE* __restrict__ Y, int T, int k, int d) {
  pdl_trigger();
  pdl_wait();
  const int per_row = d / 8;
  const int rows = k + n_shared;
  const long long total = (long long)T * per_row;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const long long t = i / per_row;
    const int c = static_cast<int>(i % per_row) * 8;
    Raw8<TE> r[R];
#pragma unroll
    for (int q = 0; q < R; ++q)
      if (q < rows)
        r[q].load(q < k ? slot + (t * k + q) * d + c : shared + ((long long)(q - k) * T + t) * d + c);
    float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
    for (int q = 0; q < R; ++q)
      if (q < rows) r[q].add_to(acc);
    store8(Y + t * d + c, acc);
  }
}

}  // namespace

int route_blocks(long long n_entries) { return static_cast<int>((n_entries + CHUNK - 1) / CHUNK); }

cudaError_t launch_route(const int32_t* topk_idx, long long n, int E, int32_t* blk_counts, int32_t* counts,
                         int32_t* offsets, int32_t* perm, int32_t* inv_perm, cudaStream_t s) {
  const int nblk = route_blocks(n);
  if (nblk == 0) {
    // No entries: counts = 0, offsets = 0.
    cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int32_t) * E, s);
    if (e != cudaSuccess) return e;
    return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), s);
  }
  if (n <= SMALL_MAX) {
    KernelScope ks("route", s);
    return launch_kernel(route_small_kernel, dim3(1), dim3(CHUNK), 0, s, topk_idx, static_cast<int>(n), E, counts,
                         offsets, perm, inv_perm);
  }
  {
    KernelScope ks("route_count", s);
    cudaError_t e = launch_kernel(route_count_kernel, dim3(nblk), dim3(CHUNK), 0, s, topk_idx, n, E, blk_counts);
    if (e != cudaSuccess) return e;
  }
  {
    KernelScope ks("route_scatter", s);
    cudaError_t e = launch_kernel(route_scatter_kernel, dim3(nblk), dim3(CHUNK), 0, s, topk_idx, n, E,
                                  (const int32_t*)blk_counts, nblk, counts, offsets, perm, inv_perm);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

// Id of the current CUDA context (driver entry points reached through the
// runtime, so the library needs no link against libcuda).  False when there is
// no current context yet or the entry points are missing.
static bool current_context_id(unsigned long long* id) {
  using GetCurrentFn = CUresult (*)(CUcontext*);
  using GetIdFn = CUresult (*)(CUcontext, unsigned long long*);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(f);
  });
  if (!get_current || !get_id) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// Device address of g_route_noalloc_cells for the current device.  The host-side
// name of a __device__ array is only a stand-in, so the address is looked up
// with the device current and cached per device, keyed on the context's id: a
// cudaDeviceReset destroys the context (and the array with it), and the next
// call then looks the address up again in the new context.
static cudaError_t noalloc_cells(int32_t** out) {
  constexpr int MAX_DEVICES = 64;
  struct Entry {
    int32_t* ptr;
    unsigned long long ctx;
  };
  static std::mutex mu;
  static Entry cache[MAX_DEVICES] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= MAX_DEVICES) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  unsigned long long ctx = 0;
  const bool known_ctx = current_context_id(&ctx);
  if (!cache[dev].ptr || !known_ctx || cache[dev].ctx != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_route_noalloc_cells);
    if (e != cudaSuccess) return e;
    unsigned long long ctx_now = 0;
    cache[dev] = Entry{static_cast<int32_t*>(p), current_context_id(&ctx_now) ? ctx_now : 0ull};
  }
  *out = cache[dev].ptr;
  return cudaSuccess;
}

cudaError_t launch_route_noalloc(const int32_t* topk_idx, long long n, int E, int32_t* counts, int32_t* offsets,
                                 int32_t* perm, int32_t* inv_perm, cudaStream_t s) {
  if ((long long)route_blocks(n) * E > EC2MOE_ROUTE_NOALLOC_MAX_CELLS) return cudaErrorInvalidValue;
  int32_t* cells = nullptr;
  cudaError_t e = noalloc_cells(&cells);
  if (e != cudaSuccess) return e;
  return launch_route(topk_idx, n, E, cells, counts, offsets, perm, inv_perm, s);
}

cudaError_t launch_gather(const void* src, void* dst, const int32_t* perm, long long rows, int k, int width, bool bf16,
                          cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  const int row_bytes = width * (bf16 ? 2 : 4);
  const int warps_per_block = 8;
  long long blocks = (rows + warps_per_block - 1) / warps_per_block;
  const long long cap = (long long)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  {
    KernelScope ks("gather_rows", s);
    cudaError_t e = launch_kernel(gather_rows_kernel, dim3(static_cast<int>(blocks)), dim3(warps_per_block * 32), 0, s,
                                  static_cast<const uint8_t*>(src), static_cast<uint8_t*>(dst), perm, rows, k, row_bytes);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_gather_rel(const void* src, void* dst, const int32_t* topk_idx, const int32_t* counts,
                              const int32_t* rel, int32_t* perm, int32_t* offsets, int E, long long n, int k,
                              int width, bool bf16, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int row_bytes = width * (bf16 ? 2 : 4);
  const int warps_per_block = 8;
  long long blocks = (n + warps_per_block - 1) / warps_per_block;
  const long long cap = (long long)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  KernelScope ks("gather_rows", s);
  return launch_kernel(gather_rel_kernel, dim3(static_cast<int>(blocks)), dim3(warps_per_block * 32), 0, s,
                       static_cast<const uint8_t*>(src), static_cast<uint8_t*>(dst), topk_idx, counts, rel, perm,
                       offsets, E, n, k, row_bytes);
}

__global__ void sum_counts_kernel(const int32_t* __restrict__ parts, int n_parts, int E, int32_t* __restrict__ counts) {
  pdl_trigger();
  pdl_wait();
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < E; e += gridDim.x * blockDim.x) {
    int32_t c = 0;
    for (int p = 0; p < n_parts; ++p) c += parts[(size_t)p * E + e];
    counts[e] = c;
  }
}

cudaError_t read_route_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_route_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_route_error, &zero, sizeof(unsigned int));
}

cudaError_t launch_sum_counts(const int32_t* parts, int n_parts, int E, int32_t* counts, cudaStream_t s) {
  KernelScope ks("sum_counts", s);
  cudaError_t e = launch_kernel(sum_counts_kernel, dim3(1), dim3(128), 0, s, parts, n_parts, E, counts);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Split-K sums into bf16.  A block covers 64 (row, 4-column) items with 4
// threads each: thread group g adds the planes s = g, g + 4, ... (8 loads in
// flight), then the four group sums are added in group order and rounded
// once -- a fixed order, so the result does not depend on the launch.
constexpr int SUM_ITEMS = 64;
constexpr int SUM_GROUPS = 4;
__global__ void __launch_bounds__(SUM_ITEMS * SUM_GROUPS)
    splitk_sum_kernel(const float* __restrict__ partial, int S, long long rows, int N,
                      __nv_bfloat16* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  __shared__ float4 part[SUM_GROUPS][SUM_ITEMS];
  const int it = threadIdx.x % SUM_ITEMS, grp = threadIdx.x / SUM_ITEMS;
  const long long per_row = N / 4;
  const long long total = rows * per_row;
  const long long plane = rows * N;
  for (long long base = (long long)blockIdx.x * SUM_ITEMS; base < total; base += (long long)gridDim.x * SUM_ITEMS) {
    const long long i = base + it;
    const long long at = i < total ? (i / per_row) * N + (i % per_row) * 4 : 0;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    if (i < total) {
      for (int s0 = grp; s0 < S; s0 += 8 * SUM_GROUPS) {
        float4 v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int s = s0 + j * SUM_GROUPS;
          v[j] = s < S ? *reinterpret_cast<const float4*>(partial + s * plane + at) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          acc.x += v[j].x;
          acc.y += v[j].y;
          acc.z += v[j].z;
          acc.w += v[j].w;
        }
      }
    }
    part[grp][it] = acc;
    __syncthreads();
    if (grp == 0 && i < total) {
      float4 t = part[0][it];
#pragma unroll
      for (int g = 1; g < SUM_GROUPS; ++g) {
        t.x += part[g][it].x;
        t.y += part[g][it].y;
        t.z += part[g][it].z;
        t.w += part[g][it].w;
      }
      uint2 o;
      o.x = pack_bf16x2(t.x, t.y);
      o.y = pack_bf16x2(t.z, t.w);
      *reinterpret_cast<uint2*>(out + at) = o;
    }
    __syncthreads();
  }
}

cudaError_t launch_splitk_sum(const float* partial, int S, long long rows, int N, void* out, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  const long long total = rows * (N / 4);
  long long blocks = (total + SUM_ITEMS - 1) / SUM_ITEMS;
  const long long cap = (long long)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  KernelScope ks("lr_reduce", s);
  cudaError_t e = launch_kernel(splitk_sum_kernel, dim3(static_cast<int>(blocks)), dim3(SUM_ITEMS * SUM_GROUPS), 0, s,
                                partial, S, rows, N, static_cast<__nv_bfloat16*>(out));
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Split-K expert outputs (bf16 layers): for every token and 8-column chunk,
// the k slots' fp32 partial sums over the K ranges are added (range order),
// weighted by the slot's gate weight (slot order), plus the shared experts'
// rows; one bf16 rounding at the end.  A decode step has only T * d / 8
// threads, so latency decides: every slot's row position is read first, and
// the S <= COMBINE_MAX_S range loads of a slot are issued together.
constexpr int COMBINE_MAX_S = 8;
constexpr int COMBINE_MAX_K = 8;
__global__ void splitk_combine_kernel(const float* __restrict__ partial, int S, long long part_rows,
                                      const int32_t* __restrict__ offsets, const int32_t* __restrict__ idx,
                                      const int32_t* __restrict__ rel, int rel_mode, const float* __restrict__ w,
                                      const __nv_bfloat16* __restrict__ shared, int n_shared,
                                      __nv_bfloat16* __restrict__ Y, int T, int k, int d) {
  pdl_trigger();
  pdl_wait();
  const int per_row = d / 8;
  const long long total = (long long)T * per_row;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const long long t = i / per_row;
    const int c = static_cast<int>(i % per_row) * 8;
    float acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.0f;
    long long pos[COMBINE_MAX_K];
    float wt[COMBINE_MAX_K];
#pragma unroll
    for (int slot = 0; slot < COMBINE_MAX_K; ++slot) {
      pos[slot] = 0;
      wt[slot] = 0.0f;
      if (slot < k) {
        const long long entry = t * k + slot;
        pos[slot] = rel_mode ? (long long)offsets[idx[entry]] + rel[entry] : (long long)rel[entry];
        wt[slot] = w[entry];
      }
    }
#pragma unroll
    for (int slot = 0; slot < COMBINE_MAX_K; ++slot) {
      if (slot >= k) break;
      float v[COMBINE_MAX_S][8];
#pragma unroll
      for (int s = 0; s < COMBINE_MAX_S; ++s)
        if (s < S) load8(partial + ((long long)s * part_rows + pos[slot]) * d + c, v[s]);
      float sum[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) sum[j] = 0.0f;
#pragma unroll
      for (int s = 0; s < COMBINE_MAX_S; ++s)
        if (s < S) {
#pragma unroll
          for (int j = 0; j < 8; ++j) sum[j] += v[s][j];
        }
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = fmaf(wt[slot], sum[j], acc[j]);
    }
    for (int j = 0; j < n_shared; ++j) {
      float v[8];
      load8(shared + ((long long)j * T + t) * d + c, v);
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] += v[q];
    }
    store8(Y + t * d + c, acc);
  }
}

cudaError_t launch_splitk_combine(const float* partial, int split_k, long long part_rows, const int32_t* offsets,
                                  const int32_t* idx, const int32_t* rel, bool rel_mode, const float* w,
                                  const void* shared, int n_shared, void* Y, int T, int k, int d, cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  if (split_k < 1 || split_k > COMBINE_MAX_S || k < 1 || k > COMBINE_MAX_K) return cudaErrorInvalidValue;
  const long long total = (long long)T * (d / 8);
  long long blocks = (total + 255) / 256;
  const long long cap = (long long)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  KernelScope ks("combine", s);
  cudaError_t e = launch_kernel(splitk_combine_kernel, dim3(static_cast<int>(blocks)), dim3(256), 0, s, partial, split_k,
                                part_rows, offsets, idx, rel, rel_mode ? 1 : 0, w,
                                static_cast<const __nv_bfloat16*>(shared), shared ? n_shared : 0,
                                static_cast<__nv_bfloat16*>(Y), T, k, d);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_combine(const void* slot, const void* shared, int n_shared, void* Y, int T, int k, int d, bool bf16,
                           cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  if (k < 1 || k > CB_MAX_K || n_shared < 0 || n_shared > CB_MAX_SHARED) return cudaErrorInvalidValue;
  const long long total = (long long)T * (d / 8);
  long long blocks = (total + 255) / 256;
  const long long cap = (long long)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  KernelScope ks("combine", s);
  const int ns = shared ? n_shared : 0;
  const int rows = k + ns;
  cudaError_t e;
  if (bf16) {
    const auto* sl = static_cast<const __nv_bfloat16*>(slot);
    const auto* sh = static_cast<const __nv_bfloat16*>(shared);
    auto* y = static_cast<__nv_bfloat16*>(Y);
    const dim3 g(static_cast<int>(blocks));
    if (rows <= 2) e = launch_kernel(combine_kernel<__nv_bfloat16, 2>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else if (rows <= 4) e = launch_kernel(combine_kernel<__nv_bfloat16, 4>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else if (rows <= 8) e = launch_kernel(combine_kernel<__nv_bfloat16, 8>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else e = launch_kernel(combine_kernel<__nv_bfloat16, 12>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
  } else {
    const auto* sl = static_cast<const float*>(slot);
    const auto* sh = static_cast<const float*>(shared);
    auto* y = static_cast<float*>(Y);
    const dim3 g(static_cast<int>(blocks));
    if (rows <= 2) e = launch_kernel(combine_kernel<float, 2>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else if (rows <= 4) e = launch_kernel(combine_kernel<float, 4>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else if (rows <= 8) e = launch_kernel(combine_kernel<float, 8>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
    else e = launch_kernel(combine_kernel<float, 12>, g, dim3(256), 0, s, sl, sh, ns, y, T, k, d);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace ec2moe
