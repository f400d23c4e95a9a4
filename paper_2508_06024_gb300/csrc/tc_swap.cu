// Grouped bf16 GEMM for decode-sized expert groups (at most 16 rows each) on
// the tensor cores with the operands swapped (Eq. 1, each E_i an FFN):
//
//   C_g^T = B_g A_g^T : 128 weight rows of expert g fill the MMA's M side
//                       (TMEM lanes), the group's <= 16 token rows its N side.
//
// With one or two tokens per expert the usual orientation (tokens on M)
// spends a 128-row MMA on one row, and only (experts with rows) x (N tiles)
// CTAs exist, fewer than the SMs.  Swapped, the work is streaming each
// expert's weights once: a unit is (group, 128 weight rows, K range), a
// persistent CTA per SM walks the units of the groups that hold rows, and
// one 18 KB stage carries 16 KB of weights and the group's 2 KB of token
// rows (TMA, 128-byte swizzle), so ten stages keep ~160 KB of weights in
// flight per SM.  SwiGLU tiles stack 64 W1 rows over the same 64 W3 rows, so
// one accumulator holds both halves of 64 output columns; the epilogue pairs
// them through shared memory.  The down projection of a decode step splits
// K (EPI_PARTIAL) so that (experts x d_model / 128 x ranges) units fill the
// SMs; the fixed-order split-K reduce applies the gate weights (Eq. 1).
//
// Roles: warp 0 loads (one thread), warp 1 issues the MMAs (one thread),
// warps 2-5 read the accumulator (TMEM lane quadrant = warp % 4) and store.
// Every wait is bounded; a timeout sets the error word and the CTA drains.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdlib.h>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace ec2moe {

// bit 0: a bounded wait timed out; bit 1: a group range (offsets) or a
// scatter destination (perm) outside the rows of the call was skipped
__device__ unsigned int g_swap_error;

namespace {

using namespace tc;

constexpr int SW_M = 128;    // weight rows per tile: MMA M, TMEM lanes
constexpr int SW_N = 16;     // token rows per group: MMA N, TMEM columns per accumulator
constexpr int SW_BK = 64;    // K per stage: one 128-byte swizzle row of bf16
constexpr int SW_UK = 16;    // K of one tcgen05.mma kind::f16
constexpr int SW_STAGES = 10;
constexpr int SW_ACC = 4;            // accumulators in TMEM
constexpr int SW_TMEM_COLS = 64;     // SW_ACC * SW_N, a power of two >= 32
constexpr int SW_EPI_WARPS = 4;
constexpr int SW_THREADS = 64 + 32 * SW_EPI_WARPS;
constexpr int SW_MAX_GROUPS = 136;
constexpr int SW_XCH_PITCH = SW_N + 1;  // floats per row of the SwiGLU exchange (no bank conflicts)

constexpr int SW_W_BYTES = SW_M * SW_BK * 2;  // 16 KB
constexpr int SW_X_BYTES = SW_N * SW_BK * 2;  // 2 KB
constexpr int SW_STAGE_BYTES = SW_W_BYTES + SW_X_BYTES;
constexpr int SW_OFF_X = SW_STAGES * SW_W_BYTES;
constexpr int SW_OFF_BARS = SW_OFF_X + SW_STAGES * SW_X_BYTES;
constexpr int SW_N_BARS = 2 * SW_STAGES + 2 * SW_ACC + 1;
constexpr int SW_OFF_SLOT = SW_OFF_BARS + SW_N_BARS * 8;  // TMEM address, abort flag, active-group count
constexpr int SW_OFF_LIST = SW_OFF_SLOT + 16;             // per active group: id, first row, rows
constexpr int SW_OFF_XCH = (SW_OFF_LIST + 3 * SW_MAX_GROUPS * 4 + 15) & ~15;
constexpr int SW_SMEM = SW_OFF_XCH + 64 * SW_XCH_PITCH * 4 + 1024;  // + alignment slack
static_assert(SW_OFF_X % 1024 == 0 && SW_OFF_BARS % 8 == 0 && SW_OFF_XCH % 16 == 0, "shared layout alignment");
static_assert(SW_SMEM <= 232448, "shared memory per CTA");
static_assert(SW_ACC * SW_N <= SW_TMEM_COLS, "TMEM columns");

struct SwParams {
  const int32_t* offsets;
  int G, M, a_shared;
  long long a_row_base, out_row_base;
  int N, K, b_group_rows;
  void* out;
  long long ldo;
  const int32_t* perm;
  const float* scale;
  float* partial;
  long long part_rows;
  int split_k, kb_per_split;
  int n_blk;  // weight tiles per group along N
  long long timeout;
  long long row_limit;  // rows of the call: group ranges and scatter destinations lie in [0, row_limit)
};

struct SwUnit {
  int a, nb, ks;  // active-group index, weight tile, K range
};
__device__ __forceinline__ SwUnit decode_unit(int u, const SwParams& p) {
  const int per = p.n_blk * p.split_k;
  const int rem = u % per;
  return SwUnit{u / per, rem / p.split_k, rem % p.split_k};
}

template <int EPI>
__global__ void __launch_bounds__(SW_THREADS, 1)
    swap_gemm_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                     const __grid_constant__ CUtensorMap tmW2, const SwParams p) {
  constexpr bool GLU = EPI == EPI_SWIGLU;
  constexpr int TN = GLU ? SW_M / 2 : SW_M;  // output columns per weight tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sW = smem;
  uint8_t* sX = smem + SW_OFF_X;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + SW_OFF_BARS);
  uint64_t* empty = full + SW_STAGES;
  uint64_t* tfull = empty + SW_STAGES;
  uint64_t* tempty = tfull + SW_ACC;
  uint64_t* drain = tempty + SW_ACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + SW_OFF_SLOT);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* n_active = reinterpret_cast<int*>(tmem_slot + 2);
  int* g_id = reinterpret_cast<int*>(smem + SW_OFF_LIST);
  int* g_r0 = g_id + SW_MAX_GROUPS;
  int* g_rows = g_r0 + SW_MAX_GROUPS;
  float* xch = reinterpret_cast<float*>(smem + SW_OFF_XCH);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // Barrier set-up, TMEM allocation and descriptor prefetch overlap the
  // previous kernel; everything that reads its results comes after pdl_wait.
  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < SW_STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < SW_ACC; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), SW_EPI_WARPS);
    }
    mbar_init(smem_u32(drain), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {
    pdl_wait();
    // The groups that hold rows, in ascending order; all row counts are
    // fetched before the ballots, so this costs about one memory latency.
    constexpr int CH = (SW_MAX_GROUPS + 31) / 32;
    int r0v[CH], mgv[CH];
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const int g = c * 32 + lane;
      r0v[c] = 0;
      mgv[c] = 0;
      if (g < p.G) {
        if (p.offsets) {
          r0v[c] = p.offsets[g];
          mgv[c] = p.offsets[g + 1] - r0v[c];
          if (r0v[c] < 0 || mgv[c] < 0 || static_cast<long long>(r0v[c]) + mgv[c] > p.row_limit) {
            // not a range of this call's rows: the group is skipped
            atomicOr(&g_swap_error, 2u);
            r0v[c] = 0;
            mgv[c] = 0;
          }
        } else {
          r0v[c] = g * p.M;
          mgv[c] = p.M;
        }
      }
    }
    int base = 0;
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const bool act = mgv[c] > 0;
      const unsigned bal = __ballot_sync(0xffffffffu, act);
      if (act) {
        const int i = base + __popc(bal & ((1u << lane) - 1u));
        g_id[i] = c * 32 + lane;
        g_r0[i] = r0v[c];
        g_rows[i] = mgv[c] < SW_N ? mgv[c] : SW_N;  // the host guarantees at most SW_N rows
      }
      base += __popc(bal);
    }
    if (lane == 0) *n_active = base;
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
    if (GLU) tma_prefetch_desc(&tmW2);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(SW_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  const uint32_t tmem_base = *tmem_slot;
  const int units = *n_active * p.n_blk * p.split_k;
  const int num_kb = (p.K + SW_BK - 1) / SW_BK;
  const long long budget = p.timeout;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0;  // bit s: stage s holds a copy the consumer has not released
      uint32_t issued_phase = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const SwUnit un = decode_unit(u, p);
        const int r0 = g_r0[un.a];
        const int x_row = static_cast<int>(p.a_row_base) + (p.offsets ? r0 : (p.a_shared ? 0 : r0));
        const int w_row = g_id[un.a] * p.b_group_rows + un.nb * TN;
        const int kb0 = un.ks * p.kb_per_split;
        const int kb1 = kb0 + p.kb_per_split < num_kb ? kb0 + p.kb_per_split : num_kb;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, budget, abort_flag, &g_swap_error)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          mbar_expect_tx(fb, SW_STAGE_BYTES);
          const uint32_t dw = smem_u32(sW + stage * SW_W_BYTES);
          if (GLU) {
            // rows 0-63 of the tile: W1, rows 64-127: W3, same output columns
            tma_load_2d(dw, &tmW, kb * SW_BK, w_row, fb);
            tma_load_2d(dw + SW_W_BYTES / 2, &tmW2, kb * SW_BK, w_row, fb);
          } else {
            tma_load_2d(dw, &tmW, kb * SW_BK, w_row, fb);
          }
          tma_load_2d(smem_u32(sX + stage * SW_X_BYTES), &tmX, kb * SW_BK, x_row, fb);
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == SW_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok || *abort_flag) {
        // Let every copy this CTA started land before shared memory is released.
        for (int s = 0; s < SW_STAGES; ++s)
          if (issued & (1u << s)) mbar_drain(smem_u32(&full[s]), (issued_phase >> s) & 1u, DRAIN_CYCLES);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      constexpr uint32_t IDESC = idesc_bf16(SW_M, SW_N);
      const uint64_t dw0 = sdesc_sw128(smem_u32(sW));
      const uint64_t dx0 = sdesc_sw128(smem_u32(sX));
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true, any = false;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++it) {
        const SwUnit un = decode_unit(u, p);
        const int kb0 = un.ks * p.kb_per_split;
        const int kb1 = kb0 + p.kb_per_split < num_kb ? kb0 + p.kb_per_split : num_kb;
        const int acc = it % SW_ACC;
        const uint32_t acc_phase = static_cast<uint32_t>(it / SW_ACC) & 1u;
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1u, budget, abort_flag, &g_swap_error)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * SW_N);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, budget, abort_flag, &g_swap_error)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // stage-0 descriptors plus the stage offset; each K = 16 step adds
          // 32 bytes (2 in the address field, which cannot carry: shared
          // addresses are below 256 KB)
          const uint64_t da = dw0 + static_cast<uint64_t>(stage) * (SW_W_BYTES >> 4);
          const uint64_t db = dx0 + static_cast<uint64_t>(stage) * (SW_X_BYTES >> 4);
          umma_bf16(d_tmem, da, db, IDESC, kb != kb0 ? 1u : 0u);
#pragma unroll
          for (int kk = 1; kk < SW_BK / SW_UK; ++kk) umma_bf16(d_tmem, da + 2 * kk, db + 2 * kk, IDESC, 1u);
          any = true;
          umma_commit(smem_u32(&empty[stage]));
          if (++stage == SW_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(smem_u32(&tfull[acc]));
      }
      if ((!ok || *abort_flag) && any) {
        // All MMAs issued so far must finish before TMEM is freed.
        umma_commit(smem_u32(drain));
        mbar_drain(smem_u32(drain), 0, DRAIN_CYCLES);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    int it = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
      const SwUnit un = decode_unit(u, p);
      const int acc = it % SW_ACC;
      const uint32_t acc_phase = static_cast<uint32_t>(it / SW_ACC) & 1u;
      const int r0 = g_r0[un.a];
      const int mg = g_rows[un.a];
      // output column of this thread's TMEM lane (SwiGLU: lanes 64-127 hold
      // the W3 half of lanes 0-63's columns)
      const int col = un.nb * TN + (GLU ? (q & 1) * 32 : q * 32) + lane;
      bool ok = mbar_wait(smem_u32(&tfull[acc]), acc_phase, budget, abort_flag, &g_swap_error);
      if (GLU) {
        // the four warps meet at named barriers below: agree on the outcome
        uint32_t all_ok;
        asm volatile(
            "{\n .reg .pred p, r;\n setp.ne.u32 p, %1, 0;\n"
            " bar.red.and.pred r, 1, 128, p;\n selp.u32 %0, 1, 0, r;\n}"
            : "=r"(all_ok)
            : "r"(ok ? 1u : 0u)
            : "memory");
        ok = all_ok != 0;
      }
      if (!ok) break;
      tc_fence_after();
      float v[SW_N];
      tmem_ld16(tmem_base + static_cast<uint32_t>(acc * SW_N) + (static_cast<uint32_t>(q * 32) << 16), v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
      const long long row_base = p.out_row_base + r0;
      if (GLU) {
        // W3 lanes hand their values to the W1 lanes of the same columns.
        // The barrier at the top of the next unit orders the next writes
        // after these reads.
        float* xr = xch + ((q & 1) * 32 + lane) * SW_XCH_PITCH;
        if (q >= 2) {
#pragma unroll
          for (int j = 0; j < SW_N; ++j) xr[j] = v[j];
        }
        asm volatile("bar.sync 2, 128;" ::: "memory");
        if (q < 2 && col < p.N) {
          __nv_bfloat16* o = static_cast<__nv_bfloat16*>(p.out);
#pragma unroll
          for (int j = 0; j < SW_N; ++j)
            if (j < mg) o[(row_base + j) * p.ldo + col] = __float2bfloat16_rn(silu_bf16out(v[j]) * xr[j]);
        }
      } else if (col < p.N) {
        if (EPI == EPI_PARTIAL) {
          float* dst = p.partial + (static_cast<long long>(un.ks) * p.part_rows + row_base) * p.N + col;
#pragma unroll
          for (int j = 0; j < SW_N; ++j)
            if (j < mg) dst[static_cast<long long>(j) * p.N] = v[j];
        } else {
          __nv_bfloat16* o = static_cast<__nv_bfloat16*>(p.out);
#pragma unroll
          for (int j = 0; j < SW_N; ++j) {
            if (j >= mg) break;
            const long long out_row = row_base + j;
            float y = v[j];
            long long dest = out_row;
            if (EPI == EPI_GELU) y = gelu_bf16out(y);
            if (EPI == EPI_SCATTER) {
              dest = p.perm ? p.perm[out_row] : out_row;
              if (dest < 0 || dest >= p.row_limit) {
                atomicOr(&g_swap_error, 2u);
                continue;
              }
              if (p.scale) y *= p.scale[dest];
            }
            o[dest * p.ldo + col] = __float2bfloat16_rn(y);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(SW_TMEM_COLS)
                 : "memory");
  }
}

bool swap_env_enabled() {
  static const bool on = [] {
    const char* e = getenv("EC2MOE_GEMM_SWAP");
    return !(e && e[0] == '0');
  }();
  return on;
}

template <int EPI>
cudaError_t launch_epi(const CUtensorMap& mX, const CUtensorMap& mW, const CUtensorMap& mW2, const SwParams& p,
                       int grid, cudaStream_t s) {
  const void* kfn = reinterpret_cast<const void*>(swap_gemm_kernel<EPI>);
  cudaError_t e = ensure_smem_attr(kfn, SW_SMEM);
  if (e != cudaSuccess) return e;
  return launch_kernel(swap_gemm_kernel<EPI>, dim3(grid), dim3(SW_THREADS), (size_t)SW_SMEM, s, mX, mW, mW2, p);
}

}  // namespace

bool swap_gemm_enabled() { return swap_env_enabled(); }

int swap_split_factor(long long tiles, int K, int max_split) {
  const int num_kb = (K + SW_BK - 1) / SW_BK;
  const long long sms = sm_count();
  int best = 1;
  double best_eff = -1.0;
  for (int sp = 1; sp <= max_split && sp <= num_kb; ++sp) {
    const int per = (num_kb + sp - 1) / sp;
    if ((num_kb + per - 1) / per != sp) continue;  // an empty K range: not this split
    const long long units = tiles * sp;
    const long long waves = (units + sms - 1) / sms;
    const double eff = (double)units / (double)(waves * sms) - 0.002 * sp;  // fewer ranges on ties
    if (eff > best_eff) {
      best_eff = eff;
      best = sp;
    }
  }
  return best;
}

long long swap_tiles_per_group(int N, int epi) {
  const int tn = epi == EPI_SWIGLU ? SW_M / 2 : SW_M;
  return (N + tn - 1) / tn;
}

bool gemm_swap_supported(const GemmArgs& a, int epi) {
  if (!swap_env_enabled()) return false;
  if (epi != EPI_STORE && epi != EPI_GELU && epi != EPI_SWIGLU && epi != EPI_SCATTER && epi != EPI_PARTIAL)
    return false;
  if (a.group_rows_bound < 1 || a.group_rows_bound > SWAP_MAX_ROWS) return false;
  if (a.G < 1 || a.G > SW_MAX_GROUPS || a.N < 1 || a.K < 1 || a.K % 8 != 0) return false;
  if (epi == EPI_PARTIAL && (!a.partial || a.split_k < 1)) return false;
  if (reinterpret_cast<uintptr_t>(a.A) % 16 != 0 || reinterpret_cast<uintptr_t>(a.B) % 16 != 0) return false;
  if (epi == EPI_SWIGLU && reinterpret_cast<uintptr_t>(a.B2) % 16 != 0) return false;
  return true;
}

cudaError_t launch_gemm_swap(const GemmArgs& a, int epi, cudaStream_t s) {
  if (!gemm_swap_supported(a, epi)) return cudaErrorInvalidValue;
  const int tn = epi == EPI_SWIGLU ? SW_M / 2 : SW_M;
  CUtensorMap mX, mW, mW2;
  if (!make_tensor_map_bf16(&mX, a.A, a.a_rows, a.K, SW_N)) return cudaErrorInvalidValue;
  if (!make_tensor_map_bf16(&mW, a.B, a.b_rows, a.K, tn)) return cudaErrorInvalidValue;
  if (epi == EPI_SWIGLU) {
    if (!make_tensor_map_bf16(&mW2, a.B2, a.b_rows, a.K, tn)) return cudaErrorInvalidValue;
  } else {
    mW2 = mW;
  }
  SwParams p;
  p.offsets = a.offsets;
  p.G = a.G;
  p.M = a.M;
  p.a_shared = a.a_shared;
  p.a_row_base = a.a_row_base;
  p.out_row_base = a.out_row_base;
  p.N = a.N;
  p.K = a.K;
  p.b_group_rows = a.b_group_rows;
  p.out = a.out;
  p.ldo = a.ldo;
  p.perm = a.perm;
  p.scale = a.scale;
  p.partial = a.partial;
  p.part_rows = a.part_rows;
  p.timeout = a.timeout_cycles;
  p.row_limit = a.max_rows > 0 ? a.max_rows : (1LL << 62);
  p.n_blk = static_cast<int>((a.N + tn - 1) / tn);
  p.split_k = epi == EPI_PARTIAL ? a.split_k : 1;
  const int num_kb = (a.K + SW_BK - 1) / SW_BK;
  p.kb_per_split = (num_kb + p.split_k - 1) / p.split_k;
  // the reduce reads split_k ranges: every one must be written
  if ((num_kb + p.kb_per_split - 1) / p.kb_per_split != p.split_k) return cudaErrorInvalidValue;
  // grid: one CTA per SM at most, no more than the units expected (groups
  // with rows <= min(G, rows, the caller's estimate))
  long long groups = a.G;
  if (a.max_rows > 0 && a.max_rows < groups) groups = a.max_rows;
  if (a.g_active > 0 && a.g_active < groups) groups = a.g_active;
  const long long units = groups * p.n_blk * p.split_k;
  const long long sms = sm_count();
  const int grid = static_cast<int>(units < 1 ? 1 : (units < sms ? units : sms));
  KernelScope ks(a.name ? a.name : "gemm_swap", s);
  cudaError_t e;
  switch (epi) {
    case EPI_GELU: e = launch_epi<EPI_GELU>(mX, mW, mW2, p, grid, s); break;
    case EPI_SWIGLU: e = launch_epi<EPI_SWIGLU>(mX, mW, mW2, p, grid, s); break;
    case EPI_SCATTER: e = launch_epi<EPI_SCATTER>(mX, mW, mW2, p, grid, s); break;
    case EPI_PARTIAL: e = launch_epi<EPI_PARTIAL>(mX, mW, mW2, p, grid, s); break;
    default: e = launch_epi<EPI_STORE>(mX, mW, mW2, p, grid, s); break;
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t read_swap_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_swap_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_swap_error, &zero, sizeof(unsigned int));
}

}  // namespace ec2moe
