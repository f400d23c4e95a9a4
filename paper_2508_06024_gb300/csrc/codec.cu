// Fused low-rank codec of the layer path on the sm_103a tensor cores: the
// end-cloud encoder Z = U^T X V and decoder X_hat = U_hat Z V_hat^T with the
// token-side projections U = U_hat = I, as two chained tcgen05 GEMMs in one
// kernel.  Each CTA owns one 128-row tile of tokens and one BN-column chunk of
// d_model:
//   1. Z_tile = X_tile V_enc^T (N = r) into TMEM (TMA-fed, 128-byte swizzle);
//   2. the epilogue warps round Z to bf16 (the transmitted tensor), write it
//      to global (chunk 0's CTA) and into shared memory in the swizzled
//      K-major layout the second MMA reads as its A operand;
//   3. X_hat chunk = Z_tile V_dec[chunk]^T (N = BN) into TMEM;
//   4. the X_hat chunk is rounded to bf16 into a row-major tile in the
//      (then idle) pipeline buffers, and each epilogue warp copies whole row
//      segments (BN * 2 contiguous bytes) to the row's (token, slot)
//      positions in expert order (offsets[e] + the row's position relative
//      to its expert, from the routing the gate kernel filled) and to the
//      tail rows the shared experts read.
// Z is recomputed by the d / BN CTAs of a token tile (cheap at r <= 256);
// nothing but the routing metadata depends on the previous kernel, so under
// programmatic dependent launch both GEMMs run before griddepcontrol.wait.
//
// Warps: 0 TMA producer, 1 TMEM allocator + MMA issuer, 2..17 epilogue (warp
// w reads TMEM lanes 32*(w%4) .. +31).  Every mbarrier wait is bounded; on
// a timeout the device error word is set, in-flight copies and MMAs are
// drained (bounded) and the kernel returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace ec2moe {

__device__ unsigned int g_codec_error;  // bit 0: a bounded wait timed out

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int UK = 16;
constexpr int EPI_WARPS = 16;
constexpr int NUM_THREADS = 64 + 32 * EPI_WARPS;
constexpr int X_ACC_COL = 256;  // TMEM column of the X_hat accumulator (Z uses [0, r))

struct CParams {
  int T, d, k, E;
  __nv_bfloat16* Z;
  __nv_bfloat16* out;
  long long ldo;
  const int32_t* rel;
  const int32_t* counts;
  const int32_t* topk_idx;
  int32_t* perm_out;
  int32_t* offsets_out;
  long long self_row_base;
  long long timeout;
  int n_chunks;
};

template <int BN, int R>
struct CCfg {
  static constexpr int A_BYTES = BM * BK * 2;                 // X box
  static constexpr int B_ROWS = R > BN ? R : BN;
  static constexpr int B_BYTES = B_ROWS * BK * 2;              // V_enc box (R rows) or V_dec box (BN rows)
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int Z_BYTES = BM * R * 2;                   // R / 64 swizzle atoms of 16 KB
  static constexpr int PARTS_X = 4;
  static constexpr int PART_X = BN / PARTS_X;                  // X_hat columns per epilogue warp
  static constexpr int PART_Z = R / 4;                         // Z columns per epilogue warp
  static constexpr int CW = 16;
  static constexpr int TILE_PITCH = BN * 2 + 16;               // bf16 X_hat tile row (padded against bank conflicts)
  static constexpr int DST_BYTES = BM * 8 * 4;                 // destination rows of each tile row (k <= 8)
  static constexpr int MISC = 1024;                            // barriers, TMEM slot, flags, offsets
  static constexpr int FIXED = 1024 + Z_BYTES + DST_BYTES + MISC;
  static constexpr int STAGES_FIT = (220 * 1024 - FIXED) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 4 ? 4 : STAGES_FIT;
  static constexpr int SMEM = FIXED + STAGES * STAGE_BYTES;
  static_assert(STAGES >= 2, "codec pipeline needs two stages");
  static_assert(SMEM <= 232448, "shared memory per CTA");
  static_assert(PART_X % CW == 0 && PART_Z % CW == 0 && R % 64 == 0, "column split");
  static_assert(STAGES * STAGE_BYTES >= BM * TILE_PITCH, "X_hat tile fits in the pipeline buffers");
  static_assert(BN <= 256, "one 16-byte piece per lane covers a row segment");
};

template <int BN, int R>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    codec_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmVe,
                 const __grid_constant__ CUtensorMap tmVd, const CParams p) {
  using C = CCfg<BN, R>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stages = smem;
  uint8_t* zs = smem + C::STAGES * C::STAGE_BYTES;
  int* s_dst = reinterpret_cast<int*>(zs + C::Z_BYTES);  // [BM][8]
  uint64_t* bars = reinterpret_cast<uint64_t*>(zs + C::Z_BYTES + C::DST_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::STAGES;
  uint64_t* zfull = bars + 2 * C::STAGES;
  uint64_t* zready = zfull + 1;
  uint64_t* xfull = zfull + 2;
  uint64_t* drain = zfull + 3;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(zfull + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* s_off = reinterpret_cast<int*>(tmem_slot + 4);  // [E + 1]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  pdl_trigger();
  const int m_tile = blockIdx.x / p.n_chunks;
  const int n_chunk = blockIdx.x % p.n_chunks;
  const int m0 = m_tile * BM;
  const int n0 = n_chunk * BN;
  const int K1 = (p.d + BK - 1) / BK;
  constexpr int K2 = R / BK;
  const long long budget = p.timeout;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    mbar_init(smem_u32(zfull), 1);
    mbar_init(smem_u32(zready), EPI_WARPS);
    mbar_init(smem_u32(xfull), 1);
    mbar_init(smem_u32(drain), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmVe);
    tma_prefetch_desc(&tmVd);
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
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;
      bool ok = true;
      const int n_loads = K1 + K2;
      for (int i = 0; i < n_loads && ok; ++i) {
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, budget, abort_flag, &g_codec_error)) {
          ok = false;
          break;
        }
        const uint32_t fb = smem_u32(&full[stage]);
        uint8_t* st = stages + stage * C::STAGE_BYTES;
        if (i < K1) {
          mbar_expect_tx(fb, C::A_BYTES + R * BK * 2);
          tma_load_2d(smem_u32(st), &tmX, i * BK, m0, fb);
          tma_load_2d(smem_u32(st + C::A_BYTES), &tmVe, i * BK, 0, fb);
        } else {
          mbar_expect_tx(fb, BN * BK * 2);
          tma_load_2d(smem_u32(st + C::A_BYTES), &tmVd, (i - K1) * BK, n0, fb);
        }
        issued |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok || *abort_flag) {
        for (int s = 0; s < C::STAGES; ++s)
          if (issued & (1u << s)) mbar_drain(smem_u32(&full[s]), (issued_phase >> s) & 1u, DRAIN_CYCLES);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC_Z = idesc_bf16(BM, R);
      constexpr uint32_t IDESC_X = idesc_bf16(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, any = false;
      // Z = X V_enc^T
      for (int kb = 0; kb < K1 && ok; ++kb) {
        if (!mbar_wait(smem_u32(&full[stage]), phase, budget, abort_flag, &g_codec_error)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* st = stages + stage * C::STAGE_BYTES;
        const uint64_t da = sdesc_sw128(smem_u32(st));
        const uint64_t db = sdesc_sw128(smem_u32(st + C::A_BYTES));
#pragma unroll
        for (int kk = 0; kk < BK / UK; ++kk)
          umma_bf16(tmem_base, da + 2 * kk, db + 2 * kk, IDESC_Z, (kb | kk) != 0 ? 1u : 0u);
        any = true;
        umma_commit(smem_u32(&empty[stage]));
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (ok) {
        umma_commit(smem_u32(zfull));
        // X_hat = Z V_dec^T once the epilogue has put Z (bf16) in shared memory
        ok = mbar_wait(smem_u32(zready), 0, budget, abort_flag, &g_codec_error);
        tc_fence_after();
      }
      for (int kb = 0; kb < K2 && ok; ++kb) {
        if (!mbar_wait(smem_u32(&full[stage]), phase, budget, abort_flag, &g_codec_error)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* st = stages + stage * C::STAGE_BYTES;
        const uint64_t da = sdesc_sw128(smem_u32(zs + kb * (BM * 128)));
        const uint64_t db = sdesc_sw128(smem_u32(st + C::A_BYTES));
#pragma unroll
        for (int kk = 0; kk < BK / UK; ++kk)
          umma_bf16(tmem_base + X_ACC_COL, da + 2 * kk, db + 2 * kk, IDESC_X, (kb | kk) != 0 ? 1u : 0u);
        umma_commit(smem_u32(&empty[stage]));
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (ok) umma_commit(smem_u32(xfull));
      if ((!ok || *abort_flag) && any) {
        umma_commit(smem_u32(drain));
        mbar_drain(smem_u32(drain), 0, DRAIN_CYCLES);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const int part = (warp - 2) >> 2;
    const int row = q * 32 + lane;
    const long long grow = m0 + row;
    const bool valid = grow < p.T;
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    bool ok = mbar_wait(smem_u32(zfull), 0, budget, abort_flag, &g_codec_error);
    if (ok) {
      tc_fence_after();
      // Z columns [part * PART_Z, +PART_Z) of this row: bf16 into the swizzled
      // A-operand layout (atom c / 64, 16-byte chunk ((c % 64) / 8) ^ (row % 8))
      // and, from chunk 0's CTA, to global.
#pragma unroll 1
      for (int cz = 0; cz < C::PART_Z; cz += C::CW) {
        const int c = part * C::PART_Z + cz;
        uint32_t r[C::CW];
        tmem_ld16_nw(t_row + c, r);
        tmem_wait();
        U4 q0{pack_bf16x2(__uint_as_float(r[0]), __uint_as_float(r[1])),
              pack_bf16x2(__uint_as_float(r[2]), __uint_as_float(r[3])),
              pack_bf16x2(__uint_as_float(r[4]), __uint_as_float(r[5])),
              pack_bf16x2(__uint_as_float(r[6]), __uint_as_float(r[7]))};
        U4 q1{pack_bf16x2(__uint_as_float(r[8]), __uint_as_float(r[9])),
              pack_bf16x2(__uint_as_float(r[10]), __uint_as_float(r[11])),
              pack_bf16x2(__uint_as_float(r[12]), __uint_as_float(r[13])),
              pack_bf16x2(__uint_as_float(r[14]), __uint_as_float(r[15]))};
        uint8_t* atom = zs + (c / 64) * (BM * 128) + row * 128;
        const int ch = (c % 64) / 8;
        *reinterpret_cast<U4*>(atom + (((ch + 0) ^ (row & 7)) * 16)) = q0;
        *reinterpret_cast<U4*>(atom + (((ch + 1) ^ (row & 7)) * 16)) = q1;
        if (n_chunk == 0 && valid) {
          U4* zg = reinterpret_cast<U4*>(p.Z + grow * R + c);
          zg[0] = q0;
          zg[1] = q1;
        }
      }
      // make the generic-proxy stores visible to the tensor core's reads
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(zready));
    }
    // Routing metadata comes from the gate kernel: wait for it here only.
    pdl_wait();
    if (warp == 2)
      warp_exclusive_scan<5>(p.E, lane, [&](int e) { return p.counts[e]; }, s_off,
                             blockIdx.x == 0 ? p.offsets_out : nullptr);
    asm volatile("bar.sync 1, %0;" ::"r"(EPI_WARPS * 32) : "memory");
    // Destination rows of this tile row (one thread per row writes them).
    if (part == 0) {
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        if (valid && r < p.k) {
          const long long entry = grow * p.k + r;
          const int dst = s_off[p.topk_idx[entry]] + p.rel[entry];
          if (n_chunk == 0) p.perm_out[dst] = static_cast<int32_t>(entry);
          s_dst[row * 8 + r] = dst;
        }
      }
    }
    if (ok) ok = mbar_wait(smem_u32(xfull), 0, budget, abort_flag, &g_codec_error);
    if (ok) {
      // Every MMA has completed, so the pipeline buffers are free: round this
      // warp's 32 rows x PART_X columns into the row-major bf16 tile.
      tc_fence_after();
      constexpr int NCH = C::PART_X / C::CW;
      uint8_t* trow = stages + row * C::TILE_PITCH + part * C::PART_X * 2;
      uint32_t rv[2][C::CW];
#pragma unroll 1
      for (int cp = 0; cp < NCH; cp += 2) {
        tmem_ld16_nw(t_row + X_ACC_COL + part * C::PART_X + cp * C::CW, rv[0]);
        if (cp + 1 < NCH) tmem_ld16_nw(t_row + X_ACC_COL + part * C::PART_X + (cp + 1) * C::CW, rv[1]);
        tmem_wait();
#pragma unroll
        for (int slot = 0; slot < 2; ++slot) {
          if (cp + slot >= NCH) break;
          const uint32_t* rr = rv[slot];
#pragma unroll
          for (int j = 0; j < C::CW / 8; ++j) {
            U4 q4{pack_bf16x2(__uint_as_float(rr[8 * j + 0]), __uint_as_float(rr[8 * j + 1])),
                  pack_bf16x2(__uint_as_float(rr[8 * j + 2]), __uint_as_float(rr[8 * j + 3])),
                  pack_bf16x2(__uint_as_float(rr[8 * j + 4]), __uint_as_float(rr[8 * j + 5])),
                  pack_bf16x2(__uint_as_float(rr[8 * j + 6]), __uint_as_float(rr[8 * j + 7]))};
            *reinterpret_cast<U4*>(trow + ((cp + slot) * C::CW + 8 * j) * 2) = q4;
          }
        }
      }
      tc_fence_before();
    }
    // The tile is complete unless a wait of some warp timed out, which set
    // the abort flag before this barrier.
    asm volatile("bar.sync 1, %0;" ::"r"(EPI_WARPS * 32) : "memory");
    if (ok && !*abort_flag) {
      // Row segments: warp w copies rows w, w + 16, ...; lane l carries
      // columns n0 + 8l .. +7 (16 bytes), so a row segment is one coalesced
      // store per destination.
      const int ew = warp - 2;
      const int col = n0 + 8 * lane;
      const bool lane_on = 8 * lane < BN && col < p.d;
#pragma unroll 1
      for (int tr = ew; tr < BM; tr += EPI_WARPS) {
        const long long g = m0 + tr;
        if (g >= p.T) break;  // uniform; later rows are further out
        if (lane_on) {
          const U4 q4 = *reinterpret_cast<const U4*>(stages + tr * C::TILE_PITCH + 16 * lane);
          for (int r = 0; r < p.k; ++r)
            *reinterpret_cast<U4*>(p.out + (long long)s_dst[tr * 8 + r] * p.ldo + col) = q4;
          if (p.self_row_base >= 0) *reinterpret_cast<U4*>(p.out + (p.self_row_base + g) * p.ldo + col) = q4;
        }
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

template <int BN, int R>
cudaError_t launch_bn_r(const CodecArgs& a, cudaStream_t s) {
  using C = CCfg<BN, R>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(codec_kernel<BN, R>), C::SMEM);
  if (e != cudaSuccess) return e;
  CUtensorMap mX, mVe, mVd;
  if (!make_tensor_map_bf16(&mX, a.X, a.T, a.d, BM)) return cudaErrorInvalidValue;
  if (!make_tensor_map_bf16(&mVe, a.V_enc, R, a.d, R)) return cudaErrorInvalidValue;
  if (!make_tensor_map_bf16(&mVd, a.V_dec, a.d, R, BN)) return cudaErrorInvalidValue;
  CParams p;
  p.T = a.T;
  p.d = a.d;
  p.k = a.k;
  p.E = a.E;
  p.Z = static_cast<__nv_bfloat16*>(a.Z);
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ldo = a.d;
  p.rel = a.rel;
  p.counts = a.counts;
  p.topk_idx = a.topk_idx;
  p.perm_out = a.perm_out;
  p.offsets_out = a.offsets_out;
  p.self_row_base = a.self_row_base;
  p.timeout = a.timeout_cycles;
  p.n_chunks = (a.d + BN - 1) / BN;
  const int m_tiles = (a.T + BM - 1) / BM;
  KernelScope ks("lr_codec", s);
  return launch_kernel(codec_kernel<BN, R>, dim3(m_tiles * p.n_chunks), dim3(NUM_THREADS), (size_t)C::SMEM, s, mX, mVe,
                       mVd, p);
}

template <int R>
cudaError_t launch_r(const CodecArgs& a, cudaStream_t s) {
  // d-chunk width: the widest whose CTA count fills the most of the GPU in one
  // wave.  The kernel runs under programmatic dependent launch next to the
  // gate kernel, whose CTAs hold `busy_sms` SMs until it ends; a grid that
  // fits in the other SMs runs both GEMMs while the gate runs, while CTAs
  // beyond them would start only after it, on the critical path.
  const int m_tiles = (a.T + BM - 1) / BM;
  const int sms = sm_count();
  const int free_sms = sms - (a.busy_sms > 0 && a.busy_sms < sms ? a.busy_sms : 0);
  const int cands[3] = {256, 192, 128};
  int best = 256;
  double best_eff = -1.0;
  for (int pass = 0; pass < 2 && best_eff < 0.0; ++pass) {
    for (int bn : cands) {
      const long long ctas = (long long)m_tiles * ((a.d + bn - 1) / bn);
      if (pass == 0 && ctas > free_sms) continue;  // first choice: fits beside the gate
      const long long waves = (ctas + sms - 1) / sms;
      const double eff = (double)ctas / (double)(waves * sms) * (bn == 256 ? 1.0 : (bn == 192 ? 0.98 : 0.95));
      if (eff > best_eff + 1e-9) {
        best_eff = eff;
        best = bn;
      }
    }
  }
  switch (best) {
    case 256: return launch_bn_r<256, R>(a, s);
    case 192: return launch_bn_r<192, R>(a, s);
    default: return launch_bn_r<128, R>(a, s);
  }
}

}  // namespace

// Every CTA of a token tile recomputes Z (reading the tile's X rows and all of
// V_enc), so the fused kernel pays off only while a tile has few d-chunks: up
// to d = 1024 (four chunks of 256).  Wider layers run the two GEMMs apart.
bool codec_fused_supported(int d, int r) { return (r == 128 || r == 256) && d % 64 == 0 && d >= 128 && d <= 1024; }

cudaError_t launch_codec_fused(const CodecArgs& a, cudaStream_t s) {
  if (!codec_fused_supported(a.d, a.r) || a.k < 1 || a.k > 8 || a.E > 128) return cudaErrorInvalidValue;
  if (a.T <= 0) return cudaSuccess;
  return a.r == 128 ? launch_r<128>(a, s) : launch_r<256>(a, s);
}

cudaError_t read_codec_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_codec_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_codec_error, &zero, sizeof(unsigned int));
}

}  // namespace ec2moe
