// Grouped bf16 GEMM on the sm_103a tensor cores: tcgen05.mma with the fp32
// accumulator in tensor memory (TMEM), operands staged by TMA into 128-byte
// swizzled shared memory, and a persistent warp-specialised CTA per SM.
//
// Used for the expert FFN projections (Eq. 1 experts, steps 4-5) and the
// low-rank codec projections (Z = X V_enc^T, X_hat = Z V_dec^T).  Every group g
// computes  C_g = A_g B_g^T  with A_g [M_g, K] (rows of A) and B_g [N, K]
// (rows of a weight matrix stored [out, in]), and the epilogue applies the
// step-specific op (plain store, GELU, SwiGLU, or gate-scale + scatter to the
// token's slot for the combine of Eq. 1).
//
// CTA layout (576 threads):
//   warp 0      TMA producer (one elected lane)
//   warp 1      TMEM allocator + MMA issuer (one elected lane)
//   warps 2..17 epilogue: TMEM -> registers -> shared staging -> global.
//               Warp w may only read TMEM lanes 32*(w%4) .. +31 (rows of the
//               128-row tile); the four warps of a lane quadrant split the
//               tile's columns and, for contiguous or per-row destinations,
//               stage 64-column slabs together (named barrier per quadrant)
//               to store whole 128-byte row segments.
// Pipelines: STAGES shared-memory stages (full/empty mbarriers) and two TMEM
// accumulators (tmem_full/tmem_empty) so the epilogue of tile i overlaps the
// main loop of tile i+1.
//
// CTA pairs (PAIR): a cluster of two CTAs on two SMs computes one 256-row tile
// with tcgen05.mma.cta_group::2 (M = 256).  Each CTA stages its own 128 rows
// of A and its half of the B tile (for SwiGLU: the even CTA the W1 rows, the
// odd one the W3 rows), so a CTA moves 2/3 of the operand bytes per k-block of
// an unpaired 128 x 256 tile and the same shared memory holds 1.5x the stages.
// The even CTA issues the MMAs.  Both CTAs' copies of a stage complete on the
// even CTA's full barrier (the odd CTA's tensor copies name the peer barrier,
// .cta_group::2), which the even CTA arms for the bytes of both.  MMA
// completion is committed to both CTAs' empty and accumulator-full barriers
// (multicast); both CTAs' epilogue warps release an accumulator on the even
// CTA's tmem_empty barrier.  TMEM is allocated for the pair (cta_group::2), and
// a cluster barrier precedes its release.  After an abort the odd CTA cannot
// observe its own copies, so it waits a fixed, bounded time for them to land.
//
// Two pairs per cluster (QUAD, opt-in): four CTAs, pair p = CTAs 2p and
// 2p + 1, both pairs on the same 256 rows of A and on N tiles 2j and 2j + 1.
// Each CTA loads 64 of its 128 A rows and multicasts them to the CTA of the
// same pair rank in the other pair; a destination's bytes complete on the full
// barrier of its own pair's even CTA.  Stage-freeing commits go to all four
// CTAs and each empty barrier counts both pairs' commits.
//
// Every mbarrier wait is bounded by a clock64 budget.  A wait that gives up
// sets the device error word, raises a CTA-wide abort flag that ends every
// other wait at once, waits (again bounded) for the CTA's own TMA copies and
// MMAs still in flight, frees TMEM and returns.  The warps of a quadrant agree
// on the outcome of their accumulator wait (bar.red.and) before they meet at
// their named barriers, so a timeout never leaves one of them behind.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <stdlib.h>

#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace ec2moe {

// bit 0: a bounded wait timed out; bit 1: a group range (offsets) or a
// scatter destination (perm) outside the rows of the call was skipped
__device__ unsigned int g_tc_error;

namespace {

using namespace tc;

constexpr int BM = 128;   // tile rows (MMA M, TMEM lanes)
constexpr int BK = 64;    // K per stage: one 128-byte swizzle row of bf16
constexpr int UK = 16;    // K of one tcgen05.mma kind::f16
constexpr int EPI_WARPS = 16;                    // four per TMEM lane quadrant
constexpr int NUM_THREADS = 64 + 32 * EPI_WARPS;  // producer + MMA warps + epilogue
constexpr int MAX_GROUPS = 136;

struct Params {
  const int32_t* offsets;
  int G, M, a_shared;
  long long a_row_base, out_row_base;
  int N, K, b_group_rows;
  void* out;
  long long ldo;
  const int32_t* perm;
  const float* scale;
  int rep_k;
  long long self_row_base;
  const int32_t* rep_counts;
  const int32_t* rep_idx;
  int32_t* rep_perm_out;
  int32_t* rep_offsets_out;
  int rep_E;
  long long timeout;
  int n_tiles_n;
  int split_k, kb_per_split;
  float* partial;
  long long part_rows;
  long long row_limit;  // rows of the call: group ranges and scatter destinations lie in [0, row_limit)
};

// ------------------------------------------------------------------ tile schedule
struct TileCoord {
  int g, m_blk, n_blk;
};

// Linear tile order: group-major, then n block, then m block, so CTAs that run
// at the same time share the group's weight tiles and activation rows in L2.
__device__ __forceinline__ TileCoord decode_tile(int tile, const int* tile_prefix, int n_tiles_n, int& cursor) {
  while (tile >= tile_prefix[cursor + 1] * n_tiles_n) ++cursor;
  const int mt = tile_prefix[cursor + 1] - tile_prefix[cursor];
  const int rem = tile - tile_prefix[cursor] * n_tiles_n;
  return TileCoord{cursor, rem % mt, rem / mt};
}

constexpr int pow2_at_least(int x) { return x <= 32 ? 32 : (x <= 64 ? 64 : (x <= 128 ? 128 : (x <= 256 ? 256 : 512))); }

template <int BN, int EPI, int STAGES, bool PAIR>
struct Cfg {
  static constexpr int CTA_B_ROWS = PAIR ? BN / 2 : BN;  // rows of the B tile this CTA stages
  static constexpr int TILE_M = PAIR ? 2 * BM : BM;      // rows of one (pair) tile
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = CTA_B_ROWS * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int BN_OUT = (EPI == EPI_SWIGLU) ? BN / 2 : BN;
  // columns of a tile split among the warps of a lane quadrant: PARTS parts
  // of PART columns (a multiple of the 16-column TMEM load)
  static constexpr int PARTS = (BN_OUT % 64 == 0) ? 4 : ((BN_OUT % 48 == 0) ? 3 : ((BN_OUT % 32 == 0) ? 2 : 1));
  static constexpr int PART = BN_OUT / PARTS;
  static constexpr int CW = 16;  // columns per TMEM load
  static_assert(PART % CW == 0, "epilogue chunks must tile each part exactly");
  static constexpr int TMEM_COLS = pow2_at_least(2 * BN);  // two accumulators
  // mbarriers: full[S], empty[S], tmem_full[2], tmem_empty[2], drain
  static constexpr int N_BARS = 2 * STAGES + 5;
  static constexpr int STG_PITCH = CW * 2 + 16;          // bytes per staged row (padded)
  // Row-segment epilogue (contiguous or per-row destinations): the four warps
  // of a lane quadrant stage 32 rows x 64 columns (bf16, 128-byte rows,
  // 16-byte chunks XOR-swizzled by row) and store whole 128-byte row
  // segments (EPI_REPLICATE: to each of the row's destinations); EPI_PARTIAL
  // writes fp32 from registers.
  static constexpr bool ROWSEG = (EPI == EPI_STORE || EPI == EPI_GELU || EPI == EPI_SWIGLU || EPI == EPI_SCATTER ||
                                  EPI == EPI_REPLICATE) &&
                                 BN_OUT % 64 == 0;
  static constexpr int SLAB = 64;
  static constexpr int STG_BYTES =
      ROWSEG ? 4 * 32 * SLAB * 2 : (EPI == EPI_PARTIAL ? 0 : EPI_WARPS * 32 * STG_PITCH);
  static constexpr int OFF_INTS = 132;  // expert offsets of EPI_REPLICATE's relative mode (<= 128 + 1, padded)
  // byte offsets from the 1024-aligned base: operand stages, barriers, TMEM
  // slot + abort flag (16 bytes), tile prefix, group first rows, expert
  // offsets, then the epilogue staging (128-byte aligned: its rows are
  // written with 16-byte vector stores)
  static constexpr int OFF_BARS = STAGES * STAGE_BYTES;
  static constexpr int OFF_SLOT = OFF_BARS + N_BARS * 8;
  static constexpr int OFF_PREFIX = OFF_SLOT + 16;
  static constexpr int OFF_ROW0 = OFF_PREFIX + (MAX_GROUPS + 1) * 4;
  static constexpr int OFF_SOFF = OFF_ROW0 + (MAX_GROUPS + 1) * 4;
  // EPI_REPLICATE with the row-segment epilogue: the tile's destination rows
  // [row][slot] (-1: no row), written once per tile by the first warp of each
  // lane quadrant and read by all four
  static constexpr int DST_BYTES = (EPI == EPI_REPLICATE && ROWSEG) ? BM * 8 * 4 : 0;
  static constexpr int OFF_DST = OFF_SOFF + OFF_INTS * 4;
  static constexpr int OFF_STG = (OFF_DST + DST_BYTES + 127) / 128 * 128;
  static constexpr int SMEM = 1024 + OFF_STG + STG_BYTES;
  static_assert(OFF_BARS % 8 == 0 && OFF_STG % 128 == 0, "shared memory alignment");
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

template <int BN, int EPI, int STAGES, bool PAIR, bool QUAD = false>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmB2, const Params p) {
  static_assert(!QUAD || PAIR, "two pairs per cluster need CTA pairs");
  using C = Cfg<BN, EPI, STAGES, PAIR>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BARS);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* tfull = bars + 2 * STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tfull + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_SLOT);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* tile_prefix = reinterpret_cast<int*>(smem + C::OFF_PREFIX);
  int* row0 = reinterpret_cast<int*>(smem + C::OFF_ROW0);
  int* s_off = reinterpret_cast<int*>(smem + C::OFF_SOFF);  // [C::OFF_INTS]
  int* s_dst = reinterpret_cast<int*>(smem + C::OFF_DST);    // [BM][8] (EPI_REPLICATE, row segments)
  uint8_t* stg_all = smem + C::OFF_STG;                      // epilogue staging

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // PAIR: rank in the CTA pair (0 issues the MMAs), the pair's even CTA in
  // the cluster, the cluster's tile stream.  QUAD: the cluster holds two pairs
  // (CTAs 0-1 and 2-3) on the same 256 rows of A and neighbouring N tiles;
  // each CTA loads half of its 128 A rows and multicasts them to the CTA of
  // the same pair rank in the other pair.
  const uint32_t crank = PAIR ? cluster_ctarank() : 0u;
  const uint32_t rank = crank & 1u;
  const uint32_t leader = crank & ~1u;
  const int pp = QUAD ? static_cast<int>(crank >> 1) : 0;
  const int ntn = QUAD ? p.n_tiles_n / 2 : p.n_tiles_n;  // N tiles of a cluster tile's stream
  const int tile_first = PAIR ? static_cast<int>(cluster_id_x()) : static_cast<int>(blockIdx.x);
  const int tile_step = PAIR ? static_cast<int>(cluster_count_x()) : static_cast<int>(gridDim.x);
  // Barrier set-up, TMEM allocation and descriptor prefetch overlap the
  // previous kernel; everything that reads its results comes after pdl_wait.
  pdl_trigger();

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      // QUAD: a stage is free once both pairs' MMAs have read it (the other
      // pair multicasts into it)
      mbar_init(smem_u32(&empty[s]), QUAD ? 2 : 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), PAIR ? 2 * EPI_WARPS : EPI_WARPS);
    }
    mbar_init(smem_u32(drain), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {
    pdl_wait();
    // Per-group first rows and tile prefix (m tiles), one warp-wide scan.
    warp_exclusive_scan<(MAX_GROUPS + 31) / 32>(
        p.G, lane,
        [&](int g) {
          int r0 = g * p.M, mg = p.M;
          if (p.offsets) {
            r0 = p.offsets[g];
            mg = p.offsets[g + 1] - r0;
            if (r0 < 0 || mg < 0 || static_cast<long long>(r0) + mg > p.row_limit) {
              // not a range of this call's rows: the group is skipped
              atomicOr(&g_tc_error, 2u);
              r0 = 0;
              mg = 0;
            }
          }
          row0[g] = r0;
          return (mg + C::TILE_M - 1) / C::TILE_M;
        },
        tile_prefix);
    if (EPI == EPI_REPLICATE && p.rep_counts)
      warp_exclusive_scan<(MAX_GROUPS + 31) / 32>(p.rep_E, lane, [&](int e) { return p.rep_counts[e]; }, s_off,
                                                   blockIdx.x == 0 ? p.rep_offsets_out : nullptr);
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (EPI == EPI_SWIGLU) tma_prefetch_desc(&tmB2);
  }
  if (warp == 1) {
    if (PAIR) {
      // the pair's columns, allocated by one warp of each CTA together
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                   "r"(C::TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                   "r"(C::TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  // PAIR: both CTAs' barriers are initialised before either arrives remotely
  if (PAIR) cluster_sync_all();
  tc_fence_after();
  pdl_wait();
  const uint32_t tmem_base = *tmem_slot;
  // Split-K (EPI_PARTIAL): tile t covers output tile t / split_k and the
  // k-blocks [ks * kb_per_split, ...) with ks = t % split_k.
  const int n_tiles = tile_prefix[p.G] * ntn * p.split_k;
  const int num_kb = (p.K + BK - 1) / BK;
  const long long budget = p.timeout;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0;  // bit s: stage s holds a copy the consumer has not released
      uint32_t issued_phase = 0;
      int cursor = 0;
      bool ok = true;
      for (int tile = tile_first; tile < n_tiles && ok; tile += tile_step) {
        const TileCoord tc = decode_tile(tile / p.split_k, tile_prefix, ntn, cursor);
        const int n_blk = QUAD ? 2 * tc.n_blk + pp : tc.n_blk;
        const int a_row = static_cast<int>(p.a_row_base) + (p.offsets ? row0[tc.g] : (p.a_shared ? 0 : row0[tc.g])) +
                          tc.m_blk * C::TILE_M + static_cast<int>(rank) * BM;
        const int b_row = tc.g * p.b_group_rows + n_blk * C::BN_OUT;
        const int kb0 = (tile % p.split_k) * p.kb_per_split;
        const int kb1 = kb0 + p.kb_per_split < num_kb ? kb0 + p.kb_per_split : num_kb;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, budget, abort_flag, &g_tc_error)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          if (PAIR) {
            // both halves complete on the even CTA's full barrier
            if (rank == 0) mbar_expect_tx(fb, 2 * C::STAGE_BYTES);
            const uint32_t fb0 = rank == 0 ? fb : map_to_rank(fb, leader);
            if (QUAD) {
              // rows [pp * 64, pp * 64 + 64) of this CTA's 128, to both pairs
              tma_load_2d_mc_pair(smem_u32(sA + stage * C::A_BYTES + pp * (BM / 2) * BK * 2), &tmA, kb * BK,
                                  a_row + pp * (BM / 2), fb0, static_cast<uint16_t>(0x5u << rank));
            } else {
              tma_load_2d_to_pair_bar(smem_u32(sA + stage * C::A_BYTES), &tmA, kb * BK, a_row, fb0);
            }
            // SwiGLU: the even CTA stages the W1 rows of the tile, the odd CTA the W3 rows
            const CUtensorMap* tb = (EPI == EPI_SWIGLU && rank) ? &tmB2 : &tmB;
            tma_load_2d_to_pair_bar(smem_u32(sB + stage * C::B_BYTES), tb, kb * BK,
                                    b_row + (EPI == EPI_SWIGLU ? 0 : static_cast<int>(rank) * C::CTA_B_ROWS), fb0);
          } else {
            mbar_expect_tx(fb, C::STAGE_BYTES);
            tma_load_2d(smem_u32(sA + stage * C::A_BYTES), &tmA, kb * BK, a_row, fb);
            if (EPI == EPI_SWIGLU) {
              tma_load_2d(smem_u32(sB + stage * C::B_BYTES), &tmB, kb * BK, b_row, fb);
              tma_load_2d(smem_u32(sB + stage * C::B_BYTES + C::B_BYTES / 2), &tmB2, kb * BK, b_row, fb);
            } else {
              tma_load_2d(smem_u32(sB + stage * C::B_BYTES), &tmB, kb * BK, b_row, fb);
            }
          }
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok || *abort_flag) {
        // Let every copy this CTA started land before shared memory is released.
        if (PAIR && rank != 0) {
          // its copies complete on the even CTA's barriers: wait a fixed time
          if (issued) {
            const unsigned long long t0 = globaltimer_ns();
            while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
          }
        } else {
          for (int s = 0; s < STAGES; ++s)
            if (issued & (1u << s)) mbar_drain(smem_u32(&full[s]), (issued_phase >> s) & 1u, DRAIN_CYCLES);
        }
        if (QUAD) {
          // the other pair's multicasts into this CTA's stages are not all
          // counted on barriers this CTA waited on: a fixed time to land too
          const unsigned long long t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
        }
      }
    }
  } else if (warp == 1) {
    if (PAIR && rank != 0) {
      // odd CTA of a pair: the even CTA issues the pair's MMAs
    } else if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      constexpr uint32_t IDESC = idesc_bf16(C::TILE_M, BN);
      constexpr uint64_t DA_STAGE = C::A_BYTES >> 4;
      constexpr uint64_t DB_STAGE = C::B_BYTES >> 4;
      const uint64_t da0 = sdesc_sw128(smem_u32(sA));
      const uint64_t db0 = sdesc_sw128(smem_u32(sB));
      const uint32_t full0 = smem_u32(&full[0]);
      const uint32_t empty0 = smem_u32(&empty[0]);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      int cursor = 0;
      bool ok = true, any = false;
      for (int tile = tile_first; tile < n_tiles && ok; tile += tile_step, ++it) {
        (void)decode_tile(tile / p.split_k, tile_prefix, ntn, cursor);
        const int kb0 = (tile % p.split_k) * p.kb_per_split;
        const int kb1 = kb0 + p.kb_per_split < num_kb ? kb0 + p.kb_per_split : num_kb;
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        // PAIR: the odd CTA's epilogue warps release the accumulator remotely
        const bool freed = PAIR ? mbar_wait_cluster(smem_u32(&tempty[acc]), acc_phase ^ 1u, budget, abort_flag, &g_tc_error)
                                : mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1u, budget, abort_flag, &g_tc_error);
        if (!freed) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(full0 + 8u * stage, phase, budget, abort_flag, &g_tc_error)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // Descriptors of this stage: the stage-0 descriptors plus the stage
          // offset; each K = 16 step adds 32 bytes (2 in the address field).
          // The address field (bits 0-13) cannot carry: shared addresses are
          // below 256 KB.
          const uint64_t da = da0 + static_cast<uint64_t>(stage) * DA_STAGE;
          const uint64_t db = db0 + static_cast<uint64_t>(stage) * DB_STAGE;
          if (PAIR) {
            umma_bf16_pair(d_tmem, da, db, IDESC, kb != kb0 ? 1u : 0u);
#pragma unroll
            for (int kk = 1; kk < BK / UK; ++kk) umma_bf16_pair(d_tmem, da + 2 * kk, db + 2 * kk, IDESC, 1u);
          } else {
            umma_bf16(d_tmem, da, db, IDESC, kb != kb0 ? 1u : 0u);
#pragma unroll
            for (int kk = 1; kk < BK / UK; ++kk) umma_bf16(d_tmem, da + 2 * kk, db + 2 * kk, IDESC, 1u);
          }
          any = true;
          // QUAD: both pairs' producers wait for this stage
          if (PAIR) umma_commit_pair_mc(empty0 + 8u * stage, QUAD ? 0xF : 0x3);
          else umma_commit(empty0 + 8u * stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if (PAIR) umma_commit_pair_mc(smem_u32(&tfull[acc]), static_cast<uint16_t>(0x3u << leader));
        else umma_commit(smem_u32(&tfull[acc]));
      }
      if ((!ok || *abort_flag) && any) {
        // All MMAs issued so far must finish before TMEM is freed.
        if (PAIR) umma_commit_pair(smem_u32(drain));
        else umma_commit(smem_u32(drain));
        mbar_drain(smem_u32(drain), 0, DRAIN_CYCLES);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;              // TMEM lane quadrant this warp may access
    const int part = (warp - 2) >> 2;    // which part of the tile's columns
    const int row_in_tile = q * 32 + lane;
    int it = 0;
    int cursor = 0;
    for (int tile = tile_first; tile < n_tiles; tile += tile_step, ++it) {
      const TileCoord tc = decode_tile(tile / p.split_k, tile_prefix, ntn, cursor);
      const int n_blk = QUAD ? 2 * tc.n_blk + pp : tc.n_blk;
      const int ks = tile % p.split_k;
      (void)ks;
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      // Row metadata first: its global loads overlap the tile's main loop.
      // (a group's tiles exist only if the prologue accepted its range)
      const int mg = p.offsets ? (p.offsets[tc.g + 1] - p.offsets[tc.g]) : p.M;
      const int local = tc.m_blk * C::TILE_M + static_cast<int>(rank) * BM + row_in_tile;
      bool valid = local < mg;
      const long long out_row = p.out_row_base + row0[tc.g] + local;
      long long dest = out_row;
      float sc = 1.0f;
      if (EPI == EPI_SCATTER && valid) {
        dest = p.perm ? p.perm[out_row] : out_row;
        if (dest < 0 || dest >= p.row_limit) {
          atomicOr(&g_tc_error, 2u);
          valid = false;
          dest = 0;
        } else if (p.scale) {
          sc = p.scale[dest];
        }
      }
      // EPI_REPLICATE: this row's destinations, read once per tile (with the
      // row-segment epilogue by the quadrant's first warp only, into s_dst;
      // the other three read them there after the first slab's barrier, and
      // the last slab's barrier orders the next tile's writes after every read)
      int rdst[8];
      if (EPI == EPI_REPLICATE && C::ROWSEG) {
        if (part == 0) {
          int* sd = s_dst + row_in_tile * 8;
#pragma unroll
          for (int r = 0; r < 8; ++r) {
            if (r >= p.rep_k) break;
            int dst = -1;
            if (valid) {
              const long long entry = out_row * p.rep_k + r;
              dst = p.perm[entry];
              if (p.rep_counts) {
                dst += s_off[p.rep_idx[entry]];
                p.rep_perm_out[dst] = static_cast<int32_t>(entry);
              }
            }
            sd[r] = dst;
          }
        }
      } else if (EPI == EPI_REPLICATE) {
#pragma unroll
        for (int r = 0; r < 8; ++r) {
          rdst[r] = 0;
          if (valid && r < p.rep_k) {
            const long long entry = out_row * p.rep_k + r;
            int dst = p.perm[entry];
            if (p.rep_counts) {
              dst += s_off[p.rep_idx[entry]];
              p.rep_perm_out[dst] = static_cast<int32_t>(entry);
            }
            rdst[r] = dst;
          }
        }
      }
      bool ok = mbar_wait(smem_u32(&tfull[acc]), acc_phase, budget, abort_flag, &g_tc_error);
      if (C::ROWSEG) {
        // the quadrant's four warps take the same path (they meet at named barriers)
        uint32_t all_ok;
        asm volatile(
            "{\n .reg .pred p, r;\n setp.ne.u32 p, %1, 0;\n"
            " bar.red.and.pred r, %2, 128, p;\n selp.u32 %0, 1, 0, r;\n}"
            : "=r"(all_ok)
            : "r"(ok ? 1u : 0u), "r"(1 + q)
            : "memory");
        ok = all_ok != 0;
      }
      if (!ok) break;
      tc_fence_after();
      const uint32_t t_row = tmem_base + static_cast<uint32_t>(acc * BN) + (static_cast<uint32_t>(q * 32) << 16);
      if constexpr (C::ROWSEG) {
        // Slabs of 64 output columns: warp `part` rounds its 16 columns of the
        // slab for the quadrant's 32 rows into the quadrant's staging slab,
        // then each warp stores 8 of the 32 rows as 128-byte row segments (4
        // rows per store instruction).  The destination row of staged row rr
        // comes from lane rr, which owns that row in every warp of the quadrant.
        uint8_t* slab = stg_all + q * (32 * C::SLAB * 2);
        constexpr int NSLAB = C::BN_OUT / C::SLAB;
#pragma unroll 1
        for (int sl = 0; sl < NSLAB; ++sl) {
          const int c0 = sl * C::SLAB + part * 16;
          uint32_t rv[16], ru[16];
          tmem_ld_nw<16>(t_row + c0, rv);
          if (EPI == EPI_SWIGLU) tmem_ld_nw<16>(t_row + c0 + BN / 2, ru);
          tmem_wait();
          float v[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            v[i] = __uint_as_float(rv[i]);
            if (EPI == EPI_SWIGLU) v[i] = silu_bf16out(v[i]) * __uint_as_float(ru[i]);
            else if (EPI == EPI_GELU) v[i] = gelu_bf16out(v[i]);
            else if (EPI == EPI_SCATTER) v[i] *= sc;
          }
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            U4 q4{pack_bf16x2(v[8 * j + 0], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                  pack_bf16x2(v[8 * j + 4], v[8 * j + 5]), pack_bf16x2(v[8 * j + 6], v[8 * j + 7])};
            *reinterpret_cast<U4*>(slab + lane * 128 + (((2 * part + j) ^ (lane & 7)) * 16)) = q4;
          }
          asm volatile("bar.sync %0, 128;" ::"r"(1 + q) : "memory");
          const int seg = lane & 7;
          const int col = n_blk * C::BN_OUT + sl * C::SLAB + seg * 8;
#pragma unroll
          for (int pass = 0; pass < 2; ++pass) {
            const int rr = part * 8 + pass * 4 + (lane >> 3);
            const bool rvalid = __shfl_sync(0xffffffffu, valid ? 1 : 0, rr) != 0;
            const U4 q4 = *reinterpret_cast<const U4*>(slab + rr * 128 + ((seg ^ (rr & 7)) * 16));
            __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(p.out);
            if (EPI == EPI_REPLICATE) {
              // the row's expert-order slots, then (optionally) its own row
              const int* sd = s_dst + (q * 32 + rr) * 8;  // staged row rr is row q * 32 + rr of the tile
#pragma unroll
              for (int r = 0; r < 8; ++r) {
                if (r >= p.rep_k) break;  // uniform across the warp
                const int dr = sd[r];
                if (rvalid && dr >= 0 && col < p.N) *reinterpret_cast<U4*>(ob + (long long)dr * p.ldo + col) = q4;
              }
              if (rvalid && col < p.N && p.self_row_base >= 0)
                *reinterpret_cast<U4*>(ob + (p.self_row_base + out_row - lane + rr) * p.ldo + col) = q4;
            } else {
              const long long drow = __shfl_sync(0xffffffffu, dest, rr);
              if (rvalid && col < p.N) *reinterpret_cast<U4*>(ob + drow * p.ldo + col) = q4;
            }
          }
          asm volatile("bar.sync %0, 128;" ::"r"(1 + q) : "memory");
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          // PAIR: both CTAs release the accumulator on the even CTA's barrier
          if (PAIR) mbar_arrive_remote(map_to_rank(smem_u32(&tempty[acc]), leader));
          else mbar_arrive(smem_u32(&tempty[acc]));
        }
        continue;
      }
      // Each chunk of 32 rows x CW columns is staged in shared memory (thread =
      // row) and written back with CW/8 lanes per row, so a warp store writes
      // whole 32-byte sectors of 16 rows instead of 16-byte pieces of 32 rows.
      uint8_t* stg = stg_all + (warp - 2) * 32 * C::STG_PITCH;
      constexpr int SEGS = C::CW / 8;           // 16-byte segments per row
      constexpr int ROWS_PER_PASS = 32 / SEGS;  // rows a warp store covers
      // Two chunks' TMEM loads are issued before one wait (half as many waits);
      // a part with an odd number of chunks ends on a single chunk.  Warps
      // beyond PARTS (narrow tiles) have no columns.
      constexpr int NCH = C::PART / C::CW;
      const int nch_mine = part < C::PARTS ? NCH : 0;
      uint32_t rv[2][C::CW], ru[2][C::CW];
#pragma unroll 1
      for (int ci = 0; ci < nch_mine; ++ci) {
        const int c0 = part * C::PART + ci * C::CW;
        const int slot = ci & 1;
        if (slot == 0) {
          tmem_ld_nw<C::CW>(t_row + c0, rv[0]);
          if (EPI == EPI_SWIGLU) tmem_ld_nw<C::CW>(t_row + c0 + BN / 2, ru[0]);
          if (ci + 1 < nch_mine) {
            tmem_ld_nw<C::CW>(t_row + c0 + C::CW, rv[1]);
            if (EPI == EPI_SWIGLU) tmem_ld_nw<C::CW>(t_row + c0 + C::CW + BN / 2, ru[1]);
          }
          tmem_wait();
        }
        const int col = n_blk * C::BN_OUT + c0;
        float v[C::CW];
#pragma unroll
        for (int i = 0; i < C::CW; ++i) v[i] = __uint_as_float(slot ? rv[1][i] : rv[0][i]);
        if (EPI == EPI_SWIGLU) {
#pragma unroll
          for (int i = 0; i < C::CW; ++i) v[i] = silu_bf16out(v[i]) * __uint_as_float(slot ? ru[1][i] : ru[0][i]);
        } else if (EPI == EPI_GELU) {
#pragma unroll
          for (int i = 0; i < C::CW; ++i) v[i] = gelu_bf16out(v[i]);
        } else if (EPI == EPI_SCATTER) {
#pragma unroll
          for (int i = 0; i < C::CW; ++i) v[i] *= sc;
        }
        if (col >= p.N) continue;  // uniform across the warp
        if (EPI == EPI_PARTIAL) {
          // fp32 partial sums, 64 contiguous bytes per row and chunk
          if (valid) {
            float4* dstp = reinterpret_cast<float4*>(p.partial + (ks * p.part_rows + out_row) * p.N + col);
#pragma unroll
            for (int j = 0; j < C::CW / 4; ++j) dstp[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
          }
          continue;
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < SEGS; ++j) {
          U4 q4{pack_bf16x2(v[8 * j + 0], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                pack_bf16x2(v[8 * j + 4], v[8 * j + 5]), pack_bf16x2(v[8 * j + 6], v[8 * j + 7])};
          *reinterpret_cast<U4*>(stg + lane * C::STG_PITCH + 16 * j) = q4;
        }
        __syncwarp();
        const int sg = lane % SEGS;
#pragma unroll
        for (int pass = 0; pass < SEGS; ++pass) {
          const int rr = pass * ROWS_PER_PASS + lane / SEGS;  // staged row this lane writes
          const bool rvalid = __shfl_sync(0xffffffffu, valid ? 1 : 0, rr) != 0;
          const U4 q4 = *reinterpret_cast<const U4*>(stg + rr * C::STG_PITCH + 16 * sg);
          if (EPI == EPI_REPLICATE) {
            const long long orow_r = __shfl_sync(0xffffffffu, out_row, rr);
            __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(p.out);
#pragma unroll
            for (int r = 0; r < 8; ++r) {
              const int dr = __shfl_sync(0xffffffffu, rdst[r], rr);
              if (rvalid && r < p.rep_k) *reinterpret_cast<U4*>(ob + (long long)dr * p.ldo + col + 8 * sg) = q4;
            }
            if (rvalid && p.self_row_base >= 0)
              *reinterpret_cast<U4*>(ob + (p.self_row_base + orow_r) * p.ldo + col + 8 * sg) = q4;
          } else {
            const long long drow = __shfl_sync(0xffffffffu, dest, rr);
            if (rvalid)
              *reinterpret_cast<U4*>(reinterpret_cast<__nv_bfloat16*>(p.out) + drow * p.ldo + col + 8 * sg) = q4;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (PAIR) mbar_arrive_remote(map_to_rank(smem_u32(&tempty[acc]), leader));
        else mbar_arrive(smem_u32(&tempty[acc]));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // PAIR: the even CTA's MMAs write both CTAs' TMEM; neither releases its
  // columns before both are done with them
  if (PAIR) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::TMEM_COLS)
                   : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::TMEM_COLS)
                   : "memory");
  }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// Map kinds: bf16 with the 128-byte swizzle, or fp32 unswizzled (rows of
// 64 x 4 = 256 bytes in shared memory).
enum MapKind { MAP_BF16_SW128 = 0, MAP_F32_PLAIN = 1 };

bool encode_map(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows, int kind);

// Encoded tensor maps are cached by (device, address, shape, box, kind):
// encoding costs host time on every launch otherwise.  A map only describes
// an address and a layout, so a hit stays valid even if the memory was
// reallocated.
struct MapKey {
  int dev;
  const void* ptr;
  long long rows, cols;
  int box_rows;
  int kind;
  bool operator==(const MapKey& o) const {
    return dev == o.dev && ptr == o.ptr && rows == o.rows && cols == o.cols && box_rows == o.box_rows &&
           kind == o.kind;
  }
};

// 2-D tensor map over a row-major [rows, cols] matrix, box = 64 columns x
// box_rows rows, zero fill out of bounds.
bool make_map(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows,
              int kind = MAP_BF16_SW128) {
  constexpr int SLOTS = 64;
  static std::mutex mu;
  static MapKey keys[SLOTS];
  static CUtensorMap maps[SLOTS];
  static bool used[SLOTS] = {};
  static int next = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  const MapKey key{dev, ptr, rows, cols, box_rows, kind};
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < SLOTS; ++i)
      if (used[i] && keys[i] == key) {
        *m = maps[i];
        return true;
      }
  }
  if (!encode_map(m, ptr, rows, cols, box_rows, kind)) return false;
  std::lock_guard<std::mutex> lock(mu);
  keys[next] = key;
  maps[next] = *m;
  used[next] = true;
  next = (next + 1) % SLOTS;
  return true;
}

bool encode_map(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows, int kind) {
  auto fn = encode_fn();
  if (!fn) return false;
  const bool f32 = kind == MAP_F32_PLAIN;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * (f32 ? 4 : 2)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  f32 ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

const char* kernel_name(int epi) {
  switch (epi) {
    case EPI_GELU: return "gemm_tc_gelu";
    case EPI_SWIGLU: return "gemm_tc_swiglu";
    case EPI_SCATTER: return "gemm_tc_scatter";
    case EPI_REPLICATE: return "gemm_tc_replicate";
    default: return "gemm_tc_store";
  }
}

// Clusters of `cdim` CTAs (2: one pair, 4: two pairs) of `kernel` that fit on
// the device at once (cached per device and kernel); 0 when the query fails.
int max_pair_clusters(const void* kernel, int smem, int cdim) {
  struct Entry {
    int dev;
    const void* kernel;
    int n;
  };
  static std::mutex mu;
  static Entry cache[32];
  static int used = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (cache[i].dev == dev && cache[i].kernel == kernel) return cache[i].n;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(cdim * sm_count());
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cdim;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    n = 0;
  }
  if (used < 32) cache[used++] = Entry{dev, kernel, n};
  return n;
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pairs(void (*kernel)(KArgs...), int clusters, int cdim, size_t smem, cudaStream_t s,
                         Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(cdim * clusters);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cdim;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = next_launch_pdl() ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

template <int BN, int EPI, int STAGES, bool PAIR = false, bool QUAD = false>
cudaError_t launch_cfg(const GemmArgs& a, cudaStream_t s) {
  using C = Cfg<BN, EPI, STAGES, PAIR>;
  const void* kfn = reinterpret_cast<const void*>(tc_gemm_kernel<BN, EPI, STAGES, PAIR, QUAD>);
  cudaError_t attr_err = ensure_smem_attr(kfn, C::SMEM);
  if (attr_err != cudaSuccess) return attr_err;
  CUtensorMap mA, mB, mB2;
  const int b_box = (EPI == EPI_SWIGLU || PAIR) ? BN / 2 : BN;
  if (!make_map(&mA, a.A, a.a_rows, a.K, QUAD ? BM / 2 : BM)) return cudaErrorInvalidValue;
  if (!make_map(&mB, a.B, a.b_rows, a.K, b_box)) return cudaErrorInvalidValue;
  if (EPI == EPI_SWIGLU) {
    if (!make_map(&mB2, a.B2, a.b_rows, a.K, b_box)) return cudaErrorInvalidValue;
  } else {
    mB2 = mB;
  }
  Params p;
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
  p.rep_k = a.rep_k;
  p.self_row_base = a.self_row_base;
  p.rep_counts = a.rep_counts;
  p.rep_idx = a.rep_idx;
  p.rep_perm_out = a.rep_perm_out;
  p.rep_offsets_out = a.rep_offsets_out;
  p.rep_E = a.rep_E;
  p.timeout = a.timeout_cycles;
  p.n_tiles_n = (a.N + C::BN_OUT - 1) / C::BN_OUT;
  p.split_k = EPI == EPI_PARTIAL && a.split_k > 1 ? a.split_k : 1;
  {
    const int num_kb = (a.K + BK - 1) / BK;
    p.kb_per_split = (num_kb + p.split_k - 1) / p.split_k;
    p.split_k = (num_kb + p.kb_per_split - 1) / p.kb_per_split;  // no empty K range
  }
  p.partial = a.partial;
  p.part_rows = a.part_rows;
  p.row_limit = a.max_rows > 0 ? a.max_rows : (1LL << 62);
  const long long m_tiles_max = a.max_rows / C::TILE_M + a.G;
  long long tiles = m_tiles_max * p.n_tiles_n * p.split_k;
  if (PAIR) {
    // QUAD: a cluster tile is two N tiles (p.n_tiles_n is even)
    if (QUAD) tiles /= 2;
    const int cdim = QUAD ? 4 : 2;
    int clusters = max_pair_clusters(kfn, C::SMEM, cdim);
    if (clusters < 1) return cudaErrorInvalidConfiguration;
    if (tiles < clusters) clusters = static_cast<int>(tiles < 1 ? 1 : tiles);
    KernelScope ks(a.name ? a.name : kernel_name(EPI), s);
    cudaError_t le = launch_pairs(tc_gemm_kernel<BN, EPI, STAGES, PAIR, QUAD>, clusters, cdim, (size_t)C::SMEM, s, mA,
                                  mB, mB2, p);
    if (le != cudaSuccess) return le;
    return cudaGetLastError();
  }
  int grid = static_cast<int>(tiles < sm_count() ? tiles : sm_count());
  if (grid < 1) grid = 1;
  KernelScope ks(a.name ? a.name : kernel_name(EPI), s);
  cudaError_t le = launch_kernel(tc_gemm_kernel<BN, EPI, STAGES, PAIR>, dim3(grid), dim3(NUM_THREADS), (size_t)C::SMEM,
                                 s, mA, mB, mB2, p);
  if (le != cudaSuccess) return le;
  return cudaGetLastError();
}

// Smem budget of the operand pipeline: as many stages as fit in ~200 KB
// (b_rows: rows of the B tile one CTA stages).
constexpr int stages_for(int b_rows) {
  return (200 * 1024) / (BM * BK * 2 + b_rows * BK * 2) > 8 ? 8 : (200 * 1024) / (BM * BK * 2 + b_rows * BK * 2);
}

template <int EPI>
cudaError_t launch_epi(const GemmArgs& a, int bn, bool pair, bool quad, cudaStream_t s) {
  if (pair) {
    if constexpr (EPI == EPI_STORE || EPI == EPI_GELU || EPI == EPI_SWIGLU || EPI == EPI_SCATTER ||
                  EPI == EPI_REPLICATE) {
      if (bn == 256 && quad) return launch_cfg<256, EPI, stages_for(128), true, true>(a, s);
      if (bn == 256) return launch_cfg<256, EPI, stages_for(128), true>(a, s);
      if (bn == 128) return launch_cfg<128, EPI, stages_for(64), true>(a, s);
    }
    return cudaErrorInvalidValue;
  }
  switch (bn) {
    case 32:
      if constexpr (EPI != EPI_SWIGLU) return launch_cfg<32, EPI, stages_for(32)>(a, s);
      break;
    case 64: return launch_cfg<64, EPI, stages_for(64)>(a, s);
    case 128: return launch_cfg<128, EPI, stages_for(128)>(a, s);
    case 192: return launch_cfg<192, EPI, stages_for(192)>(a, s);
    case 256: return launch_cfg<256, EPI, stages_for(256)>(a, s);
  }
  return cudaErrorInvalidValue;
}

// N-tile choice.  Each candidate is scored by its wave efficiency (tiles over
// whole waves of one tile per SM, or per CTA pair) times a per-tile efficiency
// that falls with the tile width (narrow tiles move more operand bytes per
// FLOP).  The m-tile count of a grouped GEMM is only known on the device; half
// a partial tile per group is expected.
int choose_bn(const GemmArgs& a, int epi, bool pair = false) {
  const int ga = a.g_active > 0 ? a.g_active : a.G;
  const int tm = pair ? 2 * BM : BM;
  const double m_tiles = (double)a.max_rows / tm + (a.G > 1 ? 0.5 * ga : 0.0) + (a.G == 1 && a.max_rows % tm ? 1 : 0);
  const int sms = pair ? sm_count() / 2 : sm_count();
  const int cands[5] = {256, 192, 128, 64, 32};
  const double tile_eff[5] = {1.0, 0.97, 0.9, 0.75, 0.6};
  int pick = 0;
  double best = -1.0;
  for (int i = 0; i < 5; ++i) {
    const int bn = cands[i];
    if (pair && bn != 256 && bn != 128) continue;
    const int out = (epi == EPI_SWIGLU) ? bn / 2 : bn;
    if (epi == EPI_SWIGLU && bn < 64) continue;
    if (out > a.N && !(out == 32 || (epi == EPI_SWIGLU && bn == 64))) continue;  // no wider than N
    const double tiles = m_tiles * ((a.N + out - 1) / out);
    const double waves = tiles / sms;
    const double wave_eff = tiles / (sms * (waves <= 1.0 ? 1.0 : static_cast<double>((long long)(waves + 0.999))));
    const double useful = (double)a.N / (((a.N + out - 1) / out) * out);  // columns wasted on a partial N tile
    const double score = wave_eff * tile_eff[i] * useful;
    if (score > best + 1e-9) {
      best = score;
      pick = bn;
    }
  }
  return pick;
}

}  // namespace

bool make_tensor_map_bf16(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows) {
  return make_map(m, ptr, rows, cols, box_rows, MAP_BF16_SW128);
}

bool make_tensor_map_f32(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows) {
  return make_map(m, ptr, rows, cols, box_rows, MAP_F32_PLAIN);
}

// Whether a grouped GEMM runs on CTA pairs (256-row tiles): for the row-
// segment epilogues, when the groups are tall enough that 256-row tiles waste
// at most ~10% more rows than 128-row ones (the Mixtral-shaped and
// fine-grained layers; the Switch-shaped one, with ~341 rows per expert, keeps
// single CTAs).  EC2MOE_GEMM_PAIR=0 / =1 in the environment forbids / forces
// pairs (A/B comparisons; both compute the same result).
bool use_pairs(const GemmArgs& a, int epi) {
  if (!(epi == EPI_STORE || epi == EPI_GELU || epi == EPI_SWIGLU || epi == EPI_SCATTER || epi == EPI_REPLICATE))
    return false;
  static const int forced = [] {
    const char* v = getenv("EC2MOE_GEMM_PAIR");
    return v ? (v[0] == '1' ? 1 : (v[0] == '0' ? 0 : 2)) : 2;
  }();
  if (forced == 0) return false;
  if (forced == 1) return true;
  const int ga = a.g_active > 0 ? a.g_active : a.G;
  const double rows = (double)a.max_rows / ga;  // expected rows per group
  if (rows < 2 * BM) return false;
  const double pad1 = std::ceil(rows / BM) * BM, pad2 = std::ceil(rows / (2 * BM)) * (2 * BM);
  return pad2 <= 1.1 * pad1;
}

// Whether a pair GEMM runs two pairs per cluster on neighbouring N tiles of
// the same rows, each CTA loading half of its A rows and multicasting them to
// the other pair (QUAD): 256-column tiles and an even N-tile count.
// EC2MOE_GEMM_QUAD=0 / =1 in the environment forbids / allows it (A/B
// comparisons; both compute the same result).
bool use_quad(const GemmArgs& a, int epi, int bn) {
  // 0: never; 1: every eligible GEMM; 2: the scattering (down) projections only
  static const int allowed = [] {
    const char* v = getenv("EC2MOE_GEMM_QUAD");
    return v ? (v[0] == '1' ? 1 : (v[0] == 'd' ? 2 : 0)) : 0;
  }();
  if (!allowed || bn != 256 || (allowed == 2 && epi != EPI_SCATTER)) return false;
  const int bn_out = epi == EPI_SWIGLU ? bn / 2 : bn;
  const int n_tiles_n = (a.N + bn_out - 1) / bn_out;
  return n_tiles_n % 2 == 0;
}

cudaError_t launch_gemm_tc(const GemmArgs& a, int epi, cudaStream_t s) {
  if (a.G < 1 || a.G > MAX_GROUPS || a.N % 32 != 0 || a.K % 8 != 0) return cudaErrorInvalidValue;
  bool pair = use_pairs(a, epi);
  int bn = choose_bn(a, epi, pair);
  const int bn_out = epi == EPI_SWIGLU ? bn / 2 : bn;
  if (pair && (bn_out % 64 != 0)) {
    pair = false;
    bn = choose_bn(a, epi, false);
  }
  const bool quad = pair && use_quad(a, epi, bn);
  switch (epi) {
    case EPI_STORE: return launch_epi<EPI_STORE>(a, bn, pair, quad, s);
    case EPI_GELU: return launch_epi<EPI_GELU>(a, bn, pair, quad, s);
    case EPI_SWIGLU: return launch_epi<EPI_SWIGLU>(a, bn, pair, quad, s);
    case EPI_SCATTER: return launch_epi<EPI_SCATTER>(a, bn, pair, quad, s);
    case EPI_REPLICATE: return launch_epi<EPI_REPLICATE>(a, bn, pair, quad, s);
    case EPI_PARTIAL:
      if (!a.partial || a.N % 4 != 0) return cudaErrorInvalidValue;
      return bn >= 256 ? launch_cfg<256, EPI_PARTIAL, stages_for(256)>(a, s)
                       : launch_cfg<128, EPI_PARTIAL, stages_for(128)>(a, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t read_tc_error(unsigned int* word) {
  unsigned int zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(word, g_tc_error, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_tc_error, &zero, sizeof(unsigned int));
}

// About two seconds at the GB300's maximum SM clock unless changed with
// ec2moe_set_wait_budget.
namespace {
std::atomic<long long> g_wait_budget{4000000000LL};
}
long long default_timeout_cycles() { return g_wait_budget.load(); }
void set_timeout_cycles(long long cycles) { g_wait_budget.store(cycles); }

}  // namespace ec2moe
