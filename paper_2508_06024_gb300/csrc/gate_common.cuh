// Definitions shared by the two gate translation units (gate.cu: SIMT gates
// and the dispatch; gate_tc.cu: the tensor-core gate).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace ec2moe {
namespace gatek {

constexpr int MAX_TOPK = 8;

struct KParams {
  const void* X;
  const float* W_local;
  const float* b_local;
  const float* W_global;
  const float* b_global;
  uint32_t mask_bits[4];
  int T, d, E, K, k, renorm;
  int top_groups;  // > 0 and < live groups: per token only the top_groups groups by m keep their experts
  int32_t* topk_idx;
  float* topk_w;
  int32_t* route_counts;  // fused routing: per-expert row counters (zero at launch); nullptr = gate only
  int32_t* route_rel;     // fused routing: [T*k] row of each entry relative to its expert's first row
  // L2 prefetch of the decode up projection's first weight tiles by the
  // small-batch decision kernel (GateArgs::pf_*); pf_w1 == nullptr: none
  const void* pf_w1;
  const void* pf_w3;
  int pf_dff, pf_tile_rows, pf_row_bytes;
};

// Tensor-core gate (bf16, at most 80 gate rows) with its prep kernel; sets
// *handled when it took the call (else the caller runs a SIMT gate).
cudaError_t launch_gate_tensor(const GateArgs& a, KParams p, int O, bool bf16, cudaStream_t s, bool* routed, int* held_sms,
                               bool* handled);

}  // namespace gatek
}  // namespace ec2moe
