// Small device helpers shared by the kernels of libec2moe.so.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ec2moe {

struct alignas(16) U4 { uint32_t x, y, z, w; };

// Programmatic dependent launch: let the next kernel in the stream start its
// independent prologue now / wait until the previous kernel's results are
// complete and visible (a no-op when launched without the attribute).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// Round-to-nearest-even pack of two floats into bf16x2 (lo in the low half).
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// 8 consecutive elements as floats from a bf16 or fp32 row (16-byte aligned).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float* v) {
  U4 q = *reinterpret_cast<const U4*>(p);
  v[0] = bf16_lo(q.x); v[1] = bf16_hi(q.x); v[2] = bf16_lo(q.y); v[3] = bf16_hi(q.y);
  v[4] = bf16_lo(q.z); v[5] = bf16_hi(q.z); v[6] = bf16_lo(q.w); v[7] = bf16_hi(q.w);
}
__device__ __forceinline__ void load8(const float* p, float* v) {
  float4 a = *reinterpret_cast<const float4*>(p);
  float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float* v) {
  U4 q{pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7])};
  *reinterpret_cast<U4*>(p) = q;
}
__device__ __forceinline__ void store8(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}

// GELU(u) = u * Phi(u) = u/2 (1 + erf(u / sqrt 2)), the exact form.
__device__ __forceinline__ float gelu_erf(float u) { return 0.5f * u * (1.0f + erff(u * 0.70710678118654752f)); }
// SiLU(u) = u / (1 + e^-u).
__device__ __forceinline__ float silu(float u) { return u / (1.0f + expf(-u)); }

// GELU for epilogues whose output is rounded to bf16 (relative step 2^-8):
// the tanh form GELU(u) ~ u/2 (1 + tanh(sqrt(2/pi) (u + 0.044715 u^3)))
// (Hendrycks & Gimpel, 2016) on the SFU's tanh.approx.f32 (absolute error
// about 2^-11).  Against the exact u Phi(u) the form is off by at most
// 4.8e-4 and the SFU adds at most 2.5e-4 |u|, about the error of the
// Abramowitz & Stegun erfc form this replaced (6.9e-4 at most), at six fp32
// instructions and one SFU op per element instead of eleven and one.
__device__ __forceinline__ float gelu_bf16out(float u) {
  const float a = 0.7978845608028654f * fmaf(0.044715f * u, u * u, u);
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(a));
  const float h = 0.5f * u;
  return fmaf(h, t, h);
}

// SiLU for bf16-output epilogues: fast exp and division (relative error ~1e-7).
__device__ __forceinline__ float silu_bf16out(float u) { return __fdividef(u, 1.0f + __expf(-u)); }

// Exclusive prefix sum of n <= 32 * CHUNKS values by one warp (all 32 lanes
// call it): out[i] = value(0) + ... + value(i - 1) for i <= n, so out[n] is
// the total, which every lane returns.  All values are fetched before the
// scan, so reading them from global memory costs about one memory latency
// instead of n dependent ones.  copy (optional, global) receives out[0..n].
template <int CHUNKS, typename F>
__device__ __forceinline__ int warp_exclusive_scan(int n, int lane, F value, int* out, int* copy = nullptr) {
  int v[CHUNKS];
#pragma unroll
  for (int c = 0; c < CHUNKS; ++c) v[c] = c * 32 + lane < n ? value(c * 32 + lane) : 0;
  int carry = 0;
#pragma unroll
  for (int c = 0; c < CHUNKS; ++c) {
    if (c * 32 >= n) break;  // uniform
    int x = v[c];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    const int i = c * 32 + lane;
    if (i < n) {
      out[i] = carry + x - v[c];
      if (copy) copy[i] = carry + x - v[c];
    }
    carry += __shfl_sync(0xffffffffu, x, 31);
  }
  if (lane == 0) {
    out[n] = carry;
    if (copy) copy[n] = carry;
  }
  return carry;
}

}  // namespace ec2moe
