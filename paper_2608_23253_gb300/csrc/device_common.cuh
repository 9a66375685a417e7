// Device helpers shared by the kernels of libe2s.so.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace e2s {

constexpr float kNegBig = -1.0e30f;   // finite "minus infinity" for (max, sum) merges

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Hardware base-2 exponential (MUFU ex2, flush-to-zero; max relative error
// about 2^-22) and reciprocal.
__device__ __forceinline__ float fast_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float fast_rcp(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Merge two online-softmax partials (m, l) in the log2 domain:
// l * 2^m + l2 * 2^m2 = l' * 2^max(m, m2).  One exp2 per merge.
__device__ __forceinline__ void lse_merge(float& m, float& l, float m2, float l2) {
  const float mx = fmaxf(m, m2);
  const float e = fast_ex2(fminf(m, m2) - mx);
  l = (m >= m2) ? fmaf(l2, e, l) : fmaf(l, e, l2);
  m = mx;
}

// Order-preserving map of a float to uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t ordered_key(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Workspace entry of the Eq. 8 normalisation statistics of one (image, layer,
// head) row of visual scores, from S = sum a, M = max a*log2e and
// E = sum 2^(a*log2e - M): (S, M, 1/E, 1/S), a reciprocal 0 when its sum is not
// positive.
__device__ __forceinline__ float4 stats_entry(float S, float M, float E) {
  return make_float4(S, M, E > 0.f ? 1.f / E : 0.f, S > 0.f ? 1.f / S : 0.f);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch: let the next kernel on the stream be
// scheduled now / wait until the previous kernel's writes are visible.
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Block-wide reductions for blockDim.x a multiple of 32 (<= 1024).
template <typename F>
__device__ __forceinline__ float warp_reduce(float v, F op) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

template <typename F>
__device__ float block_reduce(float v, F op, float* red /* >= 32 floats */) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  v = warp_reduce(v, op);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float r = red[0];
  for (int i = 1; i < nw; ++i) r = op(r, red[i]);
  return r;
}

// Upper-bound search: largest b in [0, B) with off[b] <= x (off ascending, off[0] = 0).
__device__ __forceinline__ int find_segment(const int32_t* off, int B, int x) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(off + mid) <= x) lo = mid; else hi = mid - 1;
  }
  return lo;
}

}  // namespace e2s
