// Plain SIMT text-to-visual score (Sec. 3.1 Eq. 1 and the causal-prefix
// probability reading).  One CTA per (image, layer, query head); fp32 FMA
// dot products.  Selected with E2S_SIMT_SCORE; it exists to cross-check the
// tensor-core kernel on the GPU with an independent, simple formulation.
#include <cuda_runtime.h>

#include "device_common.cuh"

namespace e2s {
namespace {

constexpr int kSimtThreads = 256;

__device__ __forceinline__ float dot_row(const float* __restrict__ qrow,
                                         const uint16_t* __restrict__ krow) {
  const uint4* k4 = reinterpret_cast<const uint4*>(krow);
  float acc = 0.f;
#pragma unroll 4
  for (int i = 0; i < 16; ++i) {
    const uint4 w = __ldg(k4 + i);
    const float* qq = qrow + 8 * i;
    acc = fmaf(qq[0], bf16_lo(w.x), acc);
    acc = fmaf(qq[1], bf16_hi(w.x), acc);
    acc = fmaf(qq[2], bf16_lo(w.y), acc);
    acc = fmaf(qq[3], bf16_hi(w.y), acc);
    acc = fmaf(qq[4], bf16_lo(w.z), acc);
    acc = fmaf(qq[5], bf16_hi(w.z), acc);
    acc = fmaf(qq[6], bf16_lo(w.w), acc);
    acc = fmaf(qq[7], bf16_hi(w.w), acc);
  }
  return acc;
}

__global__ void __launch_bounds__(kSimtThreads)
    score_simt_kernel(const LayoutArgs la, int mode, const uint16_t* __restrict__ q,
                      int64_t q_stride, const uint16_t* __restrict__ k, int64_t k_stride,
                      float* __restrict__ a_out, float4* __restrict__ stats,
                      uint32_t* counters, uint32_t* status) {
  extern __shared__ float sm[];
  float* Qs = sm;                               // [max_text][128]
  float* lse = Qs + (size_t)la.max_text * 128;  // [max_text]
  float* red = lse + la.max_text;               // [64]

  pdl_launch_dependents();
  if (counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      counters[i] = 0u;
  const int unit = blockIdx.x;
  const int h = unit % la.H;
  const int l = (unit / la.H) % la.L;
  const int b = unit / (la.H * la.L);
  const int kvh = h / (la.H / la.H_kv);
  const int S = __ldg(la.n_sys + b), NV = __ldg(la.n_vis + b), NT = __ldg(la.n_text + b);
  const int t0 = __ldg(la.tok_off + b), x0 = __ldg(la.text_off + b), v0 = __ldg(la.vis_off + b);
  const int T = S + NV + NT;
  const bool ok = S >= 0 && NV >= 0 && NT >= 1 && NT <= la.max_text && T <= la.max_T &&
                  __ldg(la.tok_off + b + 1) - t0 == T && t0 >= 0 && t0 + T <= la.sum_T &&
                  __ldg(la.text_off + b + 1) - x0 == NT && x0 >= 0 && x0 + NT <= la.sum_text &&
                  __ldg(la.vis_off + b + 1) - v0 == NV && v0 >= 0 && v0 + NV <= la.sum_vis;
  if (!ok) {
    if (threadIdx.x == 0) E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
    return;
  }
  const float scale = rsqrtf(128.f);
  const float scale_log2 = 1.4426950408889634f * scale;

  for (int i = threadIdx.x; i < NT * 128; i += blockDim.x) {
    const int t = i >> 7, c = i & 127;
    Qs[i] = __uint_as_float((uint32_t)__ldg(q + ((size_t)l * la.sum_text + x0 + t) * q_stride +
                                              (size_t)h * 128 + c)
                            << 16);
  }
  __syncthreads();
  const uint16_t* kb = k + ((size_t)l * la.sum_T + t0) * k_stride + (size_t)kvh * 128;

  if (mode == E2S_SCORE_CAUSAL_PROB) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int t = 0; t < NT; ++t) {
      const int last = S + NV + t;
      float m = kNegBig, s = 0.f;
      for (int j = threadIdx.x; j <= last; j += blockDim.x)
        lse_merge(m, s, dot_row(Qs + t * 128, kb + (size_t)j * k_stride) * scale_log2, 1.f);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
      }
      if (lane == 0) {
        red[2 * warp] = m;
        red[2 * warp + 1] = s;
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        float M = red[0], Ls = red[1];
        for (int w = 1; w < nw; ++w) lse_merge(M, Ls, red[2 * w], red[2 * w + 1]);
        lse[t] = M + log2f(Ls);
      }
      __syncthreads();
    }
  }
  const float inv_nt = 1.f / (float)NT;
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    const uint16_t* krow = kb + (size_t)(S + n) * k_stride;
    float acc = 0.f;
    for (int t = 0; t < NT; ++t) {
      const float x = dot_row(Qs + t * 128, krow);
      if (mode == E2S_SCORE_CAUSAL_PROB)
        acc += exp2f(fmaf(x, scale_log2, -lse[t]));
      else
        acc = fmaf(x, scale, acc);
    }
    a_out[((size_t)l * la.H + h) * (size_t)la.sum_vis + v0 + n] = acc * inv_nt;
  }
  // statistics of this (layer, head)'s visual scores, in a fixed reduction order
  __syncthreads();
  const float* arow = a_out + ((size_t)l * la.H + h) * (size_t)la.sum_vis + v0;
  float ls = 0.f, lm = kNegBig;
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    ls += arow[n];
    lm = fmaxf(lm, arow[n] * 1.4426950408889634f);
  }
  const float S_ = block_reduce(ls, [](float x, float y) { return x + y; }, red);
  const float M_ = block_reduce(lm, [](float x, float y) { return fmaxf(x, y); }, red);
  float le = 0.f;
  for (int n = threadIdx.x; n < NV; n += blockDim.x)
    le += fast_ex2(fmaf(arow[n], 1.4426950408889634f, -M_));
  const float E_ = block_reduce(le, [](float x, float y) { return x + y; }, red);
  if (threadIdx.x == 0) stats[((size_t)b * la.L + l) * la.H + h] = stats_entry(S_, M_, E_);
}

}  // namespace

cudaError_t launch_score_simt(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                              const void* k, int64_t k_stride, float* a_out, float4* stats,
                              uint32_t* counters, uint32_t* status, cudaStream_t st) {
  const size_t smem = ((size_t)la.max_text * 129 + 64) * sizeof(float);
  const unsigned grid = (unsigned)((size_t)la.B * la.L * la.H);
  return launch_kernel(score_simt_kernel, dim3(grid), dim3(kSimtThreads), smem, st, 0, false, la,
                       mode, static_cast<const uint16_t*>(q), q_stride,
                       static_cast<const uint16_t*>(k), k_stride, a_out, stats, counters,
                       status);
}

}  // namespace e2s
