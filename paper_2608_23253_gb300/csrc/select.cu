// Standalone spatial novelty + Top-K (Sec. 4.3, Eqs. 20-23): one CTA per
// image runs select_image over the image's priorities.
#include <cuda_runtime.h>

#include <algorithm>

#include "select_core.cuh"

namespace e2s {
namespace {

constexpr int kSelThreads = 1024;

__global__ void __launch_bounds__(kSelThreads)
    select_kernel(const LayoutArgs la, float lambda, int G, uint32_t flags,
                  const float* __restrict__ q, const int32_t* __restrict__ cand,
                  const int32_t* __restrict__ keep_count, const int32_t* __restrict__ keep_off,
                  int32_t sum_keep, int32_t* __restrict__ keep_idx, float* __restrict__ q_tilde,
                  uint32_t* status) {
  extern __shared__ uint32_t keys[];  // [max_vis] keys, then [max_vis] cell ids
  __shared__ SelectSmem ss;
  pdl_launch_dependents();
  pdl_wait();   // q comes from the previous kernel
  const int b = blockIdx.x;
  if (!select_args_ok(la, b, cand != nullptr, keep_count, keep_off, sum_keep)) {
    if (threadIdx.x == 0) E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
    return;
  }
  const int v0 = __ldg(la.vis_off + b);
  const float lam = (flags & (E2S_NO_NOVELTY | E2S_VANILLA)) ? 0.f : lambda;
  select_image(q + v0, cand ? cand + v0 : nullptr, __ldg(la.n_vis + b), __ldg(la.grid_h + b),
               __ldg(la.grid_w + b), G, lam, __ldg(keep_count + b), keys,
               reinterpret_cast<uint8_t*>(keys + la.max_vis), ss,
               q_tilde ? q_tilde + v0 : nullptr, keep_idx + __ldg(keep_off + b), status);
}

}  // namespace

cudaError_t launch_select(const LayoutArgs& la, float lambda, int G, uint32_t flags,
                          const float* q, const int32_t* cand, const int32_t* keep_count,
                          const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                          float* q_tilde, uint32_t* status, cudaStream_t st) {
  const size_t smem = (size_t)std::max(la.max_vis, 1) * 5;
  return launch_kernel(select_kernel, dim3(la.B), dim3(kSelThreads), smem, st, 0, true, la, lambda,
                       G, flags, q, cand, keep_count, keep_off, sum_keep, keep_idx, q_tilde,
                       status);
}

}  // namespace e2s
