// Internal declarations shared by the translation units of libe2s.so.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/e2s.h"

namespace e2s {

// Workspace layout: [0, 256) status word + reserved; then per-(image, layer,
// head) normalisation statistics (float2).
constexpr size_t kStatusBytes = 256;
inline size_t stats_bytes(const e2s_layout* L) {
  size_t n = (size_t)L->B * (size_t)L->L * (size_t)L->H * 2 * sizeof(float);
  return (n + 255) & ~(size_t)255;
}
inline uint32_t* status_word(void* ws) { return reinterpret_cast<uint32_t*>(ws); }
inline float2* stats_ptr(void* ws) {
  return reinterpret_cast<float2*>(reinterpret_cast<char*>(ws) + kStatusBytes);
}

// Device-side error recording: bit `code` of the status word.
#define E2S_DEV_FLAG(status, code) atomicOr((status), 1u << (code))

// Resolved score settings shared by both score kernels.
struct LayoutArgs {
  const int32_t* tok_off;
  const int32_t* n_sys;
  const int32_t* n_vis;
  const int32_t* n_text;
  const int32_t* grid_h;
  const int32_t* grid_w;
  const int32_t* vis_off;
  const int32_t* text_off;
  int B, L, H, H_kv;
  int max_T, max_vis, max_text;
  int sum_T, sum_vis, sum_text;
};

inline LayoutArgs layout_args(const e2s_layout* l) {
  LayoutArgs a;
  a.tok_off = l->tok_off; a.n_sys = l->n_sys; a.n_vis = l->n_vis; a.n_text = l->n_text;
  a.grid_h = l->grid_h; a.grid_w = l->grid_w; a.vis_off = l->vis_off; a.text_off = l->text_off;
  a.B = l->B; a.L = l->L; a.H = l->H; a.H_kv = l->H_kv;
  a.max_T = l->max_T; a.max_vis = l->max_vis; a.max_text = l->max_text;
  a.sum_T = l->sum_T; a.sum_vis = l->sum_vis; a.sum_text = l->sum_text;
  return a;
}

// Launchers (return a CUDA error code; validation happened in the API layer).
cudaError_t launch_score_tc(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                            const void* k, int64_t k_stride, float* a_out, uint32_t* status,
                            cudaStream_t st, int* unsupported);
cudaError_t launch_score_simt(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                              const void* k, int64_t k_stride, float* a_out, uint32_t* status,
                              cudaStream_t st);
cudaError_t launch_fuse(const LayoutArgs& la, int norm_softmax, uint32_t flags, const float* a,
                        const float* prior, float* mass_out, float* fused_out, float* q_out,
                        float2* stats, uint32_t* status, cudaStream_t st);
// Same two kernels as launch_fuse, with the scratch in a static device array
// (no workspace).  *too_big is set when B * L * H exceeds its capacity.
cudaError_t launch_fuse_noalloc(const LayoutArgs& la, int norm_softmax, uint32_t flags,
                                const float* a, const float* prior, float* mass_out,
                                float* fused_out, float* q_out, cudaStream_t st, int* too_big);
cudaError_t launch_select(const LayoutArgs& la, float lambda, int G, uint32_t flags,
                          const float* q, const int32_t* cand, const int32_t* keep_count,
                          const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                          float* q_tilde, uint32_t* status, cudaStream_t st);

constexpr int kMaxCompactTensors = 32;
cudaError_t launch_compact(const LayoutArgs& la, const int32_t* keep_idx, const int32_t* keep_off,
                           int32_t sum_keep, int32_t n_tensors, const void* const* src,
                           void* const* dst, const int64_t* row_bytes, int32_t* pos_ids,
                           uint32_t* status, cudaStream_t st);

// Number of SMs of the current device (cached per call by the runtime).
int sm_count();

}  // namespace e2s
