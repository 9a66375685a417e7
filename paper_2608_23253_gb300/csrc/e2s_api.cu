// C ABI of libe2s.so: argument validation and dispatch to the kernels.
// Validation here is host-side only (sizes, pointers, alignment, enums);
// the kernels re-check the device layout arrays and report through the
// status word in the workspace.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.h"

namespace e2s {

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
  return n > 0 ? n : 1;
}

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

e2s_status check_layout(const e2s_layout* L) {
  if (!L) return E2S_ERR_INVALID_ARG;
  if (L->B < 1 || L->L < 1 || L->H < 1 || L->H_kv < 1) return E2S_ERR_SHAPE;
  if (L->H % L->H_kv) return E2S_ERR_SHAPE;
  if (L->d != 128) return E2S_ERR_UNSUPPORTED;
  if (!L->tok_off || !L->n_sys || !L->n_vis || !L->n_text || !L->grid_h || !L->grid_w ||
      !L->vis_off || !L->text_off)
    return E2S_ERR_INVALID_ARG;
  if (L->max_T < 0 || L->max_vis < 0 || L->max_text < 1 || L->sum_T < 0 || L->sum_vis < 0 ||
      L->sum_text < L->B)
    return E2S_ERR_SHAPE;
  if (L->max_vis > L->max_T || L->max_text > L->max_T || L->sum_vis > L->sum_T ||
      L->sum_text > L->sum_T || L->max_T > L->sum_T)
    return E2S_ERR_SHAPE;
  if (L->max_vis > 8192) return E2S_ERR_UNSUPPORTED;
  if (L->max_text > 256) return E2S_ERR_UNSUPPORTED;
  return E2S_OK;
}

e2s_status check_params(const e2s_params* P) {
  if (!P) return E2S_ERR_INVALID_ARG;
  if (P->score_mode != E2S_SCORE_EQ1 && P->score_mode != E2S_SCORE_CAUSAL_PROB)
    return E2S_ERR_INVALID_ARG;
  if (P->norm_mode < E2S_NORM_DEFAULT || P->norm_mode > E2S_NORM_RENORM) return E2S_ERR_INVALID_ARG;
  if (P->score_mode == E2S_SCORE_EQ1 && P->norm_mode == E2S_NORM_RENORM) return E2S_ERR_UNSUPPORTED;
  if (P->G < 1 || P->G > 8) return E2S_ERR_INVALID_ARG;
  if (!(P->lambda >= 0.f && P->lambda <= 1.f)) return E2S_ERR_INVALID_ARG;
  const uint32_t known = E2S_NO_RELIABILITY | E2S_NO_LAYER_FUSION | E2S_NO_CONFLICT |
                         E2S_NO_NOVELTY | E2S_VANILLA | E2S_SIMT_SCORE;
  if (P->flags & ~known) return E2S_ERR_INVALID_ARG;
  return E2S_OK;
}

int norm_is_softmax(const e2s_params* P) {
  if (P->norm_mode == E2S_NORM_SOFTMAX) return 1;
  if (P->norm_mode == E2S_NORM_RENORM) return 0;
  return P->score_mode == E2S_SCORE_EQ1 ? 1 : 0;
}

e2s_status check_ws(const e2s_layout* L, void* ws, size_t ws_bytes) {
  if (!ws) return E2S_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return E2S_ERR_WORKSPACE;
  if (ws_bytes < kStatusBytes + stats_bytes(L) + decide_scratch_bytes(L)) return E2S_ERR_WORKSPACE;
  return E2S_OK;
}

e2s_status from_cuda(cudaError_t e) { return e == cudaSuccess ? E2S_OK : E2S_ERR_CUDA; }

#define E2S_TRY(x)                    \
  do {                                \
    const e2s_status s_ = (x);        \
    if (s_ != E2S_OK) return s_;      \
  } while (0)

e2s_status check_score_args(const e2s_layout* layout, const void* q_text, int64_t q_row_stride,
                            const void* k, int64_t k_row_stride, const float* a_out) {
  if (!q_text || !k || (!a_out && layout->sum_vis > 0)) return E2S_ERR_INVALID_ARG;
  if (q_row_stride < (int64_t)layout->H * layout->d ||
      k_row_stride < (int64_t)layout->H_kv * layout->d)
    return E2S_ERR_SHAPE;
  if (!aligned16(q_text) || !aligned16(k) || (q_row_stride % 8) || (k_row_stride % 8))
    return E2S_ERR_ALIGNMENT;
  return E2S_OK;
}

// Score launch shared by e2s_score and e2s_decide; the decision scratch it
// zeroes may be null.  With lse_text (the *_lse entry points) only a single
// pass over the visual key tiles runs, in the streaming kernel (at batch 1 it
// measured 14.8 us against 16.8 us for the cluster-per-unit kernel, and the
// whole step 27.2 against 29.7 us).
e2s_status run_score(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                     int64_t q_row_stride, const void* k, int64_t k_row_stride, float* a_out,
                     void* ws, uint32_t* counters, cudaStream_t st,
                     const float* lse_text = nullptr, bool pdl = false) {
  const LayoutArgs la = layout_args(layout);
  if (lse_text)
    return from_cuda(launch_score_stream(la, params->score_mode, q_text, q_row_stride, k,
                                         k_row_stride, a_out, stats_ptr(ws), counters,
                                         status_word(ws), st, lse_text, pdl));
  if (params->flags & E2S_SIMT_SCORE)
    return from_cuda(launch_score_simt(la, params->score_mode, q_text, q_row_stride, k,
                                       k_row_stride, a_out, stats_ptr(ws), counters,
                                       status_word(ws), st));
  int unsupported = 0;
  const cudaError_t e =
      launch_score_tc(la, params->score_mode, q_text, q_row_stride, k, k_row_stride, a_out,
                      stats_ptr(ws), counters, status_word(ws), st, &unsupported, pdl);
  if (unsupported) return E2S_ERR_UNSUPPORTED;
  return from_cuda(e);
}

e2s_status check_decide_args(const e2s_layout* layout, const e2s_params* params,
                             const void* q_text, int64_t q_row_stride, const void* k,
                             int64_t k_row_stride, const float* prior, const float* a_out,
                             const float* mass_out, const float* fused_out, const float* q_out,
                             const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                             const int32_t* keep_idx, void* ws, size_t ws_bytes) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  E2S_TRY(check_score_args(layout, q_text, q_row_stride, k, k_row_stride, a_out));
  if (layout->sum_vis > 0 && (!fused_out || !q_out)) return E2S_ERR_INVALID_ARG;
  if (!keep_count || !keep_off || sum_keep < 0) return E2S_ERR_INVALID_ARG;
  if (sum_keep > 0 && !keep_idx) return E2S_ERR_INVALID_ARG;
  if (!aligned16(prior) || !aligned16(mass_out) || !aligned16(fused_out)) return E2S_ERR_ALIGNMENT;
  if (!decide_fits(layout_args(layout))) return E2S_ERR_UNSUPPORTED;
  return E2S_OK;
}

// Score (zeroing the arrival counters), then the token-parallel decision.
e2s_status run_decide(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                      int64_t q_row_stride, const void* k, int64_t k_row_stride,
                      const int32_t* cand, const float* prior, float* a_out, float* mass_out,
                      float* fused_out, float* q_out, const int32_t* keep_count,
                      const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                      float* q_tilde_out, void* ws, cudaStream_t st,
                      const float* lse_text = nullptr, bool pdl_first = false) {
  uint32_t* scratch = decide_scratch_ptr(ws, layout);
  E2S_TRY(run_score(layout, params, q_text, q_row_stride, k, k_row_stride, a_out, ws, scratch,
                    st, lse_text, pdl_first));
  int unsupported = 0;
  const cudaError_t e =
      launch_decide(layout_args(layout), norm_is_softmax(params), params->flags, params->lambda,
                    params->G, a_out, stats_ptr(ws), prior, cand, mass_out, fused_out, q_out,
                    q_tilde_out, keep_count, keep_off, sum_keep, keep_idx, scratch,
                    status_word(ws), st, &unsupported);
  if (unsupported) return E2S_ERR_UNSUPPORTED;
  return from_cuda(e);
}

// The text rows' lse given: causal-probability scores on the streaming kernel.
e2s_status check_lse_args(const e2s_layout* layout, const e2s_params* params,
                          const float* lse_text) {
  if (!lse_text) return E2S_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(lse_text) & 3u) != 0) return E2S_ERR_ALIGNMENT;
  if (params->score_mode != E2S_SCORE_CAUSAL_PROB || (params->flags & E2S_SIMT_SCORE))
    return E2S_ERR_UNSUPPORTED;
  if (!score_stream_fits(layout_args(layout))) return E2S_ERR_UNSUPPORTED;
  return E2S_OK;
}

e2s_status check_compact_args(const e2s_layout* layout, const int32_t* keep_idx,
                              const int32_t* keep_off, int32_t sum_keep, int32_t n_tensors,
                              const void* const* src, void* const* dst,
                              const int64_t* row_bytes) {
  if (!keep_off || sum_keep < 0 || sum_keep > layout->sum_vis) return E2S_ERR_SHAPE;
  if (sum_keep > 0 && !keep_idx) return E2S_ERR_INVALID_ARG;
  if (n_tensors < 0 || n_tensors > kMaxCompactTensors) return E2S_ERR_INVALID_ARG;
  if (n_tensors > 0 && (!src || !dst || !row_bytes)) return E2S_ERR_INVALID_ARG;
  for (int i = 0; i < n_tensors; ++i) {
    if (!src[i] || !dst[i]) return E2S_ERR_INVALID_ARG;
    if (row_bytes[i] <= 0) return E2S_ERR_SHAPE;
    if ((row_bytes[i] & 15) || !aligned16(src[i]) || !aligned16(dst[i])) return E2S_ERR_ALIGNMENT;
  }
  return E2S_OK;
}

// e2s_prune / e2s_prune_lse (lse_text nullable here).
e2s_status prune_impl(const e2s_layout* layout, const e2s_params* params,
                      const void* q_text, int64_t q_row_stride, const void* k,
                      int64_t k_row_stride, const float* lse_text, const int32_t* cand,
                      const float* prior, float* a_out, float* mass_out, float* fused_out,
                      float* q_out, const int32_t* keep_count, const int32_t* keep_off,
                      int32_t sum_keep, int32_t* keep_idx, float* q_tilde_out,
                      int32_t n_tensors, const void* const* src, void* const* dst,
                      const int64_t* row_bytes, int32_t* pos_ids_out, void* ws,
                      size_t ws_bytes, void* stream) {
  E2S_TRY(check_decide_args(layout, params, q_text, q_row_stride, k, k_row_stride, prior, a_out,
                            mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                            ws, ws_bytes));
  E2S_TRY(check_compact_args(layout, keep_idx, keep_off, sum_keep, n_tensors, src, dst,
                             row_bytes));
  if (lse_text != nullptr) E2S_TRY(check_lse_args(layout, params, lse_text));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the step's first kernel waits on the kernel before it programmatically
  // (the compaction of a previous step signals its dependents as it ends), so
  // that its launch overlaps that kernel's tail: 24.7 -> 23.5 us per step of
  // back-to-back LLaVA batch-1 steps.  The standalone calls keep plain launches:
  // a score behind a kernel that signals early would hold SMs while it runs.
  E2S_TRY(run_decide(layout, params, q_text, q_row_stride, k, k_row_stride, cand, prior, a_out,
                     mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                     q_tilde_out, ws, st, lse_text, true));
  if (n_tensors == 0 && !pos_ids_out) return E2S_OK;
  // the score kernel signals its dependents only after its own wait on the
  // kernel before it, so the sources are complete before the compaction (which
  // copies the system and text rows before its wait) may start
  return from_cuda(launch_compact(layout_args(layout), keep_idx, keep_off, sum_keep, n_tensors,
                                  src, dst, row_bytes, pos_ids_out, status_word(ws), st, 1));
}

}  // namespace
}  // namespace e2s

using namespace e2s;

extern "C" {

size_t e2s_workspace_size(const e2s_layout* layout, const e2s_params* params) {
  (void)params;
  if (check_layout(layout) != E2S_OK) return 0;
  return kStatusBytes + stats_bytes(layout) + decide_scratch_bytes(layout);
}

e2s_status e2s_score(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                     int64_t q_row_stride, const void* k, int64_t k_row_stride, float* a_out,
                     void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  E2S_TRY(check_score_args(layout, q_text, q_row_stride, k, k_row_stride, a_out));
  return run_score(layout, params, q_text, q_row_stride, k, k_row_stride, a_out, ws, nullptr,
                   static_cast<cudaStream_t>(stream));
}

e2s_status e2s_score_lse(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                         int64_t q_row_stride, const void* k, int64_t k_row_stride,
                         const float* lse_text, float* a_out, void* ws, size_t ws_bytes,
                         void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  E2S_TRY(check_score_args(layout, q_text, q_row_stride, k, k_row_stride, a_out));
  E2S_TRY(check_lse_args(layout, params, lse_text));
  return run_score(layout, params, q_text, q_row_stride, k, k_row_stride, a_out, ws, nullptr,
                   static_cast<cudaStream_t>(stream), lse_text);
}

e2s_status e2s_attention(const e2s_layout* layout, const void* q, int64_t q_row_stride,
                         const void* k, int64_t k_row_stride, const void* v,
                         int64_t v_row_stride, void* o_out, int64_t o_row_stride, float* lse_out,
                         float* a_out, void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  if (!q || !k || !v || !o_out) return E2S_ERR_INVALID_ARG;
  const int64_t hd = (int64_t)layout->H * layout->d, kvd = (int64_t)layout->H_kv * layout->d;
  if (q_row_stride < hd || o_row_stride < hd || k_row_stride < kvd || v_row_stride < kvd)
    return E2S_ERR_SHAPE;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o_out) ||
      (q_row_stride % 8) || (k_row_stride % 8) || (v_row_stride % 8) || (o_row_stride % 8) ||
      (reinterpret_cast<uintptr_t>(lse_out) & 3u) || (reinterpret_cast<uintptr_t>(a_out) & 3u))
    return E2S_ERR_ALIGNMENT;
  if (a_out != nullptr && layout->max_text > 128) return E2S_ERR_UNSUPPORTED;
  return from_cuda(launch_attention(layout_args(layout), q, q_row_stride, k, k_row_stride, v,
                                    v_row_stride, o_out, o_row_stride, lse_out, a_out,
                                    stats_ptr(ws), a_out ? decide_scratch_ptr(ws, layout) : nullptr,
                                    attn_sched_ptr(ws), status_word(ws),
                                    static_cast<cudaStream_t>(stream)));
}

e2s_status e2s_decide_attn(const e2s_layout* layout, const e2s_params* params, const void* q,
                           int64_t q_row_stride, const void* k, int64_t k_row_stride,
                           const void* v, int64_t v_row_stride, void* o_out, int64_t o_row_stride,
                           float* lse_out, const int32_t* cand, const float* prior, float* a_out,
                           float* mass_out, float* fused_out, float* q_out,
                           const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                           int32_t* keep_idx, float* q_tilde_out, void* ws, size_t ws_bytes,
                           void* stream) {
  E2S_TRY(check_params(params));
  if (params->score_mode != E2S_SCORE_CAUSAL_PROB) return E2S_ERR_UNSUPPORTED;
  if (!a_out && layout && layout->sum_vis > 0) return E2S_ERR_INVALID_ARG;
  if (layout && layout->sum_vis > 0 && (!fused_out || !q_out)) return E2S_ERR_INVALID_ARG;
  if (!keep_count || !keep_off || sum_keep < 0) return E2S_ERR_INVALID_ARG;
  if (sum_keep > 0 && !keep_idx) return E2S_ERR_INVALID_ARG;
  if (!aligned16(prior) || !aligned16(mass_out) || !aligned16(fused_out)) return E2S_ERR_ALIGNMENT;
  E2S_TRY(e2s_attention(layout, q, q_row_stride, k, k_row_stride, v, v_row_stride, o_out,
                        o_row_stride, lse_out, a_out, ws, ws_bytes, stream));
  if (!decide_fits(layout_args(layout))) return E2S_ERR_UNSUPPORTED;
  int unsupported = 0;
  const cudaError_t e = launch_decide(
      layout_args(layout), norm_is_softmax(params), params->flags, params->lambda, params->G,
      a_out, stats_ptr(ws), prior, cand, mass_out, fused_out, q_out, q_tilde_out, keep_count,
      keep_off, sum_keep, keep_idx, decide_scratch_ptr(ws, layout), status_word(ws),
      static_cast<cudaStream_t>(stream), &unsupported);
  if (unsupported) return E2S_ERR_UNSUPPORTED;
  return from_cuda(e);
}

e2s_status e2s_decide_lse(const e2s_layout* layout, const e2s_params* params,
                          const void* q_text, int64_t q_row_stride, const void* k,
                          int64_t k_row_stride, const float* lse_text, const int32_t* cand,
                          const float* prior, float* a_out, float* mass_out, float* fused_out,
                          float* q_out, const int32_t* keep_count, const int32_t* keep_off,
                          int32_t sum_keep, int32_t* keep_idx, float* q_tilde_out, void* ws,
                          size_t ws_bytes, void* stream) {
  E2S_TRY(check_decide_args(layout, params, q_text, q_row_stride, k, k_row_stride, prior, a_out,
                            mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                            ws, ws_bytes));
  E2S_TRY(check_lse_args(layout, params, lse_text));
  return run_decide(layout, params, q_text, q_row_stride, k, k_row_stride, cand, prior, a_out,
                    mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                    q_tilde_out, ws, static_cast<cudaStream_t>(stream), lse_text);
}

e2s_status e2s_decide(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                      int64_t q_row_stride, const void* k, int64_t k_row_stride,
                      const int32_t* cand, const float* prior, float* a_out, float* mass_out,
                      float* fused_out, float* q_out, const int32_t* keep_count,
                      const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                      float* q_tilde_out, void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_decide_args(layout, params, q_text, q_row_stride, k, k_row_stride, prior, a_out,
                            mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                            ws, ws_bytes));
  return run_decide(layout, params, q_text, q_row_stride, k, k_row_stride, cand, prior, a_out,
                    mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                    q_tilde_out, ws, static_cast<cudaStream_t>(stream));
}

e2s_status e2s_prune(const e2s_layout* layout, const e2s_params* params, const void* q_text,
                     int64_t q_row_stride, const void* k, int64_t k_row_stride,
                     const int32_t* cand, const float* prior, float* a_out, float* mass_out,
                     float* fused_out, float* q_out, const int32_t* keep_count,
                     const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                     float* q_tilde_out, int32_t n_tensors, const void* const* src,
                     void* const* dst, const int64_t* row_bytes, int32_t* pos_ids_out, void* ws,
                     size_t ws_bytes, void* stream) {
  return prune_impl(layout, params, q_text, q_row_stride, k, k_row_stride, nullptr, cand, prior,
                    a_out, mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                    q_tilde_out, n_tensors, src, dst, row_bytes, pos_ids_out, ws, ws_bytes,
                    stream);
}

e2s_status e2s_prune_lse(const e2s_layout* layout, const e2s_params* params,
                         const void* q_text, int64_t q_row_stride, const void* k,
                         int64_t k_row_stride, const float* lse_text, const int32_t* cand,
                         const float* prior, float* a_out, float* mass_out, float* fused_out,
                         float* q_out, const int32_t* keep_count, const int32_t* keep_off,
                         int32_t sum_keep, int32_t* keep_idx, float* q_tilde_out,
                         int32_t n_tensors, const void* const* src, void* const* dst,
                         const int64_t* row_bytes, int32_t* pos_ids_out, void* ws,
                         size_t ws_bytes, void* stream) {
  if (!lse_text) return E2S_ERR_INVALID_ARG;
  return prune_impl(layout, params, q_text, q_row_stride, k, k_row_stride, lse_text, cand, prior,
                    a_out, mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                    q_tilde_out, n_tensors, src, dst, row_bytes, pos_ids_out, ws, ws_bytes,
                    stream);
}

e2s_status e2s_fuse(const e2s_layout* layout, const e2s_params* params, const float* a,
                    const int32_t* cand, const float* prior, float* mass_out, float* fused_out,
                    float* q_out, void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  if (layout->sum_vis > 0 && (!a || !fused_out || !q_out)) return E2S_ERR_INVALID_ARG;
  if (!aligned16(prior) || !aligned16(mass_out) || !aligned16(fused_out)) return E2S_ERR_ALIGNMENT;
  int unsupported = 0;
  const cudaError_t e = launch_evidence(layout_args(layout), norm_is_softmax(params),
                                        params->flags, params->lambda, params->G, a, prior, cand,
                                        mass_out, fused_out, q_out, nullptr, nullptr, nullptr, 0,
                                        nullptr, 0, status_word(ws),
                                        static_cast<cudaStream_t>(stream), &unsupported);
  if (unsupported) return E2S_ERR_UNSUPPORTED;
  return from_cuda(e);
}

e2s_status e2s_fuse_select(const e2s_layout* layout, const e2s_params* params, const float* a,
                           const int32_t* cand, const float* prior, float* mass_out,
                           float* fused_out, float* q_out, const int32_t* keep_count,
                           const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                           float* q_tilde_out, void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  if (layout->sum_vis > 0 && (!a || !fused_out || !q_out)) return E2S_ERR_INVALID_ARG;
  if (!keep_count || !keep_off || sum_keep < 0) return E2S_ERR_INVALID_ARG;
  if (sum_keep > 0 && !keep_idx) return E2S_ERR_INVALID_ARG;
  if (!aligned16(prior) || !aligned16(mass_out) || !aligned16(fused_out)) return E2S_ERR_ALIGNMENT;
  int unsupported = 0;
  const cudaError_t e = launch_evidence(layout_args(layout), norm_is_softmax(params),
                                        params->flags, params->lambda, params->G, a, prior, cand,
                                        mass_out, fused_out, q_out, q_tilde_out, keep_count,
                                        keep_off, sum_keep, keep_idx, 1, status_word(ws),
                                        static_cast<cudaStream_t>(stream), &unsupported);
  if (unsupported) return E2S_ERR_UNSUPPORTED;
  return from_cuda(e);
}

e2s_status e2s_fuse_noalloc(const e2s_layout* layout, const e2s_params* params, const float* a,
                            const int32_t* cand, const float* prior, float* mass_out,
                            float* fused_out, float* q_out, void* stream) {
  (void)cand;
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  if (layout->sum_vis > 0 && (!a || !fused_out || !q_out)) return E2S_ERR_INVALID_ARG;
  if (!aligned16(prior) || !aligned16(mass_out) || !aligned16(fused_out)) return E2S_ERR_ALIGNMENT;
  int too_big = 0;
  const cudaError_t e = launch_fuse_noalloc(layout_args(layout), norm_is_softmax(params),
                                            params->flags, a, prior, mass_out, fused_out, q_out,
                                            static_cast<cudaStream_t>(stream), &too_big);
  if (too_big) return E2S_ERR_WORKSPACE;
  return from_cuda(e);
}

e2s_status e2s_select(const e2s_layout* layout, const e2s_params* params, const float* q,
                      const int32_t* cand, const int32_t* keep_count, const int32_t* keep_off,
                      int32_t sum_keep, int32_t* keep_idx, float* q_tilde_out, void* ws,
                      size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_params(params));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  if (!keep_count || !keep_off || sum_keep < 0) return E2S_ERR_INVALID_ARG;
  if (layout->sum_vis > 0 && !q) return E2S_ERR_INVALID_ARG;
  if (sum_keep > 0 && !keep_idx) return E2S_ERR_INVALID_ARG;
  return from_cuda(launch_select(layout_args(layout), params->lambda, params->G, params->flags, q,
                                 cand, keep_count, keep_off, sum_keep, keep_idx, q_tilde_out,
                                 status_word(ws), static_cast<cudaStream_t>(stream)));
}

e2s_status e2s_compact(const e2s_layout* layout, const int32_t* keep_idx, const int32_t* keep_off,
                       int32_t sum_keep, int32_t n_tensors, const void* const* src,
                       void* const* dst, const int64_t* row_bytes, int32_t* pos_ids_out,
                       void* ws, size_t ws_bytes, void* stream) {
  E2S_TRY(check_layout(layout));
  E2S_TRY(check_ws(layout, ws, ws_bytes));
  E2S_TRY(check_compact_args(layout, keep_idx, keep_off, sum_keep, n_tensors, src, dst,
                             row_bytes));
  if (n_tensors == 0 && !pos_ids_out) return E2S_OK;
  return from_cuda(launch_compact(layout_args(layout), keep_idx, keep_off, sum_keep, n_tensors,
                                  src, dst, row_bytes, pos_ids_out, status_word(ws),
                                  static_cast<cudaStream_t>(stream), 0));
}

e2s_status e2s_read_status(const void* ws, void* stream) {
  if (!ws) return E2S_ERR_WORKSPACE;
  uint32_t word = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&word, ws, sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return E2S_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return E2S_ERR_CUDA;
  for (int c = 1; c < 32; ++c)
    if (word & (1u << c)) return static_cast<e2s_status>(c);
  return E2S_OK;
}

e2s_status e2s_clear_status(void* ws, void* stream) {
  if (!ws) return E2S_ERR_WORKSPACE;
  return from_cuda(cudaMemsetAsync(ws, 0, kClearBytes, static_cast<cudaStream_t>(stream)));
}

const char* e2s_status_string(e2s_status s) {
  switch (s) {
    case E2S_OK: return "E2S_OK";
    case E2S_ERR_INVALID_ARG: return "E2S_ERR_INVALID_ARG";
    case E2S_ERR_SHAPE: return "E2S_ERR_SHAPE";
    case E2S_ERR_ALIGNMENT: return "E2S_ERR_ALIGNMENT";
    case E2S_ERR_UNSUPPORTED: return "E2S_ERR_UNSUPPORTED";
    case E2S_ERR_WORKSPACE: return "E2S_ERR_WORKSPACE";
    case E2S_ERR_CUDA: return "E2S_ERR_CUDA";
    case E2S_ERR_TIMEOUT: return "E2S_ERR_TIMEOUT";
  }
  return "E2S_ERR_UNKNOWN";
}

int32_t e2s_version(void) { return 103; }

}  // extern "C"
