// Internal declarations shared by the translation units of libe2s.so.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/e2s.h"

namespace e2s {

// Workspace layout: [0, 256) status word, attention item counter and
// finished-CTA count (words 1 and 2), reserved; then one float4 of
// normalisation statistics per (image, layer, head) -- (S, M, 1/E, 1/S) with
// S = sum of a, M = max of a*log2e, E = sum of 2^(a*log2e - M) over the image's
// visual tokens (stats_entry), written by the score kernels; then the decision scratch of e2s_decide: per image 64
// cell arg-max keys (uint64), then one arrival counter per image (uint32).
// The score kernels zero the decision scratch when they are given it.
constexpr size_t kStatusBytes = 256;
constexpr int kDecideCells = 64;                          // G <= 8
constexpr int kDecideWordsPerImage = 2 * kDecideCells + 1;  // uint32 words to zero
inline size_t stats_bytes(const e2s_layout* L) {
  size_t n = (size_t)L->B * (size_t)L->L * (size_t)L->H * 4 * sizeof(float);
  return (n + 255) & ~(size_t)255;
}
inline size_t decide_scratch_bytes(const e2s_layout* L) {
  return ((size_t)L->B * kDecideWordsPerImage * sizeof(uint32_t) + 255) & ~(size_t)255;
}
inline uint32_t* status_word(void* ws) { return reinterpret_cast<uint32_t*>(ws); }
// Words 1 and 2 of the status area: the attention kernel's shared item counter
// and its count of finished CTAs (zero between calls).
inline uint32_t* attn_sched_ptr(void* ws) { return reinterpret_cast<uint32_t*>(ws) + 1; }
// Words 3 and 4: the streaming score kernel's shared unit counter and its
// count of finished CTAs (zero between calls); status is word 0.
inline uint32_t* stream_sched_ptr(uint32_t* status) { return status + 3; }
constexpr size_t kClearBytes = 32;   // bytes of the status area zeroed before first use
inline float4* stats_ptr(void* ws) {
  return reinterpret_cast<float4*>(reinterpret_cast<char*>(ws) + kStatusBytes);
}
// Start of the decision scratch: B * 64 cell keys, then B counters.
inline uint32_t* decide_scratch_ptr(void* ws, const e2s_layout* L) {
  return reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(ws) + kStatusBytes + stats_bytes(L));
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
// The score kernels also write the per-(image, layer, head) statistics into
// `stats` and zero B * kDecideWordsPerImage words of decision scratch at
// `counters` (nullable).
cudaError_t launch_score_tc(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                            const void* k, int64_t k_stride, float* a_out, float4* stats,
                            uint32_t* counters, uint32_t* status, cudaStream_t st,
                            int* unsupported, bool pdl = false);
// Streaming score kernel (long sequences, GQA; at most 128 text rows).  With
// lse_in (natural-log lse of every text row, [L][H][sum_text]) it skips the
// normaliser sweep and streams only the visual key tiles.
bool score_stream_fits(const LayoutArgs& la);
cudaError_t launch_score_stream(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                                const void* k, int64_t k_stride, float* a_out, float4* stats,
                                uint32_t* counters, uint32_t* status, cudaStream_t st,
                                const float* lse_in = nullptr, bool pdl = false);
// Cluster-per-unit score kernel for small batches (key tiles split over the
// cluster's CTAs): its cluster size and tiles per CTA, or false when it does
// not take the launch.  lse_in as for launch_score_stream.
bool score_split_plan(const LayoutArgs& la, int mode, bool lse, int* cluster, int* tpc);
cudaError_t launch_score_split(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                               const void* k, int64_t k_stride, float* a_out, float4* stats,
                               uint32_t* counters, uint32_t* status, cudaStream_t st,
                               const float* lse_in, int cluster, int tpc, bool pdl = false);
// The pruning layer's causal attention (O and the row lse) with the text rows'
// score a and its Eq. 8 statistics as a by-product when a_out is given.
// sched: two workspace words, zero on entry and on return (the item counter
// the CTAs share).
cudaError_t launch_attention(const LayoutArgs& la, const void* q, int64_t q_stride, const void* k,
                             int64_t k_stride, const void* v, int64_t v_stride, void* o_out,
                             int64_t o_stride, float* lse_out, float* a_out, float4* stats,
                             uint32_t* counters, uint32_t* sched, uint32_t* status,
                             cudaStream_t st);
// Persistent single-CTA-per-unit score kernel and its applicability tests.
bool score_unit_fits(const LayoutArgs& la, int mode);
bool score_unit_single_group(const LayoutArgs& la, int mode);
cudaError_t launch_score_unit(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                              const void* k, int64_t k_stride, float* a_out, float4* stats,
                              uint32_t* counters, uint32_t* status, cudaStream_t st,
                              bool pdl = false);
cudaError_t launch_score_simt(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                              const void* k, int64_t k_stride, float* a_out, float4* stats,
                              uint32_t* counters, uint32_t* status, cudaStream_t st);
cudaError_t launch_fuse(const LayoutArgs& la, int norm_softmax, uint32_t flags, const float* a,
                        const float* prior, float* mass_out, float* fused_out, float* q_out,
                        float2* stats, uint32_t* status, cudaStream_t st);
// One cluster per image: evidence, fusion and (do_select) the Top-K, no scratch.
cudaError_t launch_evidence(const LayoutArgs& la, int norm_softmax, uint32_t flags, float lambda,
                            int G, const float* a, const float* prior, const int32_t* cand,
                            float* mass_out, float* fused_out, float* q_out, float* q_tilde,
                            const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                            int32_t* keep_idx, int do_select, uint32_t* status, cudaStream_t st,
                            int* unsupported);
// Token-parallel evidence, fusion and select, reading the statistics the score
// kernel left in the workspace; the last CTA of every image runs the select.
bool decide_fits(const LayoutArgs& la);
cudaError_t launch_decide(const LayoutArgs& la, int norm_softmax, uint32_t flags, float lambda,
                          int G, const float* a, const float4* stats, const float* prior,
                          const int32_t* cand, float* mass_out, float* fused_out, float* q_out,
                          float* q_tilde, const int32_t* keep_count, const int32_t* keep_off,
                          int32_t sum_keep, int32_t* keep_idx, uint32_t* scratch,
                          uint32_t* status, cudaStream_t st, int* unsupported);
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
// early: copy the selection-independent rows before waiting on the previous
// kernel (only when the sources were complete before that kernel's
// predecessor started, as in e2s_prune).
cudaError_t launch_compact(const LayoutArgs& la, const int32_t* keep_idx, const int32_t* keep_off,
                           int32_t sum_keep, int32_t n_tensors, const void* const* src,
                           void* const* dst, const int64_t* row_bytes, int32_t* pos_ids,
                           uint32_t* status, cudaStream_t st, int early);

// Number of SMs of the current device (cached per call by the runtime).
int sm_count();

// Launch with the attributes the kernels of this library use: an optional
// thread-block cluster, and programmatic dependent launch (pdl) -- the kernel
// may be scheduled while the previous kernel on the stream is still running
// and must execute griddepcontrol.wait before it reads that kernel's outputs.
// Every kernel prefers the maximum shared-memory carve-out, so consecutive
// kernels of a decision never reconfigure the L1 / shared-memory split.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t st, int cluster, bool pdl, Args&&... args) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  if (cluster > 8) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (cluster > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = (unsigned)cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

}  // namespace e2s
