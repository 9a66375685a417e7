// Compaction of the retained rows: system rows, the kept visual rows and the
// text rows of every image are gathered, in order, into the shortened
// sequence that the next decoder layer consumes.  One warp per (tensor,
// output row); 16-byte streaming loads and stores, fully coalesced; each
// CTA first stages every image's constants in shared memory.
#include <cuda_runtime.h>

#include <algorithm>

#include "device_common.cuh"
#include "sm100_ptx.cuh"

namespace e2s {
namespace {

constexpr int kCompactThreads = 256;
constexpr long long kPrefetchBytes = 48ll << 20;   // candidate rows prefetched into L2

struct TensorSet {
  const char* src[kMaxCompactTensors];
  char* dst[kMaxCompactTensors];
  int64_t row_bytes[kMaxCompactTensors];
};

// Largest b with out_off(b) <= r, out_off(b) = tok_off[b] - vis_off[b] + keep_off[b].
__device__ __forceinline__ int out_image(const LayoutArgs& la, const int32_t* keep_off, int r) {
  int lo = 0, hi = la.B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    const int off = __ldg(la.tok_off + mid) - __ldg(la.vis_off + mid) + __ldg(keep_off + mid);
    if (off <= r) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Per-image constants of the gather: the image's first output row, its
// system / visual / text counts, its keep list and its first input row.
struct ImgRows {
  int out0, S, NV, NT, ko, Kb, tok;
};
constexpr int kTabImages = 256;   // images whose constants a CTA stages in shared memory

__device__ __forceinline__ ImgRows img_rows(const LayoutArgs& la, const int32_t* keep_off, int b) {
  ImgRows t;
  t.S = __ldg(la.n_sys + b);
  t.NV = __ldg(la.n_vis + b);
  t.NT = __ldg(la.n_text + b);
  t.ko = __ldg(keep_off + b);
  t.Kb = __ldg(keep_off + b + 1) - t.ko;
  t.tok = __ldg(la.tok_off + b);
  t.out0 = t.tok - __ldg(la.vis_off + b) + t.ko;
  return t;
}

// Every image's constants into shared memory (whole block; la.B <= kTabImages).
__device__ __forceinline__ void stage_images(const LayoutArgs& la, const int32_t* keep_off,
                                             ImgRows* tab) {
  for (int b = threadIdx.x; b < la.B; b += blockDim.x) tab[b] = img_rows(la, keep_off, b);
  __syncthreads();
}

// One (tensor, output row) pair per warp, grid-stride.  visual < 0: every
// row; visual == 0: system and text rows only; visual == 1: kept visual rows
// only.  tab (nullable): the images' constants in shared memory, so that a
// pair's source row costs a shared-memory search instead of a chain of
// dependent global loads.
// RV: 16-byte vectors per lane in flight (RV * 512 bytes of a row per warp).
template <int RV>
__device__ __forceinline__ void compact_rows(const LayoutArgs& la, const int32_t* keep_idx,
                                             const int32_t* keep_off, int n_tensors,
                                             const TensorSet& ts, int32_t* pos_ids,
                                             long long total_rows, uint32_t* status, int visual,
                                             bool spread, const ImgRows* tab) {
  const int lane = threadIdx.x & 31;
  const long long warps = (long long)gridDim.x * (blockDim.x >> 5);
  // with no tensors the pass still writes the position ids
  const long long pairs = total_rows * (n_tensors > 0 ? n_tensors : 1);
  // spread: warp w of CTA c starts at pair w * gridDim.x + c, so consecutive
  // pairs (an image's kept rows are consecutive) land on different SMs -- for
  // kept rows already in L2, on the step's critical path; otherwise
  // neighbouring rows stay in one CTA (DRAM locality)
  const long long first = spread ? (long long)(threadIdx.x >> 5) * gridDim.x + blockIdx.x
                                 : ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const bool narrow = pairs < (1ll << 31);   // 32-bit pair arithmetic
  for (long long pr = first; pr < pairs; pr += warps) {
    const int tix = narrow ? (int)((uint32_t)pr / (uint32_t)total_rows) : (int)(pr / total_rows);
    const int r = (int)(pr - (long long)tix * total_rows);
    ImgRows t;
    if (tab != nullptr) {   // largest b with tab[b].out0 <= r
      int lo = 0, hi = la.B - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (tab[mid].out0 <= r) lo = mid; else hi = mid - 1;
      }
      t = tab[lo];
    } else {
      t = img_rows(la, keep_off, out_image(la, keep_off, r));
    }
    const int S = t.S, NV = t.NV, NT = t.NT, ko = t.ko, Kb = t.Kb, out0 = t.out0;
    const int u = r - out0;
    const bool is_vis = u >= S && u < S + Kb;
    if (visual >= 0 && is_vis != (visual == 1)) continue;
    int src_local;
    bool ok = Kb >= 0 && Kb <= NV && u >= 0 && u < S + Kb + NT;
    if (u < S) {
      src_local = u;
    } else if (is_vis) {
      const int kv = __ldg(keep_idx + ko + (u - S));
      ok = ok && kv >= 0 && kv < NV;
      src_local = S + kv;
    } else {
      src_local = NV + u - Kb;
    }
    if (!ok) {
      if (lane == 0) E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
      continue;
    }
    if (tix == 0 && lane == 0 && pos_ids) pos_ids[r] = src_local;
    if (n_tensors == 0) continue;
    const long long src_row = (long long)t.tok + src_local;
    const int64_t rb = ts.row_bytes[tix];
    const uint4* s4 = reinterpret_cast<const uint4*>(ts.src[tix] + src_row * rb);
    uint4* d4 = reinterpret_cast<uint4*>(ts.dst[tix] + (long long)r * rb);
    const int n16 = (int)(rb >> 4);
    // up to 8 KiB of the row in flight per warp: all loads first, then stores
    for (int base = 0; base < n16; base += 32 * RV) {
      uint4 x[RV];
#pragma unroll
      for (int v = 0; v < RV; ++v) {
        const int i = base + v * 32 + lane;
        if (i < n16) x[v] = __ldcs(s4 + i);
      }
#pragma unroll
      for (int v = 0; v < RV; ++v) {
        const int i = base + v * 32 + lane;
        if (i < n16) __stcs(d4 + i, x[v]);
      }
    }
  }
}

// L2 prefetch of every candidate visual row of every tensor (one bulk
// prefetch per row), so that the rows the selection keeps are L2 hits.
__device__ __forceinline__ void prefetch_visual_rows(const LayoutArgs& la, int n_tensors,
                                                     const TensorSet& ts) {
  const long long total = (long long)la.sum_vis * n_tensors;
  for (long long pr = (long long)blockIdx.x * blockDim.x + threadIdx.x; pr < total;
       pr += (long long)gridDim.x * blockDim.x) {
    const int tix = (int)(pr / la.sum_vis);
    const int gv = (int)(pr - (long long)tix * la.sum_vis);
    const int b = find_segment(la.vis_off, la.B, gv);
    const long long row = (long long)__ldg(la.tok_off + b) + __ldg(la.n_sys + b) +
                          (gv - __ldg(la.vis_off + b));
    if (row < 0 || row >= la.sum_T) continue;   // inconsistent layout: the copy flags it
    ptx::prefetch_l2_bulk(ts.src[tix] + row * ts.row_bytes[tix], (uint32_t)ts.row_bytes[tix]);
  }
}

// early != 0: the system and text rows (which do not depend on the selection)
// are copied before griddepcontrol.wait, overlapping the kernel that writes
// keep_idx; the caller guarantees that the sources and keep_off were complete
// before that kernel's predecessor started.  prefetch != 0 (with early): the
// candidate visual rows are also prefetched into L2 while waiting.
template <int RV>
__global__ void __launch_bounds__(kCompactThreads)
    compact_kernel(const LayoutArgs la, const int32_t* __restrict__ keep_idx,
                   const int32_t* __restrict__ keep_off, int n_tensors, const TensorSet ts,
                   int32_t* __restrict__ pos_ids, long long total_rows, uint32_t* status,
                   int early, int prefetch) {
  __shared__ ImgRows tab_s[kTabImages];
  const ImgRows* tab = la.B <= kTabImages ? tab_s : nullptr;
  if (early) {
    if (prefetch) prefetch_visual_rows(la, n_tensors, ts);
    if (tab) stage_images(la, keep_off, tab_s);
    compact_rows<RV>(la, keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, 0, false,
                 tab);
    pdl_wait();   // keep_idx comes from the previous kernel
    compact_rows<RV>(la, keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, 1,
                 prefetch != 0, tab);
  } else {
    pdl_wait();
    if (tab) stage_images(la, keep_off, tab_s);
    compact_rows<RV>(la, keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, -1, false,
                 tab);
  }
  // the next kernel may be scheduled once this one is finishing (signalled
  // earlier, its CTAs would hold SMs while the copies run)
  pdl_launch_dependents();
}

}  // namespace

cudaError_t launch_compact(const LayoutArgs& la, const int32_t* keep_idx, const int32_t* keep_off,
                           int32_t sum_keep, int32_t n_tensors, const void* const* src,
                           void* const* dst, const int64_t* row_bytes, int32_t* pos_ids,
                           uint32_t* status, cudaStream_t st, int early) {
  const long long total_rows = (long long)la.sum_T - la.sum_vis + sum_keep;
  if (total_rows <= 0) return cudaSuccess;
  TensorSet ts = {};
  for (int i = 0; i < n_tensors; ++i) {
    ts.src[i] = static_cast<const char*>(src[i]);
    ts.dst[i] = static_cast<char*>(dst[i]);
    ts.row_bytes[i] = row_bytes[i];
  }
  // prefetching every candidate row pays while those rows fit comfortably
  // in L2 (a single image or a small batch); larger batches are bandwidth-bound
  long long row_sum = 0;
  bool rows_small = true;
  for (int i = 0; i < n_tensors; ++i) {
    row_sum += row_bytes[i];
    rows_small = rows_small && row_bytes[i] <= (1ll << 20);
  }
  const int prefetch =
      early && rows_small && (long long)la.sum_vis * row_sum <= kPrefetchBytes ? 1 : 0;
  const long long pairs = total_rows * (n_tensors > 0 ? n_tensors : 1);
  const int warps_per_block = kCompactThreads / 32;
  long long blocks = (pairs + warps_per_block - 1) / warps_per_block;
  blocks = std::min<long long>(blocks, (long long)sm_count() * 16);
  const dim3 grid((unsigned)std::max<long long>(blocks, 1));
  // 16-byte vectors per lane in flight, measured per case: all 16 (8 KiB of a
  // row per warp) when a standalone call has only a few rows per warp slot;
  // 8 when the kept rows come out of L2 after the prefetch (the batch-1
  // step, where the copies after the wait are on the critical path); 2
  // otherwise -- fewer registers, more resident warps, which measured faster
  // on every large gather (LLaVA batch 32 step 285.5 -> 278.7 us, Qwen2-VL
  // batch 16 103.0 -> 97.8 us) while 2 on the prefetched batch-1 step measured
  // 23.4 -> 26.3 us and 1 slower everywhere
  if (!early && pairs <= (long long)sm_count() * 64)
    return launch_kernel(compact_kernel<16>, grid, dim3(kCompactThreads), 0, st, 0, true, la,
                         keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, early,
                         prefetch);
  if (prefetch)
    return launch_kernel(compact_kernel<8>, grid, dim3(kCompactThreads), 0, st, 0, true, la,
                         keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, early,
                         prefetch);
  return launch_kernel(compact_kernel<2>, grid, dim3(kCompactThreads), 0, st, 0, true, la,
                       keep_idx, keep_off, n_tensors, ts, pos_ids, total_rows, status, early,
                       prefetch);
}

}  // namespace e2s
