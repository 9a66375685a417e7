// Spatial novelty and global Top-K (Sec. 4.3, Eqs. 20-23).  One CTA per
// image, everything in shared memory:
//   1. cell representative: per occupied G x G cell, arg-max of q with ties
//      to the lower index, as a 64-bit atomicMax of (ordered q bits, ~n);
//   2. q~ = (1 - lambda) q + lambda b;
//   3. exact K-th largest q~ by a 4-pass 8-bit radix select over the ordered
//      bit patterns (histogram in shared memory, digit found by a warp scan);
//   4. emission in ascending index order with block-wide prefix sums; among
//      tokens equal to the threshold the lowest indices are kept.
#include <cuda_runtime.h>

#include <algorithm>

#include "device_common.cuh"

namespace e2s {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kMaxCells = 64;

// Exclusive prefix count of `flag` over the block (in thread order) and the
// block total.  `warp_tot` is >= 32 words of shared memory.
__device__ __forceinline__ uint32_t block_excl_count(bool flag, uint32_t* warp_tot,
                                                     uint32_t& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const uint32_t bal = __ballot_sync(0xffffffffu, flag);
  const uint32_t in_warp = __popc(bal & ((1u << lane) - 1u));
  __syncthreads();
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  uint32_t before = 0, all = 0;
  for (int w = 0; w < nw; ++w) {
    const uint32_t c = warp_tot[w];
    before += (w < warp) ? c : 0u;
    all += c;
  }
  total = all;
  return before + in_warp;
}

__device__ __forceinline__ int cell_id(int r, int gh, int gw, int G) {
  const int i = r / gw, j = r - (r / gw) * gw;
  return (i * G / gh) * G + (j * G / gw);
}

__global__ void __launch_bounds__(kSelThreads)
    select_kernel(const LayoutArgs la, float lambda, int G, uint32_t flags,
                  const float* __restrict__ q, const int32_t* __restrict__ cand,
                  const int32_t* __restrict__ keep_count, const int32_t* __restrict__ keep_off,
                  int32_t sum_keep, int32_t* __restrict__ keep_idx, float* __restrict__ q_tilde,
                  uint32_t* status) {
  extern __shared__ uint32_t keys[];  // [max_vis]
  __shared__ unsigned long long cell_best[kMaxCells];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t warp_tot[32];
  __shared__ uint32_t sh_digit, sh_remaining;

  const int b = blockIdx.x;
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  const int gh = __ldg(la.grid_h + b), gw = __ldg(la.grid_w + b);
  const int K = __ldg(keep_count + b), ko = __ldg(keep_off + b);
  const bool ok = NV >= 0 && NV <= la.max_vis && v0 >= 0 && v0 + NV <= la.sum_vis &&
                  __ldg(la.vis_off + b + 1) - v0 == NV && gh > 0 && gw > 0 &&
                  (cand ? (long long)gh * gw >= NV : (long long)gh * gw == NV) && K >= 0 &&
                  ko >= 0 && __ldg(keep_off + b + 1) - ko == K && ko + K <= sum_keep;
  if (!ok) {
    if (threadIdx.x == 0) E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
    return;
  }
  const float lam = (flags & (E2S_NO_NOVELTY | E2S_VANILLA)) ? 0.f : lambda;
  const int ncell = G * G;

  // 1. cell representatives (Eqs. 20-21)
  for (int i = threadIdx.x; i < ncell; i += blockDim.x) cell_best[i] = 0ull;
  __syncthreads();
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    int r = cand ? __ldg(cand + v0 + n) : n;
    if (r < 0 || r >= gh * gw) {
      E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
      r = min(max(r, 0), gh * gw - 1);
    }
    const unsigned long long key =
        ((unsigned long long)ordered_key(q[v0 + n]) << 32) | (0xFFFFFFFFu - (uint32_t)n);
    atomicMax(&cell_best[cell_id(r, gh, gw, G)], key);
  }
  __syncthreads();
  // 2. q~ (Eq. 22)
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    int r = cand ? __ldg(cand + v0 + n) : n;
    r = min(max(r, 0), gh * gw - 1);
    const uint32_t best = (uint32_t)(cell_best[cell_id(r, gh, gw, G)] & 0xFFFFFFFFull);
    const float bind = (best == 0xFFFFFFFFu - (uint32_t)n) ? 1.f : 0.f;
    const float qt = (1.f - lam) * q[v0 + n] + lam * bind;
    keys[n] = ordered_key(qt);
    if (q_tilde) q_tilde[v0 + n] = qt;
  }
  __syncthreads();

  // 3. threshold of Top-K (Eq. 23)
  const int Kc = min(K, NV);
  const bool keep_all = Kc == NV;
  uint32_t thr = 0, need_eq = 0;
  if (!keep_all && Kc > 0) {
    uint32_t prefix = 0, mask = 0, remaining = (uint32_t)Kc;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
      __syncthreads();
      for (int n = threadIdx.x; n < NV; n += blockDim.x) {
        const uint32_t k = keys[n];
        if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        uint32_t c[8], tot = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          c[i] = hist[255 - 8 * lane - i];
          tot += c[i];
        }
        uint32_t incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        uint32_t excl = incl - tot;
        if (excl < remaining && remaining <= incl) {
          for (int i = 0; i < 8; ++i) {
            if (excl + c[i] >= remaining) {
              sh_digit = (uint32_t)(255 - 8 * lane - i);
              sh_remaining = remaining - excl;
              break;
            }
            excl += c[i];
          }
        }
      }
      __syncthreads();
      prefix |= sh_digit << shift;
      mask |= 255u << shift;
      remaining = sh_remaining;
      __syncthreads();
    }
    thr = prefix;
    need_eq = remaining;
  }

  // 4. emit ascending indices
  uint32_t base = 0, eq_seen = 0;
  if (Kc > 0) {
    for (int chunk = 0; chunk < NV; chunk += blockDim.x) {
      const int n = chunk + threadIdx.x;
      const uint32_t k = n < NV ? keys[n] : 0u;
      const bool is_eq = n < NV && !keep_all && k == thr;
      uint32_t eq_tot;
      const uint32_t rank_eq = block_excl_count(is_eq, warp_tot, eq_tot) + eq_seen;
      const bool keep = n < NV && (keep_all || k > thr || (is_eq && rank_eq < need_eq));
      uint32_t keep_tot;
      const uint32_t pos = block_excl_count(keep, warp_tot, keep_tot) + base;
      if (keep) keep_idx[ko + pos] = n;
      base += keep_tot;
      eq_seen += eq_tot;
    }
  }
  for (int s = Kc + threadIdx.x; s < K; s += blockDim.x) keep_idx[ko + s] = -1;
}

}  // namespace

cudaError_t launch_select(const LayoutArgs& la, float lambda, int G, uint32_t flags,
                          const float* q, const int32_t* cand, const int32_t* keep_count,
                          const int32_t* keep_off, int32_t sum_keep, int32_t* keep_idx,
                          float* q_tilde, uint32_t* status, cudaStream_t st) {
  const size_t smem = (size_t)std::max(la.max_vis, 1) * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  select_kernel<<<la.B, kSelThreads, smem, st>>>(la, lambda, G, flags, q, cand, keep_count,
                                                 keep_off, sum_keep, keep_idx, q_tilde, status);
  return cudaGetLastError();
}

}  // namespace e2s
