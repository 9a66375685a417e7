// Spatial novelty and global Top-K of one image, run by a whole CTA
// (Sec. 4.3, Eqs. 20-23):
//   1. cell representative: per occupied G x G cell, arg-max of q with ties
//      to the lower index, as a 64-bit atomicMax of (ordered q bits, ~n);
//   2. q~ = (1 - lambda) q + lambda b;
//   3. exact K-th largest q~ by a 4-pass 8-bit radix select over the ordered
//      bit patterns (histogram in shared memory, digit found by a warp scan);
//   4. emission in ascending index order with block-wide prefix counts; among
//      tokens equal to the threshold the lowest indices are kept.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "device_common.cuh"

namespace e2s {

constexpr int kMaxCells = 64;

constexpr int kSelDigitBits = 9;                  // radix digit of the threshold search
constexpr int kSelBuckets = 1 << kSelDigitBits;
constexpr int kSelCand = 32;                      // live keys one warp ranks directly

struct SelectSmem {
  unsigned long long cell_best[kMaxCells];
  uint32_t hist[kSelBuckets];
  uint32_t cand[kSelCand];
  uint32_t warp_tot[32];
  uint32_t w_and[32], w_or[32];   // per warp AND / OR of the keys
  uint32_t sel[4];                // digit, its keys, keys still needed, candidates gathered
};

// Per-warp AND and OR of the keys a thread wrote (identity values for none);
// the whole block calls it before the barrier that publishes the keys.
__device__ __forceinline__ void publish_key_bits(uint32_t k_and, uint32_t k_or, SelectSmem& ss) {
  k_and = __reduce_and_sync(0xffffffffu, k_and);
  k_or = __reduce_or_sync(0xffffffffu, k_or);
  if ((threadIdx.x & 31) == 0) {
    ss.w_and[threadIdx.x >> 5] = k_and;
    ss.w_or[threadIdx.x >> 5] = k_or;
  }
}

// Exclusive prefix count of `flag` over the block (in thread order) and the
// block total.  Every thread of the block must call it.
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

// n / d for 0 <= n < 2^17 and 2 <= d <= 2^13 as a multiply-high with
// m = ceil(2^32 / d): the product exceeds n/d by less than n / 2^32 < 2^-15,
// while a non-integer n/d is at least 1/d >= 2^-13 below the next integer,
// so the floor is exact.  (The multiplier of d = 1 does not fit 32 bits.)
__device__ __forceinline__ uint32_t div_multiplier(int d) {
  return d >= 2 ? (uint32_t)((0x100000000ull + (uint64_t)d - 1) / (uint64_t)d) : 0u;
}

// The G x G cell grid of one image: cell(i, j) = (i*G/h, j*G/w) of raster
// index r = i*w + j, with multiply-high divisions where they are exact.
struct CellMap {
  int gh, gw, G;
  uint32_t m_gh, m_gw;
  bool fast;
  __device__ __forceinline__ CellMap(int gh_, int gw_, int G_) : gh(gh_), gw(gw_), G(G_) {
    fast = gh >= 2 && gw >= 2 && gh <= 8192 && gw <= 8192 && (long long)gh * gw < (1 << 17);
    m_gh = fast ? div_multiplier(gh) : 0u;
    m_gw = fast ? div_multiplier(gw) : 0u;
  }
  __device__ __forceinline__ int operator()(int r) const {
    if (!fast) return cell_id(r, gh, gw, G);
    const int i = (int)__umulhi((uint32_t)r, m_gw), j = r - i * gw;
    return (int)__umulhi((uint32_t)(i * G), m_gh) * G + (int)__umulhi((uint32_t)(j * G), m_gw);
  }
};

// Cell of image-local slot n: its original raster index (cand, when given)
// mapped to the cell grid.  An out-of-range candidate raises E2S_ERR_SHAPE and
// is clamped.
__device__ __forceinline__ int token_cell(const int32_t* cand, int n, const CellMap& cm,
                                          uint32_t* status) {
  int r = cand ? __ldg(cand + n) : n;
  if (r < 0 || r >= cm.gh * cm.gw) {
    E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
    r = min(max(r, 0), cm.gh * cm.gw - 1);
  }
  return cm(r);
}

// Arg-max key of a cell: larger q wins, then the lower slot index.
__device__ __forceinline__ unsigned long long cell_key(float q, int n) {
  return ((unsigned long long)ordered_key(q) << 32) | (0xFFFFFFFFu - (uint32_t)n);
}

// Exact Kc-th largest of keys[0 .. NV) (0 < Kc < NV): its value thr and how
// many of the keys equal to it are kept (need_eq).  Radix search from the
// highest bit in which the keys differ (from the AND / OR that
// publish_key_bits left in ss), kSelDigitBits bits per pass: a histogram of
// the live keys' digit, one block-wide scan of it in descending order to find
// the digit holding the remaining-th largest live key, and the live set
// narrowed to that digit.  Once the digit's bucket holds at most kSelCand
// keys, they are gathered and one warp ranks them against each other (each
// lane compares its key with every gathered key, read as a shared-memory
// broadcast), which gives the threshold directly; one or two 9-bit passes
// usually leave that few.  Every thread of the block must call it.
static __device__ void select_threshold(const uint32_t* keys, int NV, uint32_t Kc,
                                        SelectSmem& ss, uint32_t& thr, uint32_t& need_eq) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nt = (int)blockDim.x, nw = nt >> 5;
  uint32_t all_and = 0xFFFFFFFFu, all_or = 0u;
  for (int w = 0; w < nw; ++w) {
    all_and &= ss.w_and[w];
    all_or |= ss.w_or[w];
  }
  const uint32_t diff = all_and ^ all_or;   // bits in which some keys differ
  if (diff == 0u) {                         // every key is the same
    thr = all_and;
    need_eq = Kc;
    return;
  }
  int top = 31 - __clz(diff);               // highest undecided bit
  uint32_t mask = top == 31 ? 0u : (0xFFFFFFFFu << (top + 1));
  uint32_t prefix = all_and & mask;         // live keys: (k & mask) == prefix
  uint32_t remaining = Kc;
  for (;;) {
    const int shift = max(top - (kSelDigitBits - 1), 0);
    const int nb = 1 << (top - shift + 1);
    // the previous pass read the histogram and sel before its last barrier
    for (int i = threadIdx.x; i < nb; i += nt) ss.hist[i] = 0u;
    if (threadIdx.x == 0) ss.sel[3] = 0u;
    __syncthreads();
    for (int n = threadIdx.x; n < NV; n += nt) {
      const uint32_t k = keys[n];
      if ((k & mask) == prefix) atomicAdd(&ss.hist[(k >> shift) & (uint32_t)(nb - 1)], 1u);
    }
    __syncthreads();
    // thread t owns the buckets of descending rank t*per .. t*per+per-1
    const int per = (nb + nt - 1) / nt;
    const int i0 = min((int)threadIdx.x * per, nb), i1 = min(i0 + per, nb);
    uint32_t tot = 0;
    for (int i = i0; i < i1; ++i) tot += ss.hist[nb - 1 - i];
    uint32_t incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) ss.warp_tot[warp] = incl;
    __syncthreads();
    uint32_t acc = incl - tot;
    for (int w = 0; w < warp; ++w) acc += ss.warp_tot[w];
    if (acc < remaining && remaining <= acc + tot) {   // exactly one thread
      for (int i = i0; i < i1; ++i) {
        const uint32_t h = ss.hist[nb - 1 - i];
        if (acc + h >= remaining) {
          ss.sel[0] = (uint32_t)(nb - 1 - i);
          ss.sel[1] = h;
          ss.sel[2] = remaining - acc;
          break;
        }
        acc += h;
      }
    }
    __syncthreads();
    const uint32_t cnt = ss.sel[1];
    prefix |= ss.sel[0] << shift;
    mask |= (uint32_t)(nb - 1) << shift;
    remaining = ss.sel[2];
    if (shift == 0) {   // the live keys are all equal
      thr = prefix;
      need_eq = remaining;
      return;
    }
    if (cnt <= (uint32_t)kSelCand) {
      for (int n = threadIdx.x; n < NV; n += nt) {
        const uint32_t k = keys[n];
        if ((k & mask) == prefix) ss.cand[atomicAdd(&ss.sel[3], 1u)] = k;
      }
      __syncthreads();
      if (warp == 0) {
        const uint32_t mine = (uint32_t)lane < cnt ? ss.cand[lane] : 0u;
        uint32_t gt = 0, eq = 0;
        for (uint32_t j = 0; j < cnt; ++j) {   // every lane reads the same word
          const uint32_t o = ss.cand[j];
          gt += o > mine ? 1u : 0u;
          eq += o == mine ? 1u : 0u;
        }
        // the remaining-th largest live key (equal keys write the same values)
        if ((uint32_t)lane < cnt && gt < remaining && remaining <= gt + eq) {
          ss.sel[0] = mine;
          ss.sel[1] = remaining - gt;
        }
      }
      __syncthreads();
      thr = ss.sel[0];
      need_eq = ss.sel[1];
      return;
    }
    top = shift - 1;
  }
}

// Steps 3-4 over the ordered keys of q~ (keys[0 .. NV) in shared memory).
// 3. exact K-th largest key (select_threshold);
// 4. ascending emission: each thread owns a contiguous run of slots; one
//    block-wide exclusive scan of (count above the threshold, count equal to
//    it), packed in 16-bit halves, gives every kept slot its position.  Among
//    slots equal to the threshold the lowest indices are kept.
// Every thread of the block must call it; NV <= 8192.
static __device__ void select_rank_emit(const uint32_t* keys, int NV, int K, SelectSmem& ss,
                                        int32_t* keep) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int Kc = min(K, NV);
  const bool keep_all = Kc == NV;
  uint32_t thr = 0, need_eq = 0;
  if (!keep_all && Kc > 0) {
    select_threshold(keys, NV, (uint32_t)Kc, ss, thr, need_eq);
  }

  // 4. emit ascending indices
  if (keep_all) {
    for (int n = threadIdx.x; n < NV; n += blockDim.x) keep[n] = n;
  } else if (Kc > 0) {
    const int per = (NV + (int)blockDim.x - 1) / (int)blockDim.x;
    const int lo = min(NV, (int)threadIdx.x * per), hi = min(NV, lo + per);
    uint32_t cnt = 0;   // (above threshold) | (equal to it) << 16
    for (int n = lo; n < hi; ++n) {
      const uint32_t k = keys[n];
      cnt += (k > thr) ? 1u : (k == thr ? 0x10000u : 0u);
    }
    uint32_t incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) ss.warp_tot[warp] = incl;
    __syncthreads();
    uint32_t before = incl - cnt;
    for (int w = 0; w < warp; ++w) before += ss.warp_tot[w];
    uint32_t gt = before & 0xFFFFu, eq = before >> 16;
    for (int n = lo; n < hi; ++n) {
      const uint32_t k = keys[n];
      if (k > thr) {
        keep[gt + min(eq, need_eq)] = n;
        ++gt;
      } else if (k == thr) {
        if (eq < need_eq) keep[gt + eq] = n;
        ++eq;
      }
    }
  }
  for (int s = Kc + threadIdx.x; s < K; s += blockDim.x) keep[s] = -1;
}

// Whole-CTA select for one image.  q[n], cand[n] (nullable) and q_tilde[n]
// (nullable) are indexed by the image-local slot n in [0, NV); keys (NV
// words) and cells (NV bytes) are shared scratch; keep receives K entries
// (ascending, -1 padded).
static __device__ void select_image(const float* q, const int32_t* cand, int NV, int gh, int gw,
                                    int G, float lam, int K, uint32_t* keys, uint8_t* cells,
                                    SelectSmem& ss, float* q_tilde, int32_t* keep,
                                    uint32_t* status) {
  const int ncell = G * G;
  const CellMap cm(gh, gw, G);
  // 1. cell representatives (Eqs. 20-21)
  for (int i = threadIdx.x; i < ncell; i += blockDim.x) ss.cell_best[i] = 0ull;
  __syncthreads();
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    const int g = token_cell(cand, n, cm, status);
    cells[n] = (uint8_t)g;
    atomicMax(&ss.cell_best[g], cell_key(q[n], n));
  }
  __syncthreads();
  // 2. q~ (Eq. 22)
  uint32_t k_and = 0xFFFFFFFFu, k_or = 0u;
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    const uint32_t best = (uint32_t)(ss.cell_best[cells[n]] & 0xFFFFFFFFull);
    const float bind = (best == 0xFFFFFFFFu - (uint32_t)n) ? 1.f : 0.f;
    const float qt = (1.f - lam) * q[n] + lam * bind;
    const uint32_t k = ordered_key(qt);
    keys[n] = k;
    k_and &= k;
    k_or |= k;
    if (q_tilde) q_tilde[n] = qt;
  }
  publish_key_bits(k_and, k_or, ss);
  __syncthreads();
  // 3-4. threshold of Top-K (Eq. 23) and emission
  select_rank_emit(keys, NV, K, ss, keep);
}

// The same select for a CTA that did not compute q: the cell arg-max keys
// (Eqs. 20-21) were reduced into cell_best_g[0 .. G*G) in global memory by the
// CTAs that did, and q[] was written by them; cm is the image's cell grid.  This CTA reads the keys (and
// resets them to zero for the next use) in the same phase as q, then runs
// steps 2-4.  keys (NV words) and cells (NV bytes) are shared scratch.
static __device__ void select_image_from_cells(const float* q, const int32_t* cand, int NV,
                                               const CellMap& cm, float lam, int K,
                                               unsigned long long* cell_best_g, uint32_t* keys,
                                               uint8_t* cells, SelectSmem& ss, float* q_tilde,
                                               int32_t* keep, uint32_t* status) {
  const int G = cm.G;
  for (int i = threadIdx.x; i < G * G; i += blockDim.x) {
    ss.cell_best[i] = __ldcg(cell_best_g + i);
    cell_best_g[i] = 0ull;
  }
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    keys[n] = __float_as_uint(__ldcg(q + n));
    cells[n] = (uint8_t)token_cell(cand, n, cm, status);
  }
  __syncthreads();
  // 2. q~ (Eq. 22)
  uint32_t k_and = 0xFFFFFFFFu, k_or = 0u;
  for (int n = threadIdx.x; n < NV; n += blockDim.x) {
    const uint32_t best = (uint32_t)(ss.cell_best[cells[n]] & 0xFFFFFFFFull);
    const float bind = (best == 0xFFFFFFFFu - (uint32_t)n) ? 1.f : 0.f;
    const float qt = (1.f - lam) * __uint_as_float(keys[n]) + lam * bind;
    const uint32_t k = ordered_key(qt);
    keys[n] = k;
    k_and &= k;
    k_or |= k;
    if (q_tilde) q_tilde[n] = qt;
  }
  publish_key_bits(k_and, k_or, ss);
  __syncthreads();
  select_rank_emit(keys, NV, K, ss, keep);
}

// Device-side checks of one image's select arguments.
__device__ __forceinline__ bool select_args_ok(const LayoutArgs& la, int b, bool has_cand,
                                               const int32_t* keep_count, const int32_t* keep_off,
                                               int32_t sum_keep) {
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  const int gh = __ldg(la.grid_h + b), gw = __ldg(la.grid_w + b);
  const int K = __ldg(keep_count + b), ko = __ldg(keep_off + b);
  return NV >= 0 && NV <= la.max_vis && v0 >= 0 && v0 + NV <= la.sum_vis &&
         __ldg(la.vis_off + b + 1) - v0 == NV && gh > 0 && gw > 0 &&
         (has_cand ? (long long)gh * gw >= NV : (long long)gh * gw == NV) && K >= 0 && ko >= 0 &&
         __ldg(keep_off + b + 1) - ko == K && ko + K <= sum_keep;
}

}  // namespace e2s
