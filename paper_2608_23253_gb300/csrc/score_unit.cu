// Text-to-visual score, persistent single-CTA-per-unit variant (tcgen05 +
// TMEM, TMA-staged bf16 K tiles; Sec. 3.1 Eq. 1 and its causal-prefix
// probability reading).  Used for multi-head attention (one query head per kv
// head) with at most kMaxTiles 128-key tiles per unit.
//
// One CTA per SM loops over units (image, layer, head).  All of a unit's K
// tiles sit in shared memory; its text rows are processed in column groups of
// ntg rows (tiles * ntg <= 512 TMEM columns), so the softmax of each text row
// over its full causal prefix is resolved inside the CTA with no cluster
// exchange.  Two kernels: score_unit_kernel when every unit is a single group
// (e.g. one LLaVA image with 64 text rows), score_group_kernel otherwise (its
// per-step barriers and cross-group accumulators cost the single-group case
// time when the kernel overlaps its dependents).  Per column group:
//   MMA    D[key][t] = K_tile[key][:] . Q[t][:] (M = 128, N = the group's text
//          rows, K = 128 in 8 steps), tile i into TMEM columns [i*ntg, ...).
//   pass A per-text-row maximum (running max per lane over the tiles, one
//          butterfly reduce-scatter per 16-column chunk, then the 4 quarters);
//          each warp's first chunk is folded in tile by tile as the tile's
//          MMAs complete, while later K tiles are still arriving;
//   pass B e = exp2(s - M) (one exp2 per logit), stored back for the visual
//          tiles, row sums L the same way; weight w_t = 1 / (N_T L_t);
//   pass C a[key] += sum_t e[key][t] w_t over the group's rows (EQ1:
//          sum_t s / (sqrt(d) N_T)), accumulated in registers across groups.
// While the epilogue works on one step (unit, column group), the producer
// already streams the next step's queries (and the next unit's tiles) into the
// shared memory the MMAs have released.
//
// Warp roles (576 threads): warp 0 TMA producer, warp 1 TMEM allocator and MMA
// issuer, warps 2-17 epilogue.  Epilogue warp w reads TMEM lane quarter w % 4;
// in passes A and B it owns the chunks c with c % 4 == (w - 2) / 4, in pass C
// the visual tiles i with i % 4 == (w - 2) / 4.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "sm100_ptx.cuh"

namespace e2s {

bool make_score_map(CUtensorMap* map, const void* base, int heads, int64_t rows,
                    int64_t row_stride_el, int box_rows);

namespace {

constexpr int kTileKeys = 128;
constexpr int kHalfBytes = kTileKeys * 128;
constexpr int kTileBytes = 2 * kHalfBytes;
constexpr int kMaxTiles = 6;
constexpr int kEpiWarps = 16;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kQBoxRows = 16;
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kWaitNsAfterFault = 1000000ull;
constexpr float kLog2e = 1.4426950408889634f;

struct UnitArgs {
  LayoutArgs la;
  int ntp_max;          // padded text rows of the longest image
  int ntg;              // text rows per column group (multiple of 16; tiles * ntg <= 512)
  int mode;
  int num_units;
  float scale_log2;
  float scale;
  float* a_out;
  float4* stats;        // per (image, layer, head) statistics of the visual scores
  uint32_t* counters;   // nullable: decision scratch to zero
  uint32_t* status;
};

struct UPlan {
  uint32_t q, k, bars, slot, pmax, psum, cm, w, red, total;
};

__host__ __device__ inline UPlan unit_plan(int ntg) {
  UPlan s;
  s.q = 0;
  s.k = 2u * (uint32_t)ntg * 128u;
  s.bars = s.k + (uint32_t)kMaxTiles * kTileBytes;
  s.slot = s.bars + 8u * (uint32_t)(2 * kMaxTiles + 4);
  s.pmax = (s.slot + 16u + 15u) & ~15u;      // [4][ntg]
  s.psum = s.pmax + 4u * (uint32_t)ntg * 4u;  // [4][ntg]
  s.cm = s.psum + 4u * (uint32_t)ntg * 4u;    // [ntg]
  s.w = s.cm + (uint32_t)ntg * 4u;            // [ntg]
  s.red = s.w + (uint32_t)ntg * 4u;           // [2][kEpiWarps] float2
  s.total = s.red + 2u * kEpiWarps * 8u;
  return s;
}

template <int W, int MASK, class Op>
__device__ __forceinline__ void rs_step(float (&x)[16], bool hi, Op op) {
#pragma unroll
  for (int i = 0; i < W; ++i) {
    const float send = hi ? x[i] : x[i + W];
    const float keep = hi ? x[i + W] : x[i];
    x[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, MASK));
  }
}
// lane L ends with column L >> 1 of the 16, reduced over all 32 lanes
template <class Op>
__device__ __forceinline__ float reduce_scatter16(float (&x)[16], int lane, Op op) {
  rs_step<8, 16>(x, lane & 16, op);
  rs_step<4, 8>(x, lane & 8, op);
  rs_step<2, 4>(x, lane & 4, op);
  rs_step<1, 2>(x, lane & 2, op);
  return op(x[0], __shfl_xor_sync(0xffffffffu, x[0], 1));
}
struct MaxOp {
  __device__ __forceinline__ float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct AddOp {
  __device__ __forceinline__ float operator()(float a, float b) const { return a + b; }
};

// Geometry of one unit, derived identically by every warp role.
struct UnitGeo {
  int b, l, h, S, NV, NT, ntp, t0, x0, v0, key_base, nt, vf, vl;
  bool ok;
};

__device__ __forceinline__ UnitGeo unit_geo(const UnitArgs& p, int unit) {
  const LayoutArgs& la = p.la;
  UnitGeo g;
  g.h = unit % la.H;
  g.l = (unit / la.H) % la.L;
  g.b = unit / (la.H * la.L);
  g.S = __ldg(la.n_sys + g.b);
  g.NV = __ldg(la.n_vis + g.b);
  g.NT = __ldg(la.n_text + g.b);
  g.t0 = __ldg(la.tok_off + g.b);
  g.x0 = __ldg(la.text_off + g.b);
  g.v0 = __ldg(la.vis_off + g.b);
  const int T = g.S + g.NV + g.NT;
  g.ntp = (g.NT + 15) & ~15;
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  g.key_base = causal ? 0 : g.S;
  const int span = causal ? T : g.NV;
  g.nt = (span + kTileKeys - 1) / kTileKeys;
  g.ok = g.S >= 0 && g.NV >= 0 && g.NT >= 1 && g.ntp <= p.ntp_max && T <= la.max_T &&
         g.NV <= la.max_vis && __ldg(la.tok_off + g.b + 1) - g.t0 == T && g.t0 >= 0 &&
         g.t0 + T <= la.sum_T && __ldg(la.text_off + g.b + 1) - g.x0 == g.NT && g.x0 >= 0 &&
         g.x0 + g.NT <= la.sum_text && __ldg(la.vis_off + g.b + 1) - g.v0 == g.NV &&
         g.v0 >= 0 && g.v0 + g.NV <= la.sum_vis && g.nt <= kMaxTiles &&
         g.nt * p.ntg <= 512;
  if (!g.ok) {
    g.nt = 0;
    g.ntp = 0;
  }
  g.vf = g.nt;
  g.vl = g.nt;
  for (int i = 0; i < g.nt; ++i) {
    const int k0 = g.key_base + kTileKeys * i;
    if (k0 < g.S + g.NV && k0 + kTileKeys > g.S) {
      if (g.vf == g.nt) g.vf = i;
      g.vl = i + 1;
    }
  }
  return g;
}

// Column groups of a unit: its padded text rows in groups of ntg, each group
// one pass of MMAs and epilogue over the resident K tiles.
__device__ __forceinline__ int groups_of(const UnitGeo& g, int ntg) {
  return g.nt > 0 ? max(1, (g.ntp + ntg - 1) / ntg) : 1;
}
__device__ __forceinline__ int group_cols(const UnitGeo& g, int gi, int ntg) {
  return g.nt > 0 ? min(ntg, g.ntp - gi * ntg) : 0;
}

// Single-group variant: every unit's text rows fit one group.
__global__ void __launch_bounds__(kThreads, 1)
    score_unit_kernel(const __grid_constant__ CUtensorMap tmQ,
                      const __grid_constant__ CUtensorMap tmK, const UnitArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const UPlan plan = unit_plan(p.ntp_max);
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint64_t* k_full = reinterpret_cast<uint64_t*>(smem + plan.bars);  // [kMaxTiles]
  uint64_t* q_full = k_full + kMaxTiles;
  uint64_t* mma_done = q_full + 1;
  uint64_t* smem_free = mma_done + 1;
  uint64_t* tmem_free = smem_free + 1;
  uint64_t* mma_tile = tmem_free + 1;   // [kMaxTiles]: tile i's MMAs complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float* pmax = reinterpret_cast<float*>(smem + plan.pmax);
  float* psum = reinterpret_cast<float*>(smem + plan.psum);
  float* cm = reinterpret_cast<float*>(smem + plan.cm);
  float* wcol = reinterpret_cast<float*>(smem + plan.w);
  float2* red = reinterpret_cast<float2*>(smem + plan.red);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t q_half = (uint32_t)p.ntp_max * 128u;
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  pdl_wait();   // inputs may come from the kernel before (launched with PDL)
  // only then may the next kernel be scheduled: the compaction that follows
  // in e2s_prune copies rows before its own wait
  pdl_launch_dependents();   // every CTA is resident: the next kernel may be scheduled
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  if (warp == 0 && lane == 0) {
    for (int i = 0; i < kMaxTiles; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(mma_tile + i, 1);
    }
    ptx::mbar_init(q_full, 1);
    ptx::mbar_init(mma_done, 1);
    ptx::mbar_init(smem_free, 1);
    ptx::mbar_init(tmem_free, kEpiWarps);
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    ptx::prefetch_tensormap(&tmQ);
    ptx::prefetch_tensormap(&tmK);
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, 512);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;

  if (warp == 0) {
    // ================= TMA producer
    if (lane == 0) {
      int it = 0;
      for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x, ++it) {
        const UnitGeo g = unit_geo(p, unit);
        if (!g.ok) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
        if (it > 0 && !ptx::mbar_wait(smem_free, (it - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        if (g.nt > 0) {
          ptx::mbar_arrive_expect_tx(q_full, 2u * (uint32_t)g.ntp * 128u);
          for (int half = 0; half < 2; ++half)
            for (int r = 0; r < g.ntp; r += kQBoxRows)
              ptx::tma_load_3d(q_sm + half * q_half + (uint32_t)r * 128u, &tmQ, q_full, half * 64,
                               g.h, g.l * la.sum_text + g.x0 + r);
        } else {
          ptx::mbar_arrive(q_full);
        }
        for (int i = 0; i < kMaxTiles; ++i) {
          if (i < g.nt) {
            const int row = g.l * la.sum_T + g.t0 + g.key_base + kTileKeys * i;
            ptx::mbar_arrive_expect_tx(k_full + i, kTileBytes);
            ptx::tma_load_3d(k_sm + i * kTileBytes, &tmK, k_full + i, 0, g.h, row);
            ptx::tma_load_3d(k_sm + i * kTileBytes + kHalfBytes, &tmK, k_full + i, 64, g.h, row);
          } else {
            ptx::mbar_arrive(k_full + i);   // keep every barrier's phase in step
          }
        }
      }
      // the last unit's copies are consumed by its MMAs before the MMA warp ends
    }
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0) {
      int it = 0;
      for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x, ++it) {
        const UnitGeo g = unit_geo(p, unit);
        const uint32_t ph = it & 1;
        if (!ptx::mbar_wait(q_full, ph, limit, p.status)) limit = kWaitNsAfterFault;
        if (it > 0 && !ptx::mbar_wait(tmem_free, (it - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        const uint32_t idesc = ptx::idesc_bf16_f32(128, max(g.ntp, 16));
        const uint32_t b_base = ptx::smem_addr(q_sm);
        for (int i = 0; i < kMaxTiles; ++i) {
          if (!ptx::mbar_wait(k_full + i, ph, limit, p.status)) limit = kWaitNsAfterFault;
          if (i >= g.nt) {
            ptx::mbar_arrive(mma_tile + i);   // keep every barrier's phase in step
            continue;
          }
          ptx::tc_fence_after();
          const uint32_t a_base = ptx::smem_addr(k_sm + i * kTileBytes);
          const uint32_t d = tmem + (uint32_t)(i * p.ntp_max);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t half = ks >> 2, kk = ks & 3;
            const uint64_t ad = ptx::sdesc_sw128(a_base + half * kHalfBytes + kk * 32u);
            const uint64_t bd = ptx::sdesc_sw128(b_base + half * q_half + kk * 32u);
            ptx::mma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
          }
          ptx::mma_commit(mma_tile + i);   // the epilogue's pass A may read tile i
        }
        ptx::mma_commit(mma_done);   // epilogue may read TMEM
        ptx::mma_commit(smem_free);  // producer may overwrite the tiles and Q
      }
    }
  } else {
    // ================= epilogue (16 warps)
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int grp = ew >> 2;               // 0..3
    const int row = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    int it = 0;
    for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x, ++it) {
      const UnitGeo g = unit_geo(p, unit);
      const int NT = g.NT, ntp = g.ntp, nt = g.nt;
      const int lim = g.S + g.NV;
      const int cpb = ntp >> 4;
      if (causal && nt > 0) {
        // ---- pass A: the warp's first chunk follows the MMAs tile by tile
        // (overlapping the K tiles still in flight); any further chunks run
        // once every tile is done
        auto max16 = [&](float (&mx)[16], const float (&x)[16], int c16, int lo) {
          if (lo <= c16 && c16 + 16 <= NT) {
#pragma unroll
            for (int j = 0; j < 16; ++j) mx[j] = fmaxf(mx[j], x[j]);
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (c16 + j >= lo && c16 + j < NT) mx[j] = fmaxf(mx[j], x[j]);
          }
        };
        {
          float mx[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) mx[j] = kNegBig;
          for (int i = 0; i < nt; ++i) {
            if (!ptx::mbar_wait(mma_tile + i, it & 1, limit, p.status))
              limit = kWaitNsAfterFault;
            ptx::tc_fence_after();
            if (grp < cpb) {
              float x[16];
              ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * p.ntp_max + grp * 16), x);
              max16(mx, x, grp * 16, max(g.key_base + kTileKeys * i + row - lim, 0));
            }
          }
          if (grp < cpb) {
            const float m = reduce_scatter16(mx, lane, MaxOp());
            if ((lane & 1) == 0) pmax[q4 * p.ntp_max + grp * 16 + (lane >> 1)] = m;
          }
        }
        if (!ptx::mbar_wait(mma_done, it & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        for (int c = grp + 4; c < cpb; c += 4) {
          const int c16 = c * 16;
          float mx[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) mx[j] = kNegBig;
          for (int i = 0; i < nt; ++i) {
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * p.ntp_max + c16), x);
            max16(mx, x, c16, max(g.key_base + kTileKeys * i + row - lim, 0));
          }
          const float m = reduce_scatter16(mx, lane, MaxOp());
          if ((lane & 1) == 0) pmax[q4 * p.ntp_max + c16 + (lane >> 1)] = m;
        }
        ptx::named_bar(1, kEpiThreads);
        for (int c = et; c < ntp; c += kEpiThreads) {
          const int n = p.ntp_max;
          const float m = fmaxf(fmaxf(pmax[c], pmax[n + c]), fmaxf(pmax[2 * n + c], pmax[3 * n + c]));
          cm[c] = m > 0.5f * kNegBig ? m * p.scale_log2 : kNegBig;
        }
        ptx::named_bar(1, kEpiThreads);
        // ---- pass B
        for (int c = grp; c < cpb; c += 4) {
          const int c16 = c * 16;
          float mv[16], sm[16];
          const float4* cm4 = reinterpret_cast<const float4*>(cm + c16);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const float4 c4 = cm4[v];
            mv[4 * v] = c4.x; mv[4 * v + 1] = c4.y; mv[4 * v + 2] = c4.z; mv[4 * v + 3] = c4.w;
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) sm[j] = 0.f;
          for (int i = 0; i < nt; ++i) {
            const int lo = max(g.key_base + kTileKeys * i + row - lim, 0);
            const uint32_t ta = tmem + lane_base + (uint32_t)(i * p.ntp_max + c16);
            float x[16];
            ptx::tmem_ld16(ta, x);
            if (lo <= c16 && c16 + 16 <= NT) {
#pragma unroll
              for (int j = 0; j < 16; ++j) x[j] = fast_ex2(fmaf(x[j], p.scale_log2, -mv[j]));
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j)
                x[j] = (c16 + j >= lo && c16 + j < NT) ? fast_ex2(fmaf(x[j], p.scale_log2, -mv[j]))
                                                       : 0.f;
            }
            if (i >= g.vf && i < g.vl) ptx::tmem_st16(ta, x);
#pragma unroll
            for (int j = 0; j < 16; ++j) sm[j] += x[j];
          }
          const float s = reduce_scatter16(sm, lane, AddOp());
          if ((lane & 1) == 0) psum[q4 * p.ntp_max + c16 + (lane >> 1)] = s;
        }
        ptx::tmem_wait_st();
        ptx::tc_fence_before();
        ptx::named_bar(1, kEpiThreads);
        ptx::tc_fence_after();
        for (int c = et; c < ntp; c += kEpiThreads) {
          const int n = p.ntp_max;
          const float L = ((psum[c] + psum[n + c]) + psum[2 * n + c]) + psum[3 * n + c];
          wcol[c] = (c < NT && L > 0.f) ? 1.f / ((float)NT * L) : 0.f;
        }
        ptx::named_bar(1, kEpiThreads);
      } else {
        if (!ptx::mbar_wait(mma_done, it & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        for (int c = et; c < ntp; c += kEpiThreads) wcol[c] = (c < NT) ? p.scale / (float)NT : 0.f;
        ptx::named_bar(1, kEpiThreads);
      }
      // ---- pass C, plus the statistics of the unit's visual scores, kept
      // online per lane (sum, max of a*log2e, sum of exp2 relative to it)
      float st_s = 0.f, st_m = kNegBig, st_e = 0.f;
      for (int i = g.vf + ((grp - g.vf) & 3); i < g.vl; i += 4) {
        const int key = g.key_base + kTileKeys * i + row;
        float acc0 = 0.f, acc1 = 0.f;
        for (int c16 = 0; c16 < ntp; c16 += 16) {
          float x[16];
          ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * p.ntp_max + c16), x);
          const float4* w4 = reinterpret_cast<const float4*>(wcol + c16);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const float4 w = w4[v];
            acc0 = fmaf(x[4 * v], w.x, acc0);
            acc1 = fmaf(x[4 * v + 1], w.y, acc1);
            acc0 = fmaf(x[4 * v + 2], w.z, acc0);
            acc1 = fmaf(x[4 * v + 3], w.w, acc1);
          }
        }
        if (key >= g.S && key < g.S + g.NV) {
          const float a = acc0 + acc1;
          p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + (key - g.S)] = a;
          const float al = a * kLog2e, mnew = fmaxf(st_m, al);
          st_e = st_e * fast_ex2(st_m - mnew) + fast_ex2(al - mnew);
          st_m = mnew;
          st_s += a;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float s2 = __shfl_xor_sync(0xffffffffu, st_s, o);
        const float m2 = __shfl_xor_sync(0xffffffffu, st_m, o);
        const float e2 = __shfl_xor_sync(0xffffffffu, st_e, o);
        st_s += s2;
        lse_merge(st_m, st_e, m2, e2);
      }
      if (lane == 0) {
        red[ew] = make_float2(st_s, st_m);
        red[kEpiWarps + ew] = make_float2(st_e, 0.f);
      }
      ptx::named_bar(1, kEpiThreads);
      if (et == 0 && g.ok) {   // the 16 warps in order
        float S = 0.f, M = kNegBig, E = 0.f;
        for (int w = 0; w < kEpiWarps; ++w) {
          S += red[w].x;
          lse_merge(M, E, red[w].y, red[kEpiWarps + w].x);
        }
        p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h] = stats_entry(S, M, E);
      }
      // TMEM of this unit fully read: the MMA warp may overwrite it
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(tmem_free);
      // wcol / cm are rewritten by the next unit only after a named barrier
      ptx::named_bar(1, kEpiThreads);
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

// Column-group variant: a unit's text rows are processed in groups of ntg
// (used when the longest image's padded text rows exceed ntg).
__global__ void __launch_bounds__(kThreads, 1)
    score_group_kernel(const __grid_constant__ CUtensorMap tmQ,
                      const __grid_constant__ CUtensorMap tmK, const UnitArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const UPlan plan = unit_plan(p.ntg);
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint64_t* k_full = reinterpret_cast<uint64_t*>(smem + plan.bars);  // [kMaxTiles]
  uint64_t* q_full = k_full + kMaxTiles;
  uint64_t* mma_done = q_full + 1;
  uint64_t* mma_fin = mma_done + 1;   // a step's MMAs are complete: Q (and K) may be reloaded
  uint64_t* tmem_free = mma_fin + 1;
  uint64_t* mma_tile = tmem_free + 1;   // [kMaxTiles]: tile i's MMAs complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float* pmax = reinterpret_cast<float*>(smem + plan.pmax);
  float* psum = reinterpret_cast<float*>(smem + plan.psum);
  float* cm = reinterpret_cast<float*>(smem + plan.cm);
  float* wcol = reinterpret_cast<float*>(smem + plan.w);
  float2* red = reinterpret_cast<float2*>(smem + plan.red);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t q_half = (uint32_t)p.ntg * 128u;
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  pdl_wait();   // inputs may come from the kernel before (launched with PDL)
  // only then may the next kernel be scheduled: the compaction that follows
  // in e2s_prune copies rows before its own wait
  pdl_launch_dependents();   // every CTA is resident: the next kernel may be scheduled
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  if (warp == 0 && lane == 0) {
    for (int i = 0; i < kMaxTiles; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(mma_tile + i, 1);
    }
    ptx::mbar_init(q_full, 1);
    ptx::mbar_init(mma_done, 1);
    ptx::mbar_init(mma_fin, 1);
    ptx::mbar_init(tmem_free, kEpiWarps);
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    ptx::prefetch_tensormap(&tmQ);
    ptx::prefetch_tensormap(&tmK);
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, 512);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;

  if (warp == 0) {
    // ================= TMA producer: per step (unit, column group) the group's
    // text queries; per unit (first group) every K tile
    if (lane == 0) {
      int st = 0;
      for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x) {
        const UnitGeo g = unit_geo(p, unit);
        if (!g.ok) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
        const int ng = groups_of(g, p.ntg);
        for (int gi = 0; gi < ng; ++gi, ++st) {
          // the previous step's MMAs are complete: Q and, at a unit boundary,
          // the K tiles may be overwritten
          if (st > 0 && !ptx::mbar_wait(mma_fin, (st - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          const int cols = group_cols(g, gi, p.ntg);
          if (cols > 0) {
            ptx::mbar_arrive_expect_tx(q_full, 2u * (uint32_t)cols * 128u);
            for (int half = 0; half < 2; ++half)
              for (int r = 0; r < cols; r += kQBoxRows)
                ptx::tma_load_3d(q_sm + half * q_half + (uint32_t)r * 128u, &tmQ, q_full,
                                 half * 64, g.h, g.l * la.sum_text + g.x0 + gi * p.ntg + r);
          } else {
            ptx::mbar_arrive(q_full);
          }
          if (gi > 0) continue;
          for (int i = 0; i < kMaxTiles; ++i) {
            if (i < g.nt) {
              const int row = g.l * la.sum_T + g.t0 + g.key_base + kTileKeys * i;
              ptx::mbar_arrive_expect_tx(k_full + i, kTileBytes);
              ptx::tma_load_3d(k_sm + i * kTileBytes, &tmK, k_full + i, 0, g.h, row);
              ptx::tma_load_3d(k_sm + i * kTileBytes + kHalfBytes, &tmK, k_full + i, 64, g.h,
                               row);
            } else {
              ptx::mbar_arrive(k_full + i);   // keep every barrier's phase in step
            }
          }
        }
      }
      // the last unit's copies are consumed by its MMAs before the MMA warp ends
    }
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0) {
      int st = 0, it = 0;
      for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x, ++it) {
        const UnitGeo g = unit_geo(p, unit);
        const int ng = groups_of(g, p.ntg);
        for (int gi = 0; gi < ng; ++gi, ++st) {
          if (!ptx::mbar_wait(q_full, st & 1, limit, p.status)) limit = kWaitNsAfterFault;
          if (st > 0 && !ptx::mbar_wait(tmem_free, (st - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          const int cols = group_cols(g, gi, p.ntg);
          const uint32_t idesc = ptx::idesc_bf16_f32(128, max(cols, 16));
          const uint32_t b_base = ptx::smem_addr(q_sm);
          for (int i = 0; i < kMaxTiles; ++i) {
            if (gi == 0 && !ptx::mbar_wait(k_full + i, it & 1, limit, p.status))
              limit = kWaitNsAfterFault;
            if (i >= g.nt) {
              ptx::mbar_arrive(mma_tile + i);   // keep every barrier's phase in step
              continue;
            }
            ptx::tc_fence_after();
            const uint32_t a_base = ptx::smem_addr(k_sm + i * kTileBytes);
            const uint32_t d = tmem + (uint32_t)(i * p.ntg);
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              const uint32_t half = ks >> 2, kk = ks & 3;
              const uint64_t ad = ptx::sdesc_sw128(a_base + half * kHalfBytes + kk * 32u);
              const uint64_t bd = ptx::sdesc_sw128(b_base + half * q_half + kk * 32u);
              ptx::mma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
            }
            ptx::mma_commit(mma_tile + i);   // the epilogue's pass A may read tile i
          }
          ptx::mma_commit(mma_done);   // the epilogue may read TMEM
          ptx::mma_commit(mma_fin);    // the producer may overwrite Q (and the tiles)
        }
      }
    }
  } else {
    // ================= epilogue (16 warps)
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int grp = ew >> 2;               // 0..3
    const int row = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    const int ntg = p.ntg;
    int st = 0;
    for (int unit = blockIdx.x; unit < p.num_units; unit += gridDim.x) {
      const UnitGeo g = unit_geo(p, unit);
      const int NT = g.NT, nt = g.nt;
      const int lim = g.S + g.NV;
      const int ng = groups_of(g, ntg);
      // pass C accumulators of this thread's visual tiles (at most two: tiles
      // i with i % 4 == grp), summed over the column groups
      float acc[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
      const int i_first = g.vf + ((grp - g.vf) & 3);
      for (int gi = 0; gi < ng; ++gi, ++st) {
        const int cols = group_cols(g, gi, ntg);
        const int cpb = cols >> 4;
        const int tc0 = gi * ntg;        // text row of the group's first column
        const int nt_l = NT - tc0;       // columns at or beyond nt_l are padding
        if (causal && nt > 0) {
          // ---- pass A: the warp's first chunk follows the MMAs tile by tile
          // (overlapping the K tiles still in flight); any further chunks run
          // once every tile is done.  Column c of key `key` is valid when its
          // text row tc0 + c sees the key (tc0 + c >= key - lim) and is real.
          auto max16 = [&](float (&mx)[16], const float (&x)[16], int c16, int lo) {
            if (lo <= c16 && c16 + 16 <= nt_l) {
#pragma unroll
              for (int j = 0; j < 16; ++j) mx[j] = fmaxf(mx[j], x[j]);
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j)
                if (c16 + j >= lo && c16 + j < nt_l) mx[j] = fmaxf(mx[j], x[j]);
            }
          };
          {
            float mx[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) mx[j] = kNegBig;
            for (int i = 0; i < nt; ++i) {
              if (!ptx::mbar_wait(mma_tile + i, st & 1, limit, p.status))
                limit = kWaitNsAfterFault;
              ptx::tc_fence_after();
              if (grp < cpb) {
                float x[16];
                ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * ntg + grp * 16), x);
                max16(mx, x, grp * 16, max(g.key_base + kTileKeys * i + row - lim, 0) - tc0);
              }
            }
            if (grp < cpb) {
              const float m = reduce_scatter16(mx, lane, MaxOp());
              if ((lane & 1) == 0) pmax[q4 * ntg + grp * 16 + (lane >> 1)] = m;
            }
          }
          if (!ptx::mbar_wait(mma_done, st & 1, limit, p.status)) limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          for (int c = grp + 4; c < cpb; c += 4) {
            const int c16 = c * 16;
            float mx[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) mx[j] = kNegBig;
            for (int i = 0; i < nt; ++i) {
              float x[16];
              ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * ntg + c16), x);
              max16(mx, x, c16, max(g.key_base + kTileKeys * i + row - lim, 0) - tc0);
            }
            const float m = reduce_scatter16(mx, lane, MaxOp());
            if ((lane & 1) == 0) pmax[q4 * ntg + c16 + (lane >> 1)] = m;
          }
          ptx::named_bar(1, kEpiThreads);
          for (int c = et; c < cols; c += kEpiThreads) {
            const float m =
                fmaxf(fmaxf(pmax[c], pmax[ntg + c]), fmaxf(pmax[2 * ntg + c], pmax[3 * ntg + c]));
            cm[c] = m > 0.5f * kNegBig ? m * p.scale_log2 : kNegBig;
          }
          ptx::named_bar(1, kEpiThreads);
          // ---- pass B
          for (int c = grp; c < cpb; c += 4) {
            const int c16 = c * 16;
            float mv[16], sm[16];
            const float4* cm4 = reinterpret_cast<const float4*>(cm + c16);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const float4 c4 = cm4[v];
              mv[4 * v] = c4.x; mv[4 * v + 1] = c4.y; mv[4 * v + 2] = c4.z; mv[4 * v + 3] = c4.w;
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) sm[j] = 0.f;
            for (int i = 0; i < nt; ++i) {
              const int lo = max(g.key_base + kTileKeys * i + row - lim, 0) - tc0;
              const uint32_t ta = tmem + lane_base + (uint32_t)(i * ntg + c16);
              float x[16];
              ptx::tmem_ld16(ta, x);
              if (lo <= c16 && c16 + 16 <= nt_l) {
#pragma unroll
                for (int j = 0; j < 16; ++j) x[j] = fast_ex2(fmaf(x[j], p.scale_log2, -mv[j]));
              } else {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  x[j] = (c16 + j >= lo && c16 + j < nt_l)
                             ? fast_ex2(fmaf(x[j], p.scale_log2, -mv[j]))
                             : 0.f;
              }
              if (i >= g.vf && i < g.vl) ptx::tmem_st16(ta, x);
#pragma unroll
              for (int j = 0; j < 16; ++j) sm[j] += x[j];
            }
            const float s = reduce_scatter16(sm, lane, AddOp());
            if ((lane & 1) == 0) psum[q4 * ntg + c16 + (lane >> 1)] = s;
          }
          ptx::tmem_wait_st();
          ptx::tc_fence_before();
          ptx::named_bar(1, kEpiThreads);
          ptx::tc_fence_after();
          for (int c = et; c < cols; c += kEpiThreads) {
            const float L = ((psum[c] + psum[ntg + c]) + psum[2 * ntg + c]) + psum[3 * ntg + c];
            wcol[c] = (c < nt_l && L > 0.f) ? 1.f / ((float)NT * L) : 0.f;
          }
          ptx::named_bar(1, kEpiThreads);
        } else {
          if (!ptx::mbar_wait(mma_done, st & 1, limit, p.status)) limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          for (int c = et; c < cols; c += kEpiThreads)
            wcol[c] = (c < nt_l) ? p.scale / (float)NT : 0.f;
          ptx::named_bar(1, kEpiThreads);
        }
        // ---- pass C over this group's columns, accumulated per key; after
        // the unit's last group, the scores and the partial statistics
        const bool last = gi == ng - 1;
        float ls = 0.f, lm = kNegBig, av[2] = {0.f, 0.f};
        bool has[2] = {false, false};
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int i = i_first + 4 * k;
          if (i >= g.vl) break;
          float acc0 = acc[k][0], acc1 = acc[k][1];
          for (int c16 = 0; c16 < cols; c16 += 16) {
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * ntg + c16), x);
            const float4* w4 = reinterpret_cast<const float4*>(wcol + c16);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const float4 w = w4[v];
              acc0 = fmaf(x[4 * v], w.x, acc0);
              acc1 = fmaf(x[4 * v + 1], w.y, acc1);
              acc0 = fmaf(x[4 * v + 2], w.z, acc0);
              acc1 = fmaf(x[4 * v + 3], w.w, acc1);
            }
          }
          acc[k][0] = acc0;
          acc[k][1] = acc1;
          const int key = g.key_base + kTileKeys * i + row;
          if (last && key >= g.S && key < g.S + g.NV) {
            const float a = acc0 + acc1;
            p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + (key - g.S)] = a;
            ls += a;
            lm = fmaxf(lm, a * kLog2e);
            av[k] = a;
            has[k] = true;
          }
        }
        // statistics of the unit's visual scores for Eq. 8 (red is rewritten by
        // the next step only after the barrier that ends this one)
        auto unit_stats = [&]() {
          ls = warp_reduce(ls, [](float x, float y) { return x + y; });
          lm = warp_reduce(lm, [](float x, float y) { return fmaxf(x, y); });
          if (lane == 0) red[ew] = make_float2(ls, lm);
          ptx::named_bar(1, kEpiThreads);
          float S = 0.f, M = kNegBig;
          for (int w = 0; w < kEpiWarps; ++w) {
            S += red[w].x;
            M = fmaxf(M, red[w].y);
          }
          float le = 0.f;
          if (has[0]) le += fast_ex2(fmaf(av[0], kLog2e, -M));
          if (has[1]) le += fast_ex2(fmaf(av[1], kLog2e, -M));
          le = warp_reduce(le, [](float x, float y) { return x + y; });
          if (lane == 0) red[kEpiWarps + ew] = make_float2(le, 0.f);
          ptx::named_bar(1, kEpiThreads);
          if (et == 0 && g.ok) {
            float E = 0.f;
            for (int w = 0; w < kEpiWarps; ++w) E += red[kEpiWarps + w].x;
            p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h] = stats_entry(S, M, E);
          }
        };
        // TMEM of this step fully read: the MMA warp goes on with the next
        // step while the statistics are reduced; wcol and cm are rewritten by
        // the next step only after the barrier below
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(tmem_free);
        if (last) unit_stats();
        ptx::named_bar(1, kEpiThreads);
      }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

}  // namespace

// Text rows per column group: the padded text rows of the longest image, cut
// so that the unit's tiles times the group fit the 512 TMEM columns.
static int unit_ntg(const LayoutArgs& la, int mode) {
  const int ntp_max = ((std::max(la.max_text, 1) + 15) / 16) * 16;
  const int span = (mode == E2S_SCORE_CAUSAL_PROB) ? la.max_T : la.max_vis;
  const int tiles = std::max(1, (span + kTileKeys - 1) / kTileKeys);
  return std::min(ntp_max, (512 / tiles) / 16 * 16);
}

// Whether every unit is a single column group (score_unit_kernel).
bool score_unit_single_group(const LayoutArgs& la, int mode) {
  return unit_ntg(la, mode) >= ((std::max(la.max_text, 1) + 15) / 16) * 16;
}

// Whether the persistent kernel can take this launch (see the file comment).
bool score_unit_fits(const LayoutArgs& la, int mode) {
  if (la.H != la.H_kv) return false;
  const int span = (mode == E2S_SCORE_CAUSAL_PROB) ? la.max_T : la.max_vis;
  const int tiles = (span + kTileKeys - 1) / kTileKeys;
  if (tiles > kMaxTiles) return false;
  const int ntg = unit_ntg(la, mode);
  if (ntg < 16) return false;
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  return (int)(unit_plan(ntg).total + 1024) <= optin;
}

cudaError_t launch_score_unit(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                              const void* k, int64_t k_stride, float* a_out, float4* stats,
                              uint32_t* counters, uint32_t* status, cudaStream_t st,
                              bool pdl) {
  UnitArgs p;
  p.la = la;
  p.ntp_max = ((std::max(la.max_text, 1) + 15) / 16) * 16;
  p.ntg = unit_ntg(la, mode);
  p.mode = mode;
  p.num_units = la.B * la.L * la.H;
  p.scale = 1.0f / sqrtf(128.0f);
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.a_out = a_out;
  p.stats = stats;
  p.counters = counters;
  p.status = status;
  if (p.num_units == 0 || la.sum_vis == 0) return cudaSuccess;
  CUtensorMap tmQ, tmK;
  if (!make_score_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_text, q_stride, kQBoxRows) ||
      !make_score_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTileKeys))
    return cudaErrorInvalidValue;
  const size_t smem = unit_plan(p.ntg).total + 1024;
  const dim3 grid((unsigned)std::min(p.num_units, sm_count()));
  if (p.ntg >= p.ntp_max)
    return launch_kernel(score_unit_kernel, grid, dim3(kThreads), smem, st, 0, pdl, tmQ, tmK, p);
  return launch_kernel(score_group_kernel, grid, dim3(kThreads), smem, st, 0, pdl, tmQ, tmK, p);
}

}  // namespace e2s
