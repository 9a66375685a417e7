// Text-to-visual score for small batches (Sec. 3.1 Eq. 1 and its
// causal-prefix probability reading): one thread-block cluster per (image,
// layer, query head) unit, the unit's key tiles split over the cluster's CTAs.
//
// At batch 1 a persistent one-CTA-per-unit kernel leaves SMs idle (96 units
// of LLaVA-1.5-7B on 152 SMs) and runs the whole softmax epilogue after the
// last key tile has landed.  Here each CTA holds at most kMaxTpc tiles of 128
// keys in shared memory (two CTAs per SM), so every SM loads a share of K and
// each CTA's epilogue starts as soon as its own tiles are in.  Per CTA:
//
//   sweep 1 (CAUSAL_PROB)  MMA D1[r][key] = Q2[r] . K[key] with the text rows
//          on the TMEM lanes: the queries are loaded twice (rows 0-63 and
//          64-127), each lane half takes half of every tile's key columns and
//          each of two warps per lane quarter half of that, so every text
//          row's running (max, sum of exp2) over the CTA's keys is lane-local.
//          The per-row partials (four per row) are merged in the CTA, then
//          sent to every CTA of the cluster through distributed shared memory;
//          after one cluster barrier each CTA merges the C partials of a row in
//          rank order into the row's log-sum-exp, identically in every CTA.
//   sweep 2  MMA D2[key][t] = K[key] . Q[t] for the CTA's visual tiles, the
//          keys on the lanes: a[key] = (1/N_T) sum_t exp2(s - lse_t) is
//          lane-local (one warp per lane quarter and tile).  With two tiles
//          D2 takes tile 0's TMEM columns as soon as sweep 1 has read tile 0,
//          so sweep 2's MMAs run while sweep 1 finishes and the cluster
//          exchanges its partials.
//   Eq. 8 statistics of the unit's visual scores (sum, max of a*log2e, sum of
//          exp2 relative to it): per CTA, merged in rank order by rank 0.
//
// EQ1 mode has no sweep 1 (a = sum_t s / (sqrt(d) N_T) over D2), and neither
// has CAUSAL_PROB when the caller passes each text row's lse from the layer's
// own attention pass: then only the visual key tiles are loaded.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-9 epilogue (warp w reads TMEM lane quarter w % 4).
// Every mbarrier wait is bounded and reports E2S_ERR_TIMEOUT; every thread
// passes the three cluster barriers exactly once, so a CTA that gave up on a
// wait still lets its cluster finish.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "sm100_ptx.cuh"

namespace e2s {

bool make_score_map(CUtensorMap* map, const void* base, int heads, int64_t rows,
                    int64_t row_stride_el, int box_rows);

namespace {

constexpr int kTileKeys = 128;
constexpr int kHalfBytes = kTileKeys * 128;   // 128 rows x 64 bf16 (one half of d)
constexpr int kTileBytes = 2 * kHalfBytes;    // one tile of 128 keys x 128 d
constexpr int kMaxTpc = 2;                    // key tiles per CTA
constexpr int kMaxCluster = 8;
constexpr int kRows = 64;                     // text rows per unit (loaded twice)
constexpr int kQHalf = 2 * kRows * 128;       // one half of d of the doubled queries
constexpr int kD2Stride = 64;                 // TMEM columns per sweep-2 tile
constexpr int kEpiWarps = 8;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kWaitNsAfterFault = 1000000ull;
constexpr float kLog2e = 1.4426950408889634f;

struct SplitArgs {
  LayoutArgs la;
  int mode;
  int group;        // query heads per kv head
  int cluster;      // CTAs per unit
  int tpc;          // key tiles per CTA
  int num_units;
  uint32_t tmem_cols;
  float scale;      // 1 / sqrt(d)
  float scale_log2; // log2(e) / sqrt(d)
  const float* lse_in;   // nullable: natural-log lse of every text row [L][H][sum_text]
  float* a_out;
  float4* stats;
  uint32_t* counters;    // nullable: decision scratch to zero
  uint32_t* status;
};

struct SPlan {
  uint32_t q, k, bars, slot, ms, xch, nlse, red, spart, total;
};

__host__ __device__ inline SPlan split_plan(int tpc) {
  SPlan s;
  s.q = 0;
  s.k = 2u * kQHalf;
  s.bars = s.k + (uint32_t)tpc * kTileBytes;
  s.slot = s.bars + 8u * (3 + 2 * kMaxTpc);
  s.ms = (s.slot + 16u + 15u) & ~15u;                   // float2 [2][128]
  s.xch = s.ms + 2u * 128u * 8u;                        // float2 [kMaxCluster][kRows]
  s.nlse = s.xch + (uint32_t)kMaxCluster * kRows * 8u;  // float [kRows]
  s.red = s.nlse + kRows * 4u;                          // float4 [kEpiWarps]
  s.spart = s.red + kEpiWarps * 16u;                    // float4 [kMaxCluster]
  s.total = s.spart + kMaxCluster * 16u;
  return s;
}

// Geometry of one unit as seen by one CTA of its cluster; every warp role
// derives it identically.
struct SGeo {
  int b, l, h, kvh, S, NV, NT, t0, x0, v0;
  int key_base;   // key of the unit's first tile (0: whole prefix; S: visual keys only)
  int tile0;      // the CTA's first tile within the unit
  int nti;        // tiles of this CTA
  int vfirst;     // the CTA's first visual tile (local index), nvt of them
  int nvt;
  int ntp2;       // sweep-2 columns: text rows rounded up to 16
  bool ok, prefix;
};

// With a single image the host totals of the layout are the image's
// segments (S = sum_T - sum_vis - sum_text, N_V = sum_vis, N_T = sum_text),
// so no CTA waits on a load of the layout arrays before its first copy; the
// device arrays are still checked against them (layout_mismatch).
__device__ __forceinline__ SGeo split_geo(const SplitArgs& p, int unit, int rank) {
  const LayoutArgs& la = p.la;
  SGeo g;
  g.h = unit % la.H;
  g.l = (unit / la.H) % la.L;
  g.b = unit / (la.H * la.L);
  g.kvh = g.h / p.group;
  const bool one = la.B == 1;
  g.S = one ? la.sum_T - la.sum_vis - la.sum_text : __ldg(la.n_sys + g.b);
  g.NV = one ? la.sum_vis : __ldg(la.n_vis + g.b);
  g.NT = one ? la.sum_text : __ldg(la.n_text + g.b);
  g.t0 = one ? 0 : __ldg(la.tok_off + g.b);
  g.x0 = one ? 0 : __ldg(la.text_off + g.b);
  g.v0 = one ? 0 : __ldg(la.vis_off + g.b);
  const int T = g.S + g.NV + g.NT;
  g.prefix = p.mode == E2S_SCORE_CAUSAL_PROB && p.lse_in == nullptr;
  g.key_base = g.prefix ? 0 : g.S;
  const int span = g.prefix ? T : g.NV;
  const int n_all = (span + kTileKeys - 1) / kTileKeys;
  g.ok = g.S >= 0 && g.NV >= 0 && g.NT >= 1 && g.NT <= kRows && T <= la.max_T &&
         g.NV <= la.max_vis && n_all <= p.cluster * p.tpc;
  if (!one)
    g.ok = g.ok && __ldg(la.tok_off + g.b + 1) - g.t0 == T && g.t0 >= 0 &&
           g.t0 + T <= la.sum_T && __ldg(la.text_off + g.b + 1) - g.x0 == g.NT && g.x0 >= 0 &&
           g.x0 + g.NT <= la.sum_text && __ldg(la.vis_off + g.b + 1) - g.v0 == g.NV &&
           g.v0 >= 0 && g.v0 + g.NV <= la.sum_vis;
  g.tile0 = rank * p.tpc;
  g.nti = g.ok ? max(0, min(p.tpc, n_all - g.tile0)) : 0;
  g.vfirst = g.nti;
  g.nvt = 0;
  for (int i = 0; i < g.nti; ++i) {
    const int k0 = g.key_base + kTileKeys * (g.tile0 + i);
    if (k0 < g.S + g.NV && k0 + kTileKeys > g.S) {
      if (g.nvt == 0) g.vfirst = i;
      ++g.nvt;
    }
  }
  g.ntp2 = max(16, (g.NT + 15) & ~15);
  return g;
}

// Single image: whether the device layout arrays disagree with the host
// totals the kernel computed with.
__device__ __forceinline__ bool layout_mismatch(const LayoutArgs& la, const SGeo& g) {
  return __ldg(la.n_sys) != g.S || __ldg(la.n_vis) != g.NV || __ldg(la.n_text) != g.NT ||
         __ldg(la.tok_off) != 0 || __ldg(la.tok_off + 1) != la.sum_T ||
         __ldg(la.text_off) != 0 || __ldg(la.text_off + 1) != la.sum_text ||
         __ldg(la.vis_off) != 0 || __ldg(la.vis_off + 1) != la.sum_vis;
}

__global__ void __launch_bounds__(kThreads, 2)
    score_split_kernel(const __grid_constant__ CUtensorMap tmQ,
                       const __grid_constant__ CUtensorMap tmK, const SplitArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const SPlan plan = split_plan(p.tpc);
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);
  uint64_t* d1_free = q_full + 1;       // the epilogue has read D1 (kEpiWarps arrivals)
  uint64_t* mma2_done = d1_free + 1;    // sweep 2's accumulators are complete
  uint64_t* k_full = mma2_done + 1;     // [kMaxTpc]
  uint64_t* mma1 = k_full + kMaxTpc;    // [kMaxTpc]: tile i's sweep-1 MMAs are complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float2* ms = reinterpret_cast<float2*>(smem + plan.ms);
  float2* xch = reinterpret_cast<float2*>(smem + plan.xch);
  float* nlse = reinterpret_cast<float*>(smem + plan.nlse);
  float4* red = reinterpret_cast<float4*>(smem + plan.red);
  float4* spart = reinterpret_cast<float4*>(smem + plan.spart);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const int unit = blockIdx.x / p.cluster;
  const SGeo g = split_geo(p, unit, (int)rank);
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  ptx::cluster_arrive_relaxed();   // phase 0: every CTA of the cluster is running
  pdl_wait();   // inputs may come from the kernel before (launched with PDL)
  // only then may the next kernel be scheduled: the compaction that follows
  // in e2s_prune copies rows before its own wait
  pdl_launch_dependents();
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;
  if (rank == 0 && threadIdx.x == 0 && !g.ok) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);

  if (warp == 0 && lane == 0) {
    ptx::mbar_init(q_full, 1);
    ptx::mbar_init(d1_free, kEpiWarps);
    ptx::mbar_init(mma2_done, 1);
    for (int i = 0; i < kMaxTpc; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(mma1 + i, 1);
    }
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    // ================= TMA producer: the doubled queries, then the CTA's
    // tiles, issued before the TMEM allocation and the CTA barrier
    if (g.nti > 0) {
      ptx::mbar_arrive_expect_tx(q_full, 2u * kQHalf);
      const int qrow = g.l * la.sum_text + g.x0;
      for (int half = 0; half < 2; ++half)
        for (int copy = 0; copy < 2; ++copy)
          ptx::tma_load_3d(q_sm + half * kQHalf + copy * kRows * 128, &tmQ, q_full, half * 64,
                           g.h, qrow);
      for (int i = 0; i < g.nti; ++i) {
        const int row = g.l * la.sum_T + g.t0 + g.key_base + kTileKeys * (g.tile0 + i);
        ptx::mbar_arrive_expect_tx(k_full + i, kTileBytes);
        ptx::tma_load_3d(k_sm + i * kTileBytes, &tmK, k_full + i, 0, g.kvh, row);
        ptx::tma_load_3d(k_sm + i * kTileBytes + kHalfBytes, &tmK, k_full + i, 64, g.kvh, row);
      }
    }
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, p.tmem_cols);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;
  // sweep 2's accumulators: with two prefix tiles they take tile 0's columns
  // once sweep 1 has read tile 0; with one, the columns after it
  const uint32_t d2_base = (g.prefix && g.nti == 1) ? (uint32_t)kTileKeys : 0u;

  if (warp == 0) {
    // (the producer's copies were issued above)
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0 && g.nti > 0) {
      if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
      const uint32_t q_base = ptx::smem_addr(q_sm);
      if (g.prefix) {
        const uint32_t idesc = ptx::idesc_bf16_f32(128, 128);
        for (int i = 0; i < g.nti; ++i) {
          if (!ptx::mbar_wait(k_full + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const uint32_t k_base = ptx::smem_addr(k_sm + i * kTileBytes);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t half = ks >> 2, kk = ks & 3;
            const uint64_t ad = ptx::sdesc_sw128(q_base + half * kQHalf + kk * 32u);
            const uint64_t bd = ptx::sdesc_sw128(k_base + half * kHalfBytes + kk * 32u);
            ptx::mma_bf16(tmem + (uint32_t)(i * kTileKeys), ad, bd, idesc, ks > 0 ? 1u : 0u);
          }
          ptx::mma_commit(mma1 + i);
        }
      }
    }
    ptx::cluster_wait();     // phase 0
    ptx::cluster_arrive();   // phase 1: this warp publishes nothing, so it arrives early
    if (lane == 0 && g.nti > 0) {
      const uint32_t q_base = ptx::smem_addr(q_sm);
      if (g.prefix && g.nti > 1) {
        // sweep 2 overwrites tile 0's columns once every epilogue warp has read them
        if (!ptx::mbar_wait(d1_free, 0, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
      }
      if (g.nvt > 0) {
        const uint32_t idesc = ptx::idesc_bf16_f32(128, g.ntp2);
        for (int v = 0; v < g.nvt; ++v) {
          const int i = g.vfirst + v;
          if (!g.prefix && !ptx::mbar_wait(k_full + i, 0, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const uint32_t k_base = ptx::smem_addr(k_sm + i * kTileBytes);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t half = ks >> 2, kk = ks & 3;
            const uint64_t ad = ptx::sdesc_sw128(k_base + half * kHalfBytes + kk * 32u);
            const uint64_t bd = ptx::sdesc_sw128(q_base + half * kQHalf + kk * 32u);
            ptx::mma_bf16(tmem + d2_base + (uint32_t)(v * kD2Stride), ad, bd, idesc,
                          ks > 0 ? 1u : 0u);
          }
        }
      }
      ptx::mma_commit(mma2_done);
    }
  } else {
    // ================= epilogue, part 1: sweep 1 and this CTA's row partials
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int cg = ew >> 2;                   // 0 or 1
    const int lrow = q4 * 32 + lane;          // TMEM lane
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    if (g.prefix && g.nti > 0) {
      const int t = lrow & (kRows - 1);       // text row of this lane (both lane halves)
      const int lh = lrow >> 6;               // lane half: which half of each tile's keys
      const bool tvalid = t < g.NT;
      const bool warp_live = (q4 & 1) * 32 < g.NT;   // warp-uniform
      const int lim = g.S + g.NV + t;         // last key this row sees
      float m = kNegBig, ssum = 0.f;
      for (int i = 0; i < g.nti; ++i) {
        if (i == 1) {   // tile 0 read: sweep 2's MMAs may take its columns
          ptx::tc_fence_before();
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(d1_free);
        }
        if (!ptx::mbar_wait(mma1 + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        if (warp_live) {
#pragma unroll
          for (int ch = 0; ch < 2; ++ch) {
            const int c16 = 64 * lh + 32 * cg + 16 * ch;
            const int key0 = kTileKeys * (g.tile0 + i) + c16;
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * kTileKeys + c16), x);
            if (tvalid && key0 <= lim) {
              float cmax = kNegBig;
              if (key0 + 15 <= lim) {
#pragma unroll
                for (int j = 0; j < 16; ++j) cmax = fmaxf(cmax, x[j]);
              } else {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (key0 + j <= lim) cmax = fmaxf(cmax, x[j]);
              }
              const float mnew = fmaxf(m, cmax * p.scale_log2);
              float acc0 = ssum * fast_ex2(m - mnew), acc1 = 0.f;
              if (key0 + 15 <= lim) {
#pragma unroll
                for (int j = 0; j < 16; j += 2) {
                  acc0 += fast_ex2(fmaf(x[j], p.scale_log2, -mnew));
                  acc1 += fast_ex2(fmaf(x[j + 1], p.scale_log2, -mnew));
                }
              } else {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (key0 + j <= lim) acc0 += fast_ex2(fmaf(x[j], p.scale_log2, -mnew));
              }
              ssum = acc0 + acc1;
              m = mnew;
            }
          }
        }
      }
      ms[cg * 128 + lrow] = make_float2(m, ssum);
    }
    if (la.B == 1 && blockIdx.x == 0 && et == kEpiThreads - 1 && layout_mismatch(la, g))
      E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    ptx::named_bar(1, kEpiThreads);
    ptx::cluster_wait();   // phase 0: the other CTAs' shared memory may be written
    if (g.prefix && et < kRows) {
      // this CTA's partial of row et: lane halves 0/1 x column groups 0/1
      float M = kNegBig, L = 0.f;
      if (g.nti > 0) {
        const float2 v[4] = {ms[et], ms[et + kRows], ms[128 + et], ms[128 + et + kRows]};
#pragma unroll
        for (int c = 0; c < 4; ++c) M = fmaxf(M, v[c].x);
#pragma unroll
        for (int c = 0; c < 4; ++c) L += v[c].y * fast_ex2(v[c].x - M);
      }
      for (int r = 0; r < p.cluster; ++r)
        ptx::st_dsmem_f2(xch + rank * kRows + et, (uint32_t)r, make_float2(M, L));
    }
  }
  if (warp == 0) ptx::cluster_wait();   // phase 0
  if (warp != 1) ptx::cluster_arrive(); // phase 1: the row partials are exchanged
  ptx::cluster_wait();

  if (warp >= 2) {
    // ================= epilogue, part 2: lse, sweep 2, a and the statistics
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int cg = ew >> 2;
    const int lrow = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    if (et < kRows && causal) {
      float v = -kNegBig;
      if (et < g.NT && g.ok) {
        if (g.prefix) {   // the cluster's C partials of row et, in rank order
          float M = kNegBig, L = 0.f;
          for (int r = 0; r < p.cluster; ++r) M = fmaxf(M, xch[r * kRows + et].x);
          for (int r = 0; r < p.cluster; ++r) {
            const float2 x = xch[r * kRows + et];
            L += x.y * fast_ex2(x.x - M);
          }
          v = L > 0.f ? -(M + __log2f(L)) : -kNegBig;
        } else {
          v = -__ldg(p.lse_in + ((size_t)g.l * la.H + g.h) * la.sum_text + g.x0 + et) * kLog2e;
        }
      }
      nlse[et] = v;
    }
    if (g.nvt > 0) {
      if (!ptx::mbar_wait(mma2_done, 0, limit, p.status)) limit = kWaitNsAfterFault;
      ptx::tc_fence_after();
    }
    ptx::named_bar(1, kEpiThreads);
    const int nch = g.ntp2 >> 4;
    // warp (q4, cg) sums every column of tile cg for the 32 keys of lane
    // quarter q4, so each key's a is lane-local
    float a_key = 0.f;
    if (cg < g.nvt) {
      const int v = cg;
      float acc = 0.f;
      for (int c = 0; c < nch; ++c) {
        float x[16];
        ptx::tmem_ld16(tmem + lane_base + d2_base + (uint32_t)(v * kD2Stride + c * 16), x);
        if (causal) {
          float acc1 = 0.f;
          if (c * 16 + 15 < g.NT) {
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
              acc += fast_ex2(fmaf(x[j], p.scale_log2, nlse[c * 16 + j]));
              acc1 += fast_ex2(fmaf(x[j + 1], p.scale_log2, nlse[c * 16 + j + 1]));
            }
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (c * 16 + j < g.NT) acc += fast_ex2(fmaf(x[j], p.scale_log2, nlse[c * 16 + j]));
          }
          acc += acc1;
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c * 16 + j < g.NT) acc += x[j];
        }
      }
      a_key = acc;
    }
    const float a_mul = (causal ? 1.f : p.scale) / (float)max(g.NT, 1);
    float st_s = 0.f, st_m = kNegBig, st_e = 0.f;
    if (cg < g.nvt) {
      const int key = g.key_base + kTileKeys * (g.tile0 + g.vfirst + cg) + lrow;
      if (key >= g.S && key < g.S + g.NV) {
        const float a = a_key * a_mul;
        p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + (key - g.S)] = a;
        st_s = a;
        st_m = a * kLog2e;
        st_e = 1.f;
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
    if (lane == 0) red[ew] = make_float4(st_s, st_m, st_e, 0.f);
    ptx::named_bar(1, kEpiThreads);
    if (et == 0) {   // the warps in order, then to rank 0
      float S = 0.f, M = kNegBig, E = 0.f;
      for (int w = 0; w < kEpiWarps; ++w) {
        const float4 r = red[w];
        S += r.x;
        lse_merge(M, E, r.y, r.z);
      }
      ptx::st_dsmem_f4(spart + rank, 0u, make_float4(S, M, E, 0.f));
    }
    (void)lane_base;
  }
  ptx::cluster_arrive();   // phase 2: every CTA's statistics are with rank 0
  ptx::cluster_wait();
  if (rank == 0 && threadIdx.x == 64 && g.ok) {
    float S = 0.f, M = kNegBig, E = 0.f;
    for (int r = 0; r < p.cluster; ++r) {
      const float4 v = spart[r];
      S += v.x;
      lse_merge(M, E, v.y, v.z);
    }
    p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h] = stats_entry(S, M, E);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, p.tmem_cols);
  }
}

}  // namespace

// Cluster size and tiles per CTA for a launch, or false when this kernel does
// not take it: at most 64 text rows, and one wave of two CTAs per SM.
bool score_split_plan(const LayoutArgs& la, int mode, bool lse, int* cluster, int* tpc) {
  if (la.max_text > kRows || la.max_text < 1) return false;
  if (mode != E2S_SCORE_CAUSAL_PROB && mode != E2S_SCORE_EQ1) return false;
  const bool prefix = mode == E2S_SCORE_CAUSAL_PROB && !lse;
  const int span = prefix ? la.max_T : la.max_vis;
  const int n_all = (span + kTileKeys - 1) / kTileKeys;
  if (n_all < 1) return false;
  const long long units = (long long)la.B * la.L * la.H;
  const long long slots = 2LL * sm_count();
  for (int t = 1; t <= kMaxTpc; ++t) {
    const int c = (n_all + t - 1) / t;
    if (c <= kMaxCluster && units * c <= slots) {
      *cluster = c;
      *tpc = t;
      return true;
    }
  }
  return false;
}

cudaError_t launch_score_split(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                               const void* k, int64_t k_stride, float* a_out, float4* stats,
                               uint32_t* counters, uint32_t* status, cudaStream_t st,
                               const float* lse_in, int cluster, int tpc, bool pdl) {
  SplitArgs p;
  p.la = la;
  p.mode = mode;
  p.group = la.H / la.H_kv;
  p.cluster = cluster;
  p.tpc = tpc;
  p.num_units = la.B * la.L * la.H;
  // prefix: sweep 1's tiles (at most two, 128 columns each), sweep 2's
  // accumulators in tile 0's columns or after a single tile; visual keys
  // only: sweep 2's two tiles of at most 64 columns
  const bool prefix = mode == E2S_SCORE_CAUSAL_PROB && lse_in == nullptr;
  p.tmem_cols = prefix ? 256u : (uint32_t)(kMaxTpc * kD2Stride);
  p.scale = 1.0f / sqrtf(128.0f);
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.lse_in = lse_in;
  p.a_out = a_out;
  p.stats = stats;
  p.counters = counters;
  p.status = status;
  if (p.num_units == 0 || la.sum_vis == 0) return cudaSuccess;

  int dev = 0, smem_sm = 0, reserved = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
  size_t smem = split_plan(tpc).total + 1024;   // + alignment slack
  // Never more CTAs on an SM than its TMEM holds at once (512 columns): a CTA
  // blocked in tcgen05.alloc must not wait on a CTA that waits on its cluster.
  const int max_ctas = 512 / (int)p.tmem_cols;
  const size_t floor_smem = (size_t)smem_sm / (size_t)(max_ctas + 1) - (size_t)reserved + 128;
  if (smem < floor_smem) smem = floor_smem;
  CUtensorMap tmQ, tmK;
  if (!make_score_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_text, q_stride, kRows) ||
      !make_score_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTileKeys))
    return cudaErrorInvalidValue;
  return launch_kernel(score_split_kernel, dim3((unsigned)(p.num_units * cluster)),
                       dim3(kThreads), smem, st, cluster, pdl, tmQ, tmK, p);
}

}  // namespace e2s
