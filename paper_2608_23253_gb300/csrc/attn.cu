// The pruning layer's own causal self-attention (flash-attention forward on
// tcgen05/TMEM), with the text-to-visual score of the decision as a
// by-product (Sec. 3.1; Sec. 6 names lower-overhead evidence caching as
// future work, and reading the score off the layer's attention pass is this
// library's reading of it).
//
// One CTA per (image, layer, query head, 128-row query tile).  Query tiles
// are aligned to the END of each image's sequence, so tile 0 holds the last
// 128 rows: every text row when N_T <= 128.  Key tiles are aligned the same
// way; query tile i attends to key tiles i .. n-1 (tile i is the diagonal).
// Per key tile, in ascending key order:
//   MMA   S = Q K^T (text rows on the TMEM lanes, M = N = 128), double-buffered;
//   softmax warps (two per lane quarter, 64 columns each; a row's two halves
//         exchange their maxima and, at the end, their sums through shared
//         memory): masked row maximum; the row's reference maximum m moves
//         only when the tile exceeds it by more than kLazy (log2 units), so P =
//         2^(s - m) <= 2^kLazy and O needs rescaling (by 2^(m_old - m_new), in
//         TMEM, after the previous P V) only then; P in bf16 into one of two
//         shared-memory buffers (the K-major, 128-byte-swizzled A operand), so
//         the softmax of a tile overlaps the previous tile's P V;
//   MMA   O += P V (V as the MN-major B operand straight from its TMA tile).
// Then O / l goes out in bf16 and lse = (m + log2 l) ln 2 per row.  Tile 0's
// CTA then has the final normaliser of every text row and, when the score is
// asked for, streams the image's visual key tiles once more with the keys on
// the lanes (D = K Q_text^T): a[n] = (1/N_T) sum_t 2^(s_tn - lse_t) is
// lane-local, and the Eq. 8 statistics of the unit's visual scores follow
// from the same lanes -- no other kernel reads K for the decision.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator and MMA
// issuer, warps 2-9 softmax / epilogue (warp w reads TMEM lane quarter w % 4,
// columns 64 * ((w - 2) / 4) .. of each tile).
// Every mbarrier wait is bounded and reports E2S_ERR_TIMEOUT.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "sm100_ptx.cuh"

namespace e2s {

bool make_score_map(CUtensorMap* map, const void* base, int heads, int64_t rows,
                    int64_t row_stride_el, int box_rows);

namespace {

constexpr int kTile = 128;                    // query rows and keys per tile
constexpr int kHalfBytes = kTile * 128;       // 128 rows x 64 bf16
constexpr int kTileBytes = 2 * kHalfBytes;
constexpr int kEpiWarps = 8;
constexpr float kLazy = 8.f;                  // log2 headroom of the reference maximum
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr uint32_t kColsS = 128;              // TMEM columns per S buffer
constexpr uint32_t kColO = 256;               // first TMEM column of the O accumulator
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kWaitNsAfterFault = 1000000ull;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct AttnArgs {
  LayoutArgs la;
  int group;            // query heads per kv head
  int units;            // B * L * H
  float scale_log2;     // log2(e) / sqrt(d)
  uint16_t* o_out;      // [L][sum_T] rows of (H x d) bf16
  int64_t o_stride;     // elements between consecutive rows
  float* lse_out;       // nullable [L][H][sum_T]
  float* a_out;         // nullable [L][H][sum_vis]
  float4* stats;        // per (image, layer, head), written with a_out
  uint32_t* counters;   // nullable: decision scratch to zero
  uint32_t* status;
};

struct APlan {
  uint32_t q, k, v, p, bars, slot, nlse, xch, red, total;
};

__host__ __device__ inline APlan attn_plan() {
  APlan s;
  s.q = 0;
  s.k = kTileBytes;                 // 2 stages
  s.v = s.k + 2 * kTileBytes;       // 2 stages
  s.p = s.v + 2 * kTileBytes;       // 2 buffers of P, each two 64-key halves of 128 rows
  s.bars = s.p + 2 * kTileBytes;
  s.slot = s.bars + 8u * 20u;
  s.nlse = (s.slot + 16u + 15u) & ~15u;   // float [128]
  s.xch = s.nlse + kTile * 4u;            // float [2][128]: the two column halves of a row
  s.red = s.xch + 2 * kTile * 4u;         // float4 [4]
  s.total = s.red + 4 * 16u;
  return s;
}

// MN-major 128-byte-swizzled operand descriptor (V as B): 64-element atoms
// along N are `lbo` bytes apart, 8-row atoms along K 1024 bytes apart.
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

struct AGeo {
  int b, l, h, kvh, qt, S, NV, NT, T, t0, v0;
  int nq;      // query (and key) tiles of the image
  int row0;    // image position of the tile's row 0 (may be negative)
  bool ok, work;
};

__device__ __forceinline__ AGeo attn_geo(const AttnArgs& p) {
  const LayoutArgs& la = p.la;
  AGeo g;
  const int unit = blockIdx.x % p.units;
  g.qt = blockIdx.x / p.units;
  g.h = unit % la.H;
  g.l = (unit / la.H) % la.L;
  g.b = unit / (la.H * la.L);
  g.kvh = g.h / p.group;
  g.S = __ldg(la.n_sys + g.b);
  g.NV = __ldg(la.n_vis + g.b);
  g.NT = __ldg(la.n_text + g.b);
  g.t0 = __ldg(la.tok_off + g.b);
  g.v0 = __ldg(la.vis_off + g.b);
  g.T = g.S + g.NV + g.NT;
  g.ok = g.S >= 0 && g.NV >= 0 && g.NT >= 1 && g.T <= la.max_T &&
         __ldg(la.tok_off + g.b + 1) - g.t0 == g.T && g.t0 >= 0 && g.t0 + g.T <= la.sum_T &&
         __ldg(la.vis_off + g.b + 1) - g.v0 == g.NV && g.v0 >= 0 && g.v0 + g.NV <= la.sum_vis &&
         (p.a_out == nullptr || g.NT <= kTile);
  g.nq = g.ok ? (g.T + kTile - 1) / kTile : 0;
  g.row0 = g.T - kTile * (g.qt + 1);
  g.work = g.qt < g.nq;
  return g;
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const AttnArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const APlan plan = attn_plan();
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint8_t* v_sm = smem + plan.v;
  uint8_t* p_sm = smem + plan.p;
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);
  uint64_t* k_full = q_full + 1;     // [2]
  uint64_t* k_free = k_full + 2;     // [2]
  uint64_t* v_full = k_free + 2;     // [2]
  uint64_t* v_free = v_full + 2;     // [2]
  uint64_t* s_full = v_free + 2;     // [2]
  uint64_t* s_free = s_full + 2;     // [2]
  uint64_t* p_ready = s_free + 2;    // [2] P buffer b written (and O rescaled if needed)
  uint64_t* pv_done = p_ready + 2;   // [2] the O += P V reading P buffer b is complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float* nlse = reinterpret_cast<float*>(smem + plan.nlse);
  float* xch = reinterpret_cast<float*>(smem + plan.xch);
  float4* red = reinterpret_cast<float4*>(smem + plan.red);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;
  const AGeo g = attn_geo(p);
  if (!g.ok && g.qt == 0 && threadIdx.x == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
  if (!g.work) return;   // a query tile beyond this image's rows
  const int nk = g.nq - g.qt;                     // key tiles of this query tile
  const bool sweep = p.a_out != nullptr && g.qt == 0 && g.NV > 0;
  const int nv = sweep ? (g.NV + kTile - 1) / kTile : 0;
  const int ntp2 = max(16, (g.NT + 15) & ~15);    // text columns of the score sweep

  if (warp == 0 && lane == 0) {
    ptx::mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(k_free + i, 1);
      ptx::mbar_init(v_full + i, 1);
      ptx::mbar_init(v_free + i, 1);
      ptx::mbar_init(s_full + i, 1);
      ptx::mbar_init(s_free + i, kEpiWarps);
      ptx::mbar_init(p_ready + i, kEpiWarps);
      ptx::mbar_init(pv_done + i, 1);
    }
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, 512);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;
  const int base_row = g.l * la.sum_T + g.t0;     // row of image position 0 in the maps

  if (warp == 0) {
    // ================= TMA producer
    if (lane == 0) {
      ptx::mbar_arrive_expect_tx(q_full, kTileBytes);
      ptx::tma_load_3d(q_sm, &tmQ, q_full, 0, g.h, base_row + g.row0);
      ptx::tma_load_3d(q_sm + kHalfBytes, &tmQ, q_full, 64, g.h, base_row + g.row0);
      int lk = 0, lv = 0;
      auto load_k = [&](int krow) {
        const int s = lk & 1;
        if (lk >= 2 && !ptx::mbar_wait(k_free + s, ((lk >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::mbar_arrive_expect_tx(k_full + s, kTileBytes);
        ptx::tma_load_3d(k_sm + s * kTileBytes, &tmK, k_full + s, 0, g.kvh, krow);
        ptx::tma_load_3d(k_sm + s * kTileBytes + kHalfBytes, &tmK, k_full + s, 64, g.kvh, krow);
        ++lk;
      };
      for (int jj = 0; jj < nk; ++jj) {
        const int j = g.nq - 1 - jj;
        const int krow = base_row + g.T - kTile * (j + 1);
        load_k(krow);
        const int s = lv & 1;
        if (lv >= 2 && !ptx::mbar_wait(v_free + s, ((lv >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::mbar_arrive_expect_tx(v_full + s, kTileBytes);
        ptx::tma_load_3d(v_sm + s * kTileBytes, &tmV, v_full + s, 0, g.kvh, krow);
        ptx::tma_load_3d(v_sm + s * kTileBytes + kHalfBytes, &tmV, v_full + s, 64, g.kvh, krow);
        ++lv;
      }
      for (int vt = 0; vt < nv; ++vt) load_k(base_row + g.S + kTile * vt);
    }
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0) {
      if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
      const uint32_t q_base = ptx::smem_addr(q_sm);
      const uint32_t idesc_s = ptx::idesc_bf16_f32(kTile, kTile);
      const uint32_t idesc_pv = ptx::idesc_bf16_f32(kTile, 128) | (1u << 16);   // B MN-major
      int lk = 0, lv = 0;
      auto qk = [&](int jj, uint32_t b_base, uint32_t idesc, bool keys_on_lanes) {
        const int sb = jj & 1;
        if (jj >= 2 && !ptx::mbar_wait(s_free + sb, ((jj >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        const int s = lk & 1;
        if (!ptx::mbar_wait(k_full + s, (lk >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const uint32_t k_base = ptx::smem_addr(k_sm + s * kTileBytes);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t half = ks >> 2, kk = ks & 3;
          const uint64_t qd = ptx::sdesc_sw128(b_base + half * kHalfBytes + kk * 32u);
          const uint64_t kd = ptx::sdesc_sw128(k_base + half * kHalfBytes + kk * 32u);
          ptx::mma_bf16(tmem + (uint32_t)sb * kColsS, keys_on_lanes ? kd : qd,
                        keys_on_lanes ? qd : kd, idesc, ks > 0 ? 1u : 0u);
        }
        ptx::mma_commit(k_free + s);
        ptx::mma_commit(s_full + sb);
        ++lk;
      };
      auto pv = [&](int x) {
        const int pb = x & 1;
        if (!ptx::mbar_wait(p_ready + pb, (x >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        const int s = lv & 1;
        if (!ptx::mbar_wait(v_full + s, (lv >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const uint32_t p_base = ptx::smem_addr(p_sm + pb * kTileBytes);
        const uint32_t v_base = ptx::smem_addr(v_sm + s * kTileBytes);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t half = ks >> 2, kk = ks & 3;
          const uint64_t pd = ptx::sdesc_sw128(p_base + half * kHalfBytes + kk * 32u);
          const uint64_t vd = sdesc_sw128_mn(v_base + (uint32_t)ks * 2048u, (uint32_t)kHalfBytes);
          ptx::mma_bf16(tmem + kColO, pd, vd, idesc_pv, (x > 0 || ks > 0) ? 1u : 0u);
        }
        ptx::mma_commit(v_free + s);
        ptx::mma_commit(pv_done + pb);
        ++lv;
      };
      for (int jj = 0; jj < nk; ++jj) {
        qk(jj, q_base, idesc_s, false);
        if (jj >= 1) pv(jj - 1);
      }
      pv(nk - 1);
      // score sweep: D[key][t] = K_vis Q_text^T, the text rows (the last ntp2
      // rows of the tile, an 8-row-aligned start) as N
      const uint32_t idesc_a = ptx::idesc_bf16_f32(kTile, ntp2);
      for (int vt = 0; vt < nv; ++vt)
        qk(nk + vt, q_base + (uint32_t)(kTile - ntp2) * 128u, idesc_a, true);
    }
  } else {
    // ================= softmax / epilogue: lane quarter q4, columns of half ch
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int ch = ew >> 2;                        // 0 or 1: tile columns 64 ch .. 64 ch + 63
    const int r = q4 * 32 + lane;                  // TMEM lane (query row of the tile)
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const uint32_t pair_bar = 2u + (uint32_t)q4;   // the two warps of this lane quarter
    const int qp = g.row0 + r;                     // image position of this row
    const bool rvalid = qp >= 0;
    float m = kNegBig, lsum = 0.f;                 // reference maximum and this half's sum
    for (int jj = 0; jj < nk; ++jj) {
      const int sb = jj & 1, pb = jj & 1;
      const int kbase = g.T - kTile * (g.nq - jj);   // image position of the tile's key 0
      const int c_lo = max(0, -kbase), c_hi = min(kTile - 1, qp - kbase);
      const int c0 = 64 * ch;
      const bool full = c_lo <= c0 && c_hi >= c0 + 63;
      if (!ptx::mbar_wait(s_full + sb, (jj >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
      ptx::tc_fence_after();
      const uint32_t sa = tmem + lane_base + (uint32_t)sb * kColsS + (uint32_t)c0;
      // pass 1: masked maximum of this half, then of the row (the other half's
      // through shared memory)
      float hmax = kNegBig;
      for (int c16 = 0; c16 < 64; c16 += 16) {
        float x[16];
        ptx::tmem_ld16(sa + c16, x);
        if (full) {
#pragma unroll
          for (int i = 0; i < 16; ++i) hmax = fmaxf(hmax, x[i]);
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (c0 + c16 + i >= c_lo && c0 + c16 + i <= c_hi) hmax = fmaxf(hmax, x[i]);
        }
      }
      xch[ch * kTile + r] = hmax;
      ptx::named_bar(pair_bar, 64);
      const float tmax = fmaxf(xch[r], xch[kTile + r]);
      ptx::named_bar(pair_bar, 64);   // xch is rewritten only after both halves read it
      const float tm = tmax > 0.5f * kNegBig ? tmax * p.scale_log2 : kNegBig;
      // the reference maximum moves only by more than kLazy (or from empty)
      const bool move = tm > m + kLazy || (m <= 0.5f * kNegBig && tm > 0.5f * kNegBig);
      const float mnew = move ? tm : m;
      const float alpha = move ? fast_ex2(m - mnew) : 1.f;
      if (jj >= 1 && __any_sync(0xffffffffu, move)) {
        // O of these rows is rescaled once the previous P V is complete
        const int pp = (jj - 1) & 1;
        if (!ptx::mbar_wait(pv_done + pp, ((jj - 1) >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        for (int c16 = 0; c16 < 64; c16 += 16) {
          float x[16];
          ptx::tmem_ld16(tmem + lane_base + kColO + (uint32_t)(c0 + c16), x);
#pragma unroll
          for (int i = 0; i < 16; ++i) x[i] *= alpha;
          ptx::tmem_st16(tmem + lane_base + kColO + (uint32_t)(c0 + c16), x);
        }
        ptx::tmem_wait_st();
      }
      // P buffer pb is free once the P V two tiles back is complete
      if (jj >= 2 && !ptx::mbar_wait(pv_done + pb, ((jj >> 1) - 1) & 1, limit, p.status))
        limit = kWaitNsAfterFault;
      // pass 2: P = 2^(s - m) in bf16 into this half's 64-key half of the A operand
      uint8_t* prow = p_sm + pb * kTileBytes + ch * kHalfBytes + r * 128;
      float acc = 0.f;
      for (int c16 = 0; c16 < 64; c16 += 16) {
        float x[16];
        ptx::tmem_ld16(sa + c16, x);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const bool vis = full || (c0 + c16 + i >= c_lo && c0 + c16 + i <= c_hi);
          x[i] = vis ? fast_ex2(fmaf(x[i], p.scale_log2, -mnew)) : 0.f;
          acc += x[i];
        }
#pragma unroll
        for (int h8 = 0; h8 < 2; ++h8) {
          const int chunk = (c16 >> 3) + h8;
          uint4 w;
          w.x = pack_bf16(x[8 * h8 + 0], x[8 * h8 + 1]);
          w.y = pack_bf16(x[8 * h8 + 2], x[8 * h8 + 3]);
          w.z = pack_bf16(x[8 * h8 + 4], x[8 * h8 + 5]);
          w.w = pack_bf16(x[8 * h8 + 6], x[8 * h8 + 7]);
          *reinterpret_cast<uint4*>(prow + ((chunk ^ (r & 7)) << 4)) = w;
        }
      }
      lsum = lsum * alpha + acc;
      m = mnew;
      ptx::fence_proxy_async_smem();   // P's generic-proxy stores -> the tensor core
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        ptx::mbar_arrive(s_free + sb);
        ptx::mbar_arrive(p_ready + pb);
      }
    }
    // ---- O / l and the row normaliser (the two halves' sums meet in xch)
    xch[ch * kTile + r] = lsum;
    ptx::named_bar(pair_bar, 64);
    const float ltot = xch[r] + xch[kTile + r];
    const int pl = (nk - 1) & 1;
    if (!ptx::mbar_wait(pv_done + pl, ((nk - 1) >> 1) & 1, limit, p.status))
      limit = kWaitNsAfterFault;
    ptx::tc_fence_after();
    const float inv = ltot > 0.f ? 1.f / ltot : 0.f;
    uint16_t* orow =
        p.o_out + (int64_t)(base_row + qp) * p.o_stride + (int64_t)g.h * 128 + 64 * ch;
    for (int c16 = 0; c16 < 64; c16 += 16) {
      float x[16];
      ptx::tmem_ld16(tmem + lane_base + kColO + (uint32_t)(64 * ch + c16), x);
      if (rvalid) {
        uint4 w0, w1;
        w0.x = pack_bf16(x[0] * inv, x[1] * inv);
        w0.y = pack_bf16(x[2] * inv, x[3] * inv);
        w0.z = pack_bf16(x[4] * inv, x[5] * inv);
        w0.w = pack_bf16(x[6] * inv, x[7] * inv);
        w1.x = pack_bf16(x[8] * inv, x[9] * inv);
        w1.y = pack_bf16(x[10] * inv, x[11] * inv);
        w1.z = pack_bf16(x[12] * inv, x[13] * inv);
        w1.w = pack_bf16(x[14] * inv, x[15] * inv);
        *reinterpret_cast<uint4*>(orow + c16) = w0;
        *reinterpret_cast<uint4*>(orow + c16 + 8) = w1;
      }
    }
    const float lse2 = ltot > 0.f ? m + __log2f(ltot) : -kNegBig;
    if (ch == 0) {
      if (rvalid && p.lse_out != nullptr)
        p.lse_out[((int64_t)g.l * la.H + g.h) * la.sum_T + g.t0 + qp] = lse2 * kLn2;
      nlse[r] = -lse2;
    }
    if (sweep) {
      // ---- the score from the final row normalisers: keys on the lanes,
      // column c <-> tile row kTile - ntp2 + c <-> text row c - (ntp2 - NT);
      // the two warps of a lane quarter take alternate 16-column chunks
      ptx::named_bar(1, kEpiThreads);   // nlse complete, xch free
      const int c_text = ntp2 - g.NT;
      const float inv_nt = 1.f / (float)g.NT;
      float st_s = 0.f, st_m = kNegBig, st_e = 0.f;
      for (int vt = 0; vt < nv; ++vt) {
        const int jj = nk + vt, sb = jj & 1;
        if (!ptx::mbar_wait(s_full + sb, (jj >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        float acc = 0.f;
        for (int c16 = 16 * ch; c16 < ntp2; c16 += 32) {
          float x[16];
          ptx::tmem_ld16(tmem + lane_base + (uint32_t)sb * kColsS + c16, x);
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (c16 + i >= c_text)
              acc += fast_ex2(fmaf(x[i], p.scale_log2, nlse[kTile - ntp2 + c16 + i]));
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(s_free + sb);
        xch[ch * kTile + r] = acc;
        ptx::named_bar(pair_bar, 64);
        const int key = kTile * vt + r;   // visual index of this lane's key
        if (ch == 0 && key < g.NV) {
          const float a = (xch[r] + xch[kTile + r]) * inv_nt;
          p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + key] = a;
          const float al = a * kLog2e, mn = fmaxf(st_m, al);
          st_e = st_e * fast_ex2(st_m - mn) + fast_ex2(al - mn);
          st_m = mn;
          st_s += a;
        }
        ptx::named_bar(pair_bar, 64);   // xch is rewritten by the next tile
      }
      if (ch == 0) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float s2 = __shfl_xor_sync(0xffffffffu, st_s, o);
          const float m2 = __shfl_xor_sync(0xffffffffu, st_m, o);
          const float e2 = __shfl_xor_sync(0xffffffffu, st_e, o);
          st_s += s2;
          lse_merge(st_m, st_e, m2, e2);
        }
        if (lane == 0) red[q4] = make_float4(st_s, st_m, st_e, 0.f);
      }
      ptx::named_bar(1, kEpiThreads);
      if (r == 0 && ch == 0) {   // the four lane quarters in order
        float S = 0.f, M = kNegBig, E = 0.f;
        for (int w = 0; w < 4; ++w) {
          S += red[w].x;
          lse_merge(M, E, red[w].y, red[w].z);
        }
        p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h] = stats_entry(S, M, E);
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

cudaError_t launch_attention(const LayoutArgs& la, const void* q, int64_t q_stride, const void* k,
                             int64_t k_stride, const void* v, int64_t v_stride, void* o_out,
                             int64_t o_stride, float* lse_out, float* a_out, float4* stats,
                             uint32_t* counters, uint32_t* status, cudaStream_t st) {
  AttnArgs p;
  p.la = la;
  p.group = la.H / la.H_kv;
  p.units = la.B * la.L * la.H;
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.o_out = static_cast<uint16_t*>(o_out);
  p.o_stride = o_stride;
  p.lse_out = lse_out;
  p.a_out = a_out;
  p.stats = stats;
  p.counters = counters;
  p.status = status;
  if (p.units == 0 || la.max_T == 0) return cudaSuccess;
  const int n_qt = (la.max_T + kTile - 1) / kTile;
  CUtensorMap tmQ, tmK, tmV;
  if (!make_score_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_T, q_stride, kTile) ||
      !make_score_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTile) ||
      !make_score_map(&tmV, v, la.H_kv, (int64_t)la.L * la.sum_T, v_stride, kTile))
    return cudaErrorInvalidValue;
  const size_t smem = attn_plan().total + 1024;   // + alignment slack
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  if ((size_t)optin < smem) return cudaErrorInvalidConfiguration;
  return launch_kernel(attn_kernel, dim3((unsigned)(p.units * n_qt)), dim3(kThreads), smem, st,
                       0, false, tmQ, tmK, tmV, p);
}

}  // namespace e2s
