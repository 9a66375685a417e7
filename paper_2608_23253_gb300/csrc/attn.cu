// The pruning layer's own causal self-attention (flash-attention forward on
// tcgen05/TMEM), with the text-to-visual score of the decision as a
// by-product (Sec. 3.1; Sec. 6 names lower-overhead evidence caching as
// future work, and reading the score off the layer's attention pass is this
// library's reading of it).
//
// Work item = (image, layer, query head, 128-row query tile).  Query tiles are
// aligned to the END of each image's sequence, so tile 0 holds the last 128
// rows: every text row when N_T <= 128.  Key tiles are aligned the same way;
// query tile i attends to key tiles i .. n-1 (tile i is the diagonal).  The
// kernel is persistent: one CTA per SM walks the item list in passes of
// alternating direction (tile 0 of every unit first: the heaviest items), so
// TMEM and the barriers are set up once and the loads of the next item
// overlap the end of the current one (two Q buffers).
// Per key tile, in ascending key order:
//   MMA   S = Q K^T (query rows on the TMEM lanes, M = N = 128), two S buffers;
//   softmax warps (two per lane quarter, 64 columns each): the 64 values come
//         into registers in one TMEM load and masked keys become -inf; the two
//         halves of a row exchange their maxima through shared memory; the
//         row's reference maximum m moves only when the tile exceeds it by
//         more than kLazy (log2 units), so P = 2^(s - m) <= 2^kLazy and O is
//         rescaled (by 2^(m_old - m_new), in TMEM, after the previous P V)
//         only then; P goes in bf16 pairs into one of two TMEM buffers, so the
//         softmax of a tile overlaps the previous tile's P V;
//   MMA   O += P V, P the TMEM A operand, V the MN-major B operand straight
//         from its TMA tile.
// Then O / l goes out in bf16 and lse = (m + log2 l) ln 2 per row.  A tile-0
// item then has the final normaliser of every text row and, when the score is
// asked for, streams the image's visual key tiles once more with the keys on
// the lanes (D = K Q_text^T): a[n] = (1/N_T) sum_t 2^(s_tn - lse_t) is
// lane-local, and the Eq. 8 statistics of the unit's visual scores follow
// from the same lanes -- no other kernel reads K for the decision.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator and MMA
// issuer, warps 2-9 softmax / epilogue (warp w reads TMEM lane quarter w % 4,
// columns 64 * ((w - 2) / 4) .. of each tile).  TMEM (512 columns): S buffers
// at 0 and 128, O at 256, the two P buffers (64 columns each) at 384 and 448.
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
constexpr uint32_t kColP = 384;               // two P buffers of 64 columns (bf16 pairs)
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kWaitNsAfterFault = 1000000ull;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct AttnArgs {
  LayoutArgs la;
  int group;            // query heads per kv head
  int units;            // B * L * H
  int items;            // units * query tiles of the longest image
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
  uint32_t q, k, v, bars, slot, nlse, xch, xsum, red, total;
};

constexpr int kBars = 22;

__host__ __device__ inline APlan attn_plan() {
  APlan s;
  s.q = 0;                          // 2 buffers
  s.k = 2 * kTileBytes;             // 2 stages
  s.v = s.k + 2 * kTileBytes;       // 2 stages
  s.bars = s.v + 2 * kTileBytes;
  s.slot = s.bars + 8u * kBars;
  s.nlse = (s.slot + 16u + 15u) & ~15u;   // float [128]
  s.xch = s.nlse + kTile * 4u;            // float [2][2][128]: row maxima by tile parity
  s.xsum = s.xch + 4 * kTile * 4u;        // float [2][128]: row sums, score partials
  s.red = s.xsum + 2 * kTile * 4u;        // float4 [4]
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

__device__ __forceinline__ float neg_inf() { return __int_as_float(0xff800000); }

// D (TMEM) (+)= A B with A read from TMEM (row i of A on lane i; for 16-bit
// types two consecutive K elements per 32-bit column, the lower index in the
// low half) and B from a shared-memory descriptor.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// 32 consecutive 32-bit TMEM columns of the thread's lane (32x32b shape),
// waited for in the same statement so that no use of the registers can be
// scheduled before the wait.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {"
      "%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31"
      "}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
// 64 consecutive 32-bit TMEM columns of the thread's lane (32x32b shape),
// waited for in the same statement so that no use of the registers can be
// scheduled before the wait.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {"
      "%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, "
      "%32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, "
      "%48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63"
      "}, [%64];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]),
        "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]),
        "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]),
        "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]),
        "=r"(r[62]), "=r"(r[63])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}
// Store 32 consecutive 32-bit TMEM columns of the thread's lane (32x32b
// shape); tmem_wait_st() completes the store.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {"
      "%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32"
      "};"
      :
      : "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]),
        "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]),
        "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
}
struct AGeo {
  int b, l, h, kvh, qt, S, NV, NT, T, t0, v0;
  int nq;      // query (and key) tiles of the image
  int row0;    // image position of the tile's row 0 (may be negative)
  bool ok, work;
};

// Geometry of item w: unit w % units, query tile w / units.
__device__ __forceinline__ AGeo attn_geo(const AttnArgs& p, int w) {
  const LayoutArgs& la = p.la;
  AGeo g;
  const int unit = w % p.units;
  g.qt = w / p.units;
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

// The k-th item of this CTA: passes over the item list in alternating
// direction (increasing in k, so the walk ends at the first item >= items).
__device__ __forceinline__ int attn_item(int k) {
  const int G = (int)gridDim.x, c = (int)blockIdx.x;
  return k * G + ((k & 1) ? G - 1 - c : c);
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
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);   // [2]
  uint64_t* q_free = q_full + 2;     // [2] every MMA reading Q buffer b is complete
  uint64_t* k_full = q_free + 2;     // [2]
  uint64_t* k_free = k_full + 2;     // [2]
  uint64_t* v_full = k_free + 2;     // [2]
  uint64_t* v_free = v_full + 2;     // [2]
  uint64_t* s_full = v_free + 2;     // [2]
  uint64_t* s_free = s_full + 2;     // [2]
  uint64_t* p_ready = s_free + 2;    // [2] P buffer b written (and O rescaled if needed)
  uint64_t* pv_done = p_ready + 2;   // [2] the O += P V reading P buffer b is complete
  uint64_t* o_free = pv_done + 2;    // the item's O has been read out of TMEM
  uint64_t* fin = o_free + 1;        // every MMA of the CTA is complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float* nlse = reinterpret_cast<float*>(smem + plan.nlse);
  float* xch = reinterpret_cast<float*>(smem + plan.xch);
  float* xsum = reinterpret_cast<float*>(smem + plan.xsum);
  float4* red = reinterpret_cast<float4*>(smem + plan.red);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  if (warp == 0 && lane == 0) {
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(q_full + i, 1);
      ptx::mbar_init(q_free + i, 1);
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(k_free + i, 1);
      ptx::mbar_init(v_full + i, 1);
      ptx::mbar_init(v_free + i, 1);
      ptx::mbar_init(s_full + i, 1);
      ptx::mbar_init(s_free + i, kEpiWarps);
      ptx::mbar_init(p_ready + i, kEpiWarps);
      ptx::mbar_init(pv_done + i, 1);
    }
    ptx::mbar_init(o_free, kEpiWarps);
    ptx::mbar_init(fin, 1);
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
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
      int it = 0, lk = 0, lv = 0;
      auto load_k = [&](int krow, int kvh) {
        const int s = lk & 1;
        if (lk >= 2 && !ptx::mbar_wait(k_free + s, ((lk >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::mbar_arrive_expect_tx(k_full + s, kTileBytes);
        ptx::tma_load_3d(k_sm + s * kTileBytes, &tmK, k_full + s, 0, kvh, krow);
        ptx::tma_load_3d(k_sm + s * kTileBytes + kHalfBytes, &tmK, k_full + s, 64, kvh, krow);
        ++lk;
      };
      for (int kk = 0;; ++kk) {
        const int w = attn_item(kk);
        if (w >= p.items) break;
        const AGeo g = attn_geo(p, w);
        if (!g.work) continue;
        const int nk = g.nq - g.qt;
        const int nv = p.a_out != nullptr && g.qt == 0 ? (g.NV + kTile - 1) / kTile : 0;
        const int base_row = g.l * la.sum_T + g.t0;   // row of image position 0 in the maps
        const int qb = it & 1;
        if (it >= 2 && !ptx::mbar_wait(q_free + qb, ((it >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::mbar_arrive_expect_tx(q_full + qb, kTileBytes);
        ptx::tma_load_3d(q_sm + qb * kTileBytes, &tmQ, q_full + qb, 0, g.h, base_row + g.row0);
        ptx::tma_load_3d(q_sm + qb * kTileBytes + kHalfBytes, &tmQ, q_full + qb, 64, g.h,
                         base_row + g.row0);
        for (int jj = 0; jj < nk; ++jj) {
          const int krow = base_row + g.T - kTile * (g.nq - jj);
          load_k(krow, g.kvh);
          const int s = lv & 1;
          if (lv >= 2 && !ptx::mbar_wait(v_free + s, ((lv >> 1) - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::mbar_arrive_expect_tx(v_full + s, kTileBytes);
          ptx::tma_load_3d(v_sm + s * kTileBytes, &tmV, v_full + s, 0, g.kvh, krow);
          ptx::tma_load_3d(v_sm + s * kTileBytes + kHalfBytes, &tmV, v_full + s, 64, g.kvh,
                           krow);
          ++lv;
        }
        for (int vt = 0; vt < nv; ++vt) load_k(base_row + g.S + kTile * vt, g.kvh);
        ++it;
      }
    }
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0) {
      const uint32_t idesc_s = ptx::idesc_bf16_f32(kTile, kTile);
      const uint32_t idesc_pv = ptx::idesc_bf16_f32(kTile, 128) | (1u << 16);   // B MN-major
      int it = 0, sc = 0, pc = 0, lk = 0, lv = 0;
      auto qk = [&](uint32_t b_base, uint32_t idesc, bool keys_on_lanes) {
        const int sb = sc & 1;
        if (sc >= 2 && !ptx::mbar_wait(s_free + sb, ((sc >> 1) - 1) & 1, limit, p.status))
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
        ++sc;
        ++lk;
      };
      auto pv = [&](bool first) {
        const int pb = pc & 1;
        if (!ptx::mbar_wait(p_ready + pb, (pc >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        const int s = lv & 1;
        if (!ptx::mbar_wait(v_full + s, (lv >> 1) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        // the first P V of an item overwrites O: the previous item's O must be out
        if (first && it >= 1 && !ptx::mbar_wait(o_free, (it - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const uint32_t v_base = ptx::smem_addr(v_sm + s * kTileBytes);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint64_t vd = sdesc_sw128_mn(v_base + (uint32_t)ks * 2048u, (uint32_t)kHalfBytes);
          mma_bf16_ts(tmem + kColO, tmem + kColP + (uint32_t)pb * 64u + (uint32_t)ks * 8u, vd,
                      idesc_pv, (!first || ks > 0) ? 1u : 0u);
        }
        ptx::mma_commit(v_free + s);
        ptx::mma_commit(pv_done + pb);
        ++pc;
        ++lv;
      };
      for (int kk = 0;; ++kk) {
        const int w = attn_item(kk);
        if (w >= p.items) break;
        const AGeo g = attn_geo(p, w);
        if (!g.work) continue;
        const int nk = g.nq - g.qt;
        const int nv = p.a_out != nullptr && g.qt == 0 ? (g.NV + kTile - 1) / kTile : 0;
        const int ntp2 = max(16, (g.NT + 15) & ~15);   // text columns of the score sweep
        const int qb = it & 1;
        if (!ptx::mbar_wait(q_full + qb, (it >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const uint32_t q_base = ptx::smem_addr(q_sm + qb * kTileBytes);
        for (int jj = 0; jj < nk; ++jj) {
          qk(q_base, idesc_s, false);
          if (jj >= 1) pv(jj == 1);
        }
        pv(nk == 1);
        // score sweep: D[key][t] = K_vis Q_text^T, the text rows (the last ntp2
        // rows of the tile, an 8-row-aligned start) as N
        const uint32_t idesc_a = ptx::idesc_bf16_f32(kTile, ntp2);
        for (int vt = 0; vt < nv; ++vt)
          qk(q_base + (uint32_t)(kTile - ntp2) * 128u, idesc_a, true);
        ptx::mma_commit(q_free + qb);
        ++it;
      }
      ptx::mma_commit(fin);
      if (!ptx::mbar_wait(fin, 0, limit, p.status)) limit = kWaitNsAfterFault;
    }
  } else {
    // ================= softmax / epilogue: lane quarter q4, columns of half ch
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int ch = ew >> 2;                        // 0 or 1: tile columns 64 ch .. 64 ch + 63
    const int c0 = 64 * ch;
    const int r = q4 * 32 + lane;                  // TMEM lane (query row of the tile)
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const uint32_t pair_bar = 2u + (uint32_t)q4;   // the two warps of this lane quarter
    int it = 0, sc = 0, pc = 0;
    for (int kk = 0;; ++kk) {
      const int w = attn_item(kk);
      if (w >= p.items) break;
      const AGeo g = attn_geo(p, w);
      if (!g.ok && g.qt == 0 && threadIdx.x == 64) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
      if (!g.work) continue;
      const int nk = g.nq - g.qt;
      const bool sweep = p.a_out != nullptr && g.qt == 0 && g.NV > 0;
      const int nv = sweep ? (g.NV + kTile - 1) / kTile : 0;
      const int ntp2 = max(16, (g.NT + 15) & ~15);
      const int base_row = g.l * la.sum_T + g.t0;
      const int qp = g.row0 + r;                   // image position of this row
      const bool rvalid = qp >= 0;
      float m = kNegBig, lsum = 0.f;               // reference maximum and this half's sum
      for (int jj = 0; jj < nk; ++jj) {
        const int sb = sc & 1;
        const int kbase = g.T - kTile * (g.nq - jj);   // image position of the tile's key 0
        const int c_lo = max(0, -kbase), c_hi = min(kTile - 1, qp - kbase);
        const bool full = c_lo <= c0 && c_hi >= c0 + 63;
        if (!ptx::mbar_wait(s_full + sb, (sc >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        float s[64];
        tmem_ld64(tmem + lane_base + (uint32_t)sb * kColsS + (uint32_t)c0, s);
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(s_free + sb);   // S is in registers
        ++sc;
        if (__any_sync(0xffffffffu, !full)) {
#pragma unroll
          for (int i = 0; i < 64; ++i)
            s[i] = (c0 + i >= c_lo && c0 + i <= c_hi) ? s[i] : neg_inf();
        }
        // masked maximum of this half, then of the row (the other half's
        // through shared memory; the buffer alternates with the tile)
        float mx[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) mx[i] = fmaxf(s[i], s[i + 8]);
#pragma unroll
        for (int i = 16; i < 64; ++i) mx[i & 7] = fmaxf(mx[i & 7], s[i]);
        const float hmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                 fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
        float* xb = xch + (pc & 1) * 2 * kTile;
        xb[ch * kTile + r] = hmax;
        ptx::named_bar(pair_bar, 64);
        const float tmax = fmaxf(xb[r], xb[kTile + r]);
        const float tm = tmax > 0.5f * kNegBig ? tmax * p.scale_log2 : kNegBig;
        // the reference maximum moves only by more than kLazy (or from empty)
        const bool move = tm > m + kLazy || (m <= 0.5f * kNegBig && tm > 0.5f * kNegBig);
        const float mnew = move ? tm : m;
        const float alpha = move ? fast_ex2(m - mnew) : 1.f;
        if (jj >= 1 && __any_sync(0xffffffffu, move)) {
          // O of these rows is rescaled once the previous P V is complete
          const int pp = (pc - 1) & 1;
          if (!ptx::mbar_wait(pv_done + pp, ((pc - 1) >> 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          for (int h = 0; h < 4; ++h) {
            const uint32_t oa = tmem + lane_base + kColO + (uint32_t)(c0 + 16 * h);
            float o[16];
            ptx::tmem_ld16(oa, o);
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] *= alpha;
            ptx::tmem_st16(oa, o);
          }
          ptx::tmem_wait_st();
        }
        // P buffer pb is free once the P V two tiles back is complete
        const int pb = pc & 1;
        if (pc >= 2 && !ptx::mbar_wait(pv_done + pb, ((pc >> 1) - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        // P = 2^(s - m) in bf16 pairs: key 64 ch + 2 i + e -> P column 32 ch + i
        uint32_t pk[32];
        float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float e0 = fast_ex2(fmaf(s[2 * i], p.scale_log2, -mnew));
          const float e1 = fast_ex2(fmaf(s[2 * i + 1], p.scale_log2, -mnew));
          acc0 += e0;
          acc1 += e1;
          pk[i] = pack_bf16(e0, e1);
        }
        tmem_st32(tmem + lane_base + kColP + (uint32_t)pb * 64u + (uint32_t)(32 * ch), pk);
        ptx::tmem_wait_st();
        lsum = lsum * alpha + (acc0 + acc1);
        m = mnew;
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(p_ready + pb);
        ++pc;
      }
      // ---- O / l and the row normaliser (the two halves' sums meet in xsum)
      xsum[ch * kTile + r] = lsum;
      ptx::named_bar(pair_bar, 64);
      const float ltot = xsum[r] + xsum[kTile + r];
      {
        const int pl = (pc - 1) & 1;
        if (!ptx::mbar_wait(pv_done + pl, ((pc - 1) >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
      }
      ptx::tc_fence_after();
      float o0[32], o1[32];
      tmem_ld32(tmem + lane_base + kColO + (uint32_t)c0, o0);
      tmem_ld32(tmem + lane_base + kColO + (uint32_t)(c0 + 32), o1);
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(o_free);   // the next item's P V may overwrite O
      if (rvalid) {
        const float inv = ltot > 0.f ? 1.f / ltot : 0.f;
        uint4* orow = reinterpret_cast<uint4*>(
            p.o_out + (int64_t)(base_row + qp) * p.o_stride + (int64_t)g.h * 128 + c0);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          orow[j] = make_uint4(pack_bf16(o0[8 * j] * inv, o0[8 * j + 1] * inv),
                               pack_bf16(o0[8 * j + 2] * inv, o0[8 * j + 3] * inv),
                               pack_bf16(o0[8 * j + 4] * inv, o0[8 * j + 5] * inv),
                               pack_bf16(o0[8 * j + 6] * inv, o0[8 * j + 7] * inv));
          orow[4 + j] = make_uint4(pack_bf16(o1[8 * j] * inv, o1[8 * j + 1] * inv),
                                   pack_bf16(o1[8 * j + 2] * inv, o1[8 * j + 3] * inv),
                                   pack_bf16(o1[8 * j + 4] * inv, o1[8 * j + 5] * inv),
                                   pack_bf16(o1[8 * j + 6] * inv, o1[8 * j + 7] * inv));
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
        ptx::named_bar(1, kEpiThreads);   // nlse complete, xsum read by every warp
        const int c_text = ntp2 - g.NT;
        const float inv_nt = 1.f / (float)g.NT;
        float st_s = 0.f, st_m = kNegBig, st_e = 0.f;
        for (int vt = 0; vt < nv; ++vt) {
          const int sb = sc & 1;
          if (!ptx::mbar_wait(s_full + sb, (sc >> 1) & 1, limit, p.status))
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
          ++sc;
          xsum[ch * kTile + r] = acc;
          ptx::named_bar(pair_bar, 64);
          const int key = kTile * vt + r;   // visual index of this lane's key
          if (ch == 0 && key < g.NV) {
            const float a = (xsum[r] + xsum[kTile + r]) * inv_nt;
            p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + key] = a;
            const float al = a * kLog2e, mn = fmaxf(st_m, al);
            st_e = st_e * fast_ex2(st_m - mn) + fast_ex2(al - mn);
            st_m = mn;
            st_s += a;
          }
          ptx::named_bar(pair_bar, 64);   // xsum is rewritten by the next tile
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
          for (int w4 = 0; w4 < 4; ++w4) {
            S += red[w4].x;
            lse_merge(M, E, red[w4].y, red[w4].z);
          }
          p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h] = stats_entry(S, M, E);
        }
      }
      ++it;
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
  p.items = p.units * n_qt;
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
  const int grid = std::min(p.items, sm_count());
  return launch_kernel(attn_kernel, dim3((unsigned)grid), dim3(kThreads), smem, st, 0, false,
                       tmQ, tmK, tmV, p);
}

}  // namespace e2s
