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
// kernel is persistent: one CTA per SM takes items in order (tile 0 of every
// unit first: the heaviest items) from a counter shared by all CTAs, so TMEM
// and the barriers are set up once, the CTAs stay balanced, and the loads of
// the next item overlap the end of the current one.  K and V tiles have three
// buffers each.
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
// Warp roles (384 threads): warp 0 issues O += P V, warp 1 allocates TMEM and
// issues S = Q K^T, warps 2-9 softmax / epilogue (warp w reads TMEM lane
// quarter w % 4, columns 64 * ((w - 2) / 4) .. of each tile), warp 10 loads K
// and Q, warp 11 loads V.  A thread that issues MMAs shares its SM
// sub-partition with two softmax warps; splitting the two MMA streams over two
// sub-partitions keeps their issue from falling behind the tensor pipe.  TMEM (512 columns): S buffers
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
// warp roles: the two MMA issuers sit on different SM sub-partitions (warp % 4)
// so neither shares its issue slots with more than two softmax warps
constexpr int kWarpPV = 0, kWarpQK = 1, kWarpLoadK = 10, kWarpLoadV = 11;
constexpr int kThreads = 32 * 12;
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
  uint32_t* sched;      // [0] items handed out after the first, [1] CTAs done (zero on entry)
  uint32_t* status;
};

constexpr int kStages = 3;           // K and V tile buffers each

struct APlan {
  uint32_t q, k, v, bars, slot, nlse, xch, red, total;
};

constexpr int kRing = 4;             // item slots shared by the roles
constexpr int kBars = 4 * kStages + 13 + 2 * kRing;

__host__ __device__ inline APlan attn_plan() {
  APlan s;
  s.q = 0;
  s.k = kTileBytes;
  s.v = s.k + kStages * kTileBytes;
  s.bars = s.v + kStages * kTileBytes;
  s.slot = s.bars + 8u * kBars;           // TMEM address, softmax flags [2], ring [kRing][8]
  s.nlse = (s.slot + 16u + 32u * kRing + 15u) & ~15u;   // float [128]
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

__device__ __forceinline__ float neg_inf() { return __int_as_float(0xff800000); }

// max of three (one instruction)
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Packed pairs of fp32 (one instruction per pair).
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}


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

// A ring entry: the item index (-1: no more items) and its image's geometry,
// so that only the K-load warp reads the layout arrays.
constexpr int kRingInts = 8;

__device__ __forceinline__ void ring_put(volatile int* e, int w, const AGeo& g) {
  e[0] = w;
  e[1] = g.S;
  e[2] = g.NV;
  e[3] = g.NT;
  e[4] = g.t0;
  e[5] = g.v0;
  e[6] = g.ok ? 1 : 0;
}

__device__ __forceinline__ AGeo ring_geo(const volatile int* e, const AttnArgs& p) {
  const LayoutArgs& la = p.la;
  AGeo g;
  const int w = e[0];
  const int unit = w % p.units;
  g.qt = w / p.units;
  g.h = unit % la.H;
  g.l = (unit / la.H) % la.L;
  g.b = unit / (la.H * la.L);
  g.kvh = g.h / p.group;
  g.S = e[1];
  g.NV = e[2];
  g.NT = e[3];
  g.t0 = e[4];
  g.v0 = e[5];
  g.ok = e[6] != 0;
  g.T = g.S + g.NV + g.NT;
  g.nq = g.ok ? (g.T + kTile - 1) / kTile : 0;
  g.row0 = g.T - kTile * (g.qt + 1);
  g.work = g.qt < g.nq;
  return g;
}

// Waits for ring slot k (false: the wait ran out).
__device__ __forceinline__ bool ring_wait(int k, uint64_t* item_full, uint64_t& limit,
                                          uint32_t* status) {
  if (ptx::mbar_wait(item_full + k % kRing, (k / kRing) & 1, limit, status)) return true;
  limit = kWaitNsAfterFault;
  return false;
}

// Per item: nk + nv key tiles and S tiles (nv visual key tiles of the score
// sweep), nk value tiles and P V accumulations.
enum { kOpsQK = 0, kOpsPV = 1 };

__device__ __forceinline__ int stream_ops(const AGeo& g, const AttnArgs& p, int kind) {
  const int nk = g.nq - g.qt;
  const int nv = p.a_out != nullptr && g.qt == 0 ? (g.NV + kTile - 1) / kTile : 0;
  return kind == kOpsQK ? nk + nv : nk;
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
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);
  uint64_t* q_free = q_full + 1;             // every MMA reading Q is complete
  uint64_t* k_full = q_free + 1;             // [kStages]
  uint64_t* k_free = k_full + kStages;       // [kStages]
  uint64_t* v_full = k_free + kStages;       // [kStages]
  uint64_t* v_free = v_full + kStages;       // [kStages]
  uint64_t* s_full = v_free + kStages;       // [2]
  uint64_t* s_free = s_full + 2;     // [2]
  uint64_t* p_ready = s_free + 2;    // [2] P buffer b written (and O rescaled if needed)
  uint64_t* pv_done = p_ready + 2;   // [2] the O += P V reading P buffer b is complete
  uint64_t* o_free = pv_done + 2;    // the item's O has been read out of TMEM
  uint64_t* fin = o_free + 1;        // every MMA of both issuers is complete
  uint64_t* kick = fin + 1;          // the first item's Q and first key tile have landed
  uint64_t* item_full = kick + 1;    // [kRing] ring slot written
  uint64_t* item_free = item_full + kRing;   // [kRing] ring slot read by every role
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  volatile int* sm_item = reinterpret_cast<volatile int*>(smem + plan.slot + 4);    // [2]
  volatile int* ring = reinterpret_cast<volatile int*>(smem + plan.slot + 16);      // [kRing][8]
  float* nlse = reinterpret_cast<float*>(smem + plan.nlse);
  float* xch = reinterpret_cast<float*>(smem + plan.xch);
  float4* red = reinterpret_cast<float4*>(smem + plan.red);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  uint64_t limit = kWaitNs;
  int pk_lk = 0, pk_j0 = 0;   // K-load warp: key tiles already issued, first j of item 0
  if (warp == kWarpLoadK && lane == 0) {
    ptx::prefetch_tensormap(&tmQ);
    ptx::prefetch_tensormap(&tmK);
    ptx::prefetch_tensormap(&tmV);
    ptx::mbar_init(q_full, 1);
    ptx::mbar_init(q_free, 1);
    for (int i = 0; i < kStages; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(k_free + i, 1);
      ptx::mbar_init(v_full + i, 1);
      ptx::mbar_init(v_free + i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(s_full + i, 1);
      ptx::mbar_init(s_free + i, kEpiWarps);
      ptx::mbar_init(p_ready + i, kEpiWarps);
      ptx::mbar_init(pv_done + i, 1);
    }
    ptx::mbar_init(o_free, kEpiWarps);
    ptx::mbar_init(fin, 2);
    ptx::mbar_init(kick, 1);
    for (int i = 0; i < kRing; ++i) {
      ptx::mbar_init(item_full + i, 1);
      ptx::mbar_init(item_free + i, 4);   // V loads, both MMA issuers, the softmax group
    }
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    // item 0 and, when it has work, its Q and first key tile go out before the
    // block-wide setup barrier: these loads are the first S's critical path
    const int w0 = (int)blockIdx.x;   // < items (the grid is at most the item count)
    const AGeo g0 = attn_geo(p, w0);
    if (!g0.ok && g0.qt == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    ring_put(ring, w0, g0);
    ptx::mbar_arrive(item_full);
    if (g0.work) {
      const int base_row = g0.l * la.sum_T + g0.t0;
      const int krow = base_row + g0.T - kTile * g0.nq;
      ptx::mbar_arrive_expect_tx(q_full, kTileBytes);
      ptx::tma_load_3d(q_sm, &tmQ, q_full, 0, g0.h, base_row + g0.row0);
      ptx::tma_load_3d(q_sm + kHalfBytes, &tmQ, q_full, 64, g0.h, base_row + g0.row0);
      ptx::mbar_arrive_expect_tx(k_full, kTileBytes);
      ptx::tma_load_3d(k_sm, &tmK, k_full, 0, g0.kvh, krow);
      ptx::tma_load_3d(k_sm + kHalfBytes, &tmK, k_full, 64, g0.kvh, krow);
      pk_lk = 1;
      pk_j0 = 1;
    }
  }
  if (warp == kWarpQK) ptx::tmem_alloc(tmem_slot, 512);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kWarpLoadK) {
    // ================= the item walk and TMA of each item's key tiles (then
    // the score sweep's visual key tiles) and its Q, which goes in once the
    // previous item's last S = Q K^T is complete (after the item's first two
    // key tiles).  A CTA's first item is its block index; the next ones come
    // from one counter shared by all CTAs, in item order (the heaviest query
    // tiles first), through the ring.  The first item's Q and first key tile
    // go out alone (before the setup barrier), so that the first S is not
    // queued behind every other load of the start.
    if (lane == 0) {
      int it = 0, lk = pk_lk;
      bool kicked = false;
      // the first value tile and the next key tiles wait for the first Q and
      // key tile (only this thread completes these phases: the waits cannot alias)
      auto kick_once = [&]() {
        if (kicked || lk == 0) return;
        if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
        if (!ptx::mbar_wait(k_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::mbar_arrive(kick);
        kicked = true;
      };
      auto publish = [&](int k, int w) {
        const int slot = k % kRing;
        if (k >= kRing && !ptx::mbar_wait(item_free + slot, (k / kRing - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        volatile int* e = ring + slot * kRingInts;
        if (w < p.items) {
          const AGeo g = attn_geo(p, w);
          if (!g.ok && g.qt == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
          ring_put(e, w, g);
        } else {
          e[0] = -1;
        }
        ptx::mbar_arrive(item_full + slot);
      };
      for (int k = 0;; ++k) {
        const volatile int* e = ring + (k % kRing) * kRingInts;
        if (e[0] < 0) break;
        const AGeo g = ring_geo(e, p);
        if (g.work) {
        const int nk = g.nq - g.qt;
        const int n = stream_ops(g, p, kOpsQK);
        const int base_row = g.l * la.sum_T + g.t0;   // row of image position 0 in the maps
        for (int j = k == 0 ? pk_j0 : 0; j < n; ++j) {
          kick_once();
          if (it == 0 ? j == 0 : j == min(2, n - 1)) {
            if (it >= 1 && !ptx::mbar_wait(q_free, (it - 1) & 1, limit, p.status))
              limit = kWaitNsAfterFault;
            ptx::mbar_arrive_expect_tx(q_full, kTileBytes);
            ptx::tma_load_3d(q_sm, &tmQ, q_full, 0, g.h, base_row + g.row0);
            ptx::tma_load_3d(q_sm + kHalfBytes, &tmQ, q_full, 64, g.h, base_row + g.row0);
          }
          const int s = lk % kStages;
          if (lk >= kStages && !ptx::mbar_wait(k_free + s, (lk / kStages - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          const int krow = j < nk ? base_row + g.T - kTile * (g.nq - j)
                                  : base_row + g.S + kTile * (j - nk);
          ptx::mbar_arrive_expect_tx(k_full + s, kTileBytes);
          ptx::tma_load_3d(k_sm + s * kTileBytes, &tmK, k_full + s, 0, g.kvh, krow);
          ptx::tma_load_3d(k_sm + s * kTileBytes + kHalfBytes, &tmK, k_full + s, 64, g.kvh, krow);
          ++lk;
        }
        kick_once();
        ++it;
        }
        // the next item is taken only once this item's loads are out and the
        // softmax has begun this item (every role has released item k - 1): taken
        // earlier, items would wait behind busy CTAs while others go idle
        if (k >= 1 && !ptx::mbar_wait(item_free + (k - 1) % kRing, ((k - 1) / kRing) & 1, limit,
                                      p.status))
          limit = kWaitNsAfterFault;
        publish(k + 1, (int)(gridDim.x + atomicAdd(p.sched, 1u)));
      }
      if (!kicked) ptx::mbar_arrive(kick);
    }
  } else if (warp == kWarpLoadV) {
    // ================= TMA: each item's value tiles
    if (lane == 0) {
      int lv = 0;
      for (int k = 0;; ++k) {
        const volatile int* e = ring + (k % kRing) * kRingInts;
        const bool more = ring_wait(k, item_full, limit, p.status) && e[0] >= 0;
        const AGeo g = ring_geo(e, p);
        ptx::mbar_arrive(item_free + k % kRing);
        if (!more) break;
        if (!g.work) continue;
        // the first value tile waits until the first Q and key tile have landed
        // (only here: the ring entries before it must still be released)
        if (lv == 0 && !ptx::mbar_wait(kick, 0, limit, p.status)) limit = kWaitNsAfterFault;
        const int base_row = g.l * la.sum_T + g.t0;
        for (int j = 0; j < g.nq - g.qt; ++j) {
          const int s = lv % kStages;
          if (lv >= kStages && !ptx::mbar_wait(v_free + s, (lv / kStages - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          const int krow = base_row + g.T - kTile * (g.nq - j);
          ptx::mbar_arrive_expect_tx(v_full + s, kTileBytes);
          ptx::tma_load_3d(v_sm + s * kTileBytes, &tmV, v_full + s, 0, g.kvh, krow);
          ptx::tma_load_3d(v_sm + s * kTileBytes + kHalfBytes, &tmV, v_full + s, 64, g.kvh, krow);
          ++lv;
        }
      }
    }
  } else if (warp == kWarpQK) {
    // ================= MMA: S = Q K^T for every key tile, then the score sweep
    if (lane == 0) {
      const uint32_t idesc_s = ptx::idesc_bf16_f32(kTile, kTile);
      int it = 0, sc = 0, lk = 0;
      for (int k = 0;; ++k) {
        const volatile int* e = ring + (k % kRing) * kRingInts;
        const bool more = ring_wait(k, item_full, limit, p.status) && e[0] >= 0;
        const AGeo g = ring_geo(e, p);
        ptx::mbar_arrive(item_free + k % kRing);
        if (!more) break;
        if (!g.work) continue;
        const int nk = g.nq - g.qt;
        const int n = stream_ops(g, p, kOpsQK);
        // score sweep: D[key][t] = K_vis Q_text^T, the text rows (the last ntp2
        // rows of the tile, an 8-row-aligned start) as N
        const int ntp2 = max(16, (g.NT + 15) & ~15);
        const uint32_t idesc_a = ptx::idesc_bf16_f32(kTile, ntp2);
        if (!ptx::mbar_wait(q_full, it & 1, limit, p.status)) limit = kWaitNsAfterFault;
        for (int j = 0; j < n; ++j) {
          const int sb = sc & 1, s = lk % kStages;
          if (sc >= 2 && !ptx::mbar_wait(s_free + sb, ((sc >> 1) - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          if (!ptx::mbar_wait(k_full + s, (lk / kStages) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const bool keys_on_lanes = j >= nk;
          const uint32_t q_base = ptx::smem_addr(q_sm) +
                                  (keys_on_lanes ? (uint32_t)(kTile - ntp2) * 128u : 0u);
          const uint32_t idesc = keys_on_lanes ? idesc_a : idesc_s;
          const uint32_t k_base = ptx::smem_addr(k_sm + s * kTileBytes);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t half = ks >> 2, k4 = ks & 3;
            const uint64_t qd = ptx::sdesc_sw128(q_base + half * kHalfBytes + k4 * 32u);
            const uint64_t kd = ptx::sdesc_sw128(k_base + half * kHalfBytes + k4 * 32u);
            ptx::mma_bf16(tmem + (uint32_t)sb * kColsS, keys_on_lanes ? kd : qd,
                          keys_on_lanes ? qd : kd, idesc, ks > 0 ? 1u : 0u);
          }
          ptx::mma_commit(k_free + s);
          ptx::mma_commit(s_full + sb);
          ++sc;
          ++lk;
        }
        ptx::mma_commit(q_free);   // every MMA reading this item's Q is issued
        ++it;
      }
      ptx::mma_commit(fin);
      if (!ptx::mbar_wait(fin, 0, limit, p.status)) limit = kWaitNsAfterFault;
    }
  } else if (warp == kWarpPV) {
    // ================= MMA: O += P V for every key tile
    if (lane == 0) {
      const uint32_t idesc_pv = ptx::idesc_bf16_f32(kTile, 128) | (1u << 16);   // B MN-major
      int it = 0, pc = 0, lv = 0;
      for (int k = 0;; ++k) {
        const volatile int* e = ring + (k % kRing) * kRingInts;
        const bool more = ring_wait(k, item_full, limit, p.status) && e[0] >= 0;
        const AGeo g = ring_geo(e, p);
        ptx::mbar_arrive(item_free + k % kRing);
        if (!more) break;
        if (!g.work) continue;
        for (int x = 0; x < g.nq - g.qt; ++x) {
          const int pb = pc & 1, s = lv % kStages;
          if (!ptx::mbar_wait(p_ready + pb, (pc >> 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          if (!ptx::mbar_wait(v_full + s, (lv / kStages) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          // the first P V of an item overwrites O: the previous item's O must be out
          if (x == 0 && it >= 1 && !ptx::mbar_wait(o_free, (it - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const uint32_t v_base = ptx::smem_addr(v_sm + s * kTileBytes);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t vd = sdesc_sw128_mn(v_base + (uint32_t)ks * 2048u, (uint32_t)kHalfBytes);
            mma_bf16_ts(tmem + kColO, tmem + kColP + (uint32_t)pb * 64u + (uint32_t)ks * 8u, vd,
                        idesc_pv, (x > 0 || ks > 0) ? 1u : 0u);
          }
          ptx::mma_commit(v_free + s);
          ptx::mma_commit(pv_done + pb);
          ++pc;
          ++lv;
        }
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
    for (int k = 0;; ++k) {
      // one thread takes the item from the ring for all eight warps, so they
      // always agree (their named barriers depend on it)
      if (threadIdx.x == 64) sm_item[k & 1] = ring_wait(k, item_full, limit, p.status) ? 1 : 0;
      ptx::named_bar(1, kEpiThreads);
      // every softmax warp has read entry k - 1 (it reached this barrier)
      if (threadIdx.x == 64 && k >= 1) ptx::mbar_arrive(item_free + (k - 1) % kRing);
      const volatile int* e = ring + (k % kRing) * kRingInts;
      if (sm_item[k & 1] == 0 || e[0] < 0) break;
      const AGeo g = ring_geo(e, p);
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
        for (int i = 0; i < 8; ++i) {
          mx[i] = max3f(s[i], s[i + 8], s[i + 16]);
          mx[i] = max3f(mx[i], s[i + 24], s[i + 32]);
          mx[i] = max3f(mx[i], s[i + 40], s[i + 48]);
          mx[i] = fmaxf(mx[i], s[i + 56]);
        }
        const float hmax = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]),
                                 fmaxf(mx[6], mx[7]));
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
        const uint64_t sc2 = f2_pack(p.scale_log2, p.scale_log2), nm2 = f2_pack(-mnew, -mnew);
        uint64_t acc2a = f2_pack(0.f, 0.f), acc2b = acc2a;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(s[2 * i], s[2 * i + 1]), sc2, nm2), x0, x1);
          const float e0 = fast_ex2(x0), e1 = fast_ex2(x1);
          if (i & 1) {
            acc2b = f2_add(acc2b, f2_pack(e0, e1));
          } else {
            acc2a = f2_add(acc2a, f2_pack(e0, e1));
          }
          pk[i] = pack_bf16(e0, e1);
        }
        float acc0, acc1, acc2, acc3;
        f2_unpack(acc2a, acc0, acc1);
        f2_unpack(acc2b, acc2, acc3);
        acc0 += acc2;
        acc1 += acc3;
        tmem_st32(tmem + lane_base + kColP + (uint32_t)pb * 64u + (uint32_t)(32 * ch), pk);
        ptx::tmem_wait_st();
        lsum = lsum * alpha + (acc0 + acc1);
        m = mnew;
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(p_ready + pb);
        ++pc;
      }
      // ---- O / l and the row normaliser (the two halves' sums meet in xch)
      xch[ch * kTile + r] = lsum;
      ptx::named_bar(pair_bar, 64);
      const float ltot = xch[r] + xch[kTile + r];
      ptx::named_bar(pair_bar, 64);   // xch is rewritten only after both halves read it
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
      {
        // O / l in bf16: the lane's 128 bytes of its row as eight 16-byte
        // chunks, transposed within each group of 8 lanes (three butterfly
        // exchanges) so that lane 8 g + i then holds chunk i of the group's 8
        // rows; each store instruction of the warp then writes 4 whole rows
        const float inv = ltot > 0.f ? 1.f / ltot : 0.f;
        uint32_t wd[32];
#pragma unroll
        for (int j2 = 0; j2 < 16; ++j2) {
          wd[j2] = pack_bf16(o0[2 * j2] * inv, o0[2 * j2 + 1] * inv);
          wd[16 + j2] = pack_bf16(o1[2 * j2] * inv, o1[2 * j2 + 1] * inv);
        }
#pragma unroll
        for (int d = 4; d >= 1; d >>= 1) {
          const bool upper = (lane & d) != 0;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            if ((c & d) != 0) continue;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint32_t send = upper ? wd[4 * c + q] : wd[4 * (c | d) + q];
              const uint32_t recv = __shfl_xor_sync(0xffffffffu, send, d);
              if (upper) {
                wd[4 * c + q] = recv;
              } else {
                wd[4 * (c | d) + q] = recv;
              }
            }
          }
        }
        const int grow = q4 * 32 + (lane & ~7);   // tile row of the lane group's first row
        uint16_t* obase = p.o_out + (int64_t)g.h * 128 + c0 + 8 * (lane & 7);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int qc = g.row0 + grow + c;        // image position of row grow + c
          if (qc >= 0)
            *reinterpret_cast<uint4*>(obase + (int64_t)(base_row + qc) * p.o_stride) =
                make_uint4(wd[4 * c], wd[4 * c + 1], wd[4 * c + 2], wd[4 * c + 3]);
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
        ptx::named_bar(1, kEpiThreads);   // nlse complete
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
  if (warp == kWarpQK) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
  if (threadIdx.x == 0) {
    // the last CTA out (every CTA has taken its last item) zeroes the counter
    __threadfence();
    if (atomicAdd(p.sched + 1, 1u) == gridDim.x - 1) {
      atomicExch(p.sched, 0u);
      atomicExch(p.sched + 1, 0u);
    }
  }
}

}  // namespace

cudaError_t launch_attention(const LayoutArgs& la, const void* q, int64_t q_stride, const void* k,
                             int64_t k_stride, const void* v, int64_t v_stride, void* o_out,
                             int64_t o_stride, float* lse_out, float* a_out, float4* stats,
                             uint32_t* counters, uint32_t* sched, uint32_t* status,
                             cudaStream_t st) {
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
  p.sched = sched;
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
