// Text-to-visual score, streaming variant for long sequences and grouped-query
// attention (tcgen05 + TMEM, TMA-streamed bf16 K tiles; Sec. 3.1 Eq. 1 and its
// causal-prefix probability reading).  Used when a unit's K does not fit in
// shared memory or its heads share K (GQA), for at most 128 text rows.
//
// One CTA per SM loops over units (image, layer, query heads); query head h
// reads kv head h / (H / H_kv).  When the text rows leave room, the query
// heads of one kv head are stacked into the 128 TMEM lanes (two heads of up to
// 64 rows, or four of up to 32), so that they share one stream of K tiles.
// Each key tile of 128 keys is one MMA with K = d = 128, in one of two
// orientations:
//   sweep 1 every key tile of the causal prefix (keys 0 .. S+N_V+N_T-1),
//           D[t][key] = Q[t][:] . K[key][:], text rows on the TMEM lanes:
//           each lane keeps a running (max, sum of exp2) of its row over the
//           32 columns its warp reads -- no cross-lane work; at the end the
//           four column groups merge into lse_t (log2 domain) per row;
//   sweep 2 the visual tiles again (the MMAs are recomputed from re-streamed
//           K), D[key][t] = K[key][:] . Q[t][:], keys on the TMEM lanes and
//           the text rows (rounded up to 16) on the columns: each lane sums
//           P = exp2(s - lse_t) over the text rows of its column chunks, the
//           chunk partials of a key are added in a fixed order through shared
//           memory, and a[key] = sum_t P / N_T.
// EQ1 mode has no sweep 1 and sums s / sqrt(d) / N_T in sweep 2.  Neither has
// CAUSAL_PROB when the caller supplies each text row's lse from the layer's
// own attention pass (lse_in): sweep 2 alone then streams the visual tiles.
// K tiles stream through a ring of as many stages as shared memory holds
// (TMA producer warp; deep enough to cover the load latency), the accumulator
// is double-buffered in TMEM (MMA warp), so loads, MMAs and the epilogue of
// consecutive tiles overlap.  Short units (under 24 key tiles on average)
// get a second query buffer in place of a ring stage, so the next unit's
// queries are in before the current unit ends.  With fewer than 16 units per
// CTA the units come from a counter in the workspace, handed by the producer
// to the other roles through a small shared-memory ring (heaviest images
// first below 6 units per CTA); otherwise they go round-robin.  In batches of
// mixed text length the units of at most 64 rows still run split.  Every
// image's layout is staged in shared memory once per CTA.
//
// Warp roles (608 threads): warp 0 TMA producer, warp 1 TMEM allocator and MMA
// issuer of the even tiles, warp 18 MMA issuer of the odd tiles, warps 2-17
// epilogue: warp w reads TMEM lane quarter w % 4 and column group (w - 2) / 4
// (32 keys of each tile in sweep 1, column chunks in sweep 2).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "sm100_ptx.cuh"

namespace e2s {

bool make_score_map(CUtensorMap* map, const void* base, int heads, int64_t rows,
                    int64_t row_stride_el, int box_rows);

namespace {

constexpr int kRows = 128;                    // text rows per unit (M)
constexpr int kTileKeys = 128;                // keys per tile (N)
constexpr int kHalfBytes = 128 * 128;         // 128 rows x 64 bf16
constexpr int kTileBytes = 2 * kHalfBytes;    // one 128 x 128 bf16 operand
constexpr int kMaxStages = 8;                 // K ring depth: as many as shared memory holds
constexpr int kMaxBatch = 8;                  // sweep-2 tiles of a batch unit (whole TMEM)
constexpr int kQBufs = 2;                     // query buffers at most (p.qbufs: 1 or 2)
constexpr int kTmemCols = 512;                // two 128-column accumulators, or a batch
constexpr int kEpiWarps = 16;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kMmaWarp1 = 2 + kEpiWarps;      // the second MMA issuer (odd tiles)
constexpr int kThreads = 64 + kEpiThreads + 32;
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kWaitNsAfterFault = 1000000ull;
constexpr float kLog2e = 1.4426950408889634f;

// Two fp32 lanes in one 64-bit register: packed FMA and add (fma.rn.f32x2,
// add.rn.f32x2), each lane rounded exactly as fmaf / + would round it.
__device__ __forceinline__ uint64_t f2pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// sum over 16 logits of exp2(x * s + n_j), even and odd lanes accumulated
// separately from (acc_even, acc_odd), then added
__device__ __forceinline__ float exp2_sum16(const float (&x)[16], float s, const float (&n)[16],
                                            float acc_even) {
  const uint64_t s2 = f2pack(s, s);
  uint64_t acc = f2pack(acc_even, 0.f);
#pragma unroll
  for (int j = 0; j < 16; j += 2) {
    float t0, t1;
    f2unpack(ffma2(f2pack(x[j], x[j + 1]), s2, f2pack(n[j], n[j + 1])), t0, t1);
    acc = fadd2(acc, f2pack(fast_ex2(t0), fast_ex2(t1)));
  }
  float a0, a1;
  f2unpack(acc, a0, a1);
  return a0 + a1;
}

struct StreamArgs {
  LayoutArgs la;
  int mode;
  int stages;           // K ring stages (2 .. kMaxStages)
  int group;            // query heads per kv head
  int upk;              // units per kv head: ceil(group / stacked heads)
  int num_units;
  float scale;          // 1 / sqrt(d)
  float scale_log2;     // log2(e) / sqrt(d)
  const float* lse_in;  // nullable: natural-log lse of every text row, [L][H][sum_text]
  float* a_out;
  float4* stats;        // per (image, layer, head) statistics of the visual scores
  uint32_t* counters;   // nullable: decision scratch to zero
  uint32_t* status;
  uint32_t* sched;      // nullable: [0] units handed out after the first, [1] CTAs done
  int upi;              // units per image
  int qbufs;            // query buffers: 2 lets the next unit's queries land early
  int rsplit;           // one head per unit, not SPLIT: units of <= 64 text rows run split
                        // (the query map's box is then 64 rows; the RS kernels)
  int order;            // 0: index order; 1: heaviest first if the costs are skewed;
                        // 2: heaviest first (la.B <= kOrderMax)
};

constexpr int kURing = 4;        // unit indices in flight from the producer to the other roles
constexpr int kOrderMax = 256;   // images the heaviest-first order covers

struct SPlan {
  uint32_t q, k, bars, slot, ms, lse, cps, red, imgs, ring, order, cost, ubars, total;
};

// dyn: with the unit ring, its barriers and the image order (round-robin
// launches leave them out, so their shared memory stays as small as before).
__host__ __device__ inline SPlan stream_plan(int stages, bool dyn, int qbufs) {
  SPlan s;
  s.q = 0;                                              // [kQBufs][2 halves][128 rows][128 B]
  s.k = (uint32_t)(qbufs * kTileBytes);                 // [stages][tile]
  s.bars = s.k + (uint32_t)stages * kTileBytes;         // mbarriers, see the kernel
  s.slot = s.bars + 8u * (uint32_t)(2 * kQBufs + 2 * kMaxStages + 4 + kMaxBatch + 2);
  s.ms = (s.slot + 16u + 15u) & ~15u;                   // [4][128] float2 (max, sum)
  s.lse = s.ms + 4u * kRows * 8u;                       // [128] float -lse per text row
  s.cps = s.lse + kRows * 4u;                           // [2][8 chunks][128 keys] partials
  s.red = s.cps + 2u * 8u * kTileKeys * 4u;             // [4 heads][4] float4 statistics
  s.imgs = s.red + 16u * 16u;                           // [kOrderMax] SImg image layouts
  s.ring = s.imgs + 32u * kOrderMax;                    // [kURing] int unit indices
  s.order = s.ring + 4u * kURing;                       // [kOrderMax] int images, heaviest first
  s.cost = s.order + 4u * kOrderMax;                    // [kOrderMax] float image costs
  s.ubars = s.cost + 4u * kOrderMax;                    // [2][kURing] unit-ring mbarriers
  s.total = dyn ? s.ubars + 16u * kURing : s.ring;
  return s;
}

// Text columns of the sweep-2 accumulator: the unit's rows rounded up to the
// MMA's N granularity (16), or every lane of a stack of heads.
template <int HPU>
__device__ __forceinline__ int sweep2_cols(int NT) {
  return HPU == 1 ? min(kRows, max(16, (NT + 15) & ~15)) : kRows;
}

// Geometry of one unit, derived identically by every warp role.
struct SGeo {
  int b, l, h, kvh, nh, S, NV, NT, t0, x0, v0;   // heads h .. h + nh - 1
  int n1, n2;   // key tiles of sweep 1 (whole causal prefix) and sweep 2 (visual)
  // Batch units (causal, one head, every sweep-2 accumulator fits TMEM at
  // once, every visual tile fits the K ring): sweep 1 takes n_st tiles ending
  // at key S (keys < 0 masked), the n2 visual tiles from key S and n_tt text
  // tiles, starting at key kfirst; the visual tiles stay in the ring and
  // sweep 2 issues all its MMAs at once from there.
  int n_st, n_tt, kfirst;
  bool ok, batch;
  bool sp;   // split rows: the unit's <= 64 text rows fill lanes 0-63 and again 64-127
};

// One image's layout as the units need it, staged per CTA in shared memory:
// S, N_V, N_T, first token, first text row, first visual row, and whether
// the layout arrays are consistent for it (the checks of stream_geo).
struct SImg {
  int S, NV, NT, t0, x0, v0, ok, pad;
};

template <bool SPLIT, int HPU>
__device__ __forceinline__ SImg load_image(const LayoutArgs& la, int b) {
  SImg m;
  m.S = __ldg(la.n_sys + b);
  m.NV = __ldg(la.n_vis + b);
  m.NT = __ldg(la.n_text + b);
  m.t0 = __ldg(la.tok_off + b);
  m.x0 = __ldg(la.text_off + b);
  m.v0 = __ldg(la.vis_off + b);
  const int T = m.S + m.NV + m.NT;
  m.ok = m.S >= 0 && m.NV >= 0 && m.NT >= 1 && m.NT <= (SPLIT ? kRows / 2 : kRows / HPU) &&
         T <= la.max_T && m.NV <= la.max_vis && __ldg(la.tok_off + b + 1) - m.t0 == T &&
         m.t0 >= 0 && m.t0 + T <= la.sum_T && __ldg(la.text_off + b + 1) - m.x0 == m.NT &&
         m.x0 >= 0 && m.x0 + m.NT <= la.sum_text && __ldg(la.vis_off + b + 1) - m.v0 == m.NV &&
         m.v0 >= 0 && m.v0 + m.NV <= la.sum_vis;
  m.pad = 0;
  return m;
}

// imgs: the images' layouts in shared memory (la.B <= kOrderMax), or null
// to read them from global memory.
template <int HPU, bool SPLIT, bool RS>
__device__ __forceinline__ SGeo stream_geo(const StreamArgs& p, int unit, const SImg* imgs) {
  const LayoutArgs& la = p.la;
  SGeo g;
  if (HPU == 1) {   // units are (image, layer, query head)
    g.h = unit % la.H;
    g.l = (unit / la.H) % la.L;
    g.b = unit / (la.H * la.L);
    g.kvh = g.h / p.group;
    g.nh = 1;
  } else {          // units are (image, layer, kv head, stack of query heads)
    const int ug = unit % p.upk;
    g.kvh = (unit / p.upk) % la.H_kv;
    g.l = (unit / (p.upk * la.H_kv)) % la.L;
    g.b = unit / (p.upk * la.H_kv * la.L);
    g.h = g.kvh * p.group + ug * HPU;
    g.nh = min(HPU, p.group - ug * HPU);
  }
  const SImg m = imgs ? imgs[g.b] : load_image<SPLIT, HPU>(la, g.b);
  g.S = m.S;
  g.NV = m.NV;
  g.NT = m.NT;
  g.t0 = m.t0;
  g.x0 = m.x0;
  g.v0 = m.v0;
  const int T = g.S + g.NV + g.NT;
  g.ok = m.ok != 0;
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  g.n2 = g.ok ? (g.NV + kTileKeys - 1) / kTileKeys : 0;
  g.n_st = (g.S + kTileKeys - 1) / kTileKeys;
  g.n_tt = max(0, (g.NV + g.NT + kTileKeys - 1) / kTileKeys - g.n2);
  // with the rows' lse given (from the layer's attention pass) there is no sweep 1
  const bool given = p.lse_in != nullptr;
  g.sp = SPLIT || (RS && HPU == 1 && g.NT <= kRows / 2);
  g.batch = !given && HPU == 1 && g.ok && causal && g.n2 >= 1 && g.n2 <= kMaxBatch &&
            g.n2 * sweep2_cols<HPU>(g.NT) <= kTmemCols && g.n2 + g.n_tt <= p.stages;
  g.kfirst = g.batch ? g.S - kTileKeys * g.n_st : 0;
  g.n1 = !(g.ok && causal) || given ? 0
         : g.batch ? g.n_st + g.n2 + g.n_tt : (T + kTileKeys - 1) / kTileKeys;
  return g;
}

// Relative cost of one image's units: key tiles streamed by both sweeps, each
// weighted by the text rows the epilogue sweeps (plus a fixed share for the
// MMAs and the tile's own overhead).
__device__ __forceinline__ float image_cost(const LayoutArgs& la, int b) {
  const float S = (float)__ldg(la.n_sys + b), NV = (float)__ldg(la.n_vis + b);
  const float NT = (float)__ldg(la.n_text + b);
  return (S + 2.f * NV + NT) * (NT + 64.f);
}

// Work index w (0 .. num_units - 1, in hand-out order) -> unit: with an
// order, the units of the image of rank w / upi.
__device__ __forceinline__ int unit_of(const StreamArgs& p, const int* order, int w) {
  if (!p.order) return w;
  const int r = w / p.upi;
  return order[r] * p.upi + (w - r * p.upi);
}

// HPU: query heads stacked per unit (1, 2 or 4), fixed at compile time so that
// the row mapping and the quarter sums are unrolled.  SPLIT (one head of at
// most 64 text rows): the queries fill TMEM lanes 0-63 and again 64-127, and
// in sweep 1 each half of the lanes takes half of every key tile's columns, so
// all four lane quarters (all four SM sub-partitions) share the exponentials.
// RS (one head, not SPLIT): units of at most 64 text rows run split, the
// others not (p.rsplit; the query map's box is 64 rows).  DYN: units come
// from the workspace counter through the unit ring (p.sched set); otherwise
// round-robin, and the ring's code is compiled out.
template <int HPU, bool SPLIT, bool RS, bool DYN>
__global__ void __launch_bounds__(kThreads, 1)
    score_stream_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK, const StreamArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const LayoutArgs& la = p.la;
  const SPlan plan = stream_plan(p.stages, DYN, p.qbufs);
  constexpr uint32_t q_half = kHalfBytes;   // bytes of one 64-element half of Q
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);   // [kQBufs]
  uint64_t* q_empty = q_full + kQBufs;     // [kQBufs]
  uint64_t* k_full = q_empty + kQBufs;     // [kMaxStages]
  uint64_t* k_empty = k_full + kMaxStages; // [kMaxStages]
  uint64_t* a_full = k_empty + kMaxStages; // [2] accumulator buffer ready
  uint64_t* a_empty = a_full + 2;          // [2] accumulator buffer read
  uint64_t* b_full = a_empty + 2;          // [kMaxBatch] batch sweep-2 accumulator ready
  uint64_t* b_done = b_full + kMaxBatch;   // batch sweep 2 read: TMEM free again
  uint64_t* s1_done = b_done + 1;          // a batch unit's sweep-1 accumulators all read
  uint64_t* u_full = reinterpret_cast<uint64_t*>(smem + plan.ubars);   // [kURing] unit published
  uint64_t* u_free = u_full + kURing;      // [kURing] unit index read by every consumer
  volatile int* uring = reinterpret_cast<volatile int*>(smem + plan.ring);
  int* order_s = reinterpret_cast<int*>(smem + plan.order);
  float* cost_s = reinterpret_cast<float*>(smem + plan.cost);
  SImg* imgs_s = reinterpret_cast<SImg*>(smem + plan.imgs);
  const SImg* imgs = la.B <= kOrderMax ? imgs_s : nullptr;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float2* ms = reinterpret_cast<float2*>(smem + plan.ms);
  float* nlse = reinterpret_cast<float*>(smem + plan.lse);   // -lse per text row
  float* cps = reinterpret_cast<float*>(smem + plan.cps);
  float4* red = reinterpret_cast<float4*>(smem + plan.red);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  constexpr int kRph = kRows / HPU;   // TMEM lanes per stacked head
  pdl_wait();   // inputs may come from the kernel before (launched with PDL)
  // only then may the next kernel be scheduled: the compaction that follows
  // in e2s_prune copies rows before its own wait
  pdl_launch_dependents();   // every CTA is resident: the next kernel may be scheduled
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  if (warp == 0 && lane == 0) {
    for (int i = 0; i < kQBufs; ++i) {
      ptx::mbar_init(q_full + i, 1);
      ptx::mbar_init(q_empty + i, 2);   // one commit per MMA issuer
    }
    for (int i = 0; i < kMaxStages; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(k_empty + i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(a_full + i, 1);
      ptx::mbar_init(a_empty + i, kEpiWarps);
    }
    for (int i = 0; i < kMaxBatch; ++i) ptx::mbar_init(b_full + i, 1);
    ptx::mbar_init(b_done, kEpiWarps);
    ptx::mbar_init(s1_done, kEpiWarps);
    for (int i = 0; i < (DYN ? kURing : 0); ++i) {
      ptx::mbar_init(u_full + i, 1);
      ptx::mbar_init(u_free + i, 2 + kEpiWarps);   // both MMA issuers and every epilogue warp
    }
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    ptx::prefetch_tensormap(&tmQ);
    ptx::prefetch_tensormap(&tmK);
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, kTmemCols);
  // every image's layout into shared memory once (the barrier below publishes
  // it), so that a unit's geometry is not a chain of global loads at its start
  if (imgs)
    for (int i = threadIdx.x; i < la.B; i += blockDim.x) imgs_s[i] = load_image<SPLIT, HPU>(la, i);
  if (DYN && p.order) {
    // Every CTA derives the same order.  With few units per CTA (order 2)
    // or when the costliest image costs more than twice the mean, images go
    // heaviest first (cost descending, then index), so that the last units
    // handed out are light ones; otherwise in index order, which keeps heavy
    // and light units mixed on the SMs (heaviest first measured slower there).
    for (int i = threadIdx.x; i < la.B; i += blockDim.x) cost_s[i] = image_cost(la, i);
    __syncthreads();
    float cmax = 0.f, csum = 0.f;
    for (int j = 0; j < la.B; ++j) {
      cmax = fmaxf(cmax, cost_s[j]);
      csum += cost_s[j];
    }
    const bool skewed = p.order == 2 || cmax * (float)la.B > 2.f * csum;
    for (int i = threadIdx.x; i < la.B; i += blockDim.x) {
      const float c = cost_s[i];
      int r = i;
      if (skewed) {
        r = 0;
        for (int j = 0; j < la.B; ++j) {
          const float cj = cost_s[j];
          r += (cj > c || (cj == c && j < i)) ? 1 : 0;
        }
      }
      order_s[r] = i;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;
  // consumer side of the unit ring: one thread per MMA issuer, or a whole
  // epilogue warp, whose lane 0 releases the slot once every lane has read it
  // (without the counter, units go round-robin and there is no ring)
  auto take_unit = [&](int u, bool warp_wide) -> int {
    if constexpr (!DYN) {   // round-robin
      const int w = (int)blockIdx.x + u * (int)gridDim.x;
      return w < p.num_units ? w : -1;
    }
    const int slot = u % kURing;
    if (!ptx::mbar_wait(u_full + slot, (u / kURing) & 1, limit, p.status)) {
      limit = kWaitNsAfterFault;
      return -1;
    }
    const int unit = uring[slot];
    if (warp_wide) __syncwarp();
    if (!warp_wide || lane == 0) ptx::mbar_arrive(u_free + slot);
    return unit;
  };

  if (warp == 0) {
    // ================= TMA producer: per unit the 128 text rows, then every
    // key tile of sweep 1 and of sweep 2 through the ring
    if (lane == 0) {
      // unit u of this CTA (work index w) goes into ring slot u % kURing for
      // the MMA issuers and the epilogue; -1 ends the walk
      auto publish = [&](int u, int w) {
        if constexpr (!DYN) return w < p.num_units ? w : -1;   // round-robin: no ring
        const int unit_w = w < p.num_units ? unit_of(p, order_s, w) : -1;
        const int slot = u % kURing;
        if (u >= kURing && !ptx::mbar_wait(u_free + slot, (u / kURing - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        uring[slot] = unit_w;
        ptx::mbar_arrive(u_full + slot);
        return unit_w;
      };
      int ld = 0;
      int unit = publish(0, (int)blockIdx.x);   // the CTA's own first unit
      for (int u = 0; unit >= 0; ++u) {
        const SGeo g = stream_geo<HPU, SPLIT, RS>(p, unit, imgs);
        if (!g.ok) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
        // unit u's queries go into buffer u % qbufs once the unit qbufs back is
        // done with it (with two, they land while the previous unit finishes)
        const int qb = u % p.qbufs;
        uint8_t* q_dst = q_sm + qb * kTileBytes;
        if (u >= p.qbufs && !ptx::mbar_wait(q_empty + qb, (u / p.qbufs - 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        if (g.n1 + g.n2 > 0) {
          // kRows / HPU rows of each stacked head (an absent head repeats the last one;
          // its rows are masked); with 64-row boxes (one head) two boxes: the
          // unit's first 64 rows twice when it runs split, else rows 0-63 and 64-127
          const int qrow = g.l * la.sum_text + g.x0;
          constexpr bool box64 = SPLIT || RS;
          ptx::mbar_arrive_expect_tx(q_full + qb, 2u * q_half);
#pragma unroll
          for (int hs = 0; hs < (box64 ? 2 : HPU); ++hs) {
            const int hq = box64 ? g.h : g.h + min(hs, g.nh - 1);
            const int row = qrow + (box64 && !g.sp ? hs * (kRows / 2) : 0);
            const uint32_t off = (uint32_t)(hs * (box64 ? kRows / 2 : kRph)) * 128u;
            ptx::tma_load_3d(q_dst + off, &tmQ, q_full + qb, 0, hq, row);
            ptx::tma_load_3d(q_dst + q_half + off, &tmQ, q_full + qb, 64, hq, row);
          }
        } else {
          ptx::mbar_arrive(q_full + qb);
        }
        // sweep-1 tiles, then (except in a batch unit, whose visual tiles stay
        // in the ring) the visual tiles again for sweep 2
        for (int j = 0; j < g.n1 + (g.batch ? 0 : g.n2); ++j, ++ld) {
          const int s = ld % p.stages;
          if (ld >= p.stages &&
              !ptx::mbar_wait(k_empty + s, (ld / p.stages - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          const int key0 = j < g.n1 ? g.kfirst + kTileKeys * j : g.S + kTileKeys * (j - g.n1);
          const int krow = g.l * la.sum_T + g.t0 + key0;
          ptx::mbar_arrive_expect_tx(k_full + s, (uint32_t)kTileBytes);
          ptx::tma_load_3d(k_sm + s * kTileBytes, &tmK, k_full + s, 0, g.kvh, krow);
          ptx::tma_load_3d(k_sm + s * kTileBytes + kHalfBytes, &tmK, k_full + s, 64, g.kvh, krow);
        }
        // every load of this unit issued: the next unit is taken now, and its
        // queries and first key tiles go to L2, so that its loads do not start
        // from DRAM when this unit's last MMAs retire
        // (claimed only now: claimed a unit earlier, units waited behind busy
        // CTAs -- 270 -> 286 us on the high-resolution batch)
        const int next = publish(u + 1, DYN ? (int)gridDim.x + (int)atomicAdd(p.sched, 1u)
                                            : (int)blockIdx.x + (u + 1) * (int)gridDim.x);
        unit = next;
        if (next >= 0) {
          const SGeo gn = stream_geo<HPU, SPLIT, RS>(p, next, imgs);
          if (gn.n1 + gn.n2 > 0) {
            const int qrow = gn.l * la.sum_text + gn.x0;
#pragma unroll
            for (int hs = 0; hs < (gn.sp ? 1 : RS ? 2 : HPU); ++hs) {
              const int hq = gn.h + min(hs, gn.nh - 1);
              const int row = qrow + (RS ? hs * (kRows / 2) : 0);
              ptx::tma_prefetch_3d(&tmQ, 0, hq, row);
              ptx::tma_prefetch_3d(&tmQ, 64, hq, row);
            }
            const int nt = min(gn.n1 + gn.n2, p.stages);
            for (int j = 0; j < nt; ++j) {
              const int key0 = j < gn.n1 ? gn.kfirst + kTileKeys * j : gn.S + kTileKeys * (j - gn.n1);
              const int krow = gn.l * la.sum_T + gn.t0 + key0;
              ptx::tma_prefetch_3d(&tmK, 0, gn.kvh, krow);
              ptx::tma_prefetch_3d(&tmK, 64, gn.kvh, krow);
            }
          }
        }
      }
    }
  } else if (warp == 1 || warp == kMmaWarp1) {
    // ================= MMA issuers: sweep 1 D[t][key] (text rows on the
    // lanes), sweep 2 D[key][t] (keys on the lanes).  Two threads alternate
    // tiles -- issuer m owns accumulator buffer m and the tiles tc % 2 == m --
    // so that one's waits and commits overlap the other's MMAs (an issuing
    // thread is held while the tensor pipe takes its instructions).
    const int mid = warp == 1 ? 0 : 1;
    if (lane == 0) {
      const uint32_t idesc1 = ptx::idesc_bf16_f32(kRows, kTileKeys);
      int tc = 0, u = 0, bu = 0;
      int slot = 0;          // ring stage of the next tile to consume
      uint32_t kph = 0u;     // its k_full phase
      // both operands are two 64-element halves of 128 rows (kHalfBytes apart)
      auto mma_tile = [&](uint32_t d, uint32_t a_base, uint32_t b_base, uint32_t idesc) {
        // one descriptor per operand; each K step of 16 adds its byte offset
        // (>> 4) to the 14-bit start-address field, which cannot carry for
        // shared-memory addresses below 256 KiB
        const uint64_t a0 = ptx::sdesc_sw128(a_base), b0 = ptx::sdesc_sw128(b_base);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t half = ks >> 2, kk = ks & 3;
          const uint32_t off = (half * (uint32_t)kHalfBytes + kk * 32u) >> 4;
          ptx::mma_bf16(d, a0 + off, b0 + off, idesc, ks > 0 ? 1u : 0u);
        }
      };
      for (;; ++u) {
        const int unit = take_unit(u, false);
        if (unit < 0) break;
        const SGeo g = stream_geo<HPU, SPLIT, RS>(p, unit, imgs);
        const int n2c = sweep2_cols<HPU>(g.NT);
        const uint32_t idesc2 = ptx::idesc_bf16_f32(kTileKeys, n2c);
        const int qb = u % p.qbufs;
        const uint32_t q_base = ptx::smem_addr(q_sm + qb * kTileBytes);
        if (!ptx::mbar_wait(q_full + qb, (u / p.qbufs) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        const int slot_vis = (slot + g.n_st) % p.stages;   // a batch unit's first visual tile
        for (int j = 0; j < g.n1 + (g.batch ? 0 : g.n2); ++j, ++tc) {
          const int s = slot, buf = tc & 1;
          const uint32_t ph = kph;
          if (++slot == p.stages) {
            slot = 0;
            kph ^= 1u;
          }
          if (buf != mid) continue;   // the other issuer's tile
          if (!ptx::mbar_wait(k_full + s, ph, limit, p.status)) limit = kWaitNsAfterFault;
          if (tc >= 2 && !ptx::mbar_wait(a_empty + buf, (tc / 2 - 1) & 1, limit, p.status))
            limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const uint32_t k_base = ptx::smem_addr(k_sm + s * kTileBytes);
          const uint32_t d = tmem + (uint32_t)(buf * kTileKeys);
          if (j >= g.n1)
            mma_tile(d, k_base, q_base, idesc2);
          else
            mma_tile(d, q_base, k_base, idesc1);
          const int vi = j - g.n_st;   // a batch unit keeps its visual tiles
          if (!(g.batch && vi >= 0 && vi < g.n2)) ptx::mma_commit(k_empty + s);
          ptx::mma_commit(a_full + buf);  // the epilogue may read the buffer
        }
        if (g.batch && mid == 0) {
          // every sweep-1 accumulator read: the sweep-2 accumulators of all
          // visual tiles go side by side into TMEM columns j * n2c.  The wait is
          // on a barrier that completes once per batch unit: a parity wait on
          // the other issuer's a_empty buffer could see a phase two behind
          // (that issuer not yet past its previous tile) and pass at once.
          if (!ptx::mbar_wait(s1_done, bu & 1, limit, p.status)) limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          for (int j = 0; j < kMaxBatch; ++j) {
            if (j < g.n2) {
              const int s = (slot_vis + j) % p.stages;
              mma_tile(tmem + (uint32_t)(j * n2c), ptx::smem_addr(k_sm + s * kTileBytes), q_base,
                       idesc2);
              ptx::mma_commit(k_empty + s);
              ptx::mma_commit(b_full + j);
            } else {
              ptx::mbar_arrive(b_full + j);   // keep every barrier's phase in step
            }
          }
        }
        ptx::mma_commit(q_empty + qb);   // every MMA of this issuer in the unit is done with Q
        if (g.batch) {   // the next unit's accumulators wait for the batch to be read
          if (!ptx::mbar_wait(b_done, bu & 1, limit, p.status)) limit = kWaitNsAfterFault;
          ++bu;
        }
      }
    }
  } else if (warp < 2 + kEpiWarps) {
    // ================= epilogue (16 warps)
    const int ew = warp - 2;
    const int q4 = warp & 3;                 // TMEM lane quarter: text rows 32*q4 ..
    const int cg = ew >> 2;                  // column group: keys 32*cg .. of each tile
    const int lrow = q4 * 32 + lane;         // this lane's TMEM row
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    int tc = 0, bu = 0;
    for (int u = 0;; ++u) {
      const int unit = take_unit(u, true);
      if (unit < 0) break;
      const SGeo g = stream_geo<HPU, SPLIT, RS>(p, unit, imgs);
      // TMEM row lrow holds text row t of stacked head hs (split: row lrow % 64)
      const bool sp = g.sp;
      const int hs = sp ? 0 : lrow / kRph;
      const int t = sp ? (lrow & (kRows / 2 - 1)) : lrow - hs * kRph;
      const bool rows_live =
          hs < g.nh && (sp ? (q4 & 1) * 32 : (q4 * 32) % kRph) < g.NT;   // warp-uniform
      const bool tvalid = hs < g.nh && t < g.NT;
      const int lim = tvalid ? g.S + g.NV + t : -1;   // last key this row sees
      const float inv_nt = 1.f / (float)max(g.NT, 1);
      const int NV = g.ok ? g.NV : 0;
      // ---- sweep 1: running (max, sum) per row over this warp's columns
      float m = kNegBig, ssum = 0.f;
      for (int j = 0; j < g.n1; ++j, ++tc) {
        const int buf = tc & 1;
        if (!ptx::mbar_wait(a_full + buf, (tc / 2) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        if (rows_live) {
#pragma unroll
          for (int ch = 0; ch < (sp ? 1 : 2); ++ch) {
            // 16-column chunks of this warp: 2 of its column group's 32, or
            // (split) 1 of the 64 columns of its lane half
            const int c16 = sp ? (q4 >> 1) * (kTileKeys / 2) + cg * 16 : cg * 32 + ch * 16;
            const int key0 = g.kfirst + kTileKeys * j + c16;
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(buf * kTileKeys + c16), x);
            if (key0 >= 0 && key0 + 15 <= lim) {   // the row sees the whole chunk
              float cmax = x[0];
#pragma unroll
              for (int jj = 1; jj < 16; ++jj) cmax = fmaxf(cmax, x[jj]);
              const float mnew = fmaxf(m, cmax * p.scale_log2);
              float nm[16];
#pragma unroll
              for (int jj = 0; jj < 16; ++jj) nm[jj] = -mnew;
              ssum = exp2_sum16(x, p.scale_log2, nm, ssum * fast_ex2(m - mnew));
              m = mnew;
            } else if (key0 <= lim && key0 + 15 >= 0) {   // key 0 or the row's last key inside
              float cmax = kNegBig;
#pragma unroll
              for (int jj = 0; jj < 16; ++jj)
                if (key0 + jj >= 0 && key0 + jj <= lim) cmax = fmaxf(cmax, x[jj]);
              const float mnew = fmaxf(m, cmax * p.scale_log2);
              float acc = ssum * fast_ex2(m - mnew);
#pragma unroll
              for (int jj = 0; jj < 16; ++jj)
                if (key0 + jj >= 0 && key0 + jj <= lim)
                  acc += fast_ex2(fmaf(x[jj], p.scale_log2, -mnew));
              ssum = acc;
              m = mnew;
            }
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(a_empty + buf);
      }
      // a batch unit's sweep-2 MMAs overwrite both accumulator buffers: they
      // wait until every warp has read its last sweep-1 tile
      if (g.batch && lane == 0) ptx::mbar_arrive(s1_done);
      // ---- merge the four column groups: lse per row (log2 domain), published
      // per text row for sweep 2 (or taken from the caller's attention pass)
      if (causal && p.lse_in != nullptr) {
        if (cg == 0 && (!sp || lrow < kRows / 2))
          nlse[lrow] = tvalid ? -__ldg(p.lse_in + ((size_t)g.l * la.H + g.h + hs) * la.sum_text +
                                       g.x0 + t) * kLog2e
                              : -kNegBig;
        ptx::named_bar(1, kEpiThreads);
      } else if (causal) {
        ms[cg * kRows + lrow] = make_float2(m, ssum);
        ptx::named_bar(1, kEpiThreads);
        // partials of this row: four column groups (and, split, both lane halves)
        const int nparts = sp ? 8 : 4;
        auto part = [&](int c) {
          return ms[(c & 3) * kRows + (c < 4 ? lrow : (lrow ^ (kRows / 2)))];
        };
        float M = kNegBig;
#pragma unroll
        for (int c = 0; c < nparts; ++c) M = fmaxf(M, part(c).x);
        float L = 0.f;
#pragma unroll
        for (int c = 0; c < nparts; ++c) {
          const float2 v = part(c);
          L += v.y * fast_ex2(v.x - M);
        }
        if (cg == 0 && (!sp || lrow < kRows / 2))
          nlse[lrow] = L > 0.f ? -(M + __log2f(L)) : -kNegBig;
        ptx::named_bar(1, kEpiThreads);
      }
      // ---- sweep 2: accumulator D[key][column], keys on the lanes, so each
      // key's sum over text rows is lane-local.  Warp (q4, cg) reads column
      // chunks cg and cg + 4 (16 columns each; chunk c holds text rows
      // 16c % (128 / HPU) .. of stacked head 16c / (128 / HPU)) and leaves one
      // partial per chunk and key; after the four warps of the lane quarter
      // meet, warp cg sums the chunks of head cg in order and also keeps that
      // head's statistics of Eq. 8 online (sum, max of a*log2e, sum of exp2).
      const int nch = sweep2_cols<HPU>(g.NT) >> 4;
      constexpr int kCph = kRph / 16;   // chunks per stacked head
      const int head_chunks = min(kCph, (g.NT + 15) >> 4);
      const float a_mul = causal ? inv_nt : p.scale * inv_nt;
      float st_s = 0.f, st_m = kNegBig, st_e = 0.f;
      if (g.batch) {
        // batch unit: the accumulator of visual tile j sits in columns
        // j * 16 * nch; column group cg owns the tiles j % 4 == cg and sums
        // every column of its lanes' keys -- no cross-warp reduction
        for (int j = cg; j < g.n2; j += 4) {
          if (!ptx::mbar_wait(b_full + j, bu & 1, limit, p.status)) limit = kWaitNsAfterFault;
          ptx::tc_fence_after();
          const int n = kTileKeys * j + lrow;   // visual index of this lane's key
          float a = 0.f;
          if (kTileKeys * j + q4 * 32 < NV) {   // the warp holds visual keys
            const uint32_t tb = tmem + lane_base + (uint32_t)(j * nch * 16);
            for (int c = 0; c < nch; ++c) {
              float x[16];
              ptx::tmem_ld16(tb + (uint32_t)(c * 16), x);
              const float4* l4 = reinterpret_cast<const float4*>(nlse + c * 16);
              float s0 = 0.f, s1 = 0.f;
              if (c * 16 + 15 < g.NT) {
                float nl[16];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                  const float4 v = l4[q];
                  nl[4 * q] = v.x; nl[4 * q + 1] = v.y; nl[4 * q + 2] = v.z; nl[4 * q + 3] = v.w;
                }
                s0 = exp2_sum16(x, p.scale_log2, nl, 0.f);
              } else {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                  const float4 v = l4[q];
                  const float lv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                  for (int i = 0; i < 4; ++i)
                    if (c * 16 + 4 * q + i < g.NT)
                      s0 += fast_ex2(fmaf(x[4 * q + i], p.scale_log2, lv[i]));
                }
              }
              a += s0 + s1;
            }
          }
          if (n < NV) {
            a *= a_mul;
            p.a_out[((size_t)g.l * la.H + g.h) * (size_t)la.sum_vis + g.v0 + n] = a;
            const float al = a * kLog2e, mnew = fmaxf(st_m, al);
            st_e = st_e * fast_ex2(st_m - mnew) + fast_ex2(al - mnew);
            st_m = mnew;
            st_s += a;
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(b_done);
        ++bu;
      } else
      for (int j = 0; j < g.n2; ++j, ++tc) {
        const int buf = tc & 1;
        float* cp = cps + (j & 1) * 8 * kTileKeys;
        if (!ptx::mbar_wait(a_full + buf, (tc / 2) & 1, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int c = cg + 4 * r;
          const int ct = (c * 16) % kRph, chd = (c * 16) / kRph;   // first row, head
          if (c < nch && chd < g.nh && ct < g.NT) {                 // warp-uniform
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(buf * kTileKeys + c * 16), x);
            float acc0 = 0.f, acc1 = 0.f;
            if (causal) {
              const float4* l4 = reinterpret_cast<const float4*>(nlse + c * 16);
              float lv[16];
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float4 v = l4[q];
                lv[4 * q] = v.x; lv[4 * q + 1] = v.y; lv[4 * q + 2] = v.z; lv[4 * q + 3] = v.w;
              }
              if (ct + 15 < g.NT) {
                acc0 = exp2_sum16(x, p.scale_log2, lv, 0.f);
              } else {
#pragma unroll
                for (int jj = 0; jj < 16; ++jj)
                  if (ct + jj < g.NT) acc0 += fast_ex2(fmaf(x[jj], p.scale_log2, lv[jj]));
              }
            } else {
#pragma unroll
              for (int jj = 0; jj < 16; jj += 2) {
                if (ct + jj < g.NT) acc0 += x[jj];
                if (ct + jj + 1 < g.NT) acc1 += x[jj + 1];
              }
            }
            cp[c * kTileKeys + lrow] = acc0 + acc1;
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(a_empty + buf);
        ptx::named_bar(2 + q4, 128);   // the four column groups of this lane quarter
        if (cg < g.nh) {
          const int n = kTileKeys * j + lrow;   // visual index of this lane's key
          if (n < NV) {
            const int c0 = cg * kCph;
            float a = cp[c0 * kTileKeys + lrow];
#pragma unroll
            for (int c = 1; c < kCph; ++c)
              if (c < head_chunks) a += cp[(c0 + c) * kTileKeys + lrow];
            a *= a_mul;
            p.a_out[((size_t)g.l * la.H + g.h + cg) * (size_t)la.sum_vis + g.v0 + n] = a;
            const float al = a * kLog2e, mnew = fmaxf(st_m, al);
            st_e = st_e * fast_ex2(st_m - mnew) + fast_ex2(al - mnew);
            st_m = mnew;
            st_s += a;
          }
        }
      }
      // ---- statistics of each head's visual scores: merge the lanes of the
      // head's reducing warps (one per lane quarter; in a batch unit all 16)
      // in a fixed order
      if (g.batch || cg < HPU) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float s2 = __shfl_xor_sync(0xffffffffu, st_s, o);
          const float m2 = __shfl_xor_sync(0xffffffffu, st_m, o);
          const float e2 = __shfl_xor_sync(0xffffffffu, st_e, o);
          st_s += s2;
          lse_merge(st_m, st_e, m2, e2);
        }
        if (lane == 0) red[g.batch ? ew : cg * 4 + q4] = make_float4(st_s, st_m, st_e, 0.f);
      }
      ptx::named_bar(1, kEpiThreads);
      if (et < g.nh && g.ok) {   // thread et merges stacked head et
        float S = 0.f, M = kNegBig, E = 0.f;
        const int nr = g.batch ? kEpiWarps : 4;
        for (int c = 0; c < nr; ++c) {
          const float4 r4 = red[et * 4 + c];
          S += r4.x;
          lse_merge(M, E, r4.y, r4.z);
        }
        p.stats[((size_t)g.b * la.L + g.l) * la.H + g.h + et] = stats_entry(S, M, E);
      }
      // ms, nlse, cps and red are rewritten by the next unit only after this barrier
      ptx::named_bar(1, kEpiThreads);
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
  if (DYN && threadIdx.x == 0) {
    // the last CTA out (every CTA has taken its last unit) zeroes the counter
    __threadfence();
    if (atomicAdd(p.sched + 1, 1u) == gridDim.x - 1) {
      atomicExch(p.sched, 0u);
      atomicExch(p.sched + 1, 0u);
    }
  }
}

}  // namespace

// K ring stages that fit the device's shared memory beside qbufs query
// buffers (0 if fewer than two).
static int stream_stages(int qbufs) {
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  for (int st = kMaxStages; st >= 2; --st)
    if ((int)(stream_plan(st, true, qbufs).total + 1024) <= optin) return st;
  return 0;
}

// Whether the streaming kernel can take this launch: at most 128 text rows.
bool score_stream_fits(const LayoutArgs& la) {
  return la.max_text <= kRows && la.H % la.H_kv == 0 && stream_stages(1) >= 2;
}

cudaError_t launch_score_stream(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                                const void* k, int64_t k_stride, float* a_out, float4* stats,
                                uint32_t* counters, uint32_t* status, cudaStream_t st,
                                const float* lse_in, bool pdl) {
  StreamArgs p;
  p.lse_in = lse_in;
  p.la = la;
  p.mode = mode;
  p.group = la.H / la.H_kv;
  // stack the query heads of one kv head into the 128 TMEM lanes when their
  // text rows leave room (64 rows: two heads, 32 rows: four)
  int hpu = 1;
  while (hpu < 4 && hpu * 2 <= p.group && la.max_text <= kRows / (hpu * 2)) hpu *= 2;
  // Short units (under 24 key tiles on average) take a second query buffer,
  // so that the next unit's first MMAs need not wait for its queries (LLaVA
  // batch 32: 188 -> 177 us), at the cost of a K ring stage; long units keep
  // the stage (high-resolution batch 8: 270 us with one buffer, 273 with two).
  const long long avg_tiles =
      ((long long)la.sum_T + la.sum_vis) / ((long long)std::max(la.B, 1) * kTileKeys);
  p.qbufs = avg_tiles < 24 ? 2 : 1;
  p.stages = stream_stages(p.qbufs);
  p.upk = (p.group + hpu - 1) / hpu;
  p.num_units = la.B * la.L * la.H_kv * p.upk;
  p.scale = 1.0f / sqrtf(128.0f);
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.a_out = a_out;
  p.stats = stats;
  p.counters = counters;
  p.status = status;
  p.upi = la.L * la.H_kv * p.upk;
  if (p.num_units == 0 || la.sum_vis == 0) return cudaSuccess;
  // With fewer than 16 units per CTA, units are handed out from a counter in
  // the workspace, so that CTAs that drew light units take more of them --
  // heaviest images first below 6 units per CTA (or when the image costs are
  // skewed); with more, round-robin.  Measured: Qwen2-VL batch 16 (5 units
  // per CTA) 85 -> 69 us; high-resolution batch 8 (6.7) unchanged, 272 us
  // heaviest first; LLaVA batch 32 (20) 1-2 % slower with the counter and
  // 4 % slower heaviest first.
  const int grid_n = std::min(p.num_units, sm_count());
  p.sched = status != nullptr && p.num_units < 16 * grid_n ? stream_sched_ptr(status) : nullptr;
  p.order = !p.sched || la.B <= 1 || la.B > kOrderMax ? 0 : p.num_units < 6 * grid_n ? 2 : 1;
  CUtensorMap tmQ, tmK;
  // one head of at most 64 text rows: the queries are loaded twice (SPLIT)
  const bool split = hpu == 1 && la.max_text <= kRows / 2;
  // one head per unit with longer text somewhere in the batch: the units of at
  // most 64 rows still run split (their rows loaded twice), so that all four
  // lane quarters share their sweep-1 exponentials -- when the text is short
  // on average (below 96 rows); a batch of long text only pays the branches
  // (high-resolution batch 8: +1.5 %)
  p.rsplit = hpu == 1 && !split && la.sum_text < (long long)la.B * 96 ? 1 : 0;
  if (!make_score_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_text, q_stride,
                      split || p.rsplit ? kRows / 2 : kRows / hpu) ||
      !make_score_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTileKeys))
    return cudaErrorInvalidValue;
  if (p.stages < 2) return cudaErrorInvalidValue;
  const size_t smem = stream_plan(p.stages, p.sched != nullptr, p.qbufs).total + 1024;
  const dim3 grid((unsigned)grid_n);
  const bool dyn = p.sched != nullptr;
  auto go = [&](auto kernel) {
    return launch_kernel(kernel, grid, dim3(kThreads), smem, st, 0, pdl, tmQ, tmK, p);
  };
  if (hpu == 4)
    return dyn ? go(score_stream_kernel<4, false, false, true>)
               : go(score_stream_kernel<4, false, false, false>);
  if (hpu == 2)
    return dyn ? go(score_stream_kernel<2, false, false, true>)
               : go(score_stream_kernel<2, false, false, false>);
  if (split)
    return dyn ? go(score_stream_kernel<1, true, false, true>)
               : go(score_stream_kernel<1, true, false, false>);
  if (p.rsplit)
    return dyn ? go(score_stream_kernel<1, false, true, true>)
               : go(score_stream_kernel<1, false, true, false>);
  return dyn ? go(score_stream_kernel<1, false, false, true>)
             : go(score_stream_kernel<1, false, false, false>);
}

}  // namespace e2s
