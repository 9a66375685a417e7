// Text-to-visual score on the 5th-generation tensor cores (tcgen05 + TMEM),
// with TMA-staged bf16 K tiles (Sec. 3.1 Eq. 1 and its causal-prefix
// probability reading).
//
// Work unit: (image b, layer l, kv head g, group of query heads).  The unit's
// keys are cut into 128-key tiles and split over a thread-block cluster; each
// CTA multiplies its tiles once and keeps every logit in TMEM:
//
//   MMA   D[key][col] = K_tile[key][:] . Q[col][:]   (M = 128 keys, N = padded
//         text rows of one query head, K = d = 128 in 8 steps), A = K tile and
//         B = text queries, both K-major with the 128-byte swizzle; tile i of
//         the CTA accumulates into TMEM columns [i*ncs, (i+1)*ncs).
//   pass A (CAUSAL_PROB)  per-text-row maximum over this CTA's visible keys:
//         a butterfly reduce-scatter over the warp's 32 lanes per 16-column
//         chunk, then over the four TMEM lane quarters in shared memory.
//   pass B  e = exp2(s - M) for every visible logit (one exp2 per logit),
//         written back into TMEM for the visual tiles, and the per-row sum L.
//   cluster exchange of (M, L) through distributed shared memory; every CTA
//         forms the row's log-sum-exp and a per-row weight
//         w = exp2(M_cta - lse) / N_T.
//   pass C  a[key] = sum_t e[key][t] * w[t] over the text rows (FMA only);
//         EQ1 mode: a = sum_t s[key][t] / (sqrt(d) N_T) straight from TMEM.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-9 epilogue.  Epilogue warp w reads TMEM lane quarter
// w % 4; in passes A and B it owns the 16-column chunks of parity (w - 2) / 4
// across all of the CTA's tiles (running max / sum per lane, one butterfly per
// chunk), in pass C the tiles of that parity.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "sm100_ptx.cuh"

namespace e2s {
namespace {

constexpr int kTileKeys = 128;
constexpr int kHalfBytes = kTileKeys * 128;   // 128 rows x 64 bf16 (one swizzle span)
constexpr int kTileBytes = 2 * kHalfBytes;    // 128 keys x 128 dims
constexpr int kEpiWarps = 8;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kQBoxRows = 16;
constexpr int kMaxCluster = 16;
constexpr uint64_t kWaitNs = 1000000000ull;        // first bounded wait: 1 s
constexpr uint64_t kWaitNsAfterFault = 1000000ull; // later waits after a timeout: 1 ms

struct TcArgs {
  LayoutArgs la;
  int group;           // H / H_kv
  int hpc;             // query heads per CTA
  int groups_per_kv;   // ceil(group / hpc)
  int cluster;         // CTAs per unit
  int tpc;             // tiles per CTA (capacity)
  int ntp_max;         // padded text rows, multiple of 16
  int mode;            // E2S_SCORE_*
  float scale_log2;    // log2(e) / sqrt(d)
  float scale;         // 1 / sqrt(d)
  uint32_t tmem_cols;
  float* a_out;
  float4* stats;        // per (image, layer, head) statistics of the visual scores
  uint32_t* counters;   // nullable: decision scratch to zero
  uint32_t* status;
};

struct SmemPlan {
  uint32_t q, k, bars, slot, pmax, psum, cm, part, colw, asm_, sred, spart, total;
};

__host__ __device__ inline SmemPlan smem_plan(int hpc, int ntp_max, int tpc) {
  SmemPlan s;
  const uint32_t ncs = (uint32_t)(hpc * ntp_max);
  s.q = 0;
  s.k = 2u * ncs * 128u;
  s.bars = s.k + (uint32_t)tpc * kTileBytes;
  s.slot = s.bars + 8u * (uint32_t)(1 + 2 * tpc);
  s.pmax = (s.slot + 16u + 15u) & ~15u;       // [4 lane quarters][ncs] float
  s.psum = s.pmax + 4u * ncs * 4u;            // [4 lane quarters][ncs] float
  s.cm = s.psum + 4u * ncs * 4u;              // [ncs] float: CTA max (log2 units)
  s.part = s.cm + ncs * 4u;                   // [ncs] float2: (M, L) for the cluster
  s.colw = s.part + ncs * 8u;                 // [ncs] float: pass-C weights
  s.asm_ = s.colw + ncs * 4u;                 // [hpc][tpc*128] float: this CTA's scores
  s.sred = s.asm_ + (uint32_t)hpc * (uint32_t)tpc * 128u * 4u;  // [8 warps] float2
  s.spart = s.sred + 8u * 8u;                 // [hpc] float4: CTA statistics
  s.total = s.spart + (uint32_t)hpc * 16u;
  return s;
}

// Butterfly reduce-scatter of 16 values over the 32 lanes of a warp: on
// return lane L holds, in x[0], column L >> 1 reduced over all 32 lanes.
template <int W, int MASK, class Op>
__device__ __forceinline__ void rs_step(float (&x)[16], bool hi, Op op) {
#pragma unroll
  for (int i = 0; i < W; ++i) {
    const float send = hi ? x[i] : x[i + W];
    const float keep = hi ? x[i + W] : x[i];
    x[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, MASK));
  }
}
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

__global__ void __launch_bounds__(kThreads, 2)
    score_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                    const __grid_constant__ CUtensorMap tmK, const TcArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const SmemPlan plan = smem_plan(p.hpc, p.ntp_max, p.tpc);
  uint8_t* q_sm = smem + plan.q;
  uint8_t* k_sm = smem + plan.k;
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + plan.bars);
  uint64_t* k_full = q_full + 1;
  uint64_t* mma_done = k_full + p.tpc;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float* pmax = reinterpret_cast<float*>(smem + plan.pmax);
  float* psum = reinterpret_cast<float*>(smem + plan.psum);
  float* cm = reinterpret_cast<float*>(smem + plan.cm);
  float2* part = reinterpret_cast<float2*>(smem + plan.part);
  float* colw = reinterpret_cast<float*>(smem + plan.colw);
  float* a_sm = reinterpret_cast<float*>(smem + plan.asm_);
  float2* sred = reinterpret_cast<float2*>(smem + plan.sred);
  float4* spart = reinterpret_cast<float4*>(smem + plan.spart);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const int ncs = p.hpc * p.ntp_max;
  const uint32_t q_half = (uint32_t)ncs * 128u;
  pdl_wait();   // inputs may come from the kernel before (launched with PDL)
  // only then may the next kernel be scheduled: the compaction that follows
  // in e2s_prune copies rows before its own wait
  pdl_launch_dependents();
  if (p.counters != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < la.B * kDecideWordsPerImage; i += blockDim.x)
      p.counters[i] = 0u;

  // ---- unit decomposition: (b, l, kv head, head group)
  const int unit = blockIdx.x / p.cluster;
  int rest = unit;
  const int hg = rest % p.groups_per_kv;
  rest /= p.groups_per_kv;
  const int kvh = rest % la.H_kv;
  rest /= la.H_kv;
  const int l = rest % la.L;
  const int b = rest / la.L;
  const int h0 = kvh * p.group + hg * p.hpc;
  const int nh = min(p.hpc, p.group - hg * p.hpc);

  // ---- image geometry, checked against the host-side maxima
  const int S = __ldg(la.n_sys + b), NV = __ldg(la.n_vis + b), NT = __ldg(la.n_text + b);
  const int t0 = __ldg(la.tok_off + b), x0 = __ldg(la.text_off + b), v0 = __ldg(la.vis_off + b);
  const int T = S + NV + NT;
  const int ntp = (NT + 15) & ~15;
  const bool ok = S >= 0 && NV >= 0 && NT >= 1 && ntp <= p.ntp_max && T <= la.max_T &&
                  NV <= la.max_vis && __ldg(la.tok_off + b + 1) - t0 == T && t0 >= 0 &&
                  t0 + T <= la.sum_T && __ldg(la.text_off + b + 1) - x0 == NT && x0 >= 0 &&
                  x0 + NT <= la.sum_text && __ldg(la.vis_off + b + 1) - v0 == NV && v0 >= 0 &&
                  v0 + NV <= la.sum_vis;
  if (!ok && threadIdx.x == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);

  const bool causal = p.mode == E2S_SCORE_CAUSAL_PROB;
  const int key_base = causal ? 0 : S;
  const int span = causal ? T : NV;
  const int n_tiles = ok ? (span + kTileKeys - 1) / kTileKeys : 0;
  const int per = (n_tiles + p.cluster - 1) / p.cluster;
  const int ft = min(n_tiles, (int)rank * per);
  int nt = min(n_tiles, ft + per) - ft;
  if (nt > p.tpc) {  // cannot happen when T <= max_T; never overrun the tile slots
    if (threadIdx.x == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    nt = 0;
  }
  // local tiles that hold visual keys: [vf, vl)
  int vf = nt, vl = nt;
  for (int i = 0; i < nt; ++i) {
    const int k0 = key_base + kTileKeys * (ft + i);
    if (k0 < S + NV && k0 + kTileKeys > S) {
      if (vf == nt) vf = i;
      vl = i + 1;
    }
  }

  // ---- setup: barriers, TMEM
  if (warp == 0 && lane == 0) {
    ptx::mbar_init(q_full, 1);
    for (int i = 0; i < p.tpc; ++i) {
      ptx::mbar_init(k_full + i, 1);
      ptx::mbar_init(mma_done + i, 1);
    }
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    ptx::prefetch_tensormap(&tmQ);
    ptx::prefetch_tensormap(&tmK);
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, p.tmem_cols);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint64_t limit = kWaitNs;

  if (warp == 0) {
    // ================= TMA producer
    if (lane == 0 && nt > 0) {
      ptx::mbar_arrive_expect_tx(q_full, 2u * (uint32_t)(nh * ntp) * 128u);
      for (int hh = 0; hh < nh; ++hh)
        for (int half = 0; half < 2; ++half)
          for (int r = 0; r < ntp; r += kQBoxRows)
            ptx::tma_load_3d(q_sm + half * q_half + (uint32_t)(hh * p.ntp_max + r) * 128u, &tmQ,
                             q_full, half * 64, h0 + hh, l * la.sum_text + x0 + r);
      for (int i = 0; i < nt; ++i) {
        const int row = l * la.sum_T + t0 + key_base + kTileKeys * (ft + i);
        ptx::mbar_arrive_expect_tx(k_full + i, kTileBytes);
        ptx::tma_load_3d(k_sm + i * kTileBytes, &tmK, k_full + i, 0, kvh, row);
        ptx::tma_load_3d(k_sm + i * kTileBytes + kHalfBytes, &tmK, k_full + i, 64, kvh, row);
      }
      // no copy may still be in flight when the CTA retires
      if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
      for (int i = 0; i < nt; ++i)
        if (!ptx::mbar_wait(k_full + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
    }
    __syncwarp();
    ptx::cluster_arrive();
    ptx::cluster_wait();
  } else if (warp == 1) {
    // ================= MMA issuer (one thread): every tile once, own TMEM columns
    if (lane == 0 && nt > 0) {
      const uint32_t idesc = ptx::idesc_bf16_f32(128, ntp);
      if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
      const uint32_t b_base = ptx::smem_addr(q_sm);
      for (int i = 0; i < nt; ++i) {
        if (!ptx::mbar_wait(k_full + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const uint32_t a_base = ptx::smem_addr(k_sm + i * kTileBytes);
        for (int hh = 0; hh < nh; ++hh) {
          const uint32_t d = tmem + (uint32_t)(i * ncs + hh * p.ntp_max);
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t half = ks >> 2, kk = ks & 3;
            const uint64_t ad = ptx::sdesc_sw128(a_base + half * kHalfBytes + kk * 32u);
            const uint64_t bd = ptx::sdesc_sw128(b_base + half * q_half +
                                                 (uint32_t)(hh * p.ntp_max) * 128u + kk * 32u);
            ptx::mma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
          }
        }
        ptx::mma_commit(mma_done + i);
      }
    }
    __syncwarp();
    ptx::cluster_arrive();
    ptx::cluster_wait();
  } else {
    // ================= epilogue (8 warps)
    const int ew = warp - 2;
    const int q4 = warp & 3;       // TMEM lane quarter
    const int par = ew >> 2;       // chunk parity (passes A, B) / tile parity (pass C)
    const int row = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    const int lim = S + NV;        // text row t sees key k iff k <= lim + t
    const int cpb = ntp >> 4;      // chunks per head

    if (causal) {
      // ---- pass A: per-column maximum of the visible raw logits
      for (int i = 0; i < nt; ++i)
        if (!ptx::mbar_wait(mma_done + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
      ptx::tc_fence_after();
      for (int hh = 0; hh < nh; ++hh) {
        for (int c = par; c < cpb; c += 2) {
          const int c16 = c * 16;
          const int col = hh * p.ntp_max + c16;
          float mx[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) mx[j] = kNegBig;
          for (int i = 0; i < nt; ++i) {
            const int lo = max(key_base + kTileKeys * (ft + i) + row - lim, 0);
            float x[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * ncs + col), x);
            if (lo <= c16 && c16 + 16 <= NT) {
#pragma unroll
              for (int j = 0; j < 16; ++j) mx[j] = fmaxf(mx[j], x[j]);
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j)
                if (c16 + j >= lo && c16 + j < NT) mx[j] = fmaxf(mx[j], x[j]);
            }
          }
          const float m = reduce_scatter16(mx, lane, MaxOp());
          if ((lane & 1) == 0) pmax[q4 * ncs + col + (lane >> 1)] = m;
        }
      }
      ptx::named_bar(1, kEpiThreads);
      for (int c = et; c < ncs; c += kEpiThreads) {
        const float m = fmaxf(fmaxf(pmax[c], pmax[ncs + c]), fmaxf(pmax[2 * ncs + c], pmax[3 * ncs + c]));
        cm[c] = m > 0.5f * kNegBig ? m * p.scale_log2 : kNegBig;
      }
      ptx::named_bar(1, kEpiThreads);
      // ---- pass B: e = exp2(s - M), stored back for visual tiles; row sums
      for (int hh = 0; hh < nh; ++hh) {
        for (int c = par; c < cpb; c += 2) {
          const int c16 = c * 16;
          const int col = hh * p.ntp_max + c16;
          float mv[16], sm[16];
          const float4* cm4 = reinterpret_cast<const float4*>(cm + col);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const float4 c4 = cm4[v];
            mv[4 * v] = c4.x; mv[4 * v + 1] = c4.y; mv[4 * v + 2] = c4.z; mv[4 * v + 3] = c4.w;
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) sm[j] = 0.f;
          for (int i = 0; i < nt; ++i) {
            const int lo = max(key_base + kTileKeys * (ft + i) + row - lim, 0);
            const uint32_t ta = tmem + lane_base + (uint32_t)(i * ncs + col);
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
            if (i >= vf && i < vl) ptx::tmem_st16(ta, x);
#pragma unroll
            for (int j = 0; j < 16; ++j) sm[j] += x[j];
          }
          const float sum = reduce_scatter16(sm, lane, AddOp());
          if ((lane & 1) == 0) psum[q4 * ncs + col + (lane >> 1)] = sum;
        }
      }
      ptx::tmem_wait_st();
      ptx::tc_fence_before();
      ptx::named_bar(1, kEpiThreads);
      ptx::tc_fence_after();
      for (int c = et; c < ncs; c += kEpiThreads)
        part[c] = make_float2(cm[c], ((psum[c] + psum[ncs + c]) + psum[2 * ncs + c]) + psum[3 * ncs + c]);
    }
    ptx::cluster_arrive();
    ptx::cluster_wait();
    // ---- per-column weights of pass C
    for (int c = et; c < ncs; c += kEpiThreads) {
      const int t = c % p.ntp_max;
      if (causal) {
        float2 o[kMaxCluster];
#pragma unroll
        for (int r = 0; r < kMaxCluster; ++r)
          if (r < p.cluster) o[r] = ptx::ld_dsmem_f2(part + c, (uint32_t)r);
        float M = kNegBig, Ls = 0.f;
#pragma unroll
        for (int r = 0; r < kMaxCluster; ++r)
          if (r < p.cluster) lse_merge(M, Ls, o[r].x, o[r].y);
        const float lse = M + log2f(Ls);
        colw[c] = (t < NT && Ls > 0.f) ? fast_ex2(part[c].x - lse) / (float)NT : 0.f;
      } else {
        colw[c] = (t < NT) ? p.scale / (float)NT : 0.f;
      }
    }
    ptx::named_bar(1, kEpiThreads);
    // ---- pass C: a[key] = sum_t e[key][t] w[t] for the visual tiles
    for (int i = vf + ((vf & 1) != par ? 1 : 0); i < vl; i += 2) {
      if (!causal) {
        if (!ptx::mbar_wait(mma_done + i, 0, limit, p.status)) limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
      }
      const int key = key_base + kTileKeys * (ft + i) + row;
      const bool vis = key >= S && key < S + NV;
      for (int hh = 0; hh < nh; ++hh) {
        float acc0 = 0.f, acc1 = 0.f;
        for (int c16 = 0; c16 < ntp; c16 += 16) {
          const int col = hh * p.ntp_max + c16;
          float x[16];
          ptx::tmem_ld16(tmem + lane_base + (uint32_t)(i * ncs + col), x);
          const float4* w4 = reinterpret_cast<const float4*>(colw + col);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const float4 w = w4[v];
            acc0 = fmaf(x[4 * v], w.x, acc0);
            acc1 = fmaf(x[4 * v + 1], w.y, acc1);
            acc0 = fmaf(x[4 * v + 2], w.z, acc0);
            acc1 = fmaf(x[4 * v + 3], w.w, acc1);
          }
        }
        a_sm[hh * p.tpc * kTileKeys + i * kTileKeys + row] = acc0 + acc1;
        if (vis)
          p.a_out[((size_t)l * la.H + h0 + hh) * (size_t)la.sum_vis + v0 + (key - S)] =
              acc0 + acc1;
      }
    }
    // ---- this CTA's share of the (layer, head) statistics of the visual scores
    ptx::named_bar(1, kEpiThreads);
    const int kb0 = key_base + kTileKeys * ft;
    const int i_lo = max(S, kb0) - kb0;
    const int i_hi = max(min(S + NV, kb0 + kTileKeys * nt) - kb0, i_lo);
    for (int hh = 0; hh < nh; ++hh) {
      const float* ah = a_sm + hh * p.tpc * kTileKeys;
      float ls = 0.f, lm = kNegBig;
      for (int x = i_lo + et; x < i_hi; x += kEpiThreads) {
        ls += ah[x];
        lm = fmaxf(lm, ah[x] * 1.4426950408889634f);
      }
      ls = warp_reduce(ls, [](float u, float v) { return u + v; });
      lm = warp_reduce(lm, [](float u, float v) { return fmaxf(u, v); });
      if (lane == 0) sred[ew] = make_float2(ls, lm);
      ptx::named_bar(1, kEpiThreads);
      float Sa = 0.f, Ma = kNegBig;
      for (int w = 0; w < kEpiWarps; ++w) {
        Sa += sred[w].x;
        Ma = fmaxf(Ma, sred[w].y);
      }
      ptx::named_bar(1, kEpiThreads);
      float le = 0.f;
      for (int x = i_lo + et; x < i_hi; x += kEpiThreads)
        le += fast_ex2(fmaf(ah[x], 1.4426950408889634f, -Ma));
      le = warp_reduce(le, [](float u, float v) { return u + v; });
      if (lane == 0) sred[ew] = make_float2(le, 0.f);
      ptx::named_bar(1, kEpiThreads);
      if (et == 0) {
        float Ea = 0.f;
        for (int w = 0; w < kEpiWarps; ++w) Ea += sred[w].x;
        spart[hh] = make_float4(Sa, Ma, Ea, 0.f);
      }
      ptx::named_bar(1, kEpiThreads);
    }
  }

  // ---- teardown: peers may still read `part`; rank 0 merges the statistics
  ptx::cluster_arrive();
  ptx::cluster_wait();
  if (rank == 0 && ok && threadIdx.x >= 64 && threadIdx.x - 64 < nh) {
    const int hh = threadIdx.x - 64;
    float Sa = 0.f, Ma = kNegBig, Ea = 0.f;
    for (int r = 0; r < p.cluster; ++r) {
      const float4 o = ptx::ld_dsmem_f4(spart + hh, (uint32_t)r);
      Sa += o.x;
      lse_merge(Ma, Ea, o.y, o.z);
    }
    p.stats[((size_t)b * la.L + l) * la.H + h0 + hh] = stats_entry(Sa, Ma, Ea);
  }
  ptx::cluster_arrive();
  ptx::cluster_wait();
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, p.tmem_cols);
  }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

}  // namespace

// 3-D map over rows of (heads x 128) bf16: dims (128, heads, rows), box (64, 1, box_rows).
bool make_score_map(CUtensorMap* map, const void* base, int heads, int64_t rows, int64_t row_stride_el,
              int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {128, (cuuint64_t)heads, (cuuint64_t)rows};
  cuuint64_t strides[2] = {256, (cuuint64_t)row_stride_el * 2};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)box_rows};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}


cudaError_t launch_score_tc(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                            const void* k, int64_t k_stride, float* a_out, float4* stats,
                            uint32_t* counters, uint32_t* status, cudaStream_t st,
                            int* unsupported, bool pdl) {
  *unsupported = 0;
  // kernel choice (measured): the cluster-per-unit kernel when every unit's
  // key tiles spread over at most two CTAs per SM in one wave (batch 1); the
  // persistent single-CTA kernel when every
  // unit's logits fit TMEM in one column group (short sequences, e.g. one
  // LLaVA image); the streaming kernel for longer sequences, GQA and batched
  // ragged text (up to 128 text rows); the column-group kernel above 128 text
  // rows while the K tiles fit shared memory; the cluster kernel otherwise
  int split_c = 0, split_t = 0;
  if (score_split_plan(la, mode, false, &split_c, &split_t))
    return launch_score_split(la, mode, q, q_stride, k, k_stride, a_out, stats, counters, status,
                              st, nullptr, split_c, split_t, pdl);
  const bool unit = score_unit_fits(la, mode);
  if (unit && score_unit_single_group(la, mode))
    return launch_score_unit(la, mode, q, q_stride, k, k_stride, a_out, stats, counters, status,
                             st, pdl);
  if (score_stream_fits(la))
    return launch_score_stream(la, mode, q, q_stride, k, k_stride, a_out, stats, counters, status,
                               st, nullptr, pdl);
  if (unit)
    return launch_score_unit(la, mode, q, q_stride, k, k_stride, a_out, stats, counters, status,
                             st, pdl);
  TcArgs p;
  p.la = la;
  p.group = la.H / la.H_kv;
  p.mode = mode;
  p.ntp_max = ((std::max(la.max_text, 1) + 15) / 16) * 16;
  if (p.ntp_max > 256) {
    *unsupported = 1;
    return cudaSuccess;
  }
  p.hpc = std::max(1, std::min(p.group, 256 / p.ntp_max));
  p.groups_per_kv = (p.group + p.hpc - 1) / p.hpc;
  const int ncs = p.hpc * p.ntp_max;
  const int span = (mode == E2S_SCORE_CAUSAL_PROB) ? la.max_T : la.max_vis;
  const int max_tiles = (span + kTileKeys - 1) / kTileKeys;
  if (max_tiles == 0 || la.sum_vis == 0) return cudaSuccess;
  const int tpc_tmem = std::max(1, 512 / ncs);  // every tile's logits stay in TMEM
  p.tpc = std::min({2, max_tiles, tpc_tmem});
  p.cluster = (max_tiles + p.tpc - 1) / p.tpc;
  while (p.cluster > kMaxCluster && p.tpc < tpc_tmem) {
    ++p.tpc;
    p.cluster = (max_tiles + p.tpc - 1) / p.tpc;
  }
  if (p.cluster > kMaxCluster) {
    *unsupported = 1;
    return cudaSuccess;
  }
  uint32_t cols = 32;
  while ((int)cols < p.tpc * ncs) cols <<= 1;
  p.tmem_cols = cols;
  p.scale = 1.0f / sqrtf(128.0f);
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.a_out = a_out;
  p.stats = stats;
  p.counters = counters;
  p.status = status;

  int dev = 0, smem_sm = 0, smem_optin = 0, reserved = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
  const SmemPlan plan = smem_plan(p.hpc, p.ntp_max, p.tpc);
  size_t smem = plan.total + 1024;  // + alignment slack
  // Never let more CTAs share an SM than TMEM can hold at once: a CTA blocked
  // in tcgen05.alloc must not wait on a CTA that waits on its own cluster.
  const int max_ctas = 512 / (int)p.tmem_cols;
  const size_t floor_smem = (size_t)smem_sm / (size_t)(max_ctas + 1) - (size_t)reserved + 128;
  if (smem < floor_smem) smem = floor_smem;
  if ((int)smem > smem_optin) {
    *unsupported = 1;
    return cudaSuccess;
  }
  CUtensorMap tmQ, tmK;
  if (!make_score_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_text, q_stride, kQBoxRows) ||
      !make_score_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTileKeys))
    return cudaErrorInvalidValue;
  const long long units = (long long)la.B * la.L * la.H_kv * p.groups_per_kv;
  return launch_kernel(score_tc_kernel, dim3((unsigned)(units * p.cluster)), dim3(kThreads), smem,
                       st, p.cluster, pdl, tmQ, tmK, p);
}

}  // namespace e2s
