// Per-layer evidence, layer-wise Dempster-Shafer fusion and (optionally) the
// spatial-novelty Top-K, in one launch (Sec. 4.1-4.3, Eqs. 8-23).
//
// One thread-block cluster per image; CTA r of the cluster owns a contiguous
// slice of the image's visual tokens.  For each group of evidence layers:
//   1. the slice of a[l][h][.] is staged into shared memory (coalesced);
//   2. per-(layer, head) partial normalisation statistics of Eq. 8 (sum for
//      the renormalisation, max / sum of exp2 for the softmax) are reduced
//      per warp and exchanged across the cluster through distributed shared
//      memory;
//   3. one thread per (layer, token) forms the supports p (Eq. 9), the
//      reliability rho (Eq. 10) and the layer mass (Eq. 11);
//   4. one thread per token combines the layers in order with Dempster's rule
//      and the conflict term (Eqs. 12-16).
// Then q (Eq. 19) is written; with selection enabled every CTA also stores
// its q into CTA 0's shared memory (distributed shared memory), and CTA 0
// runs select_image on the whole image.
#include <cuda_runtime.h>

#include <algorithm>

#include "select_core.cuh"
#include "sm100_ptx.cuh"

namespace e2s {
namespace {

constexpr int kEvThreads = 256;
constexpr int kEvWarps = kEvThreads / 32;
constexpr int kTokPerThread = 2;
constexpr int kMaxTs = kEvThreads * kTokPerThread;
constexpr int kMaxEvCluster = 16;
constexpr float kLog2e = 1.4426950408889634f;

struct EvArgs {
  LayoutArgs la;
  int softmax;
  uint32_t flags;
  float lam;
  int G;
  int cluster, ts, lps;
  uint32_t ts_magic;   // ceil(2^32 / ts)
  const float* a;
  const float4* prior;
  const int32_t* cand;
  float4* mass_out;
  float4* fused_out;
  float* q_out;
  float* q_tilde;
  const int32_t* keep_count;
  const int32_t* keep_off;
  int32_t sum_keep;
  int32_t* keep_idx;
  int do_select;
  uint32_t* status;
};

struct EvPlan {
  uint32_t A, part, st, ms, vs, qall, total;
};

// A: [lps][H][ts] staged scores (reused as the select's keys); part: [2][lps*H]
// float4 cluster-visible partials; st: [lps*H] merged statistics; ms: [lps][ts]
// layer masses; vs: [lps][ts] head sums of a (ablation A1); qall: [max_vis] the
// image's priorities, written into CTA 0 by every CTA of the cluster.  The
// select's keys and cell ids reuse A (max_vis * 5 bytes).
__host__ __device__ inline EvPlan ev_plan(int H, int ts, int lps, int max_vis) {
  EvPlan s;
  const uint32_t a_bytes = (uint32_t)lps * H * ts * 4u;
  const uint32_t key_bytes = (uint32_t)max_vis * 4u;
  const uint32_t sel_bytes = (uint32_t)max_vis * 5u;
  s.A = 0;
  s.part = ((a_bytes > sel_bytes ? a_bytes : sel_bytes) + 15u) & ~15u;
  s.st = s.part + 2u * (uint32_t)lps * H * 16u;
  s.ms = s.st + (uint32_t)lps * H * 16u;
  s.vs = s.ms + (uint32_t)lps * ts * 16u;     // [lps][ts] sum over heads of a
  s.qall = s.vs + (((uint32_t)lps * ts * 4u + 15u) & ~15u);
  s.total = s.qall + key_bytes;
  return s;
}

// st = (1 / sum a, max a*log2e, 1 / sum 2^(a*log2e - max), sum a) of one
// (layer, head) over the image's candidates.
__device__ __forceinline__ float support_p(float a, float4 st, int softmax, float N, float invN) {
  float r;
  if (softmax)
    r = fast_ex2(fmaf(a, kLog2e, -st.y)) * st.z;   // Eq. 8
  else
    r = st.w > 0.f ? a * st.x : invN;               // r = a / sum a
  const float x = N * r;
  return x * fast_rcp(1.f + x);                     // Eq. 9
}

__global__ void __launch_bounds__(kEvThreads) evidence_kernel(const EvArgs p) {
  extern __shared__ __align__(16) uint8_t ev_smem[];
  __shared__ SelectSmem ss;
  const LayoutArgs& la = p.la;
  const int H = la.H;
  const EvPlan plan = ev_plan(H, p.ts, p.lps, la.max_vis);
  float* A = reinterpret_cast<float*>(ev_smem + plan.A);
  float4* part = reinterpret_cast<float4*>(ev_smem + plan.part);
  float4* st = reinterpret_cast<float4*>(ev_smem + plan.st);
  float4* ms = reinterpret_cast<float4*>(ev_smem + plan.ms);
  float* vs = reinterpret_cast<float*>(ev_smem + plan.vs);
  float* qall = reinterpret_cast<float*>(ev_smem + plan.qall);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_launch_dependents();
  pdl_wait();   // a (and the other inputs) come from the previous kernel
  const uint32_t rank = ptx::cluster_ctarank();
  const int b = blockIdx.x / p.cluster;
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  const bool ok = NV >= 0 && NV <= la.max_vis && v0 >= 0 && v0 + NV <= la.sum_vis &&
                  __ldg(la.vis_off + b + 1) - v0 == NV;
  if (!ok && tid == 0 && rank == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
  const int per = ok ? (NV + p.cluster - 1) / p.cluster : 0;
  const int n0 = min(NV, (int)rank * per);
  int Ts = ok ? min(NV, n0 + per) - n0 : 0;
  if (Ts > p.ts) {  // host sizing guarantees Ts <= ts; never overrun the slice buffers
    if (tid == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    Ts = 0;
  }
  const float N = (float)NV;
  const float invN = NV > 0 ? 1.f / N : 0.f;
  const size_t plane = (size_t)la.sum_vis;
  const float inv_h = 1.f / (float)H;
  // idx / Ts and pair / Ts_pad as multiply-highs (exact for idx < 2^19 and
  // divisors <= 512; p.ts_magic is computed on the host)
  const int Ts_pad = p.ts;
  const uint32_t tsp_magic = p.ts_magic;

  // per-token fusion state: token j = tid + kEvThreads * tt of the slice
  float fI[kTokPerThread], fU[kTokPerThread], fT[kTokPerThread], Kf[kTokPerThread],
      vsum[kTokPerThread];
  bool have[kTokPerThread];
  const bool use_prior = p.prior != nullptr && !(p.flags & E2S_NO_LAYER_FUSION);
#pragma unroll
  for (int tt = 0; tt < kTokPerThread; ++tt) {
    const int j = tid + kEvThreads * tt;
    fI[tt] = 0.f; fU[tt] = 0.f; fT[tt] = 1.f; Kf[tt] = 0.f; vsum[tt] = 0.f;
    have[tt] = false;
    if (use_prior && j < Ts) {
      const float4 pr = p.prior[v0 + n0 + j];
      fI[tt] = pr.x; fU[tt] = pr.y; fT[tt] = pr.z;
      have[tt] = true;
    }
  }
  const int l_begin = (p.flags & E2S_NO_LAYER_FUSION) ? la.L - 1 : 0;

  int stage = 0;
  for (int l0 = 0; l0 < la.L; l0 += p.lps, ++stage) {
    const int nl = min(p.lps, la.L - l0);
    const int rows = nl * H;
    float4* pbuf = part + (stage & 1) * p.lps * H;
    // 1. stage the slice of a[l0 .. l0+nl)[h][.] with asynchronous copies,
    //    every one in flight before the single wait
    const float* src = p.a + (size_t)l0 * H * plane + v0 + n0;
    const int total = rows * Ts_pad;
    for (int idx = tid; idx < total; idx += kEvThreads) {
      const int r = (int)__umulhi((uint32_t)idx, tsp_magic);
      const int j = idx - r * Ts_pad;
      if (j < Ts) ptx::cp_async4(A + r * p.ts + j, src + (size_t)r * plane + j);
    }
    ptx::cp_async_wait_all();
    __syncthreads();
    // 2. partial statistics per (layer, head) row, from shared memory
    for (int r = warp; r < rows; r += kEvWarps) {
      const float* Ar = A + r * p.ts;
      float s = 0.f, m = kNegBig, e = 0.f;
      if (p.softmax) {
        for (int j = lane; j < Ts; j += 32) m = fmaxf(m, Ar[j] * kLog2e);
        m = warp_reduce(m, [](float x, float y) { return fmaxf(x, y); });
        for (int j = lane; j < Ts; j += 32) e += fast_ex2(fmaf(Ar[j], kLog2e, -m));
        e = warp_reduce(e, [](float x, float y) { return x + y; });
        if (Ts == 0) m = kNegBig;
      } else {
        for (int j = lane; j < Ts; j += 32) s += Ar[j];
        s = warp_reduce(s, [](float x, float y) { return x + y; });
      }
      if (lane == 0) pbuf[r] = make_float4(s, m, e, 0.f);
    }
    ptx::cluster_arrive();
    ptx::cluster_wait();
    for (int r = tid; r < rows; r += kEvThreads) {
      float4 o[kMaxEvCluster];
#pragma unroll
      for (int c = 0; c < kMaxEvCluster; ++c)
        if (c < p.cluster) o[c] = ptx::ld_dsmem_f4(pbuf + r, (uint32_t)c);
      float s = 0.f, m = kNegBig, e = 0.f;
#pragma unroll
      for (int c = 0; c < kMaxEvCluster; ++c)
        if (c < p.cluster) {
          s += o[c].x;
          lse_merge(m, e, o[c].y, o[c].z);
        }
      st[r] = make_float4(s != 0.f ? 1.f / s : 0.f, m, e > 0.f ? 1.f / e : 0.f, s);
    }
    __syncthreads();
    // 3. supports, reliability and mass per (layer, token): four lanes per
    //    (layer, token), one quarter of the heads each, reduced by shuffles;
    //    supports are written over the staged scores
    const int hq_len = (H + 3) >> 2;
    const int n_items = 4 * nl * Ts_pad;
    for (int base = warp * 32; base < n_items; base += kEvThreads) {  // warp-uniform trips
      const int it = base + lane;
      const int hq = it & 3;
      const int pair = it >> 2;                         // li * Ts_pad + j
      const int li = (int)__umulhi((uint32_t)pair, tsp_magic);
      const int j = pair - li * Ts_pad;
      const bool live = it < n_items && j < Ts;
      const int h_lo = hq * hq_len, h_hi = min(H, h_lo + hq_len);
      float* Ac = A + (size_t)li * H * p.ts + j;
      const float4* sl = st + li * H;
      float sum_p = 0.f, sum_a = 0.f;
      if (live)
        for (int h = h_lo; h < h_hi; ++h) {
          const float av = Ac[h * p.ts];
          const float pv = support_p(av, sl[h], p.softmax, N, invN);
          sum_a += av;
          sum_p += pv;
          Ac[h * p.ts] = pv;
        }
      sum_p += __shfl_xor_sync(0xffffffffu, sum_p, 1);
      sum_p += __shfl_xor_sync(0xffffffffu, sum_p, 2);
      sum_a += __shfl_xor_sync(0xffffffffu, sum_a, 1);
      sum_a += __shfl_xor_sync(0xffffffffu, sum_a, 2);
      const float p_bar = sum_p * inv_h;
      float clar = 0.f, dev = 0.f;
      if (live)
        for (int h = h_lo; h < h_hi; ++h) {
          const float pv = Ac[h * p.ts];
          clar += pv - 0.5f;
          dev += fabsf(pv - p_bar);
        }
      clar += __shfl_xor_sync(0xffffffffu, clar, 1);
      clar += __shfl_xor_sync(0xffffffffu, clar, 2);
      dev += __shfl_xor_sync(0xffffffffu, dev, 1);
      dev += __shfl_xor_sync(0xffffffffu, dev, 2);
      if (live && hq == 0) {
        float rho = (2.f * inv_h) * fabsf(clar) * (1.f - (2.f * inv_h) * dev);  // Eq. 10
        if (p.flags & E2S_NO_RELIABILITY) rho = 1.f;
        const float4 m4 = make_float4(rho * p_bar, rho * (1.f - p_bar), 1.f - rho, p_bar);  // Eq. 11
        ms[li * p.ts + j] = m4;
        vs[li * p.ts + j] = sum_a;
        if (p.mass_out) p.mass_out[(size_t)(l0 + li) * plane + v0 + n0 + j] = m4;
      }
    }
    __syncthreads();
    // 4. Dempster combination across the stage's layers (Eqs. 12-16)
#pragma unroll
    for (int tt = 0; tt < kTokPerThread; ++tt) {
      const int j = tid + kEvThreads * tt;
      if (j >= Ts) continue;
      for (int li = 0; li < nl; ++li) {
        if (p.flags & E2S_VANILLA) vsum[tt] += vs[li * p.ts + j];
        if (l0 + li < l_begin) continue;
        const float4 m = ms[li * p.ts + j];
        if (!have[tt]) {
          fI[tt] = m.x; fU[tt] = m.y; fT[tt] = m.z; Kf[tt] = 0.f;
          have[tt] = true;
        } else {
          const float K = fI[tt] * m.y + fU[tt] * m.x;
          const float omk = 1.f - K;
          if (omk <= 0.f) {
            fI[tt] = 0.f; fU[tt] = 0.f; fT[tt] = 1.f; Kf[tt] = 1.f;
          } else {
            const float inv = 1.f / omk;
            const float nI = (fI[tt] * m.x + fI[tt] * m.z + fT[tt] * m.x) * inv;
            const float nU = (fU[tt] * m.y + fU[tt] * m.z + fT[tt] * m.y) * inv;
            const float nT = fT[tt] * m.z * inv;
            fI[tt] = nI; fU[tt] = nU; fT[tt] = nT; Kf[tt] = K;
          }
        }
      }
    }
    __syncthreads();
  }
  // Eqs. 18-19; with selection every CTA also writes its q into CTA 0
#pragma unroll
  for (int tt = 0; tt < kTokPerThread; ++tt) {
    const int j = tid + kEvThreads * tt;
    if (j >= Ts) continue;
    const float Pl = fI[tt] + fT[tt];
    float q = (p.flags & E2S_NO_CONFLICT) ? Pl : 1.f - (1.f - Pl) * (1.f - Kf[tt]);
    if (p.flags & E2S_VANILLA) q = vsum[tt] / (float)(la.L * H);
    p.fused_out[v0 + n0 + j] = make_float4(fI[tt], fU[tt], fT[tt], Kf[tt]);
    p.q_out[v0 + n0 + j] = q;
    if (p.do_select) ptx::st_dsmem_f32(qall + n0 + j, 0u, q);
  }
  // every CTA waits here: peers may still read this CTA's partials, and CTA 0
  // needs every q before it selects
  ptx::cluster_arrive();
  ptx::cluster_wait();
  if (!p.do_select || rank != 0) return;
  if (!(ok && select_args_ok(la, b, p.cand != nullptr, p.keep_count, p.keep_off, p.sum_keep))) {
    if (tid == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    return;
  }
  const float lam = (p.flags & (E2S_NO_NOVELTY | E2S_VANILLA)) ? 0.f : p.lam;
  select_image(qall, p.cand ? p.cand + v0 : nullptr, NV, __ldg(la.grid_h + b),
               __ldg(la.grid_w + b), p.G, lam, __ldg(p.keep_count + b),
               reinterpret_cast<uint32_t*>(A), reinterpret_cast<uint8_t*>(A) + 4 * la.max_vis, ss,
               p.q_tilde ? p.q_tilde + v0 : nullptr, p.keep_idx + __ldg(p.keep_off + b),
               p.status);
}

}  // namespace

cudaError_t launch_evidence(const LayoutArgs& la, int norm_softmax, uint32_t flags, float lambda,
                            int G, const float* a, const float* prior, const int32_t* cand,
                            float* mass_out, float* fused_out, float* q_out, float* q_tilde,
                            const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                            int32_t* keep_idx, int do_select, uint32_t* status, cudaStream_t st,
                            int* unsupported) {
  *unsupported = 0;
  if (la.sum_vis == 0 && !do_select) return cudaSuccess;
  EvArgs p;
  p.la = la;
  p.softmax = norm_softmax;
  p.flags = flags;
  p.lam = lambda;
  p.G = G;
  const int mv = std::max(la.max_vis, 1);
  p.cluster = std::min(8, std::max(1, (mv + 95) / 96));
  p.ts = (mv + p.cluster - 1) / p.cluster;
  if (p.ts > kMaxTs) {
    p.cluster = kMaxEvCluster;
    p.ts = (mv + p.cluster - 1) / p.cluster;
  }
  if (p.ts > kMaxTs) {
    *unsupported = 1;
    return cudaSuccess;
  }
  p.ts = std::max(p.ts, 2);   // the multiplier of a stride of 1 does not fit 32 bits
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const size_t budget = std::min<size_t>((size_t)optin - sizeof(SelectSmem) - 64, 160u << 10);
  p.lps = 0;
  for (int lps = la.L; lps >= 1; --lps)
    if (ev_plan(la.H, p.ts, lps, la.max_vis).total <= budget) {
      p.lps = lps;
      break;
    }
  if (p.lps == 0) {
    *unsupported = 1;
    return cudaSuccess;
  }
  p.a = a;
  p.prior = reinterpret_cast<const float4*>(prior);
  p.cand = cand;
  p.mass_out = reinterpret_cast<float4*>(mass_out);
  p.fused_out = reinterpret_cast<float4*>(fused_out);
  p.q_out = q_out;
  p.q_tilde = q_tilde;
  p.keep_count = keep_count;
  p.keep_off = keep_off;
  p.sum_keep = sum_keep;
  p.keep_idx = keep_idx;
  p.do_select = do_select;
  p.status = status;
  p.ts_magic = (uint32_t)((0x100000000ull + (uint64_t)p.ts - 1) / (uint64_t)p.ts);
  const size_t smem = ev_plan(la.H, p.ts, p.lps, la.max_vis).total;
  return launch_kernel(evidence_kernel, dim3((unsigned)(la.B * p.cluster)), dim3(kEvThreads), smem,
                       st, p.cluster, true, p);
}

}  // namespace e2s
