// Evidence, layer-wise fusion and selection of e2s_decide (Sec. 4.1-4.3,
// Eqs. 8-23), token-parallel.  The normalisation statistics of Eq. 8 for
// every (image, layer, head) were produced by the score kernel, so tokens are
// independent here: a CTA takes 64 visual tokens of one image, eight lanes per
// token (one eighth of the heads each):
//   1. the image's statistics and the CTA's a[l][h][token] values are copied
//      into shared memory with asynchronous copies (16-byte copies when the
//      rows are aligned), all of a group of layers in flight at once;
//   2. per (token, layer): supports p (Eq. 9) of the lane's heads, kept in
//      registers; p_bar and the reliability terms of Eq. 10 summed over the
//      eight lanes with three shuffles; rho and the layer mass (Eq. 11);
//   3. per token: Dempster combination over the layers (Eqs. 12-16), Pl and q
//      (Eqs. 18-19);
//   4. every CTA folds its tokens' bids for their cells' representatives
//      (Eqs. 20-21) into the image's cell arg-max keys in global memory and
//      bumps the image's arrival counter; the last CTA of the image computes
//      q~ and the Top-K (Eqs. 22-23) over the whole image and re-arms the
//      keys and the counter.
#include <cuda_runtime.h>

#include <algorithm>

#include "select_core.cuh"
#include "sm100_ptx.cuh"

namespace e2s {
namespace {

constexpr int kTok = 64;                 // visual tokens per CTA
constexpr int kLanes = 8;                // lanes per token (head groups)
constexpr int kDecThreads = kLanes * kTok;
constexpr int kMaxHpl = 8;               // supports cached per lane (H <= 64)
constexpr float kLog2e = 1.4426950408889634f;
constexpr size_t kDecStageBytes = 96u << 10;   // staged scores per group of layers

struct DecArgs {
  LayoutArgs la;
  int softmax;
  uint32_t flags;
  float lam;
  int G;
  int blocks_per_image;
  int lps;   // evidence layers staged at a time
  const float* a;
  const float4* stats;
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
  unsigned long long* cell_best;   // [B][64] cell arg-max keys, zero between calls
  uint32_t* counters;              // [B] arrival counters, zero between calls
  uint32_t* status;
};

// st = (S, M, 1/E, 1/S) of one (layer, head): sum of a, max of a*log2e, the
// reciprocal of the sum of 2^(a*log2e - M), the reciprocal of S (0 if S <= 0).
__device__ __forceinline__ float support_p(float a, float4 st, int softmax, float N, float invN) {
  float r;
  if (softmax)
    r = fast_ex2(fmaf(a, kLog2e, -st.y)) * st.z;   // Eq. 8
  else
    r = st.x > 0.f ? a * st.w : invN;               // r = a / sum a
  const float x = N * r;
  return x * fast_rcp(1.f + x);                     // Eq. 9
}

__device__ __forceinline__ float lane_sum8(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  v += __shfl_xor_sync(0xffffffffu, v, 2);
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  return v;
}

__global__ void __launch_bounds__(kDecThreads) decide_kernel(const DecArgs p) {
  extern __shared__ __align__(16) uint8_t dec_smem[];
  __shared__ SelectSmem ss;
  __shared__ int is_last;
  __shared__ unsigned long long cb_s[kDecideCells];   // this CTA's cell arg-max keys
  const LayoutArgs& la = p.la;
  const int H = la.H, L = la.L;
  // [L][H] statistics, then [lps][H][kTok] staged scores (the select's scratch later)
  float4* st_s = reinterpret_cast<float4*>(dec_smem);
  float* A = reinterpret_cast<float*>(dec_smem + (size_t)L * H * 16);
  const int tid = threadIdx.x;
  for (int i = tid; i < kDecideCells; i += kDecThreads) cb_s[i] = 0ull;
  pdl_launch_dependents();
  pdl_wait();   // a and the statistics come from the score kernel

  const int b = blockIdx.x / p.blocks_per_image;
  const int blk = blockIdx.x - b * p.blocks_per_image;
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  const bool ok = NV >= 0 && NV <= la.max_vis && v0 >= 0 && v0 + NV <= la.sum_vis &&
                  __ldg(la.vis_off + b + 1) - v0 == NV;
  const int n0 = blk * kTok;
  const int ntok = ok ? max(0, min(kTok, NV - n0)) : 0;
  const size_t plane = (size_t)la.sum_vis;
  // 16-byte copies need every staged row segment 16-byte aligned
  const bool vec = ((reinterpret_cast<uintptr_t>(p.a) | ((plane & 3) << 2) |
                     ((size_t)(v0 + n0) << 2)) & 15) == 0;

  // the image's statistics (every layer) arrive with the first group of scores
  for (int i = tid; i < L * H * 4; i += kDecThreads)
    ptx::cp_async4(reinterpret_cast<float*>(st_s) + i,
                   reinterpret_cast<const float*>(p.stats + (size_t)b * L * H) + i);

  // 2-3. evidence and fusion, lanes 8j .. 8j+7 own token j
  const int j = tid / kLanes, hq = tid % kLanes;
  const bool live = j < ntok;
  const int gv = v0 + n0 + j;
  const float N = (float)NV;
  const float invN = NV > 0 ? 1.f / N : 0.f;
  const float inv_h = 1.f / (float)H;
  const int hpl = (H + kLanes - 1) / kLanes;
  const int h_lo = hq * hpl, h_cnt = max(0, min(H, h_lo + hpl) - h_lo);
  float fI = 0.f, fU = 0.f, fT = 1.f, K = 0.f, vsum = 0.f;
  bool have = false;
  if (live && p.prior != nullptr && !(p.flags & E2S_NO_LAYER_FUSION)) {
    const float4 pr = p.prior[gv];
    fI = pr.x; fU = pr.y; fT = pr.z;
    have = true;
  }
  const int l_begin = (p.flags & E2S_NO_LAYER_FUSION) ? L - 1 : 0;
  for (int l = 0; l < L; ++l) {
    const int li = l % p.lps;
    if (li == 0) {
      // 1. stage a[l .. l+lps)[h][n0 .. n0+ntok) (coalesced along the tokens)
      const int nl = min(p.lps, L - l);
      __syncthreads();   // the previous group is consumed
      if (vec) {
        for (int idx = tid; idx < nl * H * (kTok / 4); idx += kDecThreads) {
          const int jj = 4 * (idx & (kTok / 4 - 1)), lh = idx / (kTok / 4);
          const float* src = p.a + ((size_t)l * H + lh) * plane + v0 + n0 + jj;
          if (jj + 4 <= ntok) {
            ptx::cp_async16(A + lh * kTok + jj, src);
          } else {
            for (int e = 0; e < 4; ++e)
              if (jj + e < ntok) ptx::cp_async4(A + lh * kTok + jj + e, src + e);
          }
        }
      } else {
        for (int idx = tid; idx < nl * H * kTok; idx += kDecThreads) {
          const int jj = idx & (kTok - 1), lh = idx / kTok;
          if (jj < ntok)
            ptx::cp_async4(A + idx, p.a + ((size_t)l * H + lh) * plane + v0 + n0 + jj);
        }
      }
      ptx::cp_async_wait_all();
      __syncthreads();
    }
    const float* Al = A + (size_t)li * H * kTok + j;
    const float4* sl = st_s + (size_t)l * H;
    float pv[kMaxHpl];
    float sum_p = 0.f, sum_a = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxHpl; ++k) {
      pv[k] = 0.f;
      if (live && k < h_cnt) {
        const int h = h_lo + k;
        const float av = Al[h * kTok];
        sum_a += av;
        pv[k] = support_p(av, sl[h], p.softmax, N, invN);
        sum_p += pv[k];
      }
    }
    if (live)
      for (int h = h_lo + kMaxHpl; h < h_lo + h_cnt; ++h) {   // H > 64 only
        const float av = Al[h * kTok];
        sum_a += av;
        sum_p += support_p(av, sl[h], p.softmax, N, invN);
      }
    sum_p = lane_sum8(sum_p);
    sum_a = lane_sum8(sum_a);
    const float p_bar = sum_p * inv_h;
    float clar = 0.f, dev = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxHpl; ++k)
      if (live && k < h_cnt) {
        clar += pv[k] - 0.5f;
        dev += fabsf(pv[k] - p_bar);
      }
    if (live)
      for (int h = h_lo + kMaxHpl; h < h_lo + h_cnt; ++h) {
        const float v = support_p(Al[h * kTok], sl[h], p.softmax, N, invN);
        clar += v - 0.5f;
        dev += fabsf(v - p_bar);
      }
    clar = lane_sum8(clar);
    dev = lane_sum8(dev);
    float rho = (2.f * inv_h) * fabsf(clar) * (1.f - (2.f * inv_h) * dev);  // Eq. 10
    if (p.flags & E2S_NO_RELIABILITY) rho = 1.f;
    const float mI = rho * p_bar, mU = rho * (1.f - p_bar), mT = 1.f - rho;  // Eq. 11
    if (live && hq == 0 && p.mass_out)
      p.mass_out[(size_t)l * plane + gv] = make_float4(mI, mU, mT, p_bar);
    vsum += sum_a;
    if (l < l_begin) continue;
    if (!have) {                                   // Eq. 12
      fI = mI; fU = mU; fT = mT; K = 0.f;
      have = true;
    } else {                                       // Eqs. 13-16
      const float Kc = fI * mU + fU * mI;
      const float omk = 1.f - Kc;
      if (omk <= 0.f) {
        fI = 0.f; fU = 0.f; fT = 1.f; K = 1.f;
      } else {
        const float inv = 1.f / omk;
        const float nI = (fI * mI + fI * mT + fT * mI) * inv;
        const float nU = (fU * mU + fU * mT + fT * mU) * inv;
        const float nT = fT * mT * inv;
        fI = nI; fU = nU; fT = nT; K = Kc;
      }
    }
  }
  const bool select = p.keep_count != nullptr;
  const int G = p.G;
  const int gh = __ldg(la.grid_h + b), gw = __ldg(la.grid_w + b);
  if (live && hq == 0) {
    const float Pl = fI + fT;                                                   // Eq. 18
    float q = (p.flags & E2S_NO_CONFLICT) ? Pl : 1.f - (1.f - Pl) * (1.f - K);  // Eq. 19
    if (p.flags & E2S_VANILLA) q = vsum / (float)(L * H);
    p.fused_out[gv] = make_float4(fI, fU, fT, K);
    p.q_out[gv] = q;
    // 4a. this token's bid for its cell's representative (Eqs. 20-21)
    const int n = n0 + j;
    if (select && gh > 0 && gw > 0)
      atomicMax(&cb_s[token_cell(p.cand ? p.cand + v0 : nullptr, n, gh, gw, G, p.status)],
                cell_key(q, n));
  }
  if (!select) return;
  __syncthreads();
  for (int i = tid; i < G * G; i += kDecThreads)
    if (cb_s[i] != 0ull) atomicMax(p.cell_best + (size_t)b * kDecideCells + i, cb_s[i]);

  // 4b. the last CTA of the image selects; the barrier orders every thread's
  // writes before thread 0's fence and arrival
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const uint32_t ticket = atomicAdd(p.counters + b, 1u);
    is_last = ticket == (uint32_t)(p.blocks_per_image - 1);
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  if (tid == 0) p.counters[b] = 0u;   // re-armed for the next call
  unsigned long long* cells_g = p.cell_best + (size_t)b * kDecideCells;
  if (!(ok && select_args_ok(la, b, p.cand != nullptr, p.keep_count, p.keep_off, p.sum_keep))) {
    for (int i = tid; i < kDecideCells; i += kDecThreads) cells_g[i] = 0ull;
    if (tid == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    return;
  }
  const float lam = (p.flags & (E2S_NO_NOVELTY | E2S_VANILLA)) ? 0.f : p.lam;
  select_image_from_cells(p.q_out + v0, p.cand ? p.cand + v0 : nullptr, NV, gh, gw, G, lam,
                          __ldg(p.keep_count + b), cells_g, reinterpret_cast<uint32_t*>(A),
                          reinterpret_cast<uint8_t*>(A) + 4 * (size_t)la.max_vis, ss,
                          p.q_tilde ? p.q_tilde + v0 : nullptr,
                          p.keep_idx + __ldg(p.keep_off + b), p.status);
}

}  // namespace

bool decide_fits(const LayoutArgs& la) {
  return (size_t)la.H * kTok * 4 <= kDecStageBytes && (size_t)la.L * la.H * 16 <= (64u << 10);
}

cudaError_t launch_decide(const LayoutArgs& la, int norm_softmax, uint32_t flags, float lambda,
                          int G, const float* a, const float4* stats, const float* prior,
                          const int32_t* cand, float* mass_out, float* fused_out, float* q_out,
                          float* q_tilde, const int32_t* keep_count, const int32_t* keep_off,
                          int32_t sum_keep, int32_t* keep_idx, uint32_t* scratch,
                          uint32_t* status, cudaStream_t st, int* unsupported) {
  *unsupported = 0;
  if (la.max_vis == 0) return cudaSuccess;
  if (!decide_fits(la)) {
    *unsupported = 1;
    return cudaSuccess;
  }
  const size_t layer_bytes = (size_t)la.H * kTok * 4;
  DecArgs p;
  p.la = la;
  p.softmax = norm_softmax;
  p.flags = flags;
  p.lam = lambda;
  p.G = G;
  p.blocks_per_image = (la.max_vis + kTok - 1) / kTok;
  p.lps = (int)std::min<size_t>((size_t)la.L, kDecStageBytes / layer_bytes);
  p.a = a;
  p.stats = stats;
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
  p.cell_best = reinterpret_cast<unsigned long long*>(scratch);
  p.counters = scratch + (size_t)2 * kDecideCells * la.B;
  p.status = status;
  const size_t smem =
      (size_t)la.L * la.H * 16 + std::max((size_t)p.lps * layer_bytes, (size_t)la.max_vis * 5);
  return launch_kernel(decide_kernel, dim3((unsigned)(la.B * p.blocks_per_image)),
                       dim3(kDecThreads), smem, st, 0, true, p);
}

}  // namespace e2s
