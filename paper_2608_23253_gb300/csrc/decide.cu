// Evidence, layer-wise fusion and selection of e2s_decide (Sec. 4.1-4.3,
// Eqs. 8-23), token-parallel.  The normalisation statistics of Eq. 8 for
// every (image, layer, head) were produced by the score kernel, so tokens are
// independent here.  A CTA of 256 threads takes 64 visual tokens of one image
// (16 when the batch is too small to fill the GPU with 64-token CTAs):
//   1. the image's statistics and the CTA's a[l][h][token] values are copied
//      into shared memory with asynchronous copies, all in flight at once;
//   2. one thread per (token, layer) walks the H heads (with 16-token CTAs,
//      four lanes per (token, layer), each taking every fourth head, joined by
//      two shuffles): supports p (Eq. 9), written back over the staged
//      scores, p_bar, then the reliability terms of Eq. 10, rho and the layer
//      mass (Eq. 11);
//   3. one thread per token: Dempster combination of its layer masses in
//      order (Eqs. 12-16), Pl and q (Eqs. 18-19), and its bid for its cell's
//      representative (Eqs. 20-21);
//   4. every CTA folds its bids into the image's cell arg-max keys in global
//      memory and bumps the image's arrival counter; the last CTA of the image
//      computes q~ and the Top-K (Eqs. 22-23) over the whole image and re-arms
//      the keys and the counter.
// The select arguments are inputs of the call, not results of the score
// kernel, so they are checked before griddepcontrol.wait.
#include <cuda_runtime.h>

#include <algorithm>

#include "select_core.cuh"
#include "sm100_ptx.cuh"

namespace e2s {
namespace {

constexpr int kDecThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr size_t kDecSmemBudget = 160u << 10;

// Visual tokens per CTA.  64 when the batch fills the GPU; 16 for small
// batches, where the CTA's 256 threads split each (token, layer)'s heads four
// ways so the per-thread walk over the heads is four times shorter.
template <int TOK>
struct DecTile {
  static constexpr int kTok = TOK;
  // staged row stride (floats): with heads split four ways (head h = 4i + g on
  // lane group g), 24 keeps the four groups of a warp in distinct banks
  static constexpr int kRow = TOK == 64 ? 64 : 24;
  static constexpr int kHeadSplit = TOK == 64 ? 1 : 4;
  static constexpr int kLayerLanes = kDecThreads / (TOK * kHeadSplit);   // layers side by side
};

// [L][H] statistics, [L][kTok] layer masses and head sums, then the staged
// scores [L][H][kRow] (reused as the select's keys and cell ids).
template <int TOK>
__host__ __device__ inline size_t dec_smem_bytes(int L, int H, int max_vis) {
  const size_t st = (size_t)L * H * 16 + (size_t)L * TOK * 20;
  const size_t a = (size_t)L * H * DecTile<TOK>::kRow * 4;
  const size_t sel = (size_t)max_vis * 5;
  return st + (a > sel ? a : sel);
}

struct DecArgs {
  LayoutArgs la;
  int softmax;
  uint32_t flags;
  float lam;
  int G;
  int blocks_per_image;
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

template <int TOK>
__global__ void __launch_bounds__(kDecThreads) decide_kernel(const DecArgs p) {
  constexpr int kTok = DecTile<TOK>::kTok, kRow = DecTile<TOK>::kRow;
  constexpr int kSplit = DecTile<TOK>::kHeadSplit, kLayerLanes = DecTile<TOK>::kLayerLanes;
  extern __shared__ __align__(16) uint8_t dec_smem[];
  __shared__ SelectSmem ss;
  __shared__ int is_last;
  __shared__ unsigned long long cb_s[kDecideCells];   // this CTA's cell arg-max keys
  const LayoutArgs& la = p.la;
  const int H = la.H, L = la.L;
  float4* st_s = reinterpret_cast<float4*>(dec_smem);           // [L][H]
  float4* M_s = st_s + (size_t)L * H;                            // [L][kTok]
  float* SA_s = reinterpret_cast<float*>(M_s + (size_t)L * kTok);  // [L][kTok]
  float* A = SA_s + (size_t)L * kTok;                            // [L][H][kRow]
  const int tid = threadIdx.x;
  for (int i = tid; i < kDecideCells; i += kDecThreads) cb_s[i] = 0ull;

  const int b = blockIdx.x / p.blocks_per_image;
  const int blk = blockIdx.x - b * p.blocks_per_image;
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  const bool ok = NV >= 0 && NV <= la.max_vis && v0 >= 0 && v0 + NV <= la.sum_vis &&
                  __ldg(la.vis_off + b + 1) - v0 == NV;
  const int n0 = blk * kTok;
  const int ntok = ok ? max(0, min(kTok, NV - n0)) : 0;
  const size_t plane = (size_t)la.sum_vis;
  const bool select = p.keep_count != nullptr;
  const int G = p.G;
  const int gh = __ldg(la.grid_h + b), gw = __ldg(la.grid_w + b);
  const bool sel_ok =
      select && ok &&
      select_args_ok(la, b, p.cand != nullptr, p.keep_count, p.keep_off, p.sum_keep);
  const CellMap cells(gh, gw, G);
  pdl_launch_dependents();
  pdl_wait();   // a and the statistics come from the score kernel

  // 1. stage the statistics and a[l][h][n0 .. n0+ntok) (coalesced along the tokens)
  for (int i = tid; i < L * H * 4; i += kDecThreads)
    ptx::cp_async4(reinterpret_cast<float*>(st_s) + i,
                   reinterpret_cast<const float*>(p.stats + (size_t)b * L * H) + i);
  if (((v0 + n0) & 3) == 0 && (plane & 3) == 0 &&
      (reinterpret_cast<uintptr_t>(p.a) & 15) == 0) {   // 16-byte copies (4 tokens each)
    for (int idx = tid; idx < L * H * (kTok / 4); idx += kDecThreads) {
      const int jj = (idx & (kTok / 4 - 1)) * 4, lh = idx / (kTok / 4);
      const float* src = p.a + (size_t)lh * plane + v0 + n0 + jj;
      if (jj + 3 < ntok)
        ptx::cp_async16(A + lh * kRow + jj, src);
      else
        for (int t = jj; t < ntok; ++t) ptx::cp_async4(A + lh * kRow + t, src + (t - jj));
    }
  } else {
    for (int idx = tid; idx < L * H * kTok; idx += kDecThreads) {
      const int jj = idx & (kTok - 1), lh = idx / kTok;
      if (jj < ntok) ptx::cp_async4(A + lh * kRow + jj, p.a + (size_t)lh * plane + v0 + n0 + jj);
    }
  }
  ptx::cp_async_wait_all();
  __syncthreads();

  // 2. per (token, layer): supports, reliability and layer mass (Eqs. 8-11)
  const float N = (float)NV;
  const float invN = NV > 0 ? 1.f / N : 0.f;
  const float inv_h = 1.f / (float)H;
  if constexpr (kSplit == 1) {
    const int j = tid & (kTok - 1);
    for (int l = tid / kTok; l < L; l += kLayerLanes) {
      if (j >= ntok) continue;
      float* Ac = A + (size_t)l * H * kRow + j;
      const float4* sl = st_s + (size_t)l * H;
      float sum_p = 0.f, sum_a = 0.f;
#pragma unroll 8
      for (int h = 0; h < H; ++h) {
        const float av = Ac[h * kRow];
        const float pv = support_p(av, sl[h], p.softmax, N, invN);
        sum_a += av;
        sum_p += pv;
        Ac[h * kRow] = pv;
      }
      const float p_bar = sum_p * inv_h;
      float clar = 0.f, dev = 0.f;
#pragma unroll 8
      for (int h = 0; h < H; ++h) {
        const float pv = Ac[h * kRow];
        clar += pv - 0.5f;
        dev += fabsf(pv - p_bar);
      }
      float rho = (2.f * inv_h) * fabsf(clar) * (1.f - (2.f * inv_h) * dev);  // Eq. 10
      if (p.flags & E2S_NO_RELIABILITY) rho = 1.f;
      const float4 m4 = make_float4(rho * p_bar, rho * (1.f - p_bar), 1.f - rho, p_bar);  // Eq. 11
      M_s[l * kTok + j] = m4;
      SA_s[l * kTok + j] = sum_a;
      if (p.mass_out) p.mass_out[(size_t)l * plane + v0 + n0 + j] = m4;
    }
  } else {
    // lane = (token & 7) + 8 g: the four lanes of a (token, layer) take heads
    // h = g, g + 4, ... and combine their partial sums with two shuffles;
    // warp w takes tokens 8 (w & 1) .. + 7 of layer lane w >> 1
    const int lane = tid & 31, wp = tid >> 5, g = lane >> 3;
    const int j = (lane & 7) + 8 * (wp & 1);
    for (int l = wp >> 1; l < L; l += kLayerLanes) {
      float* Ac = A + (size_t)l * H * kRow + j;
      const float4* sl = st_s + (size_t)l * H;
      float sum_p = 0.f, sum_a = 0.f;
#pragma unroll 4
      for (int h = g; h < H; h += kSplit) {
        const float av = Ac[h * kRow];
        const float pv = support_p(av, sl[h], p.softmax, N, invN);
        sum_a += av;
        sum_p += pv;
        Ac[h * kRow] = pv;
      }
      sum_p += __shfl_xor_sync(0xffffffffu, sum_p, 8);
      sum_p += __shfl_xor_sync(0xffffffffu, sum_p, 16);
      sum_a += __shfl_xor_sync(0xffffffffu, sum_a, 8);
      sum_a += __shfl_xor_sync(0xffffffffu, sum_a, 16);
      const float p_bar = sum_p * inv_h;
      float clar = 0.f, dev = 0.f;
#pragma unroll 4
      for (int h = g; h < H; h += kSplit) {
        const float pv = Ac[h * kRow];
        clar += pv - 0.5f;
        dev += fabsf(pv - p_bar);
      }
      clar += __shfl_xor_sync(0xffffffffu, clar, 8);
      clar += __shfl_xor_sync(0xffffffffu, clar, 16);
      dev += __shfl_xor_sync(0xffffffffu, dev, 8);
      dev += __shfl_xor_sync(0xffffffffu, dev, 16);
      float rho = (2.f * inv_h) * fabsf(clar) * (1.f - (2.f * inv_h) * dev);  // Eq. 10
      if (p.flags & E2S_NO_RELIABILITY) rho = 1.f;
      const float4 m4 = make_float4(rho * p_bar, rho * (1.f - p_bar), 1.f - rho, p_bar);  // Eq. 11
      if (g == 0 && j < ntok) {
        M_s[l * kTok + j] = m4;
        SA_s[l * kTok + j] = sum_a;
        if (p.mass_out) p.mass_out[(size_t)l * plane + v0 + n0 + j] = m4;
      }
    }
  }
  __syncthreads();

  // 3. per token: Dempster combination over the layers (Eqs. 12-16), q (Eq. 19)
  if (tid < ntok) {
    const int j = tid, gv = v0 + n0 + j;
    float fI = 0.f, fU = 0.f, fT = 1.f, K = 0.f, vsum = 0.f;
    bool have = false;
    if (p.prior != nullptr && !(p.flags & E2S_NO_LAYER_FUSION)) {
      const float4 pr = p.prior[gv];
      fI = pr.x; fU = pr.y; fT = pr.z;
      have = true;
    }
    const int l_begin = (p.flags & E2S_NO_LAYER_FUSION) ? L - 1 : 0;
    for (int l = 0; l < L; ++l) {
      vsum += SA_s[l * kTok + j];
      if (l < l_begin) continue;
      const float4 m = M_s[l * kTok + j];
      if (!have) {                                   // Eq. 12
        fI = m.x; fU = m.y; fT = m.z; K = 0.f;
        have = true;
      } else {                                       // Eqs. 13-16
        const float Kc = fI * m.y + fU * m.x;
        const float omk = 1.f - Kc;
        if (omk <= 0.f) {
          fI = 0.f; fU = 0.f; fT = 1.f; K = 1.f;
        } else {
          const float inv = 1.f / omk;
          const float nI = (fI * m.x + fI * m.z + fT * m.x) * inv;
          const float nU = (fU * m.y + fU * m.z + fT * m.y) * inv;
          const float nT = fT * m.z * inv;
          fI = nI; fU = nU; fT = nT; K = Kc;
        }
      }
    }
    const float Pl = fI + fT;                                                   // Eq. 18
    float q = (p.flags & E2S_NO_CONFLICT) ? Pl : 1.f - (1.f - Pl) * (1.f - K);  // Eq. 19
    if (p.flags & E2S_VANILLA) q = vsum / (float)(L * H);
    p.fused_out[gv] = make_float4(fI, fU, fT, K);
    p.q_out[gv] = q;
    // bid for the cell's representative (Eqs. 20-21)
    if (sel_ok) {
      const int n = n0 + j;
      atomicMax(&cb_s[token_cell(p.cand ? p.cand + v0 : nullptr, n, cells, p.status)],
                cell_key(q, n));
    }
  }
  if (!select) return;
  __syncthreads();
  for (int i = tid; i < G * G; i += kDecThreads)
    if (cb_s[i] != 0ull) atomicMax(p.cell_best + (size_t)b * kDecideCells + i, cb_s[i]);

  // 4. the last CTA of the image selects.  The barrier orders every thread's
  // writes before thread 0's acquire-release arrival; in the last CTA the
  // arrival's acquire plus the barrier after it make every other CTA's
  // writes visible to all of its threads.
  __syncthreads();
  if (tid == 0) {
    const uint32_t ticket = ptx::atom_add_acq_rel_gpu(p.counters + b, 1u);
    is_last = ticket == (uint32_t)(p.blocks_per_image - 1);
    if (is_last) p.counters[b] = 0u;   // re-armed for the next call
  }
  __syncthreads();
  if (!is_last) return;
  unsigned long long* cells_g = p.cell_best + (size_t)b * kDecideCells;
  if (!sel_ok) {
    for (int i = tid; i < kDecideCells; i += kDecThreads) cells_g[i] = 0ull;
    if (tid == 0) E2S_DEV_FLAG(p.status, E2S_ERR_SHAPE);
    return;
  }
  const float lam = (p.flags & (E2S_NO_NOVELTY | E2S_VANILLA)) ? 0.f : p.lam;
  select_image_from_cells(p.q_out + v0, p.cand ? p.cand + v0 : nullptr, NV, cells, lam,
                          __ldg(p.keep_count + b), cells_g, reinterpret_cast<uint32_t*>(A),
                          reinterpret_cast<uint8_t*>(A) + 4 * (size_t)la.max_vis, ss,
                          p.q_tilde ? p.q_tilde + v0 : nullptr,
                          p.keep_idx + __ldg(p.keep_off + b), p.status);
}

}  // namespace

bool decide_fits(const LayoutArgs& la) {
  return dec_smem_bytes<64>(la.L, la.H, la.max_vis) <= kDecSmemBudget &&
         dec_smem_bytes<16>(la.L, la.H, la.max_vis) <= kDecSmemBudget;
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
  DecArgs p;
  p.la = la;
  p.softmax = norm_softmax;
  p.flags = flags;
  p.lam = lambda;
  p.G = G;
  // 16-token CTAs while the 64-token grid would leave most SMs idle
  const bool small = (int64_t)la.B * ((la.max_vis + 63) / 64) < (int64_t)sm_count();
  const int tok = small ? 16 : 64;
  p.blocks_per_image = (la.max_vis + tok - 1) / tok;
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
  const dim3 grid((unsigned)(la.B * p.blocks_per_image));
  if (small)
    return launch_kernel(decide_kernel<16>, grid, dim3(kDecThreads),
                         dec_smem_bytes<16>(la.L, la.H, la.max_vis), st, 0, true, p);
  return launch_kernel(decide_kernel<64>, grid, dim3(kDecThreads),
                       dec_smem_bytes<64>(la.L, la.H, la.max_vis), st, 0, true, p);
}

}  // namespace e2s
