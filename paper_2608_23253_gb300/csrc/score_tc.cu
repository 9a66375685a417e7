// Text-to-visual score on the 5th-generation tensor cores (tcgen05 + TMEM),
// with TMA-staged bf16 K tiles (Sec. 3.1 Eq. 1 and its causal-prefix
// probability reading).
//
// Work unit: (image b, layer l, kv head g, group of query heads).  A unit's
// keys are cut into 128-key tiles; a cluster of `cluster` CTAs splits the
// tiles, each CTA keeping its tiles resident in shared memory.
//
//   MMA  D[key][col] = K_tile[key][:] . Q[col][:]       (M = 128 keys,
//        N = padded text rows of one query head, K = d = 128 in 8 steps)
//        A = K tile, B = text queries, both K-major with the 128-byte swizzle,
//        fp32 accumulator in TMEM (two buffers).
//   CAUSAL_PROB phase 1: every epilogue thread owns one key (TMEM lane); per
//        16-column chunk a butterfly reduce-scatter over the warp's 32 lanes
//        turns 32 keys x 16 text rows into per-row online-softmax partials
//        (max, sum) in the log2 domain; partials are merged per warp, per CTA,
//        and then across the cluster through distributed shared memory,
//        giving each text row's log-sum-exp over its whole causal prefix.
//   phase 2: the visual tiles are multiplied again from the resident shared
//        memory copy; each thread sums exp2(s - lse) over the text rows of
//        its key and writes a = sum / N_T (EQ1 mode: the mean logit).
//
// Warp roles (192 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-5 epilogue (TMEM lane quarter = warp % 4).
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
constexpr int kEpiWarps = 4;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kQBoxRows = 16;
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
  uint32_t* status;
};

struct SmemPlan {
  uint32_t q, k, bars, slot, wstats, part, colv, total;
};

__host__ __device__ inline SmemPlan smem_plan(int hpc, int ntp_max, int tpc) {
  SmemPlan s;
  const uint32_t ncs = (uint32_t)(hpc * ntp_max);
  s.q = 0;
  s.k = 2u * ncs * 128u;
  s.bars = s.k + (uint32_t)tpc * kTileBytes;
  s.slot = s.bars + 8u * (uint32_t)(5 + tpc);
  s.wstats = (s.slot + 16u + 15u) & ~15u;
  s.part = s.wstats + (uint32_t)kEpiWarps * ncs * 8u;
  s.colv = s.part + ncs * 8u;
  s.total = s.colv + ncs * 4u;
  return s;
}

// One butterfly step of the reduce-scatter: keep W of the 2W live entries
// (upper half if `hi`), send the other W to the partner lane (xor MASK) and
// merge what comes back.
template <int W, int MASK>
__device__ __forceinline__ void rs_step(float (&m)[16], float (&s)[16], bool hi) {
#pragma unroll
  for (int i = 0; i < W; ++i) {
    const float send_m = hi ? m[i] : m[i + W];
    const float send_s = hi ? s[i] : s[i + W];
    float keep_m = hi ? m[i + W] : m[i];
    float keep_s = hi ? s[i + W] : s[i];
    const float rm = __shfl_xor_sync(0xffffffffu, send_m, MASK);
    const float rs = __shfl_xor_sync(0xffffffffu, send_s, MASK);
    lse_merge(keep_m, keep_s, rm, rs);
    m[i] = keep_m;
    s[i] = keep_s;
  }
}

// 32 lanes x 16 columns of (max, sum) partials -> lane L holds column L >> 1
// reduced over all 32 lanes (lanes L and L ^ 1 hold the same result).
__device__ __forceinline__ void reduce_scatter16(float (&m)[16], float (&s)[16], int lane) {
  rs_step<8, 16>(m, s, lane & 16);
  rs_step<4, 8>(m, s, lane & 8);
  rs_step<2, 4>(m, s, lane & 4);
  rs_step<1, 2>(m, s, lane & 2);
  const float rm = __shfl_xor_sync(0xffffffffu, m[0], 1);
  const float rs = __shfl_xor_sync(0xffffffffu, s[0], 1);
  lse_merge(m[0], s[0], rm, rs);
}

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
  uint64_t* tmem_empty = mma_done + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + plan.slot);
  float2* warp_stats = reinterpret_cast<float2*>(smem + plan.wstats);
  float2* cta_part = reinterpret_cast<float2*>(smem + plan.part);
  float* colv = reinterpret_cast<float*>(smem + plan.colv);

  const LayoutArgs& la = p.la;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const int ncs = p.hpc * p.ntp_max;
  const uint32_t q_half = (uint32_t)ncs * 128u;

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
  const int n1 = causal ? nt : 0;
  const int njobs = n1 + (vl - vf);

  // ---- setup: barriers, TMEM
  if (warp == 0 && lane == 0) {
    ptx::mbar_init(q_full, 1);
    for (int i = 0; i < p.tpc; ++i) ptx::mbar_init(k_full + i, 1);
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(mma_done + i, 1);
      ptx::mbar_init(tmem_empty + i, kEpiWarps);
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
    if (lane == 0 && njobs > 0) {
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
    // ================= MMA issuer (one thread)
    const uint32_t idesc = ptx::idesc_bf16_f32(128, ntp);
    auto issue = [&](int j, int tile) {
      const int buf = j & 1, use = j >> 1;
      if (!ptx::mbar_wait(k_full + tile, 0, limit, p.status)) limit = kWaitNsAfterFault;
      if (use > 0 && !ptx::mbar_wait(tmem_empty + buf, (use - 1) & 1, limit, p.status))
        limit = kWaitNsAfterFault;
      ptx::tc_fence_after();
      const uint32_t a_base = ptx::smem_addr(k_sm + tile * kTileBytes);
      const uint32_t b_base = ptx::smem_addr(q_sm);
      for (int hh = 0; hh < nh; ++hh) {
        const uint32_t d = tmem + (uint32_t)(buf * ncs + hh * p.ntp_max);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t half = ks >> 2, kk = ks & 3;
          const uint64_t ad = ptx::sdesc_sw128(a_base + half * kHalfBytes + kk * 32u);
          const uint64_t bd = ptx::sdesc_sw128(b_base + half * q_half +
                                               (uint32_t)(hh * p.ntp_max) * 128u + kk * 32u);
          ptx::mma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
        }
      }
      ptx::mma_commit(mma_done + buf);
    };
    if (lane == 0 && njobs > 0) {
      if (!ptx::mbar_wait(q_full, 0, limit, p.status)) limit = kWaitNsAfterFault;
      for (int j = 0; j < n1; ++j) issue(j, j);
    }
    __syncwarp();
    ptx::cluster_arrive();
    if (lane == 0)
      for (int j = n1; j < njobs; ++j) issue(j, vf + (j - n1));
    __syncwarp();
    ptx::cluster_wait();
  } else {
    // ================= epilogue (4 warps, one TMEM lane quarter each)
    const int ew = warp - 2;
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int et = threadIdx.x - 64;
    float2* my_stats = warp_stats + ew * ncs;

    if (causal) {
      for (int c = lane; c < ncs; c += 32) my_stats[c] = make_float2(kNegBig, 0.f);
      __syncwarp();
      for (int j = 0; j < n1; ++j) {
        const int buf = j & 1;
        if (!ptx::mbar_wait(mma_done + buf, (j >> 1) & 1, limit, p.status))
          limit = kWaitNsAfterFault;
        ptx::tc_fence_after();
        const int key = key_base + kTileKeys * (ft + j) + row;
        const int last_text = key - (S + NV);  // row t sees this key iff t >= last_text
        for (int hh = 0; hh < nh; ++hh) {
          for (int c16 = 0; c16 < ntp; c16 += 16) {
            float v[16], m[16], s[16];
            ptx::tmem_ld16(tmem + lane_base + (uint32_t)(buf * ncs + hh * p.ntp_max + c16), v);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int t = c16 + i;
              const bool valid = t < NT && t >= last_text;
              m[i] = valid ? v[i] * p.scale_log2 : kNegBig;
              s[i] = valid ? 1.f : 0.f;
            }
            reduce_scatter16(m, s, lane);
            if ((lane & 1) == 0) {
              float2 st = my_stats[hh * p.ntp_max + c16 + (lane >> 1)];
              lse_merge(st.x, st.y, m[0], s[0]);
              my_stats[hh * p.ntp_max + c16 + (lane >> 1)] = st;
            }
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(tmem_empty + buf);
      }
      ptx::named_bar(1, 32 * kEpiWarps);
      for (int c = et; c < ncs; c += 32 * kEpiWarps) {
        float2 acc = warp_stats[c];
        for (int w = 1; w < kEpiWarps; ++w) {
          const float2 o = warp_stats[w * ncs + c];
          lse_merge(acc.x, acc.y, o.x, o.y);
        }
        cta_part[c] = acc;
      }
    }
    ptx::cluster_arrive();
    ptx::cluster_wait();
    // per-column constants of phase 2
    for (int c = et; c < ncs; c += 32 * kEpiWarps) {
      const int t = c % p.ntp_max;
      if (causal) {
        float M = kNegBig, Ls = 0.f;
        for (int r = 0; r < p.cluster; ++r) {
          const float2 o = ptx::ld_dsmem_f2(cta_part + c, (uint32_t)r);
          lse_merge(M, Ls, o.x, o.y);
        }
        colv[c] = (t < NT && Ls > 0.f) ? M + log2f(Ls) : __int_as_float(0x7f800000);
      } else {
        colv[c] = (t < NT) ? 1.f : 0.f;
      }
    }
    ptx::named_bar(1, 32 * kEpiWarps);
    const float out_scale = causal ? 1.f / (float)NT : p.scale / (float)NT;
    for (int j = n1; j < njobs; ++j) {
      const int buf = j & 1;
      if (!ptx::mbar_wait(mma_done + buf, (j >> 1) & 1, limit, p.status))
        limit = kWaitNsAfterFault;
      ptx::tc_fence_after();
      const int tile = vf + (j - n1);
      const int key = key_base + kTileKeys * (ft + tile) + row;
      const bool vis = key >= S && key < S + NV;
      for (int hh = 0; hh < nh; ++hh) {
        float acc = 0.f;
        for (int c16 = 0; c16 < ntp; c16 += 16) {
          float v[16];
          ptx::tmem_ld16(tmem + lane_base + (uint32_t)(buf * ncs + hh * p.ntp_max + c16), v);
          const float* cv = colv + hh * p.ntp_max + c16;
          if (causal) {
#pragma unroll
            for (int i = 0; i < 16; ++i) acc += exp2f(fmaf(v[i], p.scale_log2, -cv[i]));
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) acc = fmaf(v[i], cv[i], acc);
          }
        }
        if (vis)
          p.a_out[((size_t)l * la.H + h0 + hh) * (size_t)la.sum_vis + v0 + (key - S)] =
              acc * out_scale;
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(tmem_empty + buf);
    }
  }

  // ---- teardown: peers may still read cta_part until everyone is here
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

// 3-D map over rows of (heads x 128) bf16: dims (128, heads, rows), box (64, 1, box_rows).
bool make_map(CUtensorMap* map, const void* base, int heads, int64_t rows, int64_t row_stride_el,
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

}  // namespace

cudaError_t launch_score_tc(const LayoutArgs& la, int mode, const void* q, int64_t q_stride,
                            const void* k, int64_t k_stride, float* a_out, uint32_t* status,
                            cudaStream_t st, int* unsupported) {
  *unsupported = 0;
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
  uint32_t cols = 32;
  while ((int)cols < 2 * ncs) cols <<= 1;
  p.tmem_cols = cols;
  const int span = (mode == E2S_SCORE_CAUSAL_PROB) ? la.max_T : la.max_vis;
  const int max_tiles = (span + kTileKeys - 1) / kTileKeys;
  if (max_tiles == 0 || la.sum_vis == 0) return cudaSuccess;
  p.tpc = std::min(2, max_tiles);
  p.cluster = (max_tiles + p.tpc - 1) / p.tpc;
  while (p.cluster > 8) {
    ++p.tpc;
    p.cluster = (max_tiles + p.tpc - 1) / p.tpc;
  }
  p.scale = 1.0f / sqrtf(128.0f);
  p.scale_log2 = 1.4426950408889634f / sqrtf(128.0f);
  p.a_out = a_out;
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
  if (!make_map(&tmQ, q, la.H, (int64_t)la.L * la.sum_text, q_stride, kQBoxRows) ||
      !make_map(&tmK, k, la.H_kv, (int64_t)la.L * la.sum_T, k_stride, kTileKeys))
    return cudaErrorInvalidValue;
  e = cudaFuncSetAttribute(score_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const long long units = (long long)la.B * la.L * la.H_kv * p.groups_per_kv;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(units * p.cluster));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, score_tc_kernel, tmQ, tmK, p);
}

}  // namespace e2s
