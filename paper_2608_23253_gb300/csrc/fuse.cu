// Per-layer evidence and layer-wise Dempster-Shafer fusion (Sec. 4.1-4.2).
//
//   fuse_stats_kernel  one CTA per (image, layer, head): the normalisation
//                      statistics of Eq. 8 over the image's candidate tokens
//                      (softmax: max and sum of exp; renorm: sum).
//   fuse_token_kernel  one thread per candidate token: support p (Eq. 9) per
//                      head, reliability rho (Eq. 10), layer mass (Eq. 11),
//                      recursive Dempster combination with the conflict term
//                      (Eqs. 12-16), plausibility (Eq. 18) and priority q
//                      (Eq. 19).  Reads of a[l][h][.] are coalesced across
//                      the token index.
#include <cuda_runtime.h>

#include <mutex>

#include "device_common.cuh"

namespace e2s {
namespace {

constexpr int kStatsThreads = 256;
constexpr int kTokenThreads = 128;

// Whether image b's device layout arrays agree with each other and with the
// host totals.  Both kernels take the same decision for the same image.
__device__ __forceinline__ bool image_layout_ok(const LayoutArgs& la, int b, int NV, int v0) {
  return NV >= 0 && v0 >= 0 && v0 + NV <= la.sum_vis && __ldg(la.vis_off + b + 1) - v0 == NV;
}

__global__ void __launch_bounds__(kStatsThreads)
    fuse_stats_kernel(const LayoutArgs la, int softmax, const float* __restrict__ a,
                      float2* __restrict__ stats, uint32_t* status) {
  __shared__ float red[32];
  pdl_launch_dependents();
  pdl_wait();
  const int unit = blockIdx.x;
  const int h = unit % la.H;
  const int l = (unit / la.H) % la.L;
  const int b = unit / (la.H * la.L);
  const int NV = __ldg(la.n_vis + b), v0 = __ldg(la.vis_off + b);
  if (!image_layout_ok(la, b, NV, v0)) {
    if (threadIdx.x == 0) {
      E2S_DEV_FLAG(status, E2S_ERR_SHAPE);
      stats[unit] = make_float2(0.f, 0.f);
    }
    return;
  }
  const float* row = a + ((size_t)l * la.H + h) * (size_t)la.sum_vis + v0;
  float2 out;
  if (softmax) {
    float mx = -__int_as_float(0x7f800000);
    for (int n = threadIdx.x; n < NV; n += blockDim.x) mx = fmaxf(mx, row[n]);
    mx = block_reduce(mx, [](float x, float y) { return fmaxf(x, y); }, red);
    float se = 0.f;
    for (int n = threadIdx.x; n < NV; n += blockDim.x) se += __expf(row[n] - mx);
    se = block_reduce(se, [](float x, float y) { return x + y; }, red);
    out = make_float2(mx, se);
  } else {
    float sa = 0.f;
    for (int n = threadIdx.x; n < NV; n += blockDim.x) sa += row[n];
    sa = block_reduce(sa, [](float x, float y) { return x + y; }, red);
    out = make_float2(0.f, sa);
  }
  if (threadIdx.x == 0) stats[unit] = out;
}

__device__ __forceinline__ float support_of(float a, float2 st, int softmax, float N) {
  float r;
  if (softmax)
    r = __expf(a - st.x) / st.y;         // Eq. 8
  else
    r = st.y > 0.f ? a / st.y : 1.f / N; // r = a / sum a
  const float x = N * r;
  return x / (1.f + x);                  // Eq. 9
}

__global__ void __launch_bounds__(kTokenThreads)
    fuse_token_kernel(const LayoutArgs la, int softmax, uint32_t flags,
                      const float* __restrict__ a, const float2* __restrict__ stats,
                      const float4* __restrict__ prior, float4* __restrict__ mass_out,
                      float4* __restrict__ fused_out, float* __restrict__ q_out) {
  pdl_launch_dependents();
  pdl_wait();
  const int gv = blockIdx.x * blockDim.x + threadIdx.x;
  if (gv >= la.sum_vis) return;
  const int b = find_segment(la.vis_off, la.B, gv);
  const int NV = __ldg(la.n_vis + b);
  const float N = (float)NV;
  const int H = la.H;
  const float inv_h = 1.f / (float)H;
  const size_t plane = (size_t)la.sum_vis;
  if (!image_layout_ok(la, b, NV, __ldg(la.vis_off + b))) {
    // The statistics kernel skipped this image (its entries are zero), so
    // the evidence is undefined: write the vacuous mass, no conflict, q = 0.
    if (mass_out)
      for (int l = 0; l < la.L; ++l) mass_out[(size_t)l * plane + gv] = make_float4(0.f, 0.f, 1.f, 0.f);
    fused_out[gv] = make_float4(0.f, 0.f, 1.f, 0.f);
    q_out[gv] = 0.f;
    return;
  }

  float fI = 0.f, fU = 0.f, fT = 1.f, K = 0.f;
  bool have = false;
  const bool use_prior = prior != nullptr && !(flags & E2S_NO_LAYER_FUSION);
  if (use_prior) {
    const float4 pr = prior[gv];
    fI = pr.x; fU = pr.y; fT = pr.z;
    have = true;
  }
  const int l_begin = (flags & E2S_NO_LAYER_FUSION) ? la.L - 1 : 0;
  for (int l = 0; l < la.L; ++l) {
    const float* al = a + (size_t)l * H * plane + gv;
    const float2* sl = stats + ((size_t)b * la.L + l) * H;
    float sum_p = 0.f;
    for (int h = 0; h < H; ++h) sum_p += support_of(al[h * plane], sl[h], softmax, N);
    const float p_bar = sum_p * inv_h;
    float clar = 0.f, dev = 0.f;
    for (int h = 0; h < H; ++h) {
      const float p = support_of(al[h * plane], sl[h], softmax, N);
      clar += p - 0.5f;
      dev += fabsf(p - p_bar);
    }
    // Eq. 10: clarity x consistency
    float rho = (2.f * inv_h) * fabsf(clar) * (1.f - (2.f * inv_h) * dev);
    if (flags & E2S_NO_RELIABILITY) rho = 1.f;
    // Eq. 11
    const float mI = rho * p_bar, mU = rho * (1.f - p_bar), mT = 1.f - rho;
    if (mass_out) mass_out[(size_t)l * plane + gv] = make_float4(mI, mU, mT, p_bar);
    if (l < l_begin) continue;
    if (!have) {  // Eq. 12
      fI = mI; fU = mU; fT = mT; K = 0.f;
      have = true;
    } else {      // Eqs. 13-16
      K = fI * mU + fU * mI;
      const float omk = 1.f - K;
      if (omk <= 0.f) {
        fI = 0.f; fU = 0.f; fT = 1.f; K = 1.f;
      } else {
        const float inv = 1.f / omk;
        const float nI = (fI * mI + fI * mT + fT * mI) * inv;
        const float nU = (fU * mU + fU * mT + fT * mU) * inv;
        const float nT = fT * mT * inv;
        fI = nI; fU = nU; fT = nT;
      }
    }
  }
  const float Pl = fI + fT;                                         // Eq. 18
  float q = (flags & E2S_NO_CONFLICT) ? Pl : 1.f - (1.f - Pl) * (1.f - K);  // Eq. 19
  if (flags & E2S_VANILLA) {
    float s = 0.f;
    for (int l = 0; l < la.L; ++l)
      for (int h = 0; h < H; ++h) s += a[((size_t)l * H + h) * plane + gv];
    q = s / (float)(la.L * H);
  }
  fused_out[gv] = make_float4(fI, fU, fT, K);
  q_out[gv] = q;
}

}  // namespace

cudaError_t launch_fuse(const LayoutArgs& la, int norm_softmax, uint32_t flags, const float* a,
                        const float* prior, float* mass_out, float* fused_out, float* q_out,
                        float2* stats, uint32_t* status, cudaStream_t st) {
  if (la.sum_vis == 0) return cudaSuccess;
  const unsigned units = (unsigned)((size_t)la.B * la.L * la.H);
  cudaError_t e = launch_kernel(fuse_stats_kernel, dim3(units), dim3(kStatsThreads), 0, st, 0, true,
                                la, norm_softmax, a, stats, status);
  if (e != cudaSuccess) return e;
  const unsigned blocks = (unsigned)((la.sum_vis + kTokenThreads - 1) / kTokenThreads);
  return launch_kernel(fuse_token_kernel, dim3(blocks), dim3(kTokenThreads), 0, st, 0, true, la,
                       norm_softmax, flags, a, static_cast<const float2*>(stats),
                       reinterpret_cast<const float4*>(prior), reinterpret_cast<float4*>(mass_out),
                       reinterpret_cast<float4*>(fused_out), q_out);
}

}  // namespace e2s

// ---------------------------------------------------------------------------
// Allocation-free variant (e2s_fuse_noalloc).  Some callers cannot hand us a
// workspace: code running inside a host framework whose memory pool owns the
// device heap, plug-ins called through a foreign-function interface with no
// allocator of their own, or real-time loops where any cudaMalloc is
// forbidden.  For them the statistics scratch of e2s_fuse lives in this
// file-scope device array instead.  Every GPU that loads the library holds it
// until the process exits.
namespace e2s {
namespace {

constexpr long long kNoAllocMaxUnits = 8192;   // images x layers x heads
constexpr size_t kNoAllocBytes = kStatusBytes + (size_t)kNoAllocMaxUnits * sizeof(float2);
static __device__ __align__(256) unsigned char g_fuse_scratch[kNoAllocBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_fuse_scratch on the current device.  The host-side name
// is only a stand-in, so the address is asked from the runtime once per
// device (with that device current) and cached.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_fuse_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_fuse_noalloc(const LayoutArgs& la, int norm_softmax, uint32_t flags,
                                const float* a, const float* prior, float* mass_out,
                                float* fused_out, float* q_out, cudaStream_t st, int* too_big) {
  *too_big = 0;
  if ((long long)la.B * la.L * la.H > kNoAllocMaxUnits) {
    *too_big = 1;
    return cudaSuccess;
  }
  void* base = nullptr;
  const cudaError_t e = scratch_address(&base);
  if (e != cudaSuccess) return e;
  // The statistics are fully rewritten before they are read, so nothing left
  // by an earlier call needs clearing; the status word is not read back.
  uint32_t* status = static_cast<uint32_t*>(base);
  float2* stats = reinterpret_cast<float2*>(static_cast<char*>(base) + kStatusBytes);
  return launch_fuse(la, norm_softmax, flags, a, prior, mass_out, fused_out, q_out, stats, status,
                     st);
}

}  // namespace e2s
