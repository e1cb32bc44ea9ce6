// Synthetic denoiser: posterior-mean noise of an isotropic Gaussian mixture,
// the seedable stand-in for the SD v1.5 UNet eps_theta (Sec. 3.2). Not part
// of ParaAnya; it produces the fresh eps of the misses (Eq. 6, miss branch).
//
//   v = a s^2 + 1 - a,   logit_k = (2 sqrt(a) x.mu_k - a ||mu_k||^2) / (2 v)
//   r = softmax(logit)   (the common -||x||^2 / (2 v) term cancels)
//   eps = sqrt(1 - a) / v * (x - sqrt(a) sum_k r_k mu_k)
//
// Three kernels per call:
//   k_gmm_dots     split-K partial contraction G = X M^T   [rows x K]
//   k_gmm_softmax  fixed-order split sum, logits, softmax  (one warp per row)
//   k_gmm_out      eps = a x - a sqrt(a) R M                [rows x D]
// Per-timestep scalars (sqrt(a), 1/(2v), sqrt(1-a)/v) are computed on the
// host in fp64 from alpha-bar and stored in fp32, so 1 - a never cancels in
// fp32.
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/paraanya.h"
#include "pa_internal.h"

namespace pa {
void set_error(const std::string& msg);  // pa_solver.cpp
}

namespace {

constexpr int kMaxK = 128;
constexpr int kDotThreads = 256;
constexpr int kDotRows = 16;     // rows per dots CTA
constexpr int kDotTile = 64;     // columns staged per step
constexpr int kOutCols = 128;    // columns per output CTA
constexpr int kOutRows = 32;     // rows per output CTA

struct GmmLayout {
  size_t coef, mnorm, gpart, R, rowc, total;
  int nsplit;
  int64_t split_len;
};

GmmLayout gmm_layout(int K, int64_t D, int max_rows, int T) {
  GmmLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  // split D so that the dots grid has a few waves even for small batches
  int64_t split_len = 2048;
  while (split_len > 256 && (D + split_len - 1) / split_len * ((max_rows + kDotRows - 1) / kDotRows) < 304)
    split_len /= 2;
  split_len = std::max<int64_t>(kDotTile, split_len);
  L.split_len = split_len;
  L.nsplit = (int)((D + split_len - 1) / split_len);
  L.coef = take((size_t)3 * T * sizeof(float));
  L.mnorm = take((size_t)K * sizeof(float));
  L.gpart = take((size_t)L.nsplit * max_rows * K * sizeof(float));
  L.R = take((size_t)max_rows * K * sizeof(float));
  L.rowc = take((size_t)max_rows * 2 * sizeof(float));
  L.total = o;
  return L;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ||mu_k||^2, one CTA per component, fixed-order tree.
__global__ void __launch_bounds__(256) k_gmm_norms(const float* __restrict__ mu, int64_t D,
                                                   float* __restrict__ mnorm) {
  __shared__ float s[8];
  const float* m = mu + (int64_t)blockIdx.x * D;
  float acc = 0.f;
  for (int64_t d = threadIdx.x; d < D; d += 256) acc = fmaf(m[d], m[d], acc);
  acc = warp_sum(acc);
  if ((threadIdx.x & 31) == 0) s[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += s[w];
    mnorm[blockIdx.x] = t;
  }
}

// gpart[split][r][k] = sum over this split's columns of x[r][d] mu[k][d]
__global__ void __launch_bounds__(kDotThreads) k_gmm_dots(const float* __restrict__ X,
                                                          const float* __restrict__ mu,
                                                          const int32_t* __restrict__ n_rows_dev,
                                                          int K, int64_t D, int64_t split_len,
                                                          int max_rows, float* __restrict__ gpart) {
  __shared__ float xs[kDotRows][kDotTile + 1];
  __shared__ float ms[kMaxK][kDotTile + 1];
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * kDotRows;
  if (r0 >= n_rows) return;
  const int split = blockIdx.x;
  const int64_t d0 = (int64_t)split * split_len;
  const int64_t d1 = (D < d0 + split_len) ? D : d0 + split_len;
  const int nout = kDotRows * K;  // <= 16 * 128 = 2048 -> 8 per thread
  float acc[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) acc[u] = 0.f;
  for (int64_t c0 = d0; c0 < d1; c0 += kDotTile) {
    const int w = (int)((d1 - c0) < kDotTile ? (d1 - c0) : kDotTile);
    for (int q = threadIdx.x; q < kDotRows * kDotTile; q += kDotThreads) {
      const int rr = q / kDotTile, cc = q % kDotTile;
      const int r = r0 + rr;
      xs[rr][cc] = (r < n_rows && cc < w) ? X[(int64_t)r * D + c0 + cc] : 0.f;
    }
    for (int q = threadIdx.x; q < K * kDotTile; q += kDotThreads) {
      const int k = q / kDotTile, cc = q % kDotTile;
      ms[k][cc] = (cc < w) ? mu[(int64_t)k * D + c0 + cc] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int o = threadIdx.x + u * kDotThreads;
      if (o < nout) {
        const int rr = o / K, k = o % K;
        float a = acc[u];
#pragma unroll 16
        for (int cc = 0; cc < kDotTile; ++cc) a = fmaf(xs[rr][cc], ms[k][cc], a);
        acc[u] = a;
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    const int o = threadIdx.x + u * kDotThreads;
    if (o < nout) {
      const int rr = o / K, k = o % K;
      const int r = r0 + rr;
      if (r < n_rows) gpart[((int64_t)split * max_rows + r) * K + k] = acc[u];
    }
  }
}

// One warp per row: dots (fixed-order split sum) -> logits -> softmax.
__global__ void __launch_bounds__(256) k_gmm_softmax(const float* __restrict__ gpart,
                                                     const float* __restrict__ mnorm,
                                                     const float* __restrict__ coef, int T,
                                                     const int32_t* __restrict__ miss_bt,
                                                     const int32_t* __restrict__ n_rows_dev,
                                                     int K, int nsplit, int max_rows,
                                                     float* __restrict__ R,
                                                     float* __restrict__ rowc) {
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= n_rows) return;
  const int i = miss_bt[2 * r + 1];
  const float sa = coef[i], q = coef[T + i], ac = coef[2 * T + i];
  float l[kMaxK / 32];
  float mx = -INFINITY;
#pragma unroll
  for (int u = 0; u < kMaxK / 32; ++u) {
    const int k = lane + 32 * u;
    l[u] = -INFINITY;
    if (k < K) {
      float dot = 0.f;
      for (int s = 0; s < nsplit; ++s) dot += gpart[((int64_t)s * max_rows + r) * K + k];
      l[u] = (2.f * sa * dot - sa * sa * mnorm[k]) * q;
      mx = fmaxf(mx, l[u]);
    }
  }
  mx = warp_max(mx);
  float sum = 0.f;
#pragma unroll
  for (int u = 0; u < kMaxK / 32; ++u) {
    const int k = lane + 32 * u;
    l[u] = (k < K) ? expf(l[u] - mx) : 0.f;
    sum += l[u];
  }
  sum = warp_sum(sum);
  const float inv = 1.f / sum;
#pragma unroll
  for (int u = 0; u < kMaxK / 32; ++u) {
    const int k = lane + 32 * u;
    if (k < K) R[(int64_t)r * K + k] = l[u] * inv;
  }
  if (lane == 0) {
    rowc[2 * r] = ac;
    rowc[2 * r + 1] = ac * sa;
  }
}

// eps[r][d] = ac x[r][d] - ac sqrt(a) sum_k R[r][k] mu[k][d]
__global__ void __launch_bounds__(kOutCols) k_gmm_out(const float* __restrict__ X,
                                                      const float* __restrict__ mu,
                                                      const float* __restrict__ R,
                                                      const float* __restrict__ rowc,
                                                      const int32_t* __restrict__ n_rows_dev,
                                                      int K, int64_t D, int max_rows,
                                                      float* __restrict__ eps) {
  extern __shared__ float sm[];  // ms[K][kOutCols], rs[kOutRows][K]
  float* ms = sm;
  float* rs = sm + (size_t)K * kOutCols;
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * kOutRows;
  if (r0 >= n_rows) return;
  const int64_t c = (int64_t)blockIdx.x * kOutCols + threadIdx.x;
  for (int k = 0; k < K; ++k) ms[k * kOutCols + threadIdx.x] = (c < D) ? mu[(int64_t)k * D + c] : 0.f;
  const int nr = min(kOutRows, n_rows - r0);
  for (int q = threadIdx.x; q < nr * K; q += kOutCols) rs[q] = R[(int64_t)r0 * K + q];
  __syncthreads();
  if (c >= D) return;
  for (int rr = 0; rr < nr; ++rr) {
    const int r = r0 + rr;
    float m = 0.f;
    for (int k = 0; k < K; ++k) m = fmaf(rs[rr * K + k], ms[k * kOutCols + threadIdx.x], m);
    const float ac = rowc[2 * r], acs = rowc[2 * r + 1];
    eps[(int64_t)r * D + c] = ac * X[(int64_t)r * D + c] - acs * m;
  }
}

}  // namespace

struct pa_gmm {
  int K, T, max_rows;
  int64_t D;
  const float* means;
  char* ws;
  GmmLayout L;
  cudaStream_t st;
  int64_t launches;
};

extern "C" size_t pa_gmm_workspace_bytes(int K, int64_t D, int max_rows, int T) {
  if (K < 1 || K > kMaxK || D < 1 || max_rows < 1 || T < 1 || T > 100000) return 0;
  return gmm_layout(K, D, max_rows, T).total;
}

extern "C" pa_status pa_gmm_create(pa_gmm** out, int K, int64_t D, const float* means_dev,
                                   double std, const double* alphas_cumprod, int T,
                                   int max_rows, void* workspace_dev, size_t workspace_bytes,
                                   void* stream) {
  if (!out) { pa::set_error("pa_gmm_create: out is NULL"); return PA_ERR_ARG; }
  *out = nullptr;
  if (K < 1 || K > kMaxK) { pa::set_error("pa_gmm_create: K must be in [1, 128]"); return PA_ERR_ARG; }
  if (D < 1 || max_rows < 1 || T < 1 || T > 100000 || !means_dev || !alphas_cumprod ||
      !(std >= 0.0) || !std::isfinite(std)) {
    pa::set_error("pa_gmm_create: bad size, pointer or std");
    return PA_ERR_ARG;
  }
  for (int i = 0; i <= T; ++i) {
    const double a = alphas_cumprod[i];
    if (!(a > 0.0 && a <= 1.0)) { pa::set_error("pa_gmm_create: alphas_cumprod must be in (0, 1]"); return PA_ERR_ARG; }
  }
  GmmLayout L = gmm_layout(K, D, max_rows, T);
  if (!workspace_dev || (reinterpret_cast<uintptr_t>(workspace_dev) % pa::kAlign) != 0 ||
      workspace_bytes < L.total) {
    pa::set_error("pa_gmm_create: workspace NULL, not 256-byte aligned, or smaller than pa_gmm_workspace_bytes()");
    return PA_ERR_WORKSPACE;
  }
  pa_gmm* g = new pa_gmm{};
  g->K = K; g->T = T; g->max_rows = max_rows; g->D = D; g->means = means_dev;
  g->ws = static_cast<char*>(workspace_dev); g->L = L;
  g->st = static_cast<cudaStream_t>(stream);
  std::vector<float> coef(3 * (size_t)T);
  for (int i = 0; i < T; ++i) {
    const double a = alphas_cumprod[i];
    const double v = a * std * std + (1.0 - a);
    coef[i] = (float)std::sqrt(a);
    coef[T + i] = (float)(1.0 / (2.0 * v));
    coef[2 * T + i] = (float)(std::sqrt(1.0 - a) / v);
  }
  cudaError_t e = cudaMemcpyAsync(g->ws + L.coef, coef.data(), coef.size() * sizeof(float),
                                  cudaMemcpyHostToDevice, g->st);
  if (e == cudaSuccess) {
    k_gmm_norms<<<K, 256, 0, g->st>>>(means_dev, D, reinterpret_cast<float*>(g->ws + L.mnorm));
    g->launches++;
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(g->st);
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_create: ") + cudaGetErrorString(e));
    delete g;
    return PA_ERR_CUDA;
  }
  const size_t out_smem = ((size_t)K * kOutCols + (size_t)kOutRows * K) * sizeof(float);
  if (out_smem > 48 * 1024) {
    e = cudaFuncSetAttribute(k_gmm_out, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)out_smem);
    if (e != cudaSuccess) {
      pa::set_error(std::string("pa_gmm_create: ") + cudaGetErrorString(e));
      delete g;
      return PA_ERR_CUDA;
    }
  }
  *out = g;
  return PA_OK;
}

extern "C" pa_status pa_gmm_eps(pa_gmm* g, const float* batch_x_dev, const int32_t* miss_bt_dev,
                                const int32_t* n_rows_dev, float* batch_eps_dev) {
  if (!g || !batch_x_dev || !miss_bt_dev || !n_rows_dev || !batch_eps_dev) {
    pa::set_error("pa_gmm_eps: NULL argument");
    return PA_ERR_ARG;
  }
  const GmmLayout& L = g->L;
  float* coef = reinterpret_cast<float*>(g->ws + L.coef);
  float* mnorm = reinterpret_cast<float*>(g->ws + L.mnorm);
  float* gpart = reinterpret_cast<float*>(g->ws + L.gpart);
  float* R = reinterpret_cast<float*>(g->ws + L.R);
  float* rowc = reinterpret_cast<float*>(g->ws + L.rowc);
  const int rb = (g->max_rows + kDotRows - 1) / kDotRows;
  k_gmm_dots<<<dim3(L.nsplit, rb), kDotThreads, 0, g->st>>>(batch_x_dev, g->means, n_rows_dev,
                                                           g->K, g->D, L.split_len, g->max_rows, gpart);
  k_gmm_softmax<<<(g->max_rows + 7) / 8, 256, 0, g->st>>>(gpart, mnorm, coef, g->T, miss_bt_dev,
                                                         n_rows_dev, g->K, L.nsplit, g->max_rows,
                                                         R, rowc);
  const size_t out_smem = ((size_t)g->K * kOutCols + (size_t)kOutRows * g->K) * sizeof(float);
  k_gmm_out<<<dim3((unsigned)((g->D + kOutCols - 1) / kOutCols), (g->max_rows + kOutRows - 1) / kOutRows),
              kOutCols, out_smem, g->st>>>(batch_x_dev, g->means, R, rowc, n_rows_dev, g->K, g->D,
                                            g->max_rows, batch_eps_dev);
  g->launches += 3;
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  return PA_OK;
}

extern "C" int64_t pa_gmm_launches(const pa_gmm* g) { return g ? g->launches : -1; }

extern "C" void pa_gmm_destroy(pa_gmm* g) { delete g; }
