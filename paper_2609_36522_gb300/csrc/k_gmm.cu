// Synthetic denoiser: posterior-mean noise of an isotropic Gaussian mixture,
// the seedable stand-in for the SD v1.5 UNet eps_theta (Sec. 3.2). Not part
// of ParaAnya; it produces the fresh eps of the misses (Eq. 6, miss branch).
//
//   v = a s^2 + 1 - a,   logit_k = (2 sqrt(a) x.mu_k - a ||mu_k||^2) / (2 v)
//   r = softmax(logit)   (the common -||x||^2 / (2 v) term cancels)
//   eps = sqrt(1 - a) / v * (x - sqrt(a) sum_k r_k mu_k)
//
// Three kernels per call, each with a single load phase:
//   k_gmm_dots     split-K contraction G = X M^T: a CTA stages a tile of 16
//                  rows and its D-chunk of every mean (bulk copies), one warp
//                  per row accumulates 16 components per pass, partials go to
//                  gpart[chunk][row][k]
//   k_gmm_softmax  one CTA per row: fixed-order sum of the chunk partials,
//                  logits, max-subtracted softmax
//   k_gmm_out      a CTA stages a 16-row x 256-column tile of X and the same
//                  columns of every mean, then eps = a x - a sqrt(a) R M
// Per-timestep scalars (sqrt(a), 1/(2v), sqrt(1-a)/v) are computed on the
// host in fp64 from alpha-bar and stored in fp32, so 1 - a never cancels in
// fp32. Reductions run in a fixed order: results are bitwise reproducible.
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/paraanya.h"
#include "pa_bulk.cuh"
#include "pa_internal.h"

namespace pa {
void set_error(const std::string& msg);  // pa_solver.cpp
}

namespace {

using pa::pdl_trigger;
using pa::pdl_wait;
using pa::bulk_g2s;
using pa::fence_barrier_init;
using pa::mbar_arrive_expect_tx;
using pa::mbar_init;
using pa::mbar_wait_bounded;

constexpr int kMaxK = 128;
constexpr int kThreads = 256;
constexpr int kDotRows = 16;     // rows per dots CTA (two per warp)
constexpr int kKTile = 16;       // components accumulated per pass
constexpr int kOutRows = 16;     // rows per output CTA
constexpr int kOutCols = 256;    // columns per output CTA (one per thread)
constexpr size_t kDotSmemBudget = 96 * 1024;

struct GmmLayout {
  size_t coef, mnorm, gpart, R, rowc, status, total;
  int nchunk;       // D-chunks of the dots kernel
  int chunk;        // columns per chunk
};

int dots_chunk(int K, int64_t D) {
  // largest of 512/256/128/64 columns whose (rows + K) row segments fit the budget
  int c = 512;
  while (c > 64 && (size_t)(kDotRows + K) * (c + 4) * sizeof(float) > kDotSmemBudget) c /= 2;
  while (c > 64 && (int64_t)c >= 2 * D) c /= 2;
  return c;
}

GmmLayout gmm_layout(int K, int64_t D, int max_rows, int T) {
  GmmLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  L.chunk = dots_chunk(K, D);
  L.nchunk = (int)((D + L.chunk - 1) / L.chunk);
  L.coef = take((size_t)3 * T * sizeof(float));
  L.mnorm = take((size_t)K * sizeof(float));
  L.gpart = take((size_t)L.nchunk * max_rows * K * sizeof(float));
  L.R = take((size_t)max_rows * K * sizeof(float));
  L.rowc = take((size_t)max_rows * 2 * sizeof(float));
  L.status = take(sizeof(int32_t));
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

// Stage `nrows` row segments [c0, c0 + ncol) of a row-major matrix with row
// length D into shared rows of stride `ld` floats: bulk copies counted on
// `bar`, issued by thread 0 (after the caller announced the bytes), or plain
// loads by every thread when `bulk` is false.
__device__ __forceinline__ void stage_rows(float* dst, int ld, const float* src, int64_t D, int64_t c0,
                                           int ncol, int nrows, bool bulk, uint64_t* bar) {
  if (bulk) {
    if (threadIdx.x == 0) {
      const uint32_t seg = (uint32_t)ncol * sizeof(float);
      for (int r = 0; r < nrows; ++r) bulk_g2s(dst + (size_t)r * ld, src + (int64_t)r * D + c0, seg, bar);
    }
    return;
  }
  for (int q = threadIdx.x; q < nrows * ncol; q += blockDim.x) {
    const int r = q / ncol, c = q % ncol;
    dst[(size_t)r * ld + c] = src[(int64_t)r * D + c0 + c];
  }
}

// Wait for the bulk copies of a single-phase kernel. On a timeout: record it,
// let the copies already issued land (bounded), and report false.
__device__ __forceinline__ bool wait_staged(bool bulk, uint64_t* bar, int32_t* status) {
  if (!bulk) return true;
  if (mbar_wait_bounded(bar, 0, pa::kWaitLimit)) return true;
  atomicCAS(status, 0, pa::kDevTimeout);
  mbar_wait_bounded(bar, 0, pa::kDrainLimit);
  return false;
}

// gpart[chunk][r][k] = sum over the chunk's columns of x[r][d] mu[k][d]
__global__ void __launch_bounds__(kThreads) k_gmm_dots(const float* __restrict__ X,
                                                       const float* __restrict__ mu,
                                                       const int32_t* __restrict__ n_rows_dev,
                                                       int K, int64_t D, int chunk, int max_rows,
                                                       bool bulk, float* __restrict__ gpart,
                                                       int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar;
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * kDotRows;
  if (r0 >= n_rows) return;
  const int nr = min(kDotRows, n_rows - r0);
  const int64_t c0 = (int64_t)blockIdx.x * chunk;
  const int ncol = (int)(((D - c0) < chunk) ? (D - c0) : chunk);
  const int ld = chunk + 4;  // padded row stride, keeps 16-byte alignment
  float* xs = reinterpret_cast<float*>(smem_raw);
  float* ms = xs + (size_t)kDotRows * ld;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar, (uint32_t)ncol * sizeof(float) * (uint32_t)(nr + K));
  }
  __syncthreads();
  stage_rows(ms, ld, mu, D, c0, ncol, K, bulk, &bar);  // the means do not depend on the predecessor
  pdl_wait();  // the rows come from the gather (or the caller) just before
  stage_rows(xs, ld, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar);
  const bool ok = wait_staged(bulk, &bar, status);
  __syncthreads();
  if (!ok) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int rr = warp; rr < nr; rr += kThreads / 32) {
    const float* xr = xs + (size_t)rr * ld;
    for (int k0 = 0; k0 < K; k0 += kKTile) {
      float acc[kKTile];
#pragma unroll
      for (int u = 0; u < kKTile; ++u) acc[u] = 0.f;
      for (int c = lane; c < ncol; c += 32) {
        const float xv = xr[c];
#pragma unroll
        for (int u = 0; u < kKTile; ++u)
          if (k0 + u < K) acc[u] = fmaf(xv, ms[(size_t)(k0 + u) * ld + c], acc[u]);
      }
#pragma unroll
      for (int u = 0; u < kKTile; ++u) acc[u] = warp_sum(acc[u]);
      if (lane < kKTile && k0 + lane < K) {
        float v = 0.f;
#pragma unroll
        for (int u = 0; u < kKTile; ++u) v = (lane == u) ? acc[u] : v;
        gpart[((int64_t)blockIdx.x * max_rows + r0 + rr) * K + k0 + lane] = v;
      }
    }
  }
}

// One CTA per row: dots (fixed-order chunk sum) -> logits -> softmax.
__global__ void __launch_bounds__(kThreads) k_gmm_softmax(const float* __restrict__ gpart,
                                                          const float* __restrict__ mnorm,
                                                          const float* __restrict__ coef, int T,
                                                          const int32_t* __restrict__ miss_bt,
                                                          const int32_t* __restrict__ n_rows_dev,
                                                          int K, int nchunk, int max_rows,
                                                          float* __restrict__ R,
                                                          float* __restrict__ rowc) {
  __shared__ float s_part[kThreads];
  __shared__ float s_logit[kMaxK];
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r = blockIdx.x;
  if (r >= n_rows) return;
  // thread -> (component k, chunk group g); groups take the chunks round robin
  int KB = 1;
  while (KB < K) KB <<= 1;
  const int G = kThreads / KB;
  const int k = threadIdx.x % KB, g = threadIdx.x / KB;
  const int i = miss_bt[2 * r + 1];
  const float sa = coef[i], q = coef[T + i], ac = coef[2 * T + i];
  pdl_wait();  // the partials come from the dot-product kernel
  float part = 0.f;
  if (k < K)
    for (int s = g; s < nchunk; s += G) part += gpart[((int64_t)s * max_rows + r) * K + k];
  s_part[threadIdx.x] = part;
  __syncthreads();
  if (threadIdx.x < K) {
    float dot = 0.f;
    for (int gg = 0; gg < G; ++gg) dot += s_part[gg * KB + threadIdx.x];
    s_logit[threadIdx.x] = (2.f * sa * dot - sa * sa * mnorm[threadIdx.x]) * q;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    float mx = -INFINITY;
    for (int kk = lane; kk < K; kk += 32) mx = fmaxf(mx, s_logit[kk]);
    mx = warp_max(mx);
    float sum = 0.f;
    for (int kk = lane; kk < K; kk += 32) sum += expf(s_logit[kk] - mx);
    sum = warp_sum(sum);
    const float inv = 1.f / sum;
    for (int kk = lane; kk < K; kk += 32) R[(int64_t)r * K + kk] = expf(s_logit[kk] - mx) * inv;
    if (lane == 0) {
      rowc[2 * r] = ac;
      rowc[2 * r + 1] = ac * sa;
    }
  }
}

// eps[r][c] = ac x[r][c] - ac sqrt(a) sum_k R[r][k] mu[k][c]
__global__ void __launch_bounds__(kOutCols) k_gmm_out(const float* __restrict__ X,
                                                      const float* __restrict__ mu,
                                                      const float* __restrict__ R,
                                                      const float* __restrict__ rowc,
                                                      const int32_t* __restrict__ n_rows_dev,
                                                      int K, int64_t D, int max_rows, bool bulk,
                                                      float* __restrict__ eps, int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ float s_r[kOutRows * kMaxK];
  __shared__ float s_c[kOutRows * 2];
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * kOutRows;
  if (r0 >= n_rows) return;
  const int nr = min(kOutRows, n_rows - r0);
  const int64_t c0 = (int64_t)blockIdx.x * kOutCols;
  const int ncol = (int)(((D - c0) < kOutCols) ? (D - c0) : kOutCols);
  float* ms = reinterpret_cast<float*>(smem_raw);   // [K][kOutCols]
  float* xs = ms + (size_t)K * kOutCols;            // [kOutRows][kOutCols]
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar, (uint32_t)ncol * sizeof(float) * (uint32_t)(nr + K));
  }
  __syncthreads();
  // the means and the rows (written two kernels back) do not depend on the predecessor
  stage_rows(ms, kOutCols, mu, D, c0, ncol, K, bulk, &bar);
  stage_rows(xs, kOutCols, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar);
  pdl_wait();  // the responsibilities come from the softmax kernel
  for (int q = threadIdx.x; q < nr * K; q += kOutCols) s_r[q] = R[(int64_t)r0 * K + q];
  for (int q = threadIdx.x; q < nr * 2; q += kOutCols) s_c[q] = rowc[2 * r0 + q];
  const bool ok = wait_staged(bulk, &bar, status);
  __syncthreads();
  if (!ok) return;
  const int c = threadIdx.x;
  if (c >= ncol) return;
  for (int rr = 0; rr < nr; ++rr) {
    float m = 0.f;
    for (int k = 0; k < K; ++k) m = fmaf(s_r[rr * K + k], ms[(size_t)k * kOutCols + c], m);
    eps[(int64_t)(r0 + rr) * D + c0 + c] = s_c[2 * rr] * xs[(size_t)rr * kOutCols + c] - s_c[2 * rr + 1] * m;
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
  if (e == cudaSuccess) e = cudaMemsetAsync(g->ws + L.status, 0, sizeof(int32_t), g->st);
  if (e == cudaSuccess) {
    k_gmm_norms<<<K, 256, 0, g->st>>>(means_dev, D, reinterpret_cast<float*>(g->ws + L.mnorm));
    g->launches++;
    e = cudaGetLastError();
  }
  const size_t dots_smem = (size_t)(kDotRows + K) * (L.chunk + 4) * sizeof(float);
  const size_t out_smem = (size_t)(K + kOutRows) * kOutCols * sizeof(float);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gmm_dots, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dots_smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gmm_out, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)out_smem);
  if (e == cudaSuccess) e = cudaStreamSynchronize(g->st);
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_create: ") + cudaGetErrorString(e));
    delete g;
    return PA_ERR_CUDA;
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
  int32_t* status = reinterpret_cast<int32_t*>(g->ws + L.status);
  // bulk copies need 16-byte aligned rows: D % 4 == 0 and aligned base pointers
  const bool bulk = g->D % 4 == 0 && ((reinterpret_cast<uintptr_t>(batch_x_dev) |
                                       reinterpret_cast<uintptr_t>(g->means)) & 15) == 0;
  const size_t dots_smem = (size_t)(kDotRows + g->K) * (L.chunk + 4) * sizeof(float);
  const size_t out_smem = (size_t)(g->K + kOutRows) * kOutCols * sizeof(float);
  cudaError_t e = pa::launch_ex(k_gmm_dots, dim3(L.nchunk, (g->max_rows + kDotRows - 1) / kDotRows),
                                dim3(kThreads), dots_smem, g->st, 0, batch_x_dev, g->means, n_rows_dev, g->K,
                                g->D, L.chunk, g->max_rows, bulk, gpart, status);
  if (e == cudaSuccess)
    e = pa::launch_ex(k_gmm_softmax, dim3(g->max_rows), dim3(kThreads), 0, g->st, 0, (const float*)gpart,
                      (const float*)mnorm, (const float*)coef, g->T, miss_bt_dev, n_rows_dev, g->K, L.nchunk,
                      g->max_rows, R, rowc);
  if (e == cudaSuccess)
    e = pa::launch_ex(k_gmm_out,
                      dim3((unsigned)((g->D + kOutCols - 1) / kOutCols), (g->max_rows + kOutRows - 1) / kOutRows),
                      dim3(kOutCols), out_smem, g->st, 0, batch_x_dev, g->means, (const float*)R,
                      (const float*)rowc, n_rows_dev, g->K, g->D, g->max_rows, bulk, batch_eps_dev, status);
  g->launches += 3;
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  return PA_OK;
}

extern "C" pa_status pa_gmm_check(pa_gmm* g) {
  if (!g) { pa::set_error("pa_gmm_check: NULL handle"); return PA_ERR_ARG; }
  int32_t st = 0;
  cudaError_t e = cudaMemcpyAsync(&st, g->ws + g->L.status, sizeof(st), cudaMemcpyDeviceToHost, g->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(g->st);
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_check: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  if (st == pa::kDevTimeout) { pa::set_error("pa_gmm_check: a bounded wait ran out"); return PA_ERR_TIMEOUT; }
  return PA_OK;
}

extern "C" int64_t pa_gmm_launches(const pa_gmm* g) { return g ? g->launches : -1; }

extern "C" void pa_gmm_destroy(pa_gmm* g) { delete g; }

// ---------------------------------------------------------------------------
// Allocation-free variant of pa_gmm_eps (no counterpart in the paper).
//
// Some callers cannot allocate device memory when they need the denoiser: a
// plugin that only receives buffers handed over by its host framework, a
// real-time loop that forbids cudaMalloc/cudaFree after start-up because an
// allocation may block, or code running where another allocator owns the
// device. pa_gmm_eps keeps its scratch (per-timestep coefficients, ||mu_k||^2,
// split-K partial dot products, responsibilities, a status word) in the
// workspace of a pa_gmm handle; pa_gmm_eps_noalloc keeps the same scratch in
// the fixed device array below and runs the same kernels on it.
constexpr size_t kNoAllocScratchBytes = (size_t)4 << 20;  // 4 MiB, held by every device that loads this library

// The fixed scratch. In host code `g_gmm_scratch` is only a stand-in name:
// its device address comes from cudaGetSymbolAddress, looked up per device.
static __device__ __align__(256) unsigned char g_gmm_scratch[kNoAllocScratchBytes];

namespace {

constexpr int kNoAllocMaxDevices = 64;
constexpr int kNoAllocCoefChunk = 512;                    // host coefficients staged in chunks on the stack

std::mutex g_scratch_mu;
unsigned char* g_scratch_dev[kNoAllocMaxDevices] = {};

// Device address of g_gmm_scratch for the current device, looked up once per
// device (the host-side name is only a stand-in for the device array).
pa_status scratch_for_current_device(unsigned char** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: cudaGetDevice: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kNoAllocMaxDevices) {
    pa::set_error("pa_gmm_eps_noalloc: device index beyond the supported 64");
    return PA_ERR_ARG;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_gmm_scratch);
    if (e != cudaSuccess || !p) {
      pa::set_error(std::string("pa_gmm_eps_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      return PA_ERR_CUDA;
    }
    g_scratch_dev[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_dev[dev];
  return PA_OK;
}

}  // namespace

extern "C" pa_status pa_gmm_eps_noalloc(const float* means_dev, int K, int64_t D, double std,
                                        const double* alphas_cumprod, int T,
                                        const float* batch_x_dev, const int32_t* miss_bt_dev,
                                        int n_rows, float* batch_eps_dev, void* stream) {
  if (K < 1 || K > kMaxK || D < 1 || T < 1 || n_rows < 0 || !means_dev || !alphas_cumprod ||
      !batch_x_dev || !miss_bt_dev || !batch_eps_dev || !(std >= 0.0) || !std::isfinite(std)) {
    pa::set_error("pa_gmm_eps_noalloc: bad size, pointer or std");
    return PA_ERR_ARG;
  }
  for (int i = 0; i <= T; ++i) {
    const double a = alphas_cumprod[i];
    if (!(a > 0.0 && a <= 1.0)) {
      pa::set_error("pa_gmm_eps_noalloc: alphas_cumprod must be in (0, 1]");
      return PA_ERR_ARG;
    }
  }
  if (n_rows == 0) return PA_OK;
  // scratch layout: coef[3T] | mnorm[K] | gpart[nchunk][n_rows][K] | R[n_rows][K] |
  //                 rowc[n_rows][2] | n_rows | status   (256-byte aligned pieces)
  const int chunk = dots_chunk(K, D);
  const int nchunk = (int)((D + chunk - 1) / chunk);
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  const size_t o_coef = take((size_t)3 * T * sizeof(float));
  const size_t o_mnorm = take((size_t)K * sizeof(float));
  const size_t o_gpart = take((size_t)nchunk * n_rows * K * sizeof(float));
  const size_t o_R = take((size_t)n_rows * K * sizeof(float));
  const size_t o_rowc = take((size_t)n_rows * 2 * sizeof(float));
  const size_t o_n = take(sizeof(int32_t));
  const size_t o_status = take(sizeof(int32_t));
  if (o > kNoAllocScratchBytes) {
    pa::set_error("pa_gmm_eps_noalloc: these sizes need " + std::to_string(o) +
                  " bytes of scratch, more than the fixed 4 MiB (4194304 bytes); "
                  "use pa_gmm_create + pa_gmm_eps with a caller-allocated workspace");
    return PA_ERR_ARG;
  }
  unsigned char* scratch = nullptr;
  pa_status ps = scratch_for_current_device(&scratch);
  if (ps != PA_OK) return ps;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* coef = reinterpret_cast<float*>(scratch + o_coef);
  float* mnorm = reinterpret_cast<float*>(scratch + o_mnorm);
  float* gpart = reinterpret_cast<float*>(scratch + o_gpart);
  float* R = reinterpret_cast<float*>(scratch + o_R);
  float* rowc = reinterpret_cast<float*>(scratch + o_rowc);
  int32_t* nrows_dev = reinterpret_cast<int32_t*>(scratch + o_n);
  int32_t* status = reinterpret_cast<int32_t*>(scratch + o_status);

  // Per-timestep scalars, formed in fp64 on the host in stack-sized chunks;
  // each pageable copy returns once its source has been staged.
  cudaError_t e = cudaSuccess;
  float buf[kNoAllocCoefChunk];
  for (int part = 0; part < 3 && e == cudaSuccess; ++part) {
    for (int i0 = 0; i0 < T && e == cudaSuccess; i0 += kNoAllocCoefChunk) {
      const int n = (T - i0) < kNoAllocCoefChunk ? (T - i0) : kNoAllocCoefChunk;
      for (int u = 0; u < n; ++u) {
        const double a = alphas_cumprod[i0 + u];
        const double v = a * std * std + (1.0 - a);
        buf[u] = (float)(part == 0 ? std::sqrt(a) : part == 1 ? 1.0 / (2.0 * v) : std::sqrt(1.0 - a) / v);
      }
      e = cudaMemcpyAsync(coef + (size_t)part * T + i0, buf, (size_t)n * sizeof(float),
                          cudaMemcpyHostToDevice, st);
    }
  }
  const int32_t nr = n_rows;
  if (e == cudaSuccess) e = cudaMemcpyAsync(nrows_dev, &nr, sizeof(nr), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(status, 0, sizeof(int32_t), st);  // starts at zero every call
  const size_t dots_smem = (size_t)(kDotRows + K) * (chunk + 4) * sizeof(float);
  const size_t out_smem = (size_t)(K + kOutRows) * kOutCols * sizeof(float);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gmm_dots, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dots_smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gmm_out, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)out_smem);
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  const bool bulk = D % 4 == 0 && ((reinterpret_cast<uintptr_t>(batch_x_dev) |
                                    reinterpret_cast<uintptr_t>(means_dev)) & 15) == 0;
  k_gmm_norms<<<K, 256, 0, st>>>(means_dev, D, mnorm);
  k_gmm_dots<<<dim3(nchunk, (n_rows + kDotRows - 1) / kDotRows), kThreads, dots_smem, st>>>(
      batch_x_dev, means_dev, nrows_dev, K, D, chunk, n_rows, bulk, gpart, status);
  k_gmm_softmax<<<n_rows, kThreads, 0, st>>>(gpart, mnorm, coef, T, miss_bt_dev, nrows_dev, K, nchunk,
                                             n_rows, R, rowc);
  k_gmm_out<<<dim3((unsigned)((D + kOutCols - 1) / kOutCols), (n_rows + kOutRows - 1) / kOutRows),
              kOutCols, out_smem, st>>>(batch_x_dev, means_dev, R, rowc, nrows_dev, K, D, n_rows, bulk,
                                        batch_eps_dev, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  return PA_OK;
}
