// Synthetic denoiser: posterior-mean noise of an isotropic Gaussian mixture,
// the seedable stand-in for the SD v1.5 UNet eps_theta (Sec. 3.2). Not part
// of ParaAnya; it produces the fresh eps of the misses (Eq. 6, miss branch).
//
//   v = a s^2 + 1 - a,   logit_k = (2 sqrt(a) x.mu_k - a ||mu_k||^2) / (2 v)
//   r = softmax(logit)   (the common -||x||^2 / (2 v) term cancels)
//   eps = sqrt(1 - a) / v * (x - sqrt(a) sum_k r_k mu_k)
//
// Two kernels per call, each with a single load phase:
//   k_gmm_dots     split-K contraction G = X M^T over bulk-staged 16-row tiles
//                  (register-tiled 4 rows x 8 components per thread); the last
//                  CTA of each row block sums the chunks in a fixed order and
//                  applies the logits and the max-subtracted softmax
//   k_gmm_out      eps = a x - a sqrt(a) R M over bulk-staged 16-row x
//                  256-column tiles (4 x 4 outputs per thread)
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
constexpr int kOutCols = 256;    // columns per output CTA (four per thread)
constexpr size_t kDotSmemBudget = 96 * 1024;
constexpr float kDotScale = 4294967296.f;  // 2^32: fixed-point scale of the dot-product accumulators

struct GmmLayout {
  size_t coef, mnorm, gacc, R, rowc, tickets, status, total;
  int nchunk;       // D-chunks of the dots kernel
  int chunk;        // columns per chunk
};

size_t dots_smem_bytes(int K, int chunk) {
  // the staged tiles, later reused for the column-split sums
  int KG = 1;
  while (KG * 8 < K) KG <<= 1;
  const size_t tiles = (size_t)(kDotRows + K) * (chunk + 4) * sizeof(float);
  const size_t red = (size_t)(kThreads / (4 * KG) + 1) * kDotRows * K * sizeof(float);
  return tiles > red ? tiles : red;
}

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
  L.gacc = take((size_t)max_rows * K * sizeof(long long));
  L.R = take((size_t)max_rows * K * sizeof(float));
  L.rowc = take((size_t)max_rows * 2 * sizeof(float));
  L.tickets = take((size_t)((max_rows + kDotRows - 1) / kDotRows) * sizeof(uint32_t));
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
// `bar`, issued by the lanes of warp 0 (after the caller announced the bytes),
// or plain loads by every thread when `bulk` is false.
__device__ __forceinline__ void stage_rows(float* dst, int ld, const float* src, int64_t D, int64_t c0,
                                           int ncol, int nrows, bool bulk, uint64_t* bar) {
  if (bulk) {
    if (threadIdx.x < 32) {  // the lanes of warp 0 issue the rows in parallel
      const uint32_t seg = (uint32_t)ncol * sizeof(float);
      for (int r = threadIdx.x; r < nrows; r += 32)
        bulk_g2s(dst + (size_t)r * ld, src + (int64_t)r * D + c0, seg, bar);
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

// Dot products and softmax, one kernel: a CTA stages 16 rows x `chunk`
// columns of X and the same columns of every mean, each thread accumulates a
// 4-row x 8-component block over a column split (register tiling: 12 shared
// loads per 32 FMAs), and the column splits are summed in a fixed order
// through shared memory. Chunks are combined by adding each CTA's sums,
// rounded to fixed point (2^-32), into int64 accumulators gacc[r][k] with
// atomics: integer addition is exact, so the result does not depend on the
// order in which CTAs arrive. The CTA that finishes a row block last (atomic
// ticket after a fence, nobody waits) reads the finished dot products, clears
// the accumulators for the next call, and applies the logits and the
// max-subtracted softmax -> R[r][k], rowc[r].
__global__ void __launch_bounds__(kThreads) k_gmm_dots(const float* __restrict__ X,
                                                       const float* __restrict__ mu,
                                                       const int32_t* __restrict__ n_rows_dev,
                                                       int K, int64_t D, int chunk, int nchunk, int max_rows,
                                                       bool bulk, long long* __restrict__ gacc,
                                                       uint32_t* __restrict__ tickets,
                                                       const float* __restrict__ coef, int T,
                                                       const int32_t* __restrict__ miss_bt,
                                                       const float* __restrict__ mnorm,
                                                       float* __restrict__ R, float* __restrict__ rowc,
                                                       int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_last;
  __shared__ float s_logit[kDotRows * kMaxK];
  __shared__ float s_sa[kDotRows], s_q[kDotRows], s_ac[kDotRows];
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * kDotRows;
  if (r0 >= n_rows) return;
  const int nr = min(kDotRows, n_rows - r0);
  const int64_t c0 = (int64_t)blockIdx.x * chunk;
  const int ncol = (int)(((D - c0) < chunk) ? (D - c0) : chunk);
  const int ld = chunk + 4;  // padded row stride, keeps 16-byte alignment
  float* xs = reinterpret_cast<float*>(smem_raw);
  float* ms = xs + (size_t)kDotRows * ld;
  const int tid = threadIdx.x;
  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar, (uint32_t)ncol * sizeof(float) * (uint32_t)(nr + K));
  }
  for (int q = tid; q < (kDotRows - nr) * ld; q += kThreads) xs[(size_t)nr * ld + q] = 0.f;  // rows past nr
  __syncthreads();
  stage_rows(ms, ld, mu, D, c0, ncol, K, bulk, &bar);  // the means do not depend on the predecessor
  pdl_wait();  // the rows come from the gather (or the caller) just before
  stage_rows(xs, ld, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar);
  const bool ok = wait_staged(bulk, &bar, status);
  __syncthreads();
  if (!ok) return;

  // thread -> (column split tcs, component group tkg, row group trg)
  int KG = 1;
  while (KG * 8 < K) KG <<= 1;          // component groups of 8 (power of two)
  const int CS = kThreads / (4 * KG);   // column splits
  const int tcs = tid % CS, tkg = (tid / CS) % KG, trg = tid / (CS * KG);
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int u = 0; u < 8; ++u) acc[i][u] = 0.f;
  for (int c = tcs; c < ncol; c += CS) {
    float xv[4], mv[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) xv[i] = xs[(size_t)(trg * 4 + i) * ld + c];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int k = tkg + KG * u;  // interleaved: neighbouring groups read neighbouring rows
      mv[u] = (k < K) ? ms[(size_t)k * ld + c] : 0.f;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int u = 0; u < 8; ++u) acc[i][u] = fmaf(xv[i], mv[u], acc[i][u]);
  }
  __syncthreads();  // the tiles are consumed: reuse their space for the split sums
  float* red = xs;  // [kDotRows * K][CS + 1]: split index fastest (conflict-free both ways)
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int k = tkg + KG * u;
      if (k < K) red[((size_t)(trg * 4 + i) * K + k) * (CS + 1) + tcs] = acc[i][u];
    }
  __syncthreads();
  for (int o = tid; o < nr * K; o += kThreads) {
    float a4[4] = {0.f, 0.f, 0.f, 0.f};
    const float* ro = red + (size_t)o * (CS + 1);
    for (int cs = 0, u = 0; cs < CS; ++cs, u = (u + 1) & 3) a4[u] += ro[cs];
    const float sum = (a4[0] + a4[1]) + (a4[2] + a4[3]);
    atomicAdd(reinterpret_cast<unsigned long long*>(gacc + (int64_t)r0 * K + o),
              static_cast<unsigned long long>(__float2ll_rn(sum * kDotScale)));
  }
  // the last CTA of this row block finishes the contraction and the softmax
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const unsigned int k = atomicAdd(&tickets[blockIdx.y], 1u);
    s_last = (k == gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) tickets[blockIdx.y] = 0u;  // ready for the next call
  if (tid < nr) {
    const int i = miss_bt[2 * (r0 + tid) + 1];
    s_sa[tid] = coef[i];
    s_q[tid] = coef[T + i];
    s_ac[tid] = coef[2 * T + i];
  }
  __syncthreads();
  for (int o = tid; o < nr * K; o += kThreads) {
    const int rr = o / K, k = o % K;
    long long* acc_p = gacc + (int64_t)(r0 + rr) * K + k;
    const long long v = __ldcg(acc_p);
    *acc_p = 0;  // ready for the next call
    const float dot = (float)((double)v * (1.0 / (double)kDotScale));
    const float sa = s_sa[rr];
    s_logit[rr * K + k] = (2.f * sa * dot - sa * sa * mnorm[k]) * s_q[rr];
  }
  __syncthreads();
  const int warp = tid >> 5, lane = tid & 31;
  for (int rr = warp; rr < nr; rr += kThreads / 32) {
    const float* l = s_logit + rr * K;
    float mx = -INFINITY;
    for (int k = lane; k < K; k += 32) mx = fmaxf(mx, l[k]);
    mx = warp_max(mx);
    float sum = 0.f;
    for (int k = lane; k < K; k += 32) sum += expf(l[k] - mx);
    sum = warp_sum(sum);
    const float inv = 1.f / sum;
    const int r = r0 + rr;
    for (int k = lane; k < K; k += 32) R[(int64_t)r * K + k] = expf(l[k] - mx) * inv;
    if (lane == 0) {
      rowc[2 * r] = s_ac[rr];
      rowc[2 * r + 1] = s_ac[rr] * s_sa[rr];
    }
  }
}

// eps[r][c] = ac x[r][c] - ac sqrt(a) sum_k R[r][k] mu[k][c]: a CTA stages a
// 16-row x 256-column tile of X and the same columns of every mean; each
// thread computes a 4-row x 4-column block (one 16-byte mean load and four
// broadcast responsibility loads per 16 FMAs).
__global__ void __launch_bounds__(kThreads) k_gmm_out(const float* __restrict__ X,
                                                      const float* __restrict__ mu,
                                                      const float* __restrict__ R,
                                                      const float* __restrict__ rowc,
                                                      const int32_t* __restrict__ n_rows_dev,
                                                      int K, int64_t D, int max_rows, bool bulk, bool vec_out,
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
  const int tid = threadIdx.x;
  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar, (uint32_t)ncol * sizeof(float) * (uint32_t)(nr + K));
  }
  __syncthreads();
  // the means and the rows (written two kernels back) do not depend on the predecessor
  stage_rows(ms, kOutCols, mu, D, c0, ncol, K, bulk, &bar);
  stage_rows(xs, kOutCols, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar);
  pdl_wait();  // the responsibilities come from the dot-product kernel
  for (int q = tid; q < kOutRows * K; q += kThreads) s_r[q] = (q < nr * K) ? R[(int64_t)r0 * K + q] : 0.f;
  for (int q = tid; q < kOutRows * 2; q += kThreads) s_c[q] = (q < nr * 2) ? rowc[2 * r0 + q] : 0.f;
  const bool ok = wait_staged(bulk, &bar, status);
  __syncthreads();
  if (!ok) return;
  const int cg = tid % (kOutCols / 4), rg = tid / (kOutCols / 4);  // 64 column groups x 4 row groups
  const int cc = cg * 4;
  if (cc >= ncol) return;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k = 0; k < K; ++k) {
    const float4 m = *reinterpret_cast<const float4*>(ms + (size_t)k * kOutCols + cc);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float rk = s_r[(rg * 4 + i) * K + k];
      acc[i][0] = fmaf(rk, m.x, acc[i][0]);
      acc[i][1] = fmaf(rk, m.y, acc[i][1]);
      acc[i][2] = fmaf(rk, m.z, acc[i][2]);
      acc[i][3] = fmaf(rk, m.w, acc[i][3]);
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int rr = rg * 4 + i;
    if (rr >= nr) break;
    const float ac = s_c[2 * rr], acs = s_c[2 * rr + 1];
    const float* xr = xs + (size_t)rr * kOutCols + cc;
    float* er = eps + (int64_t)(r0 + rr) * D + c0 + cc;
    if (vec_out && cc + 4 <= ncol) {
      const float4 x = *reinterpret_cast<const float4*>(xr);
      *reinterpret_cast<float4*>(er) = make_float4(ac * x.x - acs * acc[i][0], ac * x.y - acs * acc[i][1],
                                                   ac * x.z - acs * acc[i][2], ac * x.w - acs * acc[i][3]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (cc + j < ncol) er[j] = ac * xr[j] - acs * acc[i][j];
    }
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
  if (e == cudaSuccess)
    e = cudaMemsetAsync(g->ws + L.tickets, 0, (size_t)((max_rows + kDotRows - 1) / kDotRows) * sizeof(uint32_t),
                        g->st);
  if (e == cudaSuccess) e = cudaMemsetAsync(g->ws + L.gacc, 0, (size_t)max_rows * K * sizeof(long long), g->st);
  if (e == cudaSuccess) {
    k_gmm_norms<<<K, 256, 0, g->st>>>(means_dev, D, reinterpret_cast<float*>(g->ws + L.mnorm));
    g->launches++;
    e = cudaGetLastError();
  }
  const size_t dots_smem = dots_smem_bytes(K, L.chunk);
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
  long long* gacc = reinterpret_cast<long long*>(g->ws + L.gacc);
  float* R = reinterpret_cast<float*>(g->ws + L.R);
  float* rowc = reinterpret_cast<float*>(g->ws + L.rowc);
  int32_t* status = reinterpret_cast<int32_t*>(g->ws + L.status);
  // bulk copies need 16-byte aligned rows: D % 4 == 0 and aligned base pointers
  const bool bulk = g->D % 4 == 0 && ((reinterpret_cast<uintptr_t>(batch_x_dev) |
                                       reinterpret_cast<uintptr_t>(g->means)) & 15) == 0;
  uint32_t* tickets = reinterpret_cast<uint32_t*>(g->ws + L.tickets);
  const bool vec_out = g->D % 4 == 0 && (reinterpret_cast<uintptr_t>(batch_eps_dev) & 15) == 0;
  const size_t dots_smem = dots_smem_bytes(g->K, L.chunk);
  const size_t out_smem = (size_t)(g->K + kOutRows) * kOutCols * sizeof(float);
  cudaError_t e = pa::launch_ex(k_gmm_dots, dim3(L.nchunk, (g->max_rows + kDotRows - 1) / kDotRows),
                                dim3(kThreads), dots_smem, g->st, 0, batch_x_dev, g->means, n_rows_dev, g->K,
                                g->D, L.chunk, L.nchunk, g->max_rows, bulk, gacc, tickets, (const float*)coef,
                                g->T, miss_bt_dev, (const float*)mnorm, R, rowc, status);
  if (e == cudaSuccess)
    e = pa::launch_ex(k_gmm_out,
                      dim3((unsigned)((g->D + kOutCols - 1) / kOutCols), (g->max_rows + kOutRows - 1) / kOutRows),
                      dim3(kOutCols), out_smem, g->st, 0, batch_x_dev, g->means, (const float*)R,
                      (const float*)rowc, n_rows_dev, g->K, g->D, g->max_rows, bulk, vec_out, batch_eps_dev,
                      status);
  g->launches += 2;
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
  // scratch layout: coef[3T] | mnorm[K] | gacc[n_rows][K] (int64) | R[n_rows][K] |
  //                 rowc[n_rows][2] | tickets | n_rows | status   (256-byte aligned pieces)
  const int chunk = dots_chunk(K, D);
  const int nchunk = (int)((D + chunk - 1) / chunk);
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  const size_t o_coef = take((size_t)3 * T * sizeof(float));
  const size_t o_mnorm = take((size_t)K * sizeof(float));
  const size_t o_gacc = take((size_t)n_rows * K * sizeof(long long));
  const size_t o_R = take((size_t)n_rows * K * sizeof(float));
  const size_t o_rowc = take((size_t)n_rows * 2 * sizeof(float));
  const size_t o_tick = take((size_t)((n_rows + kDotRows - 1) / kDotRows) * sizeof(uint32_t));
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
  long long* gacc = reinterpret_cast<long long*>(scratch + o_gacc);
  float* R = reinterpret_cast<float*>(scratch + o_R);
  float* rowc = reinterpret_cast<float*>(scratch + o_rowc);
  uint32_t* tickets = reinterpret_cast<uint32_t*>(scratch + o_tick);
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
  if (e == cudaSuccess)  // the row-block tickets and the dot accumulators start at zero every call too
    e = cudaMemsetAsync(tickets, 0, (size_t)((n_rows + kDotRows - 1) / kDotRows) * sizeof(uint32_t), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(gacc, 0, (size_t)n_rows * K * sizeof(long long), st);
  const size_t dots_smem = dots_smem_bytes(K, chunk);
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
  const bool vec_out = D % 4 == 0 && (reinterpret_cast<uintptr_t>(batch_eps_dev) & 15) == 0;
  k_gmm_dots<<<dim3(nchunk, (n_rows + kDotRows - 1) / kDotRows), kThreads, dots_smem, st>>>(
      batch_x_dev, means_dev, nrows_dev, K, D, chunk, nchunk, n_rows, bulk, gacc, tickets, coef, T, miss_bt_dev,
      mnorm, R, rowc, status);
  k_gmm_out<<<dim3((unsigned)((D + kOutCols - 1) / kOutCols), (n_rows + kOutRows - 1) / kOutRows), kOutCols,
              out_smem, st>>>(batch_x_dev, means_dev, R, rowc, nrows_dev, K, D, n_rows, bulk, vec_out,
                              batch_eps_dev, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  return PA_OK;
}
