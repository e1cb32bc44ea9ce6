// Synthetic denoiser: posterior-mean noise of an isotropic Gaussian mixture,
// the seedable stand-in for the SD v1.5 UNet eps_theta (Sec. 3.2). Not part
// of ParaAnya; it produces the fresh eps of the misses (Eq. 6, miss branch).
//
//   v = a s^2 + 1 - a,   logit_k = (2 sqrt(a) x.mu_k - a ||mu_k||^2) / (2 v)
//   r = softmax(logit)   (the common -||x||^2 / (2 v) term cancels)
//   eps = sqrt(1 - a) / v * (x - sqrt(a) sum_k r_k mu_k)
//
// Two kernels per call:
//   dot products   G = X M^T, split over column chunks of D, either on the
//                  tensor cores (k_gmm_dots_tc: tcgen05, tf32 operands split
//                  in two parts for fp32 accuracy) or on the CUDA cores
//                  (k_gmm_dots: bulk-staged 16-row tiles, 4 rows x 8
//                  components per thread); each CTA adds its chunk sums, in
//                  2^-32 fixed point, into int64 accumulators with integer
//                  atomics (exact: the order of arrival does not matter)
//   k_gmm_out      per 16-row block: logits and max-subtracted softmax of its
//                  rows from the accumulators, then eps = a x - a sqrt(a) R M
//                  over bulk-staged 16-row x 256-column tiles (4 x 4 outputs
//                  per thread)
// The accumulators come in two sets used in turn. A call's dot-product kernel
// reads the handle's epoch e, accumulates into set e mod 2, clears the other
// set (read by the previous call's output kernel, which has completed) and
// records e for the output kernel; the output kernel reads set e mod 2 and
// advances the epoch. No kernel waits for another CTA, and the state lives on
// the device, so a captured CUDA graph replays correctly.
// Per-timestep scalars (sqrt(a), 1/(2v), sqrt(1-a)/v) are computed on the
// host in fp64 from alpha-bar and stored in fp32, so 1 - a never cancels in
// fp32. Reductions run in a fixed order: results are bitwise reproducible.
#include <cooperative_groups.h>

#include <cmath>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/paraanya.h"
#include "pa_bulk.cuh"
#include "pa_internal.h"
#include "pa_tcgen05.cuh"

namespace pa {
void set_error(const std::string& msg);  // pa_solver.cpp
}

namespace {

namespace cg = cooperative_groups;

using pa::pdl_trigger;
using pa::pdl_wait;
using pa::bulk_g2s;
using pa::fence_barrier_init;
using pa::mbar_arrive_expect_tx;
using pa::mbar_init;
using pa::mbar_wait_bounded;
using pa::smem_u32;
using pa::tc_commit;
using pa::tc_fence_after_sync;
using pa::tc_fence_before_sync;
using pa::tc_idesc_tf32;
using pa::tc_mma_tf32;
using pa::tc_smem_desc;
using pa::tmem_alloc;
using pa::tmem_dealloc;
using pa::tmem_ld16;
using pa::to_tf32;
using pa::fence_proxy_async_smem;

constexpr int kMaxK = 128;
constexpr int kThreads = 256;
constexpr int kDotRows = 16;     // rows per dots CTA (two per warp)
constexpr int kOutRows = 16;     // rows per output CTA
constexpr int kOutCols = 256;    // columns per output CTA (four per thread)
constexpr size_t kDotSmemBudget = 96 * 1024;
constexpr float kDotScale = 4294967296.f;  // 2^32: fixed-point scale of the dot-product accumulators

// tensor-core dot products: rows per CTA (the MMA's M), columns per CTA
constexpr int kTcRows = 128;
constexpr int kTcCols = 64;   // 8 MMA steps of 8 (98 KB of shared memory at K = 64: two CTAs per SM)
constexpr int kTcThreads = 256;
constexpr int kTcCluster = 8;            // column chunks per thread-block cluster ...
constexpr int kTcClusterMinChunks = 256;  // ... when there are this many chunks (fewer atomics per accumulator)
constexpr int kTcMinK = 16;               // tensor-core dot products by default above this many components

// the MMA's N: K rounded up to 16, 32, 64 or 128 (padded means are zero)
__host__ __device__ inline int tc_npad(int K) {
  int n = 16;
  while (n < K) n <<= 1;
  return n;
}
// floats of one column chunk's means image: hi and lo, Kp rows each
__host__ __device__ inline size_t tc_mu_chunk_floats(int K) { return (size_t)2 * tc_npad(K) * kTcCols; }
// The tensor-core output contraction: kOtCols columns per CTA (two CTAs per
// SM), up to 64 (padded) components; its operand images hold hi rows, then lo
// rows, of tc_npad(K) values in core-matrix order: 2 x 128 rows of
// responsibilities, 2 x kOtCols rows (columns of D) of means.
constexpr int kOtCols = 64;
constexpr int kOtThreads = 256;
constexpr int kOtMaxKp = 64;
constexpr int kRespRows = 8;  // rows per k_gmm_resp CTA, a warp each
__host__ __device__ inline size_t ot_img_floats(int K) { return (size_t)2 * kTcRows * tc_npad(K); }
__host__ __device__ inline size_t ot_mut_floats(int K) { return (size_t)2 * kOtCols * tc_npad(K); }

struct GmmLayout {
  size_t coef, mnorm, gacc, epoch, status, mu_img, mut_img, r_img, rcoef, total;
  int tc_chunks;    // column chunks of the tensor-core dot products (whole clusters)
  int nchunk;       // D-chunks of the CUDA-core dots kernel
  int chunk;        // columns per chunk
};

// Which accumulator set a call uses (see the file comment).
struct GmmEpoch {
  uint32_t epoch;   // advanced by the output kernel
  uint32_t cur;     // the epoch of the dot products just formed
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
  L.gacc = take((size_t)2 * max_rows * K * sizeof(long long));  // two sets, used in turn
  L.epoch = take(sizeof(GmmEpoch));
  L.status = take(sizeof(int32_t));
  L.tc_chunks = (int)((D + kTcCols - 1) / kTcCols + kTcCluster - 1) / kTcCluster * kTcCluster;  // whole clusters
  L.mu_img = take((size_t)L.tc_chunks * tc_mu_chunk_floats(K) * sizeof(float));
  // the tensor-core output contraction (16 < K <= 64): the means' transposed
  // split image, the responsibilities' split image and the rows' scalars
  const bool ot = K > kTcMinK && tc_npad(K) <= kOtMaxKp;
  L.mut_img = take(ot ? (size_t)((D + kOtCols - 1) / kOtCols) * ot_mut_floats(K) * sizeof(float) : 0);
  L.r_img = take(ot ? (size_t)((max_rows + kTcRows - 1) / kTcRows) * ot_img_floats(K) * sizeof(float) : 0);
  L.rcoef = take(ot ? (size_t)2 * max_rows * sizeof(float) : 0);
  L.total = o;
  return L;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
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

// Start of a dot-product kernel: the accumulator set of this call (epoch e),
// the other set cleared by all CTAs together (every CTA, also those without
// rows), and e recorded for the output kernel.
__device__ __forceinline__ long long* begin_dots(long long* gacc2, GmmEpoch* ep, int64_t set_size) {
  const uint32_t e = ep->epoch;  // advanced by the previous call's output kernel, long finished
  long long* other = gacc2 + (int64_t)((e + 1u) & 1u) * set_size;
  const int64_t cta = (int64_t)blockIdx.y * gridDim.x + blockIdx.x;
  const int64_t nthr = (int64_t)gridDim.x * gridDim.y * blockDim.x;
  for (int64_t q = cta * blockDim.x + threadIdx.x; q < set_size; q += nthr) other[q] = 0;
  if (cta == 0 && threadIdx.x == 0) ep->cur = e;
  return gacc2 + (int64_t)(e & 1u) * set_size;
}

// Dot products on the CUDA cores: a CTA stages 16 rows x `chunk` columns of
// X and the same columns of every mean, each thread accumulates a 4-row x
// 8-component block over a column split (register tiling: 12 shared loads per
// 32 FMAs), the column splits are summed in a fixed order through shared
// memory, and the chunk sums go into the accumulators (file comment).
__global__ void __launch_bounds__(kThreads) k_gmm_dots(const float* __restrict__ X,
                                                       const float* __restrict__ mu,
                                                       const int32_t* __restrict__ n_rows_dev,
                                                       int K, int64_t D, int chunk, int nchunk, int max_rows,
                                                       bool bulk, long long* __restrict__ gacc2,
                                                       GmmEpoch* ep, int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar_m, bar_x;
  long long* gacc = begin_dots(gacc2, ep, (int64_t)max_rows * K);
  const int r0 = blockIdx.y * kDotRows;
  const int64_t c0 = (int64_t)blockIdx.x * chunk;
  const int ncol = (int)(((D - c0) < chunk) ? (D - c0) : chunk);
  const int ld = chunk + 4;  // padded row stride, keeps 16-byte alignment
  float* xs = reinterpret_cast<float*>(smem_raw);
  float* ms = xs + (size_t)kDotRows * ld;
  const int tid = threadIdx.x;
  if (tid == 0) {
    mbar_init(&bar_m, 1);
    mbar_init(&bar_x, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar_m, (uint32_t)ncol * sizeof(float) * (uint32_t)K);
  }
  __syncthreads();
  stage_rows(ms, ld, mu, D, c0, ncol, K, bulk, &bar_m);  // the means do not depend on the predecessor
  pdl_wait();  // the rows and their count come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  const int n_rows = min(*n_rows_dev, max_rows);
  const int nr = min(kDotRows, n_rows - r0);
  if (nr <= 0) {  // no rows for this CTA: the means copy lands before it exits
    wait_staged(bulk, &bar_m, status);
    return;
  }
  for (int q = tid; q < (kDotRows - nr) * ld; q += kThreads) xs[(size_t)nr * ld + q] = 0.f;  // rows past nr
  if (tid == 0 && bulk) mbar_arrive_expect_tx(&bar_x, (uint32_t)ncol * sizeof(float) * (uint32_t)nr);
  __syncthreads();
  stage_rows(xs, ld, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar_x);
  const bool ok_m = wait_staged(bulk, &bar_m, status);
  const bool ok = wait_staged(bulk, &bar_x, status) && ok_m;
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
    int cs = 0;
    for (; cs + 3 < CS; cs += 4) {
      a4[0] += ro[cs];
      a4[1] += ro[cs + 1];
      a4[2] += ro[cs + 2];
      a4[3] += ro[cs + 3];
    }
    for (; cs < CS; ++cs) a4[0] += ro[cs];
    const float sum = (a4[0] + a4[1]) + (a4[2] + a4[3]);
    atomicAdd(reinterpret_cast<unsigned long long*>(gacc + (int64_t)r0 * K + o),
              static_cast<unsigned long long>(__float2ll_rn(sum * kDotScale)));
  }
}

// Output kernel. First the 16 rows' responsibilities: the finished dot
// products (accumulator set of this call), the logits with ||mu_k||^2 and the
// per-timestep scalars, and the max-subtracted softmax, while the row and mean
// tiles are in flight. Then eps[r][c] = ac x[r][c] - ac sqrt(a) sum_k
// R[r][k] mu[k][c] over a 16-row x 256-column tile: each thread computes a
// 4-row x 4-column block (one 16-byte mean load and four broadcast
// responsibility loads per 16 FMAs).
__global__ void __launch_bounds__(kThreads) k_gmm_out(const float* __restrict__ X,
                                                      const float* __restrict__ mu,
                                                      const long long* __restrict__ gacc2,
                                                      GmmEpoch* ep, const float* __restrict__ coef, int T,
                                                      const int32_t* __restrict__ miss_bt,
                                                      const float* __restrict__ mnorm,
                                                      const int32_t* __restrict__ n_rows_dev,
                                                      int K, int64_t D, int max_rows, bool bulk, bool vec_out,
                                                      float* __restrict__ eps, int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ float s_r[kOutRows * kMaxK];
  __shared__ float s_c[kOutRows * 2];
  __shared__ float s_sa[kOutRows], s_q[kOutRows];
  const int n_rows = min(*n_rows_dev, max_rows);  // written two kernels back
  const int r0 = blockIdx.y * kOutRows;
  if (r0 >= n_rows) {  // every CTA passes the dependency wait before it exits
    pdl_wait();
    return;
  }
  const int nr = min(kOutRows, n_rows - r0);
  const int64_t c0 = (int64_t)blockIdx.x * kOutCols;
  const int ncol = (int)(((D - c0) < kOutCols) ? (D - c0) : kOutCols);
  float* ms = reinterpret_cast<float*>(smem_raw);   // [K][kOutCols]
  float* xs = ms + (size_t)K * kOutCols;            // [kOutRows][kOutCols]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (bulk) mbar_arrive_expect_tx(&bar, (uint32_t)ncol * sizeof(float) * (uint32_t)(nr + K));
  }
  __syncthreads();
  // the means and the rows (written two kernels back) do not depend on the predecessor
  stage_rows(ms, kOutCols, mu, D, c0, ncol, K, bulk, &bar);
  stage_rows(xs, kOutCols, X + (int64_t)r0 * D, D, c0, ncol, nr, bulk, &bar);
  for (int rr = tid; rr < nr; rr += kThreads) {
    const int i = miss_bt[2 * (r0 + rr) + 1];
    s_sa[rr] = coef[i];
    s_q[rr] = coef[T + i];
    s_c[2 * rr] = coef[2 * T + i];
    s_c[2 * rr + 1] = coef[2 * T + i] * coef[i];
  }
  pdl_wait();  // the dot products come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  // both accumulator sets are read together with the set index and the
  // status word (one round trip): a dot-product kernel that timed out left
  // the sums incomplete
  const uint32_t cur = ep->cur;
  const int dots_status = __ldcg(status);
  const int64_t set_size = (int64_t)max_rows * K;
  __syncthreads();
  for (int q = tid; q < kOutRows * K; q += kThreads) {
    float l = 0.f;
    if (q < nr * K) {
      const int rr = q / K, k = q % K;
      const long long v0 = __ldcg(gacc2 + (int64_t)r0 * K + q);
      const long long v1 = __ldcg(gacc2 + set_size + (int64_t)r0 * K + q);
      const float dot = __ll2float_rn((cur & 1u) ? v1 : v0) * (1.f / kDotScale);  // exact scale
      const float sa = s_sa[rr];
      l = (2.f * sa * dot - sa * sa * mnorm[k]) * s_q[rr];
    }
    s_r[q] = l;
  }
  __syncthreads();
  // softmax per row: a half-warp per row when K <= 16 (two rows per warp and
  // pass), else a warp; the reductions are the same trees either way
  {
    const int width = K <= 16 ? 16 : 32, sub = lane / width, sl = lane % width;
    for (int rr0 = warp * (32 / width); rr0 < nr; rr0 += (kThreads / 32) * (32 / width)) {
      const int rr = rr0 + sub;
      const bool ok = rr < nr;
      float* l = s_r + (ok ? rr : 0) * K;
      float mx = -INFINITY;
      if (ok)
        for (int k = sl; k < K; k += width) mx = fmaxf(mx, l[k]);
      for (int o = width / 2; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float sum = 0.f;
      if (ok)
        for (int k = sl; k < K; k += width) sum += expf(l[k] - mx);
      for (int o = width / 2; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      const float inv = 1.f / sum;
      __syncwarp();
      if (ok)
        for (int k = sl; k < K; k += width) l[k] = expf(l[k] - mx) * inv;
    }
  }
  if (blockIdx.x == 0 && blockIdx.y == 0 && tid == 0) ep->epoch = cur + 1u;  // the next call's set
  const bool ok = wait_staged(bulk, &bar, status);
  if (__syncthreads_or(!ok || dots_status != 0)) {
    // a bounded wait ran out here or in the dot products: the tile is written
    // as NaN, so the failure shows in the output as well as in the status word
    for (int q = tid; q < nr * ncol; q += kThreads)
      eps[(int64_t)(r0 + q / ncol) * D + c0 + q % ncol] = __int_as_float(0x7fc00000);
    return;
  }
  // kOutCols / 4 column groups of 4 x kThreads / (kOutCols / 4) row groups of 4
  static_assert(kThreads / (kOutCols / 4) * 4 == kOutRows, "the threads cover the tile's rows");
  const int cg = tid % (kOutCols / 4), rg = tid / (kOutCols / 4);
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

// ---------------------------------------------------------------------------
// Tensor-core form of the dot products (tcgen05, kind::tf32). G = X M^T is a
// dense contraction over D: a CTA takes a block of 128 rows (M = 128, rows past
// the count are zero) and a chunk of kTcCols columns, and computes the
// 128 x Kp partial product (Kp = K rounded up to 16, 32, 64 or 128; padded
// means are zero) in TMEM with single-thread tcgen05.mma issue. fp32 accuracy
// from tf32 operands: every value is split as v = hi + lo with
// hi = tf32(v), lo = tf32(v - hi), and the product summed as
// hi*hi + hi*lo + lo*hi (the lo*lo term is below fp32 resolution). The rows are
// split by the CTA's threads into core-matrix order in shared memory; the
// means' split image is prepared once per handle (k_gmm_mu_image) and arrives
// by one bulk copy. Chunk sums go into the fixed-point accumulators as in
// k_gmm_dots (with a thread-block cluster of kTcCluster chunks, the cluster's
// partial sums are first added through distributed shared memory, which cuts
// the atomics on each accumulator by that factor).
__host__ inline size_t tc_smem_bytes(int K) {
  return ((size_t)2 * kTcRows * kTcCols + tc_mu_chunk_floats(K)) * sizeof(float);
}
// element (r, c) of a K-major tile with kTcCols columns, in core-matrix order:
// 8-row groups of (kTcCols / 4) core matrices of 8 rows x 4 values
__host__ __device__ inline int tc_off(int r, int c) {
  return ((r >> 3) * (kTcCols / 4) + (c >> 2)) * 32 + (r & 7) * 4 + (c & 3);
}

// The means' split image, once per handle: chunk ch, part (0 hi, 1 lo), in
// core-matrix order with Kp rows.
__global__ void __launch_bounds__(256) k_gmm_mu_image(const float* __restrict__ mu, int K, int64_t D,
                                                      float* __restrict__ img) {
  const int Kp = tc_npad(K);
  const int64_t ch = blockIdx.x;
  float* out = img + ch * tc_mu_chunk_floats(K);
  for (int q = threadIdx.x; q < Kp * kTcCols; q += 256) {
    const int k = q / kTcCols, c = q % kTcCols;
    const int64_t col = ch * kTcCols + c;
    const float v = (k < K && col < D) ? mu[(int64_t)k * D + col] : 0.f;
    const float hi = to_tf32(v);
    out[tc_off(k, c)] = hi;
    out[(size_t)Kp * kTcCols + tc_off(k, c)] = to_tf32(v - hi);
  }
}

template <int CL>
__global__ void __launch_bounds__(kTcThreads) k_gmm_dots_tc(const float* __restrict__ X,
                                                            const float* __restrict__ mu_img,
                                                            const int32_t* __restrict__ n_rows_dev, int K,
                                                            int64_t D, int max_rows,
                                                            long long* __restrict__ gacc2, GmmEpoch* ep,
                                                            int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar_mu;
  __shared__ __align__(8) uint64_t bar_mma;
  __shared__ uint32_t s_taddr;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  long long* gacc = begin_dots(gacc2, ep, (int64_t)max_rows * K);
  const int r0 = blockIdx.y * kTcRows;
  const int Kp = tc_npad(K);
  const uint32_t ncols = 2 * Kp < 32 ? 32u : (uint32_t)(2 * Kp);  // TMEM columns: a power of two >= 32
  const int64_t c0 = (int64_t)blockIdx.x * kTcCols;
  float* A_hi = reinterpret_cast<float*>(smem_raw);
  float* A_lo = A_hi + kTcRows * kTcCols;
  float* B_img = A_lo + kTcRows * kTcCols;  // hi then lo, Kp rows each
  if (tid == 0) {
    mbar_init(&bar_mu, 1);
    mbar_init(&bar_mma, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(&s_taddr, ncols);
    tc_fence_before_sync();
  }
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t taddr = s_taddr;
  if (tid == 0) {  // the means image does not depend on the predecessor
    const uint32_t bytes = (uint32_t)(tc_mu_chunk_floats(K) * sizeof(float));
    mbar_arrive_expect_tx(&bar_mu, bytes);
    bulk_g2s(B_img, mu_img + (size_t)blockIdx.x * tc_mu_chunk_floats(K), bytes, &bar_mu);
  }
  pdl_wait();  // the rows and their count come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  const int n_rows = min(*n_rows_dev, max_rows);
  const int nr = min(kTcRows, n_rows - r0);
  if (nr <= 0) {  // no rows for this block (the whole cluster alike): the means copy
                  // lands and TMEM is freed before the CTA exits
    if (!mbar_wait_bounded(&bar_mu, 0, pa::kDrainLimit) && tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    tc_fence_before_sync();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, ncols);
    return;
  }

  // rows -> (hi, lo) in core-matrix order: a warp step covers 8 rows x 16
  // columns; lanes 8q..8q+7 write one 128-byte core matrix (conflict-free).
  // All of a thread's loads are issued before the first conversion.
  {
    constexpr int kSteps = (kTcRows / 8) * (kTcCols / 16);
    constexpr int kPer = kSteps / (kTcThreads / 32);
    const int rin = lane & 7, kq = lane >> 3;
    float4 v[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int it = warp + u * (kTcThreads / 32);
      const int g = it / (kTcCols / 16), kb = (it % (kTcCols / 16)) * 4 + kq;
      const int r = g * 8 + rin, c = kb * 4;
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (r < nr && c0 + c < D) v[u] = __ldg(reinterpret_cast<const float4*>(X + (int64_t)(r0 + r) * D + c0 + c));
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int it = warp + u * (kTcThreads / 32);
      const int g = it / (kTcCols / 16), kb = (it % (kTcCols / 16)) * 4 + kq;
      const int r = g * 8 + rin, c = kb * 4;
      float4 hi, lo;
      hi.x = to_tf32(v[u].x); lo.x = to_tf32(v[u].x - hi.x);
      hi.y = to_tf32(v[u].y); lo.y = to_tf32(v[u].y - hi.y);
      hi.z = to_tf32(v[u].z); lo.z = to_tf32(v[u].z - hi.z);
      hi.w = to_tf32(v[u].w); lo.w = to_tf32(v[u].w - hi.w);
      const int off = tc_off(r, c);
      *reinterpret_cast<float4*>(A_hi + off) = hi;
      *reinterpret_cast<float4*>(A_lo + off) = lo;
    }
  }
  fence_proxy_async_smem();  // the tensor core reads what the threads wrote
  // every decision below is taken by the whole CTA (__syncthreads_and)
  bool ok = __syncthreads_and(mbar_wait_bounded(&bar_mu, 0, pa::kWaitLimit));
  if (!ok) {
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    mbar_wait_bounded(&bar_mu, 0, pa::kDrainLimit);  // the copy lands before the CTA moves on
  }
  if (tid == 0 && ok) {
    tc_fence_after_sync();
    // The means image's hi rows are directly followed by its lo rows, so one
    // N = 2 Kp product gives hi*hi in columns [0, Kp) and hi*lo in [Kp, 2 Kp);
    // lo*hi then accumulates into [0, Kp): two MMAs per k-step.
    const uint32_t idesc2 = tc_idesc_tf32(kTcRows, 2 * Kp), idesc1 = tc_idesc_tf32(kTcRows, Kp);
    const uint32_t a_hi = smem_u32(A_hi), a_lo = smem_u32(A_lo);
    const uint32_t b_hi = smem_u32(B_img);
    const uint32_t sbo = (kTcCols / 4) * 128;  // next 8-row group
    for (int ks = 0; ks < kTcCols / 8; ++ks) {
      const uint32_t ko = (uint32_t)ks * 256;  // two core matrices along K per step
      const uint64_t dah = tc_smem_desc(a_hi + ko, 128, sbo), dal = tc_smem_desc(a_lo + ko, 128, sbo);
      const uint64_t db = tc_smem_desc(b_hi + ko, 128, sbo);
      tc_mma_tf32(taddr, dah, db, idesc2, ks > 0 ? 1u : 0u);
      tc_mma_tf32(taddr, dal, db, idesc1, 1u);
    }
    tc_commit(&bar_mma);
  }
  if (ok && !__syncthreads_and(mbar_wait_bounded(&bar_mma, 0, pa::kWaitLimit))) {
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    mbar_wait_bounded(&bar_mma, 0, pa::kDrainLimit);  // let the MMAs finish before TMEM is freed
    ok = false;
  }
  tc_fence_after_sync();
  float* part = A_hi;  // [kTcRows][Kp]: this CTA's partial sums (the operands are consumed)
  if (warp < 4 && ok) {  // warp w reads TMEM lanes (rows) 32w .. 32w + 31
    const int row = warp * 32 + lane;
    for (int cb = 0; cb < Kp; cb += 16) {
      float v[16], w[16];
      tmem_ld16(taddr + ((uint32_t)(warp * 32) << 16) + (uint32_t)cb, v);
      tmem_ld16(taddr + ((uint32_t)(warp * 32) << 16) + (uint32_t)(Kp + cb), w);
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] += w[u];  // (hi*hi + lo*hi) + hi*lo
      if constexpr (CL > 1) {
#pragma unroll
        for (int u = 0; u < 16; ++u) part[row * Kp + cb + u] = v[u];
      } else if (row < nr) {
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const int k = cb + u;
          if (k < K)
            atomicAdd(reinterpret_cast<unsigned long long*>(gacc + (int64_t)(r0 + row) * K + k),
                      static_cast<unsigned long long>(__float2ll_rn(v[u] * kDotScale)));
        }
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(taddr, ncols);
  if constexpr (CL > 1) {
    // the CL column chunks of a cluster are added through distributed shared
    // memory in rank order; rank q then adds rows [q R, (q+1) R) to gacc
    cg::cluster_group cluster = cg::this_cluster();
    if (!ok)
      for (int q = tid; q < kTcRows * Kp; q += kTcThreads) part[q] = 0.f;
    cluster.sync();
    const int rank = (int)cluster.block_rank();
    constexpr int kRowsPer = kTcRows / CL;
    for (int o = tid; o < kRowsPer * K; o += kTcThreads) {
      const int rr = rank * kRowsPer + o / K, k = o % K;
      if (rr < nr) {
        float sum = 0.f;
        for (int q = 0; q < CL; ++q) sum += cluster.map_shared_rank(part, q)[rr * Kp + k];
        atomicAdd(reinterpret_cast<unsigned long long*>(gacc + (int64_t)(r0 + rr) * K + k),
                  static_cast<unsigned long long>(__float2ll_rn(sum * kDotScale)));
      }
    }
    cluster.sync();  // peers read this CTA's partial sums until here
  }
}

// ---------------------------------------------------------------------------
// Tensor-core form of the output contraction, for 16 < K <= 64 (with the
// tensor-core dot products, form 1). eps = a x - a sqrt(a) R M, and R M is a
// dense contraction over the components: rows x K times K x D.
// k_gmm_resp forms each row's responsibilities once -- the same logits and
// max-subtracted softmax as k_gmm_out -- and writes them as a split image
// (hi = tf32(R), lo = tf32(R - hi), in core-matrix order, K-major); then
// k_gmm_out_tc takes a block of 128 rows (M = 128; rows past the count are
// zero) and kOtCols columns: one bulk copy brings the responsibilities'
// image, another the means' transposed split image of its columns (built once
// per handle, k_gmm_mut_image: the hi rows of the kOtCols columns followed by
// their lo rows), one thread issues R_hi [M_hi; M_lo]^T (N = 2 kOtCols,
// columns [0, kOtCols) hi*hi and [kOtCols, 2 kOtCols) hi*lo) and R_lo M_hi^T
// (accumulated into [0, kOtCols)) per 8-component step into TMEM, and every
// thread reads its row's
// accumulators back (tcgen05.ld, one row per TMEM lane) and writes its
// columns of eps from the row values it loaded before the dependency wait.

// element (r, c) of a K-major tile with Kp columns, in core-matrix order
__host__ __device__ inline int ot_off(int r, int c, int Kp) {
  return ((r >> 3) * (Kp >> 2) + (c >> 2)) * 32 + (r & 7) * 4 + (c & 3);
}

// The means' transposed split image, once per handle: chunk ch of kOtCols
// columns, rows n (column ch * kOtCols + n; n >= kOtCols: the lo parts) x
// components.
__global__ void __launch_bounds__(256) k_gmm_mut_image(const float* __restrict__ mu, int K, int64_t D,
                                                       float* __restrict__ img) {
  const int Kp = tc_npad(K);
  const int64_t ch = blockIdx.x;
  float* out = img + ch * ot_mut_floats(K);
  for (int q = threadIdx.x; q < Kp * kOtCols; q += 256) {
    const int k = q / kOtCols, n = q % kOtCols;  // consecutive threads read consecutive columns
    const int64_t col = ch * kOtCols + n;
    const float v = (k < K && col < D) ? mu[(int64_t)k * D + col] : 0.f;
    const float hi = to_tf32(v);
    out[ot_off(n, k, Kp)] = hi;
    out[ot_off(n + kOtCols, k, Kp)] = to_tf32(v - hi);
  }
}

// The responsibilities of every row (a warp per row) as the split image of
// its 128-row block, and the row's scalars (a, a sqrt(a)) for the epilogue;
// rows past the count (up to the end of their block) are zero. Advances the
// accumulator epoch as k_gmm_out does.
__global__ void __launch_bounds__(kRespRows * 32) k_gmm_resp(const long long* __restrict__ gacc2, GmmEpoch* ep,
                                                             const float* __restrict__ coef, int T,
                                                             const int32_t* __restrict__ miss_bt,
                                                             const float* __restrict__ mnorm,
                                                             const int32_t* __restrict__ n_rows_dev, int K,
                                                             int max_rows, float* __restrict__ rimg,
                                                             float* __restrict__ rcoef) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * kRespRows + warp;
  const int Kp = tc_npad(K);
  const int n_rows = min(*n_rows_dev, max_rows);  // written two kernels back
  float sa = 0.f, q = 0.f, c = 0.f;
  if (r < n_rows) {
    const int i = miss_bt[2 * r + 1];
    sa = coef[i];
    q = coef[T + i];
    c = coef[2 * T + i];
  }
  pdl_wait();     // the dot products come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  const uint32_t cur = ep->cur;
  float* blk = rimg + (size_t)(r / kTcRows) * ot_img_floats(K);
  const int rr = r % kTcRows;
  float rv[2] = {0.f, 0.f};  // components lane and lane + 32
  if (r < n_rows) {
    const long long* g = gacc2 + (int64_t)(cur & 1u) * max_rows * K + (int64_t)r * K;
    float l[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int k = lane + 32 * u;
      if (k < K) {
        const float dot = __ll2float_rn(__ldcg(g + k)) * (1.f / kDotScale);  // exact scale
        l[u] = (2.f * sa * dot - sa * sa * mnorm[k]) * q;
      }
    }
    float mx = fmaxf(l[0], l[1]);  // the order of k_gmm_out's loop: k = lane, then lane + 32
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
#pragma unroll
    for (int u = 0; u < 2; ++u)
      if (lane + 32 * u < K) sum += expf(l[u] - mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float inv = 1.f / sum;
#pragma unroll
    for (int u = 0; u < 2; ++u)
      if (lane + 32 * u < K) rv[u] = expf(l[u] - mx) * inv;
    if (lane == 0) {
      rcoef[2 * r] = c;
      rcoef[2 * r + 1] = c * sa;
    }
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int k = lane + 32 * u;
    if (k < Kp) {
      const float hi = to_tf32(rv[u]);
      blk[ot_off(rr, k, Kp)] = hi;
      blk[ot_off(rr + kTcRows, k, Kp)] = to_tf32(rv[u] - hi);
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) ep->epoch = cur + 1u;  // the next call's set
}

__host__ inline size_t ot_smem_bytes(int K) {
  // both split images; at least 60 KB so that at most three CTAs (3 x 128 TMEM columns) share an SM
  const size_t b = (ot_img_floats(K) + ot_mut_floats(K)) * sizeof(float);
  return b < 60 * 1024 ? 60 * 1024 : b;
}

__global__ void __launch_bounds__(kOtThreads, 2) k_gmm_out_tc(const float* __restrict__ X,
                                                              const float* __restrict__ mut_img,
                                                              const float* __restrict__ rimg,
                                                              const float* __restrict__ rcoef,
                                                              const int32_t* __restrict__ n_rows_dev, int K,
                                                              int64_t D, int max_rows, float* __restrict__ eps,
                                                              int32_t* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar_b, bar_a, bar_mma;
  __shared__ uint32_t s_taddr;
  constexpr uint32_t kTmemCols = 2 * kOtCols;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Kp = tc_npad(K);
  const size_t img = ot_img_floats(K), mimg = ot_mut_floats(K);
  float* A = reinterpret_cast<float*>(smem_raw);  // responsibilities: hi rows, then lo rows
  float* B = A + img;                              // means of the columns: hi rows, then lo rows
  const int64_t c0 = (int64_t)blockIdx.x * kOtCols;
  const int r0 = blockIdx.y * kTcRows;
  if (tid == 0) {
    mbar_init(&bar_b, 1);
    mbar_init(&bar_a, 1);
    mbar_init(&bar_mma, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(&s_taddr, kTmemCols);
    tc_fence_before_sync();
  }
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t taddr = s_taddr;
  const uint32_t img_bytes = (uint32_t)(img * sizeof(float)), mimg_bytes = (uint32_t)(mimg * sizeof(float));
  if (tid == 0) {  // the means image does not change
    mbar_arrive_expect_tx(&bar_b, mimg_bytes);
    bulk_g2s(B, mut_img + (size_t)blockIdx.x * mimg, mimg_bytes, &bar_b);
  }
  // the rows and their count were written three kernels back: thread (warp,
  // lane) takes row 32 (warp % 4) + lane (its TMEM lane) and the 64 columns
  // of half warp / 4
  const int n_rows = min(*n_rows_dev, max_rows);
  const int nr = min(kTcRows, n_rows - r0);
  const int row = 32 * (warp & 3) + lane, half = warp >> 2;
  const int64_t cb0 = c0 + half * (kOtCols / 2);
  float4 xv[kOtCols / 8];
  if (row < nr) {
    const float4* xr = reinterpret_cast<const float4*>(X + (int64_t)(r0 + row) * D + cb0);
#pragma unroll
    for (int u = 0; u < kOtCols / 8; ++u) xv[u] = __ldg(xr + u);
  }
  pdl_wait();     // the responsibilities and the row scalars come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  if (nr <= 0) {  // no rows in this block: the means copy lands and TMEM is freed
    if (!mbar_wait_bounded(&bar_b, 0, pa::kDrainLimit) && tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    tc_fence_before_sync();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, kTmemCols);
    return;
  }
  if (tid == 0) {
    mbar_arrive_expect_tx(&bar_a, img_bytes);
    bulk_g2s(A, rimg + (size_t)blockIdx.y * img, img_bytes, &bar_a);
  }
  const bool dots_bad = __ldcg(status) != 0;  // a dot-product wait ran out: the sums are incomplete
  bool ok = __syncthreads_and(mbar_wait_bounded(&bar_b, 0, pa::kWaitLimit) &&
                              mbar_wait_bounded(&bar_a, 0, pa::kWaitLimit));
  if (!ok) {
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    mbar_wait_bounded(&bar_b, 0, pa::kDrainLimit);  // the copies land before the CTA moves on
    mbar_wait_bounded(&bar_a, 0, pa::kDrainLimit);
  }
  if (tid == 0 && ok) {
    tc_fence_after_sync();
    const uint32_t idesc2 = tc_idesc_tf32(kTcRows, 2 * kOtCols), idesc1 = tc_idesc_tf32(kTcRows, kOtCols);
    const uint32_t a_hi = smem_u32(A), a_lo = smem_u32(A + (size_t)kTcRows * Kp), b = smem_u32(B);
    const uint32_t sbo = (uint32_t)(Kp / 4) * 128;  // next 8-row group
    for (int ks = 0; ks < Kp / 8; ++ks) {
      const uint32_t ko = (uint32_t)ks * 256;  // two core matrices along K per step
      tc_mma_tf32(taddr, tc_smem_desc(a_hi + ko, 128, sbo), tc_smem_desc(b + ko, 128, sbo), idesc2,
                  ks > 0 ? 1u : 0u);
      tc_mma_tf32(taddr, tc_smem_desc(a_lo + ko, 128, sbo), tc_smem_desc(b + ko, 128, sbo), idesc1, 1u);
    }
    tc_commit(&bar_mma);
  }
  if (ok && !__syncthreads_and(mbar_wait_bounded(&bar_mma, 0, pa::kWaitLimit))) {
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    mbar_wait_bounded(&bar_mma, 0, pa::kDrainLimit);  // the MMAs finish before TMEM is freed
    ok = false;
  }
  tc_fence_after_sync();
  const bool live = row < nr;
  const float ac = live ? rcoef[2 * (r0 + row)] : 0.f, acs = live ? rcoef[2 * (r0 + row) + 1] : 0.f;
  float* er = eps + (int64_t)(r0 + row) * D + cb0;
  const uint32_t tl = taddr + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)(half * (kOtCols / 2));
#pragma unroll
  for (int cb = 0; cb < kOtCols / 2; cb += 16) {
    float v[16], w[16];
    if (ok) {  // uniform across the CTA: every lane of the warp takes part in the loads
      tmem_ld16(tl + (uint32_t)cb, v);
      tmem_ld16(tl + (uint32_t)(kOtCols + cb), w);
    }
    if (!live) continue;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const float4 x = xv[cb / 4 + g];
      float4 o;
      if (ok && !dots_bad) {
        o = make_float4(ac * x.x - acs * (v[4 * g] + w[4 * g]), ac * x.y - acs * (v[4 * g + 1] + w[4 * g + 1]),
                        ac * x.z - acs * (v[4 * g + 2] + w[4 * g + 2]), ac * x.w - acs * (v[4 * g + 3] + w[4 * g + 3]));
      } else {  // a bounded wait ran out here or before: the tile shows it
        const float nan = __int_as_float(0x7fc00000);
        o = make_float4(nan, nan, nan, nan);
      }
      *reinterpret_cast<float4*>(er + cb + 4 * g) = o;
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(taddr, kTmemCols);
}

// ---------------------------------------------------------------------------
// Single-kernel form for up to 16 components (form 2): a thread-block cluster
// of CL CTAs takes a block of RB rows; CTA q of the cluster owns columns
// [q * chunk, (q + 1) * chunk) with chunk = D / CL. Each CTA stages its chunk of
// the means (before the dependency wait: the means do not change) and of the
// rows, forms the rows' partial dot products x . mu_k over its columns in
// registers (4 rows x 4 components per warp, packed fp32 pairs, 16-byte
// shared loads), and the CL partials are summed through distributed shared
// memory in rank order -- the same sums in every CTA of the cluster. Every CTA then
// takes the logits and the max-subtracted softmax of the block's rows and
// writes eps = a x - a sqrt(a) R M for its columns from the tiles it already
// holds: no second kernel, no global accumulators, nothing read twice. The
// cluster's barriers are hardware barriers; its CTAs are co-scheduled.
constexpr int kClThreads = 256;
constexpr int kClMaxK = 16;

constexpr int kClCoefT = 2048;  // per-timestep scalars staged in shared memory up to this many timesteps

template <int CL, int RB>
struct ClShape {
  static int ld(int chunk) { return chunk + 4; }  // padded row stride: the two half-warps' rows on other banks
  static size_t coef_bytes(int T) { return T <= kClCoefT ? (size_t)3 * T * sizeof(float) : 0; }
  static size_t smem_bytes(int chunk, int T) {
    return (size_t)(kClMaxK + RB) * ld(chunk) * sizeof(float) + coef_bytes(T);
  }
};

__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
// The address of this CTA's shared variable at `saddr` in the shared memory of
// cluster CTA `rank` (a shared::cluster address).
__device__ __forceinline__ uint32_t cluster_map(uint32_t saddr, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
// A 4-byte store into a peer's shared memory that completes on the peer's
// mbarrier (both shared::cluster addresses): no round trip for the sender.
__device__ __forceinline__ void st_async_remote(uint32_t raddr, float v, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(raddr),
               "r"(__float_as_uint(v)), "r"(rbar)
               : "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

template <int CL, int RB>
__global__ void __launch_bounds__(kClThreads, 2) k_gmm_cluster(const float* __restrict__ X, const float* __restrict__ mu,
                                                            const float* __restrict__ coef, int T,
                                                            const int32_t* __restrict__ miss_bt,
                                                            const float* __restrict__ mnorm,
                                                            const int32_t* __restrict__ n_rows_dev, int K, int64_t D,
                                                            int chunk, int max_rows, float* __restrict__ eps,
                                                            int32_t* status) {
  static_assert(RB == 8 && kClThreads == 256 && CL % 2 == 0,
                "8 warps: 2 row quads x 2 component octets x 2 column halves of the 8 x 16 block");
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bar_m, bar_x, bar_p;
  __shared__ float s_all[CL][RB * kClMaxK];  // the partial dot products of every CTA, pushed by their owners
  __shared__ float s_half[2][RB * kClMaxK];  // this CTA's partials from each half of its columns
  __shared__ __align__(16) float s_rt[kClMaxK * RB];  // responsibilities [k][row]
  __shared__ float s_sa[RB], s_q[RB], s_c[RB], s_cs[RB];
  __shared__ int s_bad;
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = (int)cluster.block_rank();
  const int ld = chunk + 4;
  const int64_t c0 = (int64_t)rank * chunk;
  float* ms = reinterpret_cast<float*>(smem_raw);  // [kClMaxK][ld], rows >= K zero
  float* xs = ms + (size_t)kClMaxK * ld;           // [RB][ld]
  float* s_coef = xs + (size_t)RB * ld;            // [3][T] when T <= kClCoefT
  if (tid == 0) {
    mbar_init(&bar_m, 1);
    mbar_init(&bar_x, 1);
    mbar_init(&bar_p, 1);
    fence_barrier_init();
    mbar_arrive_expect_tx(&bar_m, (uint32_t)chunk * sizeof(float) * (uint32_t)K);
    // every CTA of the cluster stores its RB x kClMaxK partials here
    mbar_arrive_expect_tx(&bar_p, (uint32_t)(CL * RB * kClMaxK * sizeof(float)));
    s_bad = 0;
  }
  // ||mu_k||^2 of the component this thread takes in the softmax (constant)
  const float mn = (tid < RB * kClMaxK && (tid & (kClMaxK - 1)) < K) ? mnorm[tid & (kClMaxK - 1)] : 0.f;
  for (int q = tid; q < (kClMaxK - K) * ld; q += kClThreads) ms[(size_t)K * ld + q] = 0.f;
  const bool coef_staged = T <= kClCoefT;  // constants: staged before the dependency wait
  if (coef_staged)
    for (int q = tid; q < 3 * T; q += kClThreads) s_coef[q] = coef[q];
  __syncthreads();
  if (warp == 0)  // the means do not depend on the predecessor
    for (int k = lane; k < K; k += 32) bulk_g2s(ms + (size_t)k * ld, mu + (int64_t)k * D + c0, chunk * 4u, &bar_m);
  pdl_wait();     // the rows, their count and their timesteps come from the kernel just before
  pdl_trigger();  // the successor may now run its prologue
  const int n_rows = min(*n_rows_dev, max_rows);
  const int r0 = blockIdx.y * RB;
  const int nr = min(RB, n_rows - r0);
  if (nr <= 0) {  // the whole cluster has no rows (uniform): the means copy lands first
    if (!mbar_wait_bounded(&bar_m, 0, pa::kDrainLimit) && tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    return;
  }
  cluster_arrive_relaxed();  // this CTA runs: its peers may push into its shared memory after their wait
  // the row copies go out first: they need only the count, while each row's
  // coefficients wait for its timestep (one more trip to memory)
  if (warp == 0) {
    if (lane == 0) mbar_arrive_expect_tx(&bar_x, (uint32_t)chunk * sizeof(float) * (uint32_t)nr);
    __syncwarp();  // expect_tx precedes the copies
    for (int r = lane; r < nr; r += 32) bulk_g2s(xs + (size_t)r * ld, X + (int64_t)(r0 + r) * D + c0, chunk * 4u, &bar_x);
  }
  for (int q = tid; q < (RB - nr) * ld; q += kClThreads) xs[(size_t)nr * ld + q] = 0.f;  // rows past the count
  if (tid < nr) {
    const int i = miss_bt[2 * (r0 + tid) + 1];
    const float* cf = coef_staged ? s_coef : coef;
    s_sa[tid] = cf[i];
    s_q[tid] = cf[T + i];
    s_c[tid] = cf[2 * T + i];
    s_cs[tid] = cf[2 * T + i] * cf[i];
  }
  // bounded waits; a CTA whose copies did not land keeps to the cluster's
  // barriers (its peers wait for it there) and writes NaN
  bool ok = mbar_wait_bounded(&bar_m, 0, pa::kWaitLimit);
  ok = mbar_wait_bounded(&bar_x, 0, pa::kWaitLimit) && ok;
  if (!ok) {
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    s_bad = 1;
    mbar_wait_bounded(&bar_m, 0, pa::kDrainLimit);
    mbar_wait_bounded(&bar_x, 0, pa::kDrainLimit);
  }
  __syncthreads();
  // partial dot products: warp w takes rows 4 (w & 1) .. + 3, components
  // 8 ((w >> 1) & 1) .. + 7 and half w >> 2 of the CTA's columns; lane l the
  // columns 4 l + 128 i of that half (16-byte shared loads, conflict-free),
  // accumulated in packed fp32 pairs (two columns per FMA): each loaded row
  // vector feeds 8 components and each mean vector 4 rows
  {
    const int rq = (warp & 1) * 4, ko = ((warp >> 1) & 1) * 8, half = warp >> 2;
    const int hb = ((chunk >> 2) >> 1) << 2;  // where the second half starts: a multiple of 4 columns
    const int cb = half ? hb : 0, ce = half ? chunk : hb;
    float2 a2[4][8];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int u = 0; u < 8; ++u) a2[i][u] = make_float2(0.f, 0.f);
#pragma unroll 2
    for (int c = cb + lane * 4; c < ce; c += 128) {
      float4 xv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) xv[i] = *reinterpret_cast<const float4*>(xs + (size_t)(rq + i) * ld + c);
#pragma unroll
      for (int uh = 0; uh < 8; uh += 4) {
        float4 mv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) mv[u] = *reinterpret_cast<const float4*>(ms + (size_t)(ko + uh + u) * ld + c);
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            float2& acc = a2[i][uh + u];
            acc = __ffma2_rn(make_float2(xv[i].x, xv[i].y), make_float2(mv[u].x, mv[u].y), acc);
            acc = __ffma2_rn(make_float2(xv[i].z, xv[i].w), make_float2(mv[u].z, mv[u].w), acc);
          }
      }
    }
    // the 32 sums (v = 8 i + u) over the 32 lanes by a halving exchange: at
    // offset o each lane keeps half of its values (the upper half if lane bit
    // o is set) and adds its partner's copy of them, so after offsets 16, 8,
    // 4, 2, 1 lane l holds value l summed over all lanes: 31 shuffles
    float a[32];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int u = 0; u < 8; ++u) a[i * 8 + u] = a2[i][u].x + a2[i][u].y;
#pragma unroll
    for (int o = 16, n = 16; o > 0; o >>= 1, n >>= 1) {
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int v = 0; v < n; ++v) {
        const float send = up ? a[v] : a[v + n];
        const float keep = up ? a[v + n] : a[v];
        a[v] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
    s_half[half][(rq + (lane >> 3)) * kClMaxK + ko + (lane & 7)] = a[0];
  }
  __syncthreads();
  // this CTA's partial of (row, k) = idx: its two column halves, stored into
  // every CTA of the cluster (slot [this CTA's rank][idx] there), half of the
  // CTAs by each of the two threads that hold it, by asynchronous stores that
  // complete on the receiver's mbarrier: no round trip for the sender and no
  // cluster barrier; every CTA waits for its own barrier and then reads its
  // own shared memory only
  cluster_wait();  // every CTA of the cluster is running (its barrier initialised)
  {
    const int idx = tid & (RB * kClMaxK - 1);
    const float pv = s_half[0][idx] + s_half[1][idx];
    const uint32_t slot = smem_u32(&s_all[rank][idx]), bar = smem_u32(&bar_p);
    const int q0 = (tid >> 7) * (CL / 2);
#pragma unroll
    for (int q = 0; q < CL / 2; ++q) st_async_remote(cluster_map(slot, q0 + q), pv, cluster_map(bar, q0 + q));
  }
  if (!mbar_wait_bounded(&bar_p, 0, pa::kWaitLimit)) {  // every peer's partials have landed
    if (tid == 0) atomicCAS(status, 0, pa::kDevTimeout);
    s_bad = 1;
  }
  __syncthreads();
  // the complete dot products (the CL partials in rank order), the logits and
  // the max-subtracted softmax: thread t < 128 takes row t / 16, component
  // t % 16, so each row is a half-warp
  if (tid < RB * kClMaxK) {
    const int rr = tid >> 4, k = tid & 15;
    float dot = 0.f;
#pragma unroll
    for (int q = 0; q < CL; ++q) dot += s_all[q][tid];
    {
      const bool on = rr < nr && k < K;
      float l = -INFINITY;
      if (on) {
        const float sa = s_sa[rr];
        l = (2.f * sa * dot - sa * sa * mn) * s_q[rr];
      }
      float mx = l;
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float ex = on ? expf(l - mx) : 0.f;
      float sum = ex;
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      s_rt[k * RB + rr] = ex / sum;  // zero for k >= K
    }
  }
  __syncthreads();
  // eps = a x - a sqrt(a) sum_k R_k mu_k over this CTA's columns, four per thread
  const bool bad = s_bad != 0;
  for (int cq = tid * 4; cq < chunk; cq += kClThreads * 4) {
    float2 acc[RB][2];  // columns cq, cq+1 and cq+2, cq+3 of each row, packed fp32 pairs
#pragma unroll
    for (int r = 0; r < RB; ++r) acc[r][0] = acc[r][1] = make_float2(0.f, 0.f);
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
      const float4 m = *reinterpret_cast<const float4*>(ms + (size_t)k * ld + cq);
      const float2 ml = make_float2(m.x, m.y), mh = make_float2(m.z, m.w);
#pragma unroll
      for (int r = 0; r < RB; r += 4) {
        const float4 v = *reinterpret_cast<const float4*>(s_rt + k * RB + r);  // responsibilities of 4 rows
        const float w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 w2 = make_float2(w4[q], w4[q]);
          acc[r + q][0] = __ffma2_rn(w2, ml, acc[r + q][0]);
          acc[r + q][1] = __ffma2_rn(w2, mh, acc[r + q][1]);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      if (r >= nr) break;
      const float4 x = *reinterpret_cast<const float4*>(xs + (size_t)r * ld + cq);
      const float ac = s_c[r], acs = s_cs[r];
      float4 o = make_float4(ac * x.x - acs * acc[r][0].x, ac * x.y - acs * acc[r][0].y, ac * x.z - acs * acc[r][1].x,
                             ac * x.w - acs * acc[r][1].y);
      if (bad) o = make_float4(__int_as_float(0x7fc00000), __int_as_float(0x7fc00000), __int_as_float(0x7fc00000),
                               __int_as_float(0x7fc00000));
      *reinterpret_cast<float4*>(eps + (int64_t)(r0 + r) * D + c0 + cq) = o;
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
  bool tc_ok;   // the tensor-core dot products fit this device and these sizes
  bool use_tc;  // ... and are selected
  bool cl_ok;   // the single-kernel cluster form fits these sizes and this device
  bool ot_ok;   // form 1 also takes the output contraction on the tensor cores (16 < K <= 64)
  int form;     // 0 CUDA-core dots + output kernel, 1 tensor-core dots + output kernel, 2 cluster form
};

namespace {
constexpr int kClSize = 16;   // CTAs per cluster (non-portable size, opted into)
constexpr int kClRows = 8;    // rows per cluster
}  // namespace

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
  if (e == cudaSuccess) e = cudaMemsetAsync(g->ws + L.epoch, 0, sizeof(GmmEpoch), g->st);
  if (e == cudaSuccess) e = cudaMemsetAsync(g->ws + L.gacc, 0, (size_t)2 * max_rows * K * sizeof(long long), g->st);
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
  // tensor-core dot products: sm_100-family tensor cores, 16-byte rows, and
  // shared memory for the split rows and the means image of one chunk
  int dev = 0, major = 0, optin = 0;
  g->tc_ok = false;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e == cudaSuccess && major == 10 && D % 4 == 0 && (reinterpret_cast<uintptr_t>(means_dev) & 15) == 0 &&
      tc_smem_bytes(K) + 2048 <= (size_t)optin) {
    e = cudaFuncSetAttribute(k_gmm_dots_tc<kTcCluster>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)tc_smem_bytes(K));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k_gmm_dots_tc<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc_smem_bytes(K));
    if (e == cudaSuccess) {
      k_gmm_mu_image<<<L.tc_chunks, 256, 0, g->st>>>(means_dev, K, D, reinterpret_cast<float*>(g->ws + L.mu_img));
      g->launches++;
      e = cudaGetLastError();
      g->tc_ok = e == cudaSuccess;
    }
  }
  // The tensor-core output contraction beside them: 16 < K <= 64 (padded
  // components fit one image of 128 rows x 64), whole kOtCols-column chunks.
  g->ot_ok = false;
  if (e == cudaSuccess && g->tc_ok && K > kTcMinK && tc_npad(K) <= kOtMaxKp && D % kOtCols == 0 &&
      ot_smem_bytes(K) + 4096 <= (size_t)optin) {
    e = cudaFuncSetAttribute(k_gmm_out_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ot_smem_bytes(K));
    if (e == cudaSuccess) {
      k_gmm_mut_image<<<(unsigned)(D / kOtCols), 256, 0, g->st>>>(means_dev, K, D,
                                                                    reinterpret_cast<float*>(g->ws + L.mut_img));
      g->launches++;
      e = cudaGetLastError();
      g->ot_ok = e == cudaSuccess;
    }
  }
  // Default: the tensor cores for K > 16. At K <= 16 the contraction is under
  // a microsecond of CUDA-core FMA work per call and the CUDA-core kernel's
  // shorter per-CTA chain wins (measured at 4x64x64: 30.1 vs 33.1 us per
  // Picard iteration); at K = 64 the tensor cores win (151.9 vs 170.4 us at
  // 4x128x128).
  g->use_tc = g->tc_ok && K > kTcMinK;
  // The single-kernel cluster form for K <= 16 when D splits into kClSize
  // 16-byte-aligned column chunks whose tiles fit in shared memory and a
  // cluster of kClSize CTAs can be resident; then the default.
  g->cl_ok = false;
  g->form = g->use_tc ? 1 : 0;
  if (e == cudaSuccess && major == 10 && K <= kClMaxK && D % (4 * kClSize) == 0 &&
      (reinterpret_cast<uintptr_t>(means_dev) & 15) == 0) {
    const int chunk = (int)(D / kClSize);
    const size_t smem = ClShape<kClSize, kClRows>::smem_bytes(chunk, T);
    auto kern = k_gmm_cluster<kClSize, kClRows>;
    cudaFuncAttributes fa = {};
    e = cudaFuncGetAttributes(&fa, kern);
    if (e == cudaSuccess && smem + fa.sharedSizeBytes <= (size_t)optin) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(kClSize, 1, 1);
        cfg.blockDim = dim3(kClThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = kClSize;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int nclusters = 0;
        e = cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg);
        g->cl_ok = e == cudaSuccess && nclusters > 0;
        if (e != cudaSuccess) {
          (void)cudaGetLastError();  // the size is not supported here: keep the two-kernel forms
          e = cudaSuccess;
        }
      }
    }
    if (g->cl_ok) g->form = 2;
  }
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
  const float* coef = reinterpret_cast<const float*>(g->ws + L.coef);
  const float* mnorm = reinterpret_cast<const float*>(g->ws + L.mnorm);
  long long* gacc2 = reinterpret_cast<long long*>(g->ws + L.gacc);
  GmmEpoch* ep = reinterpret_cast<GmmEpoch*>(g->ws + L.epoch);
  int32_t* status = reinterpret_cast<int32_t*>(g->ws + L.status);
  // bulk copies need 16-byte aligned rows: D % 4 == 0 and aligned base pointers
  const bool bulk = g->D % 4 == 0 && ((reinterpret_cast<uintptr_t>(batch_x_dev) |
                                       reinterpret_cast<uintptr_t>(g->means)) & 15) == 0;
  const bool vec_out = g->D % 4 == 0 && (reinterpret_cast<uintptr_t>(batch_eps_dev) & 15) == 0;
  const size_t out_smem = (size_t)(g->K + kOutRows) * kOutCols * sizeof(float);
  const dim3 tc_grid(L.tc_chunks, (g->max_rows + kTcRows - 1) / kTcRows);
  cudaError_t e;
  if (g->form == 2 && bulk && vec_out) {  // one kernel: cluster of kClSize CTAs per kClRows rows
    const int chunk = (int)(g->D / kClSize);
    e = pa::launch_ex(k_gmm_cluster<kClSize, kClRows>, dim3(kClSize, (g->max_rows + kClRows - 1) / kClRows),
                      dim3(kClThreads), ClShape<kClSize, kClRows>::smem_bytes(chunk, g->T), g->st, kClSize,
                      batch_x_dev, g->means, coef, g->T, miss_bt_dev, mnorm, n_rows_dev, g->K, g->D, chunk,
                      g->max_rows, batch_eps_dev, status);
    g->launches += 1;
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
      pa::set_error(std::string("pa_gmm_eps: ") + cudaGetErrorString(e));
      return PA_ERR_CUDA;
    }
    return PA_OK;
  }
  if (g->use_tc && bulk && L.tc_chunks >= kTcClusterMinChunks)
    e = pa::launch_ex(k_gmm_dots_tc<kTcCluster>, tc_grid, dim3(kTcThreads), tc_smem_bytes(g->K), g->st,
                      kTcCluster, batch_x_dev, (const float*)(g->ws + L.mu_img), n_rows_dev, g->K, g->D,
                      g->max_rows, gacc2, ep, status);
  else if (g->use_tc && bulk)
    e = pa::launch_ex(k_gmm_dots_tc<1>, tc_grid, dim3(kTcThreads), tc_smem_bytes(g->K), g->st, 0, batch_x_dev,
                      (const float*)(g->ws + L.mu_img), n_rows_dev, g->K, g->D, g->max_rows, gacc2, ep, status);
  else
    e = pa::launch_ex(k_gmm_dots, dim3(L.nchunk, (g->max_rows + kDotRows - 1) / kDotRows), dim3(kThreads),
                      dots_smem_bytes(g->K, L.chunk), g->st, 0, batch_x_dev, g->means, n_rows_dev, g->K, g->D,
                      L.chunk, L.nchunk, g->max_rows, bulk, gacc2, ep, status);
  if (g->use_tc && g->ot_ok && bulk && vec_out) {  // responsibilities, then the contraction on the tensor cores
    const int blocks = (g->max_rows + kTcRows - 1) / kTcRows;
    float* rimg = reinterpret_cast<float*>(g->ws + L.r_img);
    float* rcoef = reinterpret_cast<float*>(g->ws + L.rcoef);
    if (e == cudaSuccess)
      e = pa::launch_ex(k_gmm_resp, dim3(blocks * (kTcRows / kRespRows)), dim3(kRespRows * 32), 0, g->st, 0,
                        (const long long*)gacc2, ep, coef, g->T, miss_bt_dev, mnorm, n_rows_dev, g->K, g->max_rows,
                        rimg, rcoef);
    if (e == cudaSuccess)
      e = pa::launch_ex(k_gmm_out_tc, dim3((unsigned)(g->D / kOtCols), blocks), dim3(kOtThreads),
                        ot_smem_bytes(g->K), g->st, 0, batch_x_dev, (const float*)(g->ws + L.mut_img),
                        (const float*)rimg, (const float*)rcoef, n_rows_dev, g->K, g->D, g->max_rows,
                        batch_eps_dev, status);
    g->launches += 3;
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
      pa::set_error(std::string("pa_gmm_eps: ") + cudaGetErrorString(e));
      return PA_ERR_CUDA;
    }
    return PA_OK;
  }
  if (e == cudaSuccess)
    e = pa::launch_ex(k_gmm_out,
                      dim3((unsigned)((g->D + kOutCols - 1) / kOutCols), (g->max_rows + kOutRows - 1) / kOutRows),
                      dim3(kThreads), out_smem, g->st, 0, batch_x_dev, g->means, (const long long*)gacc2, ep, coef,
                      g->T, miss_bt_dev, mnorm, n_rows_dev, g->K, g->D, g->max_rows, bulk, vec_out, batch_eps_dev,
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

extern "C" pa_status pa_gmm_set_form(pa_gmm* g, int form) {
  if (!g) { pa::set_error("pa_gmm_set_form: NULL handle"); return PA_ERR_ARG; }
  if (form < 0 || form > 2) { pa::set_error("pa_gmm_set_form: form must be 0, 1 or 2"); return PA_ERR_ARG; }
  if (form == 1 && !g->tc_ok) {
    pa::set_error("pa_gmm_set_form: tensor-core dot products need an sm_100-family GPU, D % 4 == 0, "
                  "16-byte aligned means and enough shared memory");
    return PA_ERR_ARG;
  }
  if (form == 2 && !g->cl_ok) {
    pa::set_error("pa_gmm_set_form: the cluster form needs K <= 16, D a multiple of 64, an sm_100-family GPU, "
                  "16-byte aligned means and enough shared memory");
    return PA_ERR_ARG;
  }
  g->use_tc = form == 1;
  g->form = form;
  return PA_OK;
}

extern "C" int pa_gmm_form(const pa_gmm* g) { return g ? g->form : -1; }

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
// its device address comes from cudaGetSymbolAddress, looked up on each call
// with the caller's device current.
static __device__ __align__(256) unsigned char g_gmm_scratch[kNoAllocScratchBytes];

namespace {

// Per-timestep scalars of the allocation-free path, formed on the device in
// fp64 from alpha-bar values that travel in the launch's own parameters (no
// host buffer, no host-to-device copy); the launch with i0 = 0 also stores the
// row count. Same expressions as pa_gmm_create's host loop, with no fused
// multiply-add, so the values round to fp32 alike.
constexpr int kNoAllocCoefChunk = 3000;  // alphas per launch: 24 KB of kernel parameters
struct AlphaChunk {
  int i0, n;
  double std;
  double a[kNoAllocCoefChunk];
};

__global__ void __launch_bounds__(256) k_noalloc_coef(AlphaChunk c, int T, int n_rows, float* __restrict__ coef,
                                                      int32_t* __restrict__ nrows_dev) {
  for (int u = threadIdx.x; u < c.n; u += blockDim.x) {
    const double a = c.a[u];
    const double v = __dadd_rn(__dmul_rn(__dmul_rn(a, c.std), c.std), 1.0 - a);
    coef[c.i0 + u] = (float)sqrt(a);
    coef[T + c.i0 + u] = (float)(1.0 / (2.0 * v));
    coef[2 * T + c.i0 + u] = (float)(sqrt(1.0 - a) / v);
  }
  if (c.i0 == 0 && threadIdx.x == 0) *nrows_dev = n_rows;
}

// Device address of g_gmm_scratch for the current device, looked up on every
// call (cheap, not a stream operation; a cached address could go stale if the
// device's context were torn down and the module reloaded elsewhere).
pa_status scratch_for_current_device(unsigned char** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_gmm_scratch);
  if (e != cudaSuccess || !p) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  *out = static_cast<unsigned char*>(p);
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
  // scratch layout: coef[3T] | mnorm[K] | gacc[2][n_rows][K] (int64) | epoch |
  //                 n_rows | status   (256-byte aligned pieces)
  const int chunk = dots_chunk(K, D);
  const int nchunk = (int)((D + chunk - 1) / chunk);
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  const size_t o_coef = take((size_t)3 * T * sizeof(float));
  const size_t o_mnorm = take((size_t)K * sizeof(float));
  const size_t o_gacc = take((size_t)2 * n_rows * K * sizeof(long long));
  const size_t o_epoch = take(sizeof(GmmEpoch));
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
  long long* gacc2 = reinterpret_cast<long long*>(scratch + o_gacc);
  GmmEpoch* ep = reinterpret_cast<GmmEpoch*>(scratch + o_epoch);
  int32_t* nrows_dev = reinterpret_cast<int32_t*>(scratch + o_n);
  int32_t* status = reinterpret_cast<int32_t*>(scratch + o_status);

  // Per-timestep scalars and the row count: small launches whose parameters
  // carry the alphas (asynchronous, nothing on the host to outlive the call).
  cudaError_t e = cudaSuccess;
  {
    AlphaChunk c;
    c.std = std;
    for (int i0 = 0; i0 < T && e == cudaSuccess; i0 += kNoAllocCoefChunk) {
      c.i0 = i0;
      c.n = (T - i0) < kNoAllocCoefChunk ? (T - i0) : kNoAllocCoefChunk;
      for (int u = 0; u < c.n; ++u) c.a[u] = alphas_cumprod[i0 + u];
      k_noalloc_coef<<<1, 256, 0, st>>>(c, T, n_rows, coef, nrows_dev);
      e = cudaGetLastError();
    }
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(status, 0, sizeof(int32_t), st);  // starts at zero every call
  if (e == cudaSuccess)  // the epoch and both accumulator sets start at zero every call too
    e = cudaMemsetAsync(ep, 0, sizeof(GmmEpoch), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(gacc2, 0, (size_t)2 * n_rows * K * sizeof(long long), st);
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
      batch_x_dev, means_dev, nrows_dev, K, D, chunk, nchunk, n_rows, bulk, gacc2, ep, status);
  k_gmm_out<<<dim3((unsigned)((D + kOutCols - 1) / kOutCols), (n_rows + kOutRows - 1) / kOutRows), kThreads,
              out_smem, st>>>(batch_x_dev, means_dev, gacc2, ep, coef, T, miss_bt_dev, mnorm, nrows_dev, K, D,
                              n_rows, bulk, vec_out, batch_eps_dev, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    pa::set_error(std::string("pa_gmm_eps_noalloc: ") + cudaGetErrorString(e));
    return PA_ERR_CUDA;
  }
  return PA_OK;
}
