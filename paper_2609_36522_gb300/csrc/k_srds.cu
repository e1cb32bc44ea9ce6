// Parareal (SRDS-style) DDIM sampling with ParaAnya's output cache on every
// network evaluation (Sec. 2.1: Parareal-based samplers; Sec. 2.2: the cache
// applies to the coarse and fine evaluations, the Parareal update unchanged).
//
// Blocks of s = ceil(sqrt(T)) sampling steps, N = ceil(T / s) blocks; block n
// covers indices [n s, e_n), e_n = min((n + 1) s, T). Fine solver F_n: the
// DDIM steps of block n. Coarse solver G_n: one DDIM jump from alpha-bar(n s)
// to alpha-bar(e_n) with eps at (u, n s).
//   iteration 0   U_0 = x_init, U_{n+1} = G_n(U_n)                 (coarse stages)
//   iteration k   F_n(U_n^{k-1}) for all n                         (s fine stages)
//                 U_{n+1}^k = G_n(U_n^k) + F_n(U_n^{k-1}) - G_n(U_n^{k-1})  (N coarse stages)
//                 err = max_n (1/D) ||U_n^k - U_n^{k-1}||^2 <= tol => converged (Eq. 2 on the
//                 block boundaries); a converged trajectory is frozen; Parareal is exact at k = N.
// Every evaluation stage: cache distance of each live row against its index's
// entry (Eq. 4), hit iff entry && delta < tau_cache (Eq. 5), misses compacted
// trajectory-major and gathered for the denoiser (k_srds_plan_gather); then
// the step (k_srds_apply) takes eps from the batch (miss, updating the entry,
// Eq. 7) or from the cache (hit, Eq. 6). The distances of a stage's rows are
// summed by the kernel that produced those rows (the previous stage's
// k_srds_apply, or k_srds_err for the first fine stage of an iteration) into
// fp64 accumulators, one set per stage parity, while the new values are in
// registers.
//
// Data (rows of D): U, Up [B][N+1][D] fp64 boundaries now and before this
// iteration; Y [B][N][D] fp64 fine states (F after the sweep); G [B][N][D]
// fp64 coarse results; Xh [B][T][D] fp64 and Eh [B][T][D] fp32 the cache;
// batch_x [B*N][D] fp32. The trajectory states are fp64: a sample passes
// through about T steps plus N corrections, one rounding each, and fp32
// states drift by ~1e-5 of the latent scale over T = 100 (measured); the
// denoiser still sees fp32 rows and returns fp32 eps.
#include <cmath>
#include <string>
#include <vector>

#include "../../include/paraanya.h"
#include "pa_internal.h"

namespace pa {
void set_error(const std::string& msg);  // pa_solver.cpp
}

namespace {

constexpr int kSThreads = 256;
constexpr int kSStrip = 1024;        // columns per error CTA
constexpr int kSMaxRows = 2048;      // B * N

enum StageKind : int32_t { kCoarseInit = 0, kFine = 1, kCoarse = 2 };

struct SCtl {
  int32_t n_miss, n_active, iter, status;
  long long nfe, hits;
};

struct SDev {
  int T, B, N, s, nstrip;
  int64_t D;
  double* U;
  double* Up;
  double* Y;
  double* G;
  double* Xh;
  float* Eh;
  int32_t* has;      // [B][T]
  float* batch_x;    // [B*N][D]
  int32_t* miss_bt;  // [B*N][2]
  int32_t* rank;     // [B*N]: miss rank, -1 hit, -2 not live
  double* part;      // [B*N][nstrip] Eq. 2 partials of the block boundaries
  double* sacc;      // [2][B*N] x kAccStride: Eq. 4 sums of the next stage's rows, set = stage number mod 2
  int32_t* active;   // [B]
  int32_t* iters;    // [B]
  float* err_log;    // [N][B]
  const double* cm1;  // [T] single steps: c_i - 1
  const double* e1;   // [T]
  const double* cjm1; // [N] block jumps: c - 1
  const double* ej;   // [N]
  SCtl* ctl;
  double tol, cache_thresh;
};

struct Stage {
  int32_t kind, j, n, iter;  // fine: j; coarse: n
};

__device__ __forceinline__ int stage_rows(const SDev& d, const Stage& st) {
  return st.kind == kFine ? d.B * d.N : d.B;
}

// Row r of a stage: trajectory b, sampling index i, its input row; false if
// the row takes no part (frozen trajectory, or past the end of a short block).
__device__ __forceinline__ bool row_info(const SDev& d, const Stage& st, int r, int& b, int& n, int& i,
                                         double*& x) {
  if (st.kind == kFine) {
    b = r / d.N;
    n = r % d.N;
    i = n * d.s + st.j;
    const int end = min((n + 1) * d.s, d.T);
    x = d.Y + ((int64_t)b * d.N + n) * d.D;
    return d.active[b] && i < end;
  }
  b = r;
  n = st.n;
  i = n * d.s;
  x = d.U + ((int64_t)b * (d.N + 1) + n) * d.D;
  return d.active[b] != 0;
}

// A CTA's partial of an Eq. 4 sum (non-negative) as it enters the fp64
// accumulator that CTAs add into in arrival order: rounded up to a multiple of
// 2^-32, so every partial sum below 2^21 is exactly representable (2^21 / 2^-32
// = 2^53) and the accumulated sum is the same whatever the order; above 2^21
// the mean distance is at least 2^21 / D, far beyond any tau_cache.
__device__ __forceinline__ double quantize_sum(double v) {
  return ceil(v * 4294967296.0) * (1.0 / 4294967296.0);
}

__device__ __forceinline__ double block_sum(double v, double* s_w) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) s_w[warp] = v;
  __syncthreads();
  double t = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kSThreads / 32; ++w) t += s_w[w];  // fixed order
  return t;
}

// One stage's plan and batch, one launch. Every CTA takes the stage's
// decision over its rows (at most 2048) with all of its warps, one 32-row chunk
// per warp at a time: a live row with an entry hits iff its distance sum / D <
// tau_cache (Eq. 5); misses get ranks in row order (trajectory-major) from the
// chunks' ballots and one scan of their miss counts. The
// same inputs give the same plan in every CTA; CTA (0, 0) publishes it (ranks,
// miss list, counters) and clears the distance set the coming apply adds into.
// Then every CTA narrows its column range of the batch row whose rank is its
// blockIdx.y, if that row holds a miss.
__global__ void __launch_bounds__(kSThreads) k_srds_plan_gather(SDev d, Stage st, int set) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  constexpr int kChunks = kSMaxRows / 32, kWarps = kSThreads / 32;
  __shared__ int s_total, s_row;
  __shared__ unsigned s_mm[kChunks], s_hm[kChunks];  // miss / hit bits of each 32-row chunk
  __shared__ int s_base[kChunks];                     // misses before each chunk
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool publish = blockIdx.x == 0 && blockIdx.y == 0;
  const int rows = stage_rows(d, st);
  const int R = d.B * d.N;
  const int nchunk = (rows + 31) / 32;
  // 1. hit/miss of every row, one warp per chunk; a row's trajectory flag, entry
  //    flag and distance sum are read together
  for (int c = warp; c < nchunk; c += kWarps) {
    const int r = c * 32 + lane;
    bool live = false, hit = false;
    if (r < rows) {
      int b, n, i;
      double* x;
      live = row_info(d, st, r, b, n, i, x);
      const bool has = i < d.T && d.has[(int64_t)b * d.T + i];
      const double sv = d.sacc[((size_t)set * R + r) * pa::kAccStride];
      hit = live && has && sv / (double)d.D < d.cache_thresh;
    }
    const unsigned mm = __ballot_sync(0xffffffffu, live && !hit), hm = __ballot_sync(0xffffffffu, hit);
    if (lane == 0) {
      s_mm[c] = mm;
      s_hm[c] = hm;
    }
  }
  __syncthreads();
  // 2. each chunk's first rank (exclusive scan of the chunk miss counts, two
  //    chunks per lane), the totals, the counters
  if (warp == 0) {
    const int c0 = 2 * lane, c1 = 2 * lane + 1;
    const int n0 = c0 < nchunk ? __popc(s_mm[c0]) : 0, n1 = c1 < nchunk ? __popc(s_mm[c1]) : 0;
    int incl = n0 + n1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int excl = incl - (n0 + n1);
    if (c0 < nchunk) s_base[c0] = excl;
    if (c1 < nchunk) s_base[c1] = excl + n0;
    const int hits = __reduce_add_sync(0xffffffffu, (c0 < nchunk ? __popc(s_hm[c0]) : 0) +
                                                        (c1 < nchunk ? __popc(s_hm[c1]) : 0));
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    if (lane == 0) {
      s_total = total;
      s_row = -1;
      if (publish) {
        d.ctl->n_miss = total;
        d.ctl->nfe += total;
        d.ctl->hits += hits;
      }
    }
    if (publish)
      for (int q = lane; q < R; q += 32) d.sacc[((size_t)(set ^ 1) * R + q) * pa::kAccStride] = 0.0;
  }
  __syncthreads();
  // 3. ranks in row order; the row of this CTA's rank
  for (int c = warp; c < nchunk; c += kWarps) {
    const int r = c * 32 + lane;
    if (r >= rows) continue;
    const unsigned mm = s_mm[c];
    const bool miss = (mm >> lane) & 1u;
    const int rank = s_base[c] + __popc(mm & ((1u << lane) - 1u));
    if (miss && rank == (int)blockIdx.y) s_row = r;  // one row holds each rank
    if (publish) {
      d.rank[r] = miss ? rank : (((s_hm[c] >> lane) & 1u) ? -1 : -2);
      if (miss) {
        int b, n, i;
        double* x;
        row_info(d, st, r, b, n, i, x);
        d.miss_bt[2 * rank] = b;
        d.miss_bt[2 * rank + 1] = i;
      }
    }
  }
  __syncthreads();
  const int m = blockIdx.y, r = s_row;
  if (m >= s_total || r < 0) return;
  int b, n, i;
  double* x;
  row_info(d, st, r, b, n, i, x);
  float* to = d.batch_x + (int64_t)m * d.D;
  for (int64_t c = (int64_t)blockIdx.x * kSThreads + tid; c < d.D; c += (int64_t)gridDim.x * kSThreads)
    to[c] = (float)x[c];
}

// The step of every live row: eps from the batch (miss: the entry becomes
// (x, eps), Eq. 7) or the cache (hit, Eq. 6); then a fine step
// Y <- Y + (c_i - 1) Y + e_i eps, or a coarse jump g = x + (c - 1) x + e eps
// with U_{n+1} = g (iteration 0) or g + F_n - G_n (later), G_n <- g.
// The next stage's rows that this stage produced also get their Eq. 4
// distance here, added into set `nset`: a fine step feeds the next fine step
// of its block; the last fine step of block 0 feeds the first coarse block,
// whose input U_0 does not change; a coarse block feeds the next one.
__global__ void __launch_bounds__(kSThreads) k_srds_apply(SDev d, Stage st, const float* __restrict__ beps,
                                                         int nset) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  __shared__ double s_w[kSThreads / 32];
  const int r = blockIdx.y;
  int b, n, i;
  double* x;
  if (!row_info(d, st, r, b, n, i, x)) return;
  const int rk = d.rank[r];
  const int64_t e_off = ((int64_t)b * d.T + i) * d.D;
  const float* eps = rk >= 0 ? beps + (int64_t)rk * d.D : d.Eh + e_off;
  if (rk >= 0 && blockIdx.x == 0 && threadIdx.x == 0) d.has[(int64_t)b * d.T + i] = 1;
  const double cm1 = st.kind == kFine ? d.cm1[i] : d.cjm1[n];
  const double ec = st.kind == kFine ? d.e1[i] : d.ej[n];
  double* Un1 = d.U + ((int64_t)b * (d.N + 1) + n + 1) * d.D;
  double* Gn = d.G + ((int64_t)b * d.N + n) * d.D;
  const double* Fn = d.Y + ((int64_t)b * d.N + n) * d.D;
  // the next stage's row fed by this one, if any: its row index, timestep and input
  int nrow = -1, i1 = 0;
  const double* nx0 = nullptr;  // the next input when it is not the value computed here
  if (st.kind == kFine) {
    if (st.j + 1 < d.s) {
      const int end = min((n + 1) * d.s, d.T);
      if (i + 1 < end) { nrow = r; i1 = i + 1; }
    } else if (n == 0) {
      nrow = b; i1 = 0; nx0 = d.U + (int64_t)b * (d.N + 1) * d.D;
    }
  } else if (n + 1 < d.N) {
    nrow = b; i1 = (n + 1) * d.s;
  }
  // an entry for timestep i1 exists if an earlier stage made it, or this row
  // (same timestep: one step per block) is a miss making it now
  const bool nhas = nrow >= 0 && ((i1 == i && rk >= 0) || d.has[(int64_t)b * d.T + i1] != 0);
  const double* xh1 = d.Xh + ((int64_t)b * d.T + i1) * d.D;
  double dist = 0.0;
  for (int64_t c = (int64_t)blockIdx.x * kSThreads + threadIdx.x; c < d.D; c += (int64_t)gridDim.x * kSThreads) {
    const double xv = x[c];
    const float ev = eps[c];
    if (rk >= 0) {
      d.Xh[e_off + c] = xv;
      d.Eh[e_off + c] = ev;
    }
    const double g = xv + fma(cm1, xv, ec * (double)ev);
    double nv;
    if (st.kind == kFine) {
      x[c] = g;
      nv = g;
    } else if (st.kind == kCoarseInit) {
      Gn[c] = g;
      Un1[c] = g;
      nv = g;
    } else {
      nv = g + (Fn[c] - Gn[c]);
      Un1[c] = nv;
      Gn[c] = g;
    }
    if (nhas) dist += fabs((nx0 ? nx0[c] : nv) - xh1[c]);
  }
  if (nhas) {
    const double t = block_sum(dist, s_w);
    if (threadIdx.x == 0) atomicAdd(d.sacc + ((size_t)nset * d.B * d.N + nrow) * pa::kAccStride, quantize_sum(t));
  }
}

// End of an iteration: partial sums of (U_{n+1} - Up_{n+1})^2 per strip
// (iterations >= 1), then Up <- U and Y_n <- U_n for the next fine sweep.
// The next fine sweep starts from Y_n = U_n: the Eq. 4 distance of its first
// stage's rows (timestep n s) is added into set `nset` here.
__global__ void __launch_bounds__(kSThreads) k_srds_err(SDev d, int iter, int nset) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  __shared__ double s_w[kSThreads / 32];
  const int r = blockIdx.y, b = r / d.N, n = r % d.N;
  if (!d.active[b]) return;
  const int64_t c0 = (int64_t)blockIdx.x * kSStrip;
  const int64_t c1 = (c0 + kSStrip < d.D) ? c0 + kSStrip : d.D;
  double* u1 = d.U + ((int64_t)b * (d.N + 1) + n + 1) * d.D;
  double* p1 = d.Up + ((int64_t)b * (d.N + 1) + n + 1) * d.D;
  const double* u0 = d.U + ((int64_t)b * (d.N + 1) + n) * d.D;
  double* y = d.Y + ((int64_t)b * d.N + n) * d.D;
  const bool nhas = d.has[(int64_t)b * d.T + n * d.s] != 0;
  const double* xh = d.Xh + ((int64_t)b * d.T + n * d.s) * d.D;
  double acc = 0.0, dist = 0.0;
  for (int64_t c = c0 + threadIdx.x; c < c1; c += kSThreads) {
    const double df = u1[c] - p1[c];
    acc = fma(df, df, acc);
    p1[c] = u1[c];
    const double v = u0[c];
    y[c] = v;
    if (nhas) dist += fabs(v - xh[c]);
  }
  const double t = block_sum(acc, s_w);
  if (threadIdx.x == 0) d.part[(int64_t)r * d.nstrip + blockIdx.x] = iter > 0 ? t : 0.0;
  if (nhas) {
    __syncthreads();  // s_w is reused
    const double t2 = block_sum(dist, s_w);
    if (threadIdx.x == 0) atomicAdd(d.sacc + ((size_t)nset * d.B * d.N + r) * pa::kAccStride, quantize_sum(t2));
  }
}

// Convergence of every trajectory after iteration `iter` (one CTA).
__global__ void __launch_bounds__(kSThreads) k_srds_finish(SDev d, int iter, cudaGraphConditionalHandle next,
                                                           int has_next) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  __shared__ int s_act;
  if (threadIdx.x == 0) s_act = 0;
  __syncthreads();
  for (int b = threadIdx.x; b < d.B; b += kSThreads) {
    if (!d.active[b]) continue;
    if (iter > 0) {
      double err = 0.0;
      for (int n = 0; n < d.N; ++n) {
        double sum = 0.0;
        const int r = b * d.N + n;
        for (int k = 0; k < d.nstrip; ++k) sum += d.part[(int64_t)r * d.nstrip + k];
        err = fmax(err, sum / (double)d.D);
      }
      d.iters[b] = iter;
      d.err_log[(int64_t)(iter - 1) * d.B + b] = (float)err;
      if (err <= d.tol || iter >= d.N) {
        d.active[b] = 0;
        continue;
      }
    }
    atomicAdd(&s_act, 1);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    d.ctl->n_active = s_act;
    d.ctl->iter = iter;
    // inside a captured generation: the next iteration's IF node runs only
    // while a trajectory is still active
    if (has_next) cudaGraphSetConditional(next, s_act > 0 ? 1u : 0u);
  }
}

// fp32 rows (pitch D) -> fp64 rows of the boundary array (pitch (N+1) D), and back.
__global__ void k_srds_load(SDev d, const float* __restrict__ src, int slot) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  const int b = blockIdx.y;
  double* to = d.U + ((int64_t)b * (d.N + 1) + slot) * d.D;
  double* to2 = d.Up + ((int64_t)b * (d.N + 1) + slot) * d.D;
  for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < d.D; c += (int64_t)gridDim.x * blockDim.x) {
    to[c] = (double)src[(int64_t)b * d.D + c];
    to2[c] = to[c];
  }
}

__global__ void k_srds_store(SDev d, float* __restrict__ dst, int slot) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  const int b = blockIdx.y;
  const double* from = d.U + ((int64_t)b * (d.N + 1) + slot) * d.D;
  for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < d.D; c += (int64_t)gridDim.x * blockDim.x)
    dst[(int64_t)b * d.D + c] = (float)from[c];
}

__global__ void k_srds_reset(SDev d) {
  pa::pdl_wait();     // everything read here comes from earlier kernels
  pa::pdl_trigger();  // the successor may now be scheduled
  for (int b = threadIdx.x; b < d.B; b += blockDim.x) {
    d.active[b] = 1;
    d.iters[b] = 0;
  }
  for (int64_t q = threadIdx.x; q < (int64_t)d.B * d.T; q += blockDim.x) d.has[q] = 0;
  if (threadIdx.x == 0) {
    SCtl c{};
    c.n_active = d.B;
    *d.ctl = c;
  }
}

struct SLayout {
  size_t U, Up, Y, G, Xh, Eh, has, batch_x, miss_bt, rank, part, sacc, active, iters, err_log, coef, ctl, total;
};

SLayout s_layout(int T, int64_t D, int B, int N, int nstrip) {
  SLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = pa::align_up(o + bytes, pa::kAlign); return at; };
  const size_t row = (size_t)D * sizeof(float), row64 = (size_t)D * sizeof(double);
  L.U = take((size_t)B * (N + 1) * row64);
  L.Up = take((size_t)B * (N + 1) * row64);
  L.Y = take((size_t)B * N * row64);
  L.G = take((size_t)B * N * row64);
  L.Xh = take((size_t)B * T * row64);
  L.Eh = take((size_t)B * T * row);
  L.has = take((size_t)B * T * sizeof(int32_t));
  L.batch_x = take((size_t)B * N * row);
  L.miss_bt = take((size_t)B * N * 2 * sizeof(int32_t));
  L.rank = take((size_t)B * N * sizeof(int32_t));
  L.part = take((size_t)B * N * nstrip * sizeof(double));
  L.sacc = take((size_t)2 * B * N * pa::kAccStride * sizeof(double));  // one 128-byte line per sum
  L.active = take((size_t)B * sizeof(int32_t));
  L.iters = take((size_t)B * sizeof(int32_t));
  L.err_log = take((size_t)N * B * sizeof(float));
  L.coef = take((size_t)(2 * T + 2 * N) * sizeof(double));
  L.ctl = take(sizeof(SCtl));
  L.total = o;
  return L;
}

void s_blocks(int T, int* s, int* N) {
  int v = 1;
  while (v * v < T) ++v;
  *s = v;
  *N = (T + v - 1) / v;
}

}  // namespace

struct pa_srds {
  SDev d;
  SLayout L;
  char* ws;
  cudaStream_t st;
  int phase;      // -1 created, 0 ready for a step, 1 stepped (waiting for eps), 2 done
  int iter;       // current iteration (0 = coarse initialisation)
  int stage;      // index within the iteration: fine stages first (iter >= 1), then coarse
  int64_t g;      // stages since pa_srds_init: the distance set of stage g is g mod 2
  int nsm;        // SMs of the device
  int64_t launches;
  SCtl* host_ctl;
  // a whole generation captured as one CUDA graph (pa_srds_loop_*): a chain
  // of IF nodes, one per Parareal iteration, each body that iteration's
  // stages; iteration i's finishing kernel sets the condition of i + 1
  cudaGraph_t loop_graph;
  cudaGraphExec_t loop_exec;
  std::vector<cudaGraphConditionalHandle> loop_cond;  // one per iteration 0..N
  cudaGraphNode_t loop_last;  // the IF node of the iteration being captured
  bool loop_capturing;
  int64_t loop_launches0;
};

namespace {

pa_status s_fail(const std::string& m, pa_status code) {
  pa::set_error(m);
  return code;
}

// Forget the captured generation graph.
void s_drop_loop(pa_srds* h) {
  if (h->loop_exec) cudaGraphExecDestroy(h->loop_exec);
  if (h->loop_graph) cudaGraphDestroy(h->loop_graph);  // and the bodies its IF nodes own
  h->loop_exec = nullptr;
  h->loop_graph = nullptr;
  h->loop_cond.clear();
  h->loop_last = nullptr;
}

// Append the IF node of iteration it to the chain and point the capture of
// the sampler's stream at its body.
cudaError_t s_open_iteration(pa_srds* h, int it) {
  cudaGraphNodeParams np = {};
  np.type = cudaGraphNodeTypeConditional;
  np.conditional.handle = h->loop_cond[it];
  np.conditional.type = cudaGraphCondTypeIf;
  np.conditional.size = 1;
  cudaGraphNode_t node = nullptr;
  const cudaGraphNode_t dep = h->loop_last;
  cudaError_t e = cudaGraphAddNode(&node, h->loop_graph, dep ? &dep : nullptr, nullptr, dep ? 1 : 0, &np);
  if (e != cudaSuccess) return e;
  h->loop_last = node;
  // relaxed: calls this thread makes meanwhile on other work must not
  // invalidate the capture
  return cudaStreamBeginCaptureToGraph(h->st, np.conditional.phGraph_out[0], nullptr, nullptr, 0,
                                       cudaStreamCaptureModeRelaxed);
}

// Let go of a generation graph whose capture the runtime invalidated,
// without destroying it: destroying such a graph crashed the host process
// inside the CUDA runtime. The graph leaks; the handle can capture again.
void s_forget_loop(pa_srds* h) {
  h->loop_exec = nullptr;
  h->loop_graph = nullptr;
  h->loop_cond.clear();
  h->loop_last = nullptr;
}

Stage current_stage(const pa_srds* h) {
  Stage st{};
  st.iter = h->iter;
  const int nfine = h->iter == 0 ? 0 : h->d.s;
  if (h->stage < nfine) {
    st.kind = kFine;
    st.j = h->stage;
  } else {
    st.kind = h->iter == 0 ? kCoarseInit : kCoarse;
    st.n = h->stage - nfine;
  }
  return st;
}

cudaError_t s_sync_ctl(pa_srds* h) {
  cudaError_t e = cudaMemcpyAsync(h->host_ctl, h->d.ctl, sizeof(SCtl), cudaMemcpyDeviceToHost, h->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
  return e;
}

}  // namespace

extern "C" size_t pa_srds_workspace_bytes(int T, int64_t D, int batch) {
  if (T < 1 || T > 100000 || D < 1 || batch < 1 || batch > pa::kMaxBatch) return 0;
  int s, N;
  s_blocks(T, &s, &N);
  if ((int64_t)batch * N > kSMaxRows) return 0;
  return s_layout(T, D, batch, N, (int)((D + kSStrip - 1) / kSStrip)).total;
}

extern "C" pa_status pa_srds_create(pa_srds** out, int T, const int64_t* latent_shape, int ndim,
                                    const double* alphas_cumprod, double tol, double cache_thresh, int batch,
                                    void* workspace_dev, size_t workspace_bytes, void* stream) {
  if (!out) return s_fail("pa_srds_create: out is NULL", PA_ERR_ARG);
  *out = nullptr;
  if (T < 1 || T > 100000 || !latent_shape || ndim < 1 || ndim > 8 || !alphas_cumprod || batch < 1 ||
      batch > pa::kMaxBatch || !(tol >= 0.0) || !(cache_thresh >= 0.0))
    return s_fail("pa_srds_create: bad size, pointer or threshold", PA_ERR_ARG);
  int64_t D = 1;
  for (int k = 0; k < ndim; ++k) {
    if (latent_shape[k] < 1) return s_fail("pa_srds_create: latent_shape entries must be >= 1", PA_ERR_ARG);
    D *= latent_shape[k];
  }
  for (int i = 0; i <= T; ++i) {
    const double a = alphas_cumprod[i];
    if (!(a > 0.0 && a <= 1.0)) return s_fail("pa_srds_create: alphas_cumprod must be in (0, 1]", PA_ERR_ARG);
  }
  int s, N;
  s_blocks(T, &s, &N);
  if ((int64_t)batch * N > kSMaxRows) return s_fail("pa_srds_create: batch * blocks exceeds 2048", PA_ERR_ARG);
  const int nstrip = (int)((D + kSStrip - 1) / kSStrip);
  const SLayout L = s_layout(T, D, batch, N, nstrip);
  if (!workspace_dev || (reinterpret_cast<uintptr_t>(workspace_dev) % pa::kAlign) != 0 || workspace_bytes < L.total)
    return s_fail("pa_srds_create: workspace NULL, not 256-byte aligned, or smaller than pa_srds_workspace_bytes()",
                  PA_ERR_WORKSPACE);
  pa_srds* h = new pa_srds{};
  h->L = L;
  h->ws = static_cast<char*>(workspace_dev);
  h->st = static_cast<cudaStream_t>(stream);
  h->phase = -1;
  char* w = h->ws;
  SDev& d = h->d;
  d.T = T; d.B = batch; d.N = N; d.s = s; d.nstrip = nstrip; d.D = D;
  d.U = reinterpret_cast<double*>(w + L.U);
  d.Up = reinterpret_cast<double*>(w + L.Up);
  d.Y = reinterpret_cast<double*>(w + L.Y);
  d.G = reinterpret_cast<double*>(w + L.G);
  d.Xh = reinterpret_cast<double*>(w + L.Xh);
  d.Eh = reinterpret_cast<float*>(w + L.Eh);
  d.has = reinterpret_cast<int32_t*>(w + L.has);
  d.batch_x = reinterpret_cast<float*>(w + L.batch_x);
  d.miss_bt = reinterpret_cast<int32_t*>(w + L.miss_bt);
  d.rank = reinterpret_cast<int32_t*>(w + L.rank);
  d.part = reinterpret_cast<double*>(w + L.part);
  d.sacc = reinterpret_cast<double*>(w + L.sacc);
  d.active = reinterpret_cast<int32_t*>(w + L.active);
  d.iters = reinterpret_cast<int32_t*>(w + L.iters);
  d.err_log = reinterpret_cast<float*>(w + L.err_log);
  double* coef = reinterpret_cast<double*>(w + L.coef);
  d.cm1 = coef;
  d.e1 = coef + T;
  d.cjm1 = coef + 2 * T;
  d.ej = coef + 2 * T + N;
  d.ctl = reinterpret_cast<SCtl*>(w + L.ctl);
  d.tol = tol;
  d.cache_thresh = cache_thresh;
  // DDIM (eta = 0) jump from a to a2: x + (c - 1) x + e eps with c = sqrt(a2 / a),
  // e = sqrt(1 - a2) - sqrt(a2 (1 - a) / a); c - 1 formed without cancellation.
  auto jump = [](double a, double a2, double* cm1, double* e) {
    const double r = a2 / a, c = std::sqrt(r);
    *cm1 = (r - 1.0) / (c + 1.0);
    *e = std::sqrt(1.0 - a2) - std::sqrt(a2) * std::sqrt(1.0 - a) / std::sqrt(a);
  };
  std::vector<double> hc(2 * (size_t)T + 2 * (size_t)N);
  for (int i = 0; i < T; ++i) jump(alphas_cumprod[i], alphas_cumprod[i + 1], &hc[i], &hc[T + i]);
  for (int n = 0; n < N; ++n) {
    const int a0 = n * s, a1 = (n + 1) * s < T ? (n + 1) * s : T;
    jump(alphas_cumprod[a0], alphas_cumprod[a1], &hc[2 * T + n], &hc[2 * T + N + n]);
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaHostAlloc(reinterpret_cast<void**>(&h->host_ctl), sizeof(SCtl), cudaHostAllocDefault);
  if (e == cudaSuccess) e = cudaMemcpyAsync(coef, hc.data(), hc.size() * sizeof(double), cudaMemcpyHostToDevice, h->st);
  if (e == cudaSuccess) e = cudaMemsetAsync(d.ctl, 0, sizeof(SCtl), h->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
  if (e != cudaSuccess) {
    if (h->host_ctl) cudaFreeHost(h->host_ctl);
    delete h;
    return s_fail(std::string("pa_srds_create: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  }
  *out = h;
  return PA_OK;
}

extern "C" pa_status pa_srds_init(pa_srds* h, const float* x_init) {
  if (!h || !x_init) return s_fail("pa_srds_init: NULL argument", PA_ERR_ARG);
  if (h->loop_capturing) return s_fail("pa_srds_init: a generation is being captured", PA_ERR_STATE);
  const SDev& d = h->d;
  // x_init (host or device) is staged in batch_x, then widened into U_0 and Up_0
  cudaError_t e = cudaMemcpyAsync(d.batch_x, x_init, (size_t)d.B * d.D * sizeof(float), cudaMemcpyDefault, h->st);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_init: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  e = pa::launch_ex(k_srds_load, dim3(32, d.B), dim3(256), 0, h->st, 0, d, (const float*)d.batch_x, 0);
  if (e == cudaSuccess) e = pa::launch_ex(k_srds_reset, dim3(1), dim3(256), 0, h->st, 0, d);
  h->launches += 2;
  if (e == cudaSuccess) e = cudaMemsetAsync(d.sacc, 0, (size_t)2 * d.B * d.N * pa::kAccStride * sizeof(double), h->st);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_init: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  h->iter = 0;
  h->stage = 0;
  h->g = 0;
  h->phase = 0;
  return PA_OK;
}

extern "C" pa_status pa_srds_step_async(pa_srds* h, const float** batch_x, const int32_t** miss_bt,
                                        const int32_t** n_miss_dev) {
  if (!h) return s_fail("pa_srds_step_async: NULL handle", PA_ERR_ARG);
  if (h->phase == 2) return PA_DONE;
  if (h->phase != 0) return s_fail("pa_srds_step_async: call order (pa_srds_init, then step / submit)", PA_ERR_STATE);
  const SDev& d = h->d;
  const Stage st = current_stage(h);
  const int rows = st.kind == kFine ? d.B * d.N : d.B;
  // every CTA plans: about two CTAs per SM in all, each narrowing a longer part of its row
  int gx = (int)((d.D + kSThreads * 4 - 1) / (kSThreads * 4));
  const int gcap = (2 * h->nsm + rows - 1) / rows;
  if (gx > gcap) gx = gcap;
  if (gx > 32) gx = 32;
  if (gx < 1) gx = 1;
  const cudaError_t e =
      pa::launch_ex(k_srds_plan_gather, dim3(gx, rows), dim3(kSThreads), 0, h->st, 0, d, st, (int)(h->g & 1));
  h->launches += 1;
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_step_async: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  if (batch_x) *batch_x = d.batch_x;
  if (miss_bt) *miss_bt = d.miss_bt;
  if (n_miss_dev) *n_miss_dev = &d.ctl->n_miss;
  h->phase = 1;
  return PA_OK;
}

extern "C" pa_status pa_srds_step(pa_srds* h, int* n_miss, const float** batch_x, const int32_t** miss_bt) {
  if (!h || !n_miss) return s_fail("pa_srds_step: NULL argument", PA_ERR_ARG);
  if (h->loop_capturing)
    return s_fail("pa_srds_step: synchronises; inside a capture use pa_srds_step_async", PA_ERR_STATE);
  if (h->phase == 2) return PA_DONE;
  if (h->phase == 0 && h->stage == 0 && h->iter > 0) {  // a new iteration: anything left to refine?
    cudaError_t e = s_sync_ctl(h);
    if (e != cudaSuccess) return s_fail(std::string("pa_srds_step: ") + cudaGetErrorString(e), PA_ERR_CUDA);
    if (h->host_ctl->status != 0) return s_fail("pa_srds_step: device-side failure", PA_ERR_DEVICE);
    if (h->host_ctl->n_active == 0) {
      h->phase = 2;
      return PA_DONE;
    }
  }
  pa_status r = pa_srds_step_async(h, batch_x, miss_bt, nullptr);
  if (r != PA_OK) return r;
  const cudaError_t e = s_sync_ctl(h);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_step: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  *n_miss = h->host_ctl->n_miss;
  return PA_OK;
}

extern "C" const int32_t* pa_srds_n_miss_dev(const pa_srds* h) { return h ? &h->d.ctl->n_miss : nullptr; }

extern "C" pa_status pa_srds_submit_eps(pa_srds* h, const float* batch_eps) {
  if (!h || !batch_eps) return s_fail("pa_srds_submit_eps: NULL argument", PA_ERR_ARG);
  if (h->phase != 1) return s_fail("pa_srds_submit_eps: no step to complete", PA_ERR_STATE);
  const SDev& d = h->d;
  const Stage st = current_stage(h);
  const int rows = st.kind == kFine ? d.B * d.N : d.B;
  // column blocks per row: four columns per thread (at most 32 blocks), or
  // more blocks when the stage has few rows (a coarse stage has only B), up to
  // about two CTAs per SM in all and one column per thread
  int gx = (int)((d.D + kSThreads * 4 - 1) / (kSThreads * 4));
  if (gx > 32) gx = 32;
  const int gsm = (2 * h->nsm + rows - 1) / rows;
  const int gmax = (int)((d.D + kSThreads - 1) / kSThreads);
  if (gsm > gx) gx = gsm < gmax ? gsm : gmax;
  if (gx < 1) gx = 1;
  const int nset = (int)((h->g + 1) & 1);  // the next stage's distance set
  cudaError_t e = pa::launch_ex(k_srds_apply, dim3(gx, rows), dim3(kSThreads), 0, h->st, 0, d, st, batch_eps, nset);
  h->launches++;
  const int nstages = (h->iter == 0 ? 0 : d.s) + d.N;
  if (++h->stage == nstages) {  // the iteration is complete
    const bool next = h->loop_capturing && h->iter + 1 <= d.N;  // captured: set the next IF node's condition
    if (e == cudaSuccess)
      e = pa::launch_ex(k_srds_err, dim3(d.nstrip, d.B * d.N), dim3(kSThreads), 0, h->st, 0, d, h->iter, nset);
    if (e == cudaSuccess)
      e = pa::launch_ex(k_srds_finish, dim3(1), dim3(kSThreads), 0, h->st, 0, d, h->iter,
                        next ? h->loop_cond[h->iter + 1] : (cudaGraphConditionalHandle)0, next ? 1 : 0);
    h->launches += 2;
    h->stage = 0;
    h->iter++;
    if (h->loop_capturing) {  // the iteration's body is complete: close it, open the next one's
      cudaGraph_t body = nullptr;
      const cudaError_t ec = cudaStreamEndCapture(h->st, &body);
      if (e == cudaSuccess) e = ec;
      if (e == cudaSuccess && h->iter <= d.N) e = s_open_iteration(h, h->iter);
      if (e != cudaSuccess) {  // nothing ran; the capture is closed and dropped
        (void)cudaGetLastError();
        h->loop_capturing = false;
        if (ec != cudaSuccess)
          s_forget_loop(h);  // an invalidated capture: destroy nothing
        else
          s_drop_loop(h);
        h->phase = -1;  // pa_srds_init must follow
        return s_fail(std::string("pa_srds_submit_eps: capture: ") + cudaGetErrorString(e), PA_ERR_CUDA);
      }
    }
  }
  h->g++;
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_submit_eps: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  h->phase = (h->iter > d.N) ? 2 : 0;
  return PA_OK;
}

extern "C" pa_status pa_srds_poll(pa_srds* h, int* n_active) {
  if (!h) return s_fail("pa_srds_poll: NULL handle", PA_ERR_ARG);
  if (h->loop_capturing) return s_fail("pa_srds_poll: synchronises; not inside a capture", PA_ERR_STATE);
  const cudaError_t e = s_sync_ctl(h);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_poll: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  const int act = h->host_ctl->n_active;
  if (n_active) *n_active = act;
  if (act == 0 && h->phase == 0) h->phase = 2;
  return act == 0 ? PA_DONE : PA_OK;
}

extern "C" pa_status pa_srds_result(pa_srds* h, float* x_out) {
  if (!h || !x_out) return s_fail("pa_srds_result: NULL argument", PA_ERR_ARG);
  if (h->loop_capturing) return s_fail("pa_srds_result: synchronises; not inside a capture", PA_ERR_STATE);
  if (h->phase != 2) return s_fail("pa_srds_result: not finished", PA_ERR_STATE);
  const SDev& d = h->d;
  // U_N narrowed to fp32 in batch_x (free once sampling is done), then copied out
  cudaError_t e = pa::launch_ex(k_srds_store, dim3(32, d.B), dim3(256), 0, h->st, 0, d, d.batch_x, d.N);
  h->launches++;
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(x_out, d.batch_x, (size_t)d.B * d.D * sizeof(float), cudaMemcpyDefault, h->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_result: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  return PA_OK;
}

extern "C" pa_status pa_srds_loop_capture_begin(pa_srds* h) {
  if (!h) return s_fail("pa_srds_loop_capture_begin: NULL handle", PA_ERR_ARG);
  if (h->loop_capturing) return s_fail("pa_srds_loop_capture_begin: a capture is already open", PA_ERR_STATE);
  if (h->phase != 0 || h->iter != 0 || h->stage != 0 || h->g != 0)
    return s_fail("pa_srds_loop_capture_begin: call right after pa_srds_init", PA_ERR_STATE);
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(h->st, &cs);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_loop_capture_begin: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  if (cs != cudaStreamCaptureStatusNone)
    return s_fail("pa_srds_loop_capture_begin: the stream is already being captured", PA_ERR_STATE);
  s_drop_loop(h);
  e = cudaGraphCreate(&h->loop_graph, 0);
  // iteration 0 (the coarse sweep) always runs; every later one only when the
  // previous one's finishing kernel found a trajectory still active
  h->loop_cond.assign((size_t)h->d.N + 1, 0);
  for (int i = 0; i <= h->d.N && e == cudaSuccess; ++i)
    e = cudaGraphConditionalHandleCreate(&h->loop_cond[i], h->loop_graph, i == 0 ? 1u : 0u,
                                         cudaGraphCondAssignDefault);
  if (e == cudaSuccess) e = s_open_iteration(h, 0);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    s_drop_loop(h);
    return s_fail(std::string("pa_srds_loop_capture_begin: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  }
  h->loop_capturing = true;
  h->loop_launches0 = h->launches;
  return PA_OK;
}

extern "C" pa_status pa_srds_loop_capture_end(pa_srds* h) {
  if (!h) return s_fail("pa_srds_loop_capture_end: NULL handle", PA_ERR_ARG);
  if (!h->loop_capturing) return s_fail("pa_srds_loop_capture_end: no capture is open", PA_ERR_STATE);
  h->loop_capturing = false;
  if (h->phase != 2) {  // a body is still open: close it, keep nothing
    cudaGraph_t body = nullptr;
    const cudaError_t ec = cudaStreamEndCapture(h->st, &body);
    (void)cudaGetLastError();
    if (ec != cudaSuccess)
      s_forget_loop(h);  // an invalidated capture: destroy nothing
    else
      s_drop_loop(h);
    h->phase = -1;  // pa_srds_init must follow
    return s_fail("pa_srds_loop_capture_end: issue every stage first (pa_srds_step_async until PA_DONE)",
                  PA_ERR_STATE);
  }
  const cudaError_t e = cudaGraphInstantiate(&h->loop_exec, h->loop_graph, 0);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    s_drop_loop(h);
    h->phase = -1;
    return s_fail(std::string("pa_srds_loop_capture_end: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  }
  // nothing ran: back to the state right after pa_srds_init
  h->iter = 0;
  h->stage = 0;
  h->g = 0;
  h->phase = 0;
  h->launches = h->loop_launches0;
  return PA_OK;
}

extern "C" pa_status pa_srds_loop_launch(pa_srds* h) {
  if (!h) return s_fail("pa_srds_loop_launch: NULL handle", PA_ERR_ARG);
  if (!h->loop_exec) return s_fail("pa_srds_loop_launch: nothing has been captured", PA_ERR_STATE);
  if (h->loop_capturing || h->phase != 0 || h->iter != 0 || h->stage != 0 || h->g != 0)
    return s_fail("pa_srds_loop_launch: call right after pa_srds_init", PA_ERR_STATE);
  const cudaError_t e = cudaGraphLaunch(h->loop_exec, h->st);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_loop_launch: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  h->phase = 2;  // the graph runs the generation to its end
  h->iter = h->d.N + 1;
  return PA_OK;
}

extern "C" pa_status pa_srds_stats(pa_srds* h, pa_srds_stats_t* out) {
  if (!h || !out) return s_fail("pa_srds_stats: NULL argument", PA_ERR_ARG);
  if (h->loop_capturing) return s_fail("pa_srds_stats: synchronises; not inside a capture", PA_ERR_STATE);
  const cudaError_t e = s_sync_ctl(h);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_stats: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  out->iters = h->host_ctl->iter;
  out->nfe = h->host_ctl->nfe;
  out->hits = h->host_ctl->hits;
  out->launches = h->launches;
  out->n_active = h->host_ctl->n_active;
  out->n_miss = h->host_ctl->n_miss;
  out->device_status = h->host_ctl->status;
  out->blocks = h->d.N;
  out->block_steps = h->d.s;
  return PA_OK;
}

extern "C" pa_status pa_srds_errors(pa_srds* h, float* err_out) {
  if (!h || !err_out) return s_fail("pa_srds_errors: NULL argument", PA_ERR_ARG);
  const cudaError_t e = cudaMemcpy(err_out, h->d.err_log, (size_t)h->d.N * h->d.B * sizeof(float),
                                   cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return s_fail(std::string("pa_srds_errors: ") + cudaGetErrorString(e), PA_ERR_CUDA);
  return PA_OK;
}

extern "C" void pa_srds_destroy(pa_srds* h) {
  if (!h) return;
  if (h->loop_capturing) {  // close the capture so that the stream stays usable
    cudaGraph_t g = nullptr;
    if (cudaStreamEndCapture(h->st, &g) != cudaSuccess) s_forget_loop(h);
    (void)cudaGetLastError();
  }
  s_drop_loop(h);
  if (h->host_ctl) cudaFreeHost(h->host_ctl);
  delete h;
}
