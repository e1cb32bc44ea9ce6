// Internal layout shared by the host state machine (pa_solver.cpp) and the
// kernels (k_solver.cu, k_update_bulk.cu). Not part of the public ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace pa {

constexpr int kMaxWindow = 1024;
constexpr int kMaxBatch = 64;
constexpr size_t kAlign = 256;
// Doubles from one fp64 accumulator (Eq. 2 / Eq. 4 sums) to the next: each
// sits on its own 128-byte line, so the atomic adds of many CTAs into
// different window positions do not queue behind one another on a line.
constexpr int kAccStride = 16;
constexpr int kBulkConfigs = 13;    // launch shapes of the bulk-copy update kernel
constexpr int kLeanConfigs = 17;    // launch shapes of the lean register update kernel (0..6, 10..16)

// Device status codes written by kernels (first error wins, atomicCAS from 0).
constexpr int kDevOk = 0;
constexpr int kDevTimeout = 1;      // a bounded mbarrier wait ran out
constexpr int kDevBadRank = 2;      // a miss rank outside [0, n_miss)
constexpr int kDevBadState = 3;     // trajectory bookkeeping inconsistent

// Per-trajectory window bookkeeping.
//  t : window start (the converged state x_t, Sec. 2.1 sliding window)
//  p : evaluation points t..t+p-1 this iteration (0 once t == T)
//  e : evaluated frontier: timesteps < e have a cache entry (Eq. 3); states
//      0..e hold real values in the state ring; states > e are "lazy" and
//      equal state e (new tail states copy the last computed state).
//  m : misses of trajectory b in the planned iteration (for the iteration log)
//  h1: hits among window positions 1..p-1 of the planned iteration (their xhat
//      rows are read for the next iteration's distances; for the byte count)
//  ne: window positions of the planned iteration that have a cache entry
//  nh: hits among them (the adaptation of tau_cache reads ne and nh)
struct Traj {
  int32_t t, p, e, done, m, h1, ne, nh;
};
constexpr int kLogFields = 8;  // iteration log entry: t, p, misses, stride, e, h1, ne, nh

// Counters read by the host (one copy, written by whichever kernel publishes
// a plan) and by the denoiser (n_miss, through its device pointer).
struct Ctl {
  int32_t n_miss;     // misses planned for the next iteration (Eq. 5)
  int32_t n_active;   // trajectories with t < T
  int32_t iter;       // iterations completed
  int32_t status;     // kDev* code
  long long nfe;
  long long hits;
  int32_t loop_passes;  // body passes of the device-driven loop since its launch
  int32_t reserved;
};

// The counters a decision starts from. Kept in two copies, like the
// trajectories: the plan of iteration k lives in copy k mod 2, so the kernel
// that decides iteration k+1 reads copy k mod 2 in all of its CTAs while one
// of them writes copy (k+1) mod 2.
struct PlanCtr {
  int32_t n_active, iter;
  long long nfe, hits;
};

struct Layout {
  size_t X, Xhat, Ehat, batch_x, coef, traj, pc, ctl, rank, miss_bt;
  size_t acc, red_err, red_del, iter_log, gbar, tau, total;
};

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

inline Layout make_layout(int T, int P, int64_t D, int B) {
  Layout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = align_up(o + bytes, kAlign); return at; };
  const size_t row = (size_t)D * sizeof(float);
  L.X = take((size_t)B * (P + 1) * row);          // state ring, slot = i mod (P+1)
  L.Xhat = take((size_t)B * P * row);             // cache inputs, slot = i mod P
  L.Ehat = take((size_t)B * P * row);             // cache outputs, slot = i mod P
  L.batch_x = take((size_t)B * P * row);          // gathered misses
  L.coef = take((size_t)3 * T * sizeof(float));   // (c_i - 1, e_i, sigma_i)
  L.traj = take((size_t)2 * B * sizeof(Traj));     // two copies (plan parity)
  L.pc = take(2 * sizeof(PlanCtr));
  L.ctl = take(sizeof(Ctl));
  L.rank = take((size_t)B * P * sizeof(int32_t));
  L.miss_bt = take((size_t)B * P * 2 * sizeof(int32_t));
  L.acc = take((size_t)2 * 2 * B * P * kAccStride * sizeof(double));  // [set][err, dist][B][P], strided
  L.red_err = take((size_t)B * P * sizeof(float));
  L.red_del = take((size_t)B * P * sizeof(float));
  L.iter_log = take((size_t)(T + 1) * B * kLogFields * sizeof(int32_t));
  L.gbar = take(128);                              // arrival counter of the fused step's grid barrier
  L.tau = take((size_t)2 * B * sizeof(double));    // tau_cache per trajectory, by plan parity
  L.total = o;
  return L;
}

// Device views of one solver's workspace.
struct Dev {
  float* X;
  float* Xhat;
  float* Ehat;
  float* batch_x;
  const float* cm1;   // c_i - 1
  const float* ecoef; // e_i
  const float* sigma; // sigma_i of stochastic steps (0 for eta = 0)
  const float* noise; // [B][T][D] draws z_i of stochastic steps, caller-owned; NULL for eta = 0
  Traj* traj;         // [2][B]: copy k mod 2 holds the plan of iteration k
  PlanCtr* pc;        // [2]
  Ctl* ctl;
  int32_t* rank;      // [B][P] rank of window position j among the misses, -1 = hit
  int32_t* miss_bt;   // [B*P][2]
  double* acc;        // [2][2][B][P] x kAccStride: sums of Eq. 2 and Eq. 4 terms; set k mod 2 in iteration k
  float* red_err;     // [B][P] the last decision's reductions (divided by D), for the host
  float* red_del;
  int32_t* iter_log;  // [T+1][B][kLogFields]
  unsigned long long* gbar;  // arrivals at the fused step's grid barrier (cleared by pa_init)
  // Triangular Anderson mixing (pa_set_anderson), in a caller-owned second
  // workspace: the Picard map's output G and residual R of every window
  // state, [2][B][P+1][D] each by iteration parity (copy k mod 2 written in
  // iteration k, slot = state mod (P+1)), and the Gram sums <dR, R>, <dR, dR>
  // per position, [2][2][B][P] x kAccStride, set k mod 2 in iteration k,
  // and the frontier state's value before the iteration, [B][D]: the mix
  // kernel overwrites state e's slot while the lazy states (past e) still
  // need its old value.
  float* taa_g;
  float* taa_r;
  double* taa_acc;
  float* taa_xe;
  int taa;            // 1: iterations mix (depth 1); 0: plain Picard
  // Online adaptation of tau_cache (pa_set_cache_adaptation): tau of every
  // trajectory, [2][B] by plan parity (copy k mod 2 is the tau of iteration
  // k's hit test); adapt = 0 keeps tau_cache fixed (thr_d is then used).
  double* tau;
  int adapt;
  double adapt_up, adapt_target, tau_min, tau_max;
  int T, P, B;
  int64_t D;
  double tol, cache_thresh;   // tau of Eq. 2 and tau_cache of Eq. 5
  // The same thresholds on the undivided sums, as the kernels compare them:
  // sum <= tol * D (Eq. 2) and sum < tau_cache * D (Eq. 5), formed in fp64 on
  // the host; both sides are non-negative doubles, so the kernels compare
  // their bit patterns as integers (the same order) and run no fp64
  // arithmetic. inv_d = 1 / D for the reductions reported to the host.
  double tol_d, thr_d, inv_d;
  int bulk_cfg;               // launch shape of the bulk-copy update kernel
  int cache_bf16;             // 1: xhat and ehat rows hold bfloat16 values (row pitch D elements)
  uint32_t wait_limit;        // polls before an mbarrier wait counts as timed out
};
constexpr uint32_t kWaitLimit = 1u << 17;  // tries of an mbarrier wait (~1.3 s with the suspend hint)

// Programmatic dependent launch (PDL). Every kernel of an iteration is
// launched with programmatic stream serialization: it does the work that does
// not read its predecessor's output, then executes pdl_wait() (predecessor
// complete, its writes visible). Each kernel triggers its successor
// (pdl_trigger) right after its own pdl_wait, never before: when a kernel
// starts, every CTA of its predecessor has passed its wait, so the kernel two
// back has completed. A kernel's prologue may therefore read anything written
// two or more kernels back, and must not write anything its predecessor reads.
// The successor is scheduled only once all of the predecessor's CTAs have
// triggered, i.e. are resident, so its waiting CTAs never keep a predecessor
// CTA from an SM.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

bool pdl_enabled();  // false when the environment sets PA_DISABLE_PDL=1

// cudaLaunchKernelEx with the PDL attribute (when enabled), an optional
// cluster width along x (0 = no cluster attribute) and, with `coop`, the
// cooperative attribute (every CTA resident at once, for a grid barrier).
template <typename... KArgs, typename... Args>
cudaError_t launch_ex_coop(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                           unsigned cluster_x, bool coop, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[3];
  unsigned n = 0;
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster_x > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (coop) {
    attr[n].id = cudaLaunchAttributeCooperative;
    attr[n].val.cooperative = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                      unsigned cluster_x, Args&&... args) {
  return launch_ex_coop(kern, grid, block, smem, st, cluster_x, false, static_cast<Args&&>(args)...);
}

// Cache entries stored as bfloat16 (a storage option, not from the paper):
// loads widen exactly, stores round to nearest even.
template <int V>
struct Bf16Row;
template <>
struct Bf16Row<4> {
  __device__ static void load(const uint16_t* p, float* a) {
    const uint2 q = *reinterpret_cast<const uint2*>(p);
    a[0] = __uint_as_float(q.x << 16);
    a[1] = __uint_as_float(q.x & 0xffff0000u);
    a[2] = __uint_as_float(q.y << 16);
    a[3] = __uint_as_float(q.y & 0xffff0000u);
  }
  __device__ static void store(uint16_t* p, const float* a) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(a[0], a[1]);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(a[2], a[3]);
    uint2 q;
    q.x = *reinterpret_cast<const uint32_t*>(&lo);
    q.y = *reinterpret_cast<const uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(p) = q;
  }
};
template <>
struct Bf16Row<1> {
  __device__ static void load(const uint16_t* p, float* a) { a[0] = __uint_as_float((uint32_t)*p << 16); }
  __device__ static void store(uint16_t* p, const float* a) {
    const __nv_bfloat16 h = __float2bfloat16_rn(a[0]);
    *p = *reinterpret_cast<const uint16_t*>(&h);
  }
};

// A CTA's partial of an Eq. 2 / Eq. 4 sum (non-negative fp32) as it enters the
// fp64 accumulators: rounded up to a multiple of 2^-32. Every term is then a
// multiple of 2^-32 and every partial sum of such terms below 2^21 is exactly
// representable in fp64 (2^21 / 2^-32 = 2^53), so the accumulated sum is exact
// -- the same whatever order the CTAs arrive in -- as long as it stays below
// 2^21; above that the sum divided by D is at least 2^21 / D (>= 32 for rows of
// up to 65536 values), far beyond any tolerance the decision compares it
// with. Rounding up keeps a nonzero partial nonzero (tol = 0 stays exact) and
// moves a sum by at most one 2^-32 per CTA.
__device__ __forceinline__ double quantize_partial(float v) {
  return ceil((double)v * 4294967296.0) * (1.0 / 4294967296.0);
}

// Eq. 2 / Eq. 5 tests on an accumulated (non-negative) sum, by bit pattern.
__device__ __forceinline__ bool sum_le(double sum, double bound) {
  return __double_as_longlong(sum) <= __double_as_longlong(bound);
}
__device__ __forceinline__ bool sum_lt(double sum, double bound) {
  return __double_as_longlong(sum) < __double_as_longlong(bound);
}

// One CTA's share of the Eq. 2 error (which = 0) or Eq. 4 distance (which =
// 1) of window position q = b*P + j, added into the accumulator set of the
// iteration's parity (exact, see quantize_partial).
__device__ __forceinline__ void red_add(const Dev& d, int par, int which, int q, float v) {
  atomicAdd(d.acc + ((size_t)(par * 2 + which) * d.B * d.P + q) * kAccStride, quantize_partial(v));
}

// A CTA's partial of a Gram sum of the Anderson mixing (<dR, R> for which = 0,
// <dR, dR> for which = 1) of window position q, into set par. The partial may
// be negative; rounded to a multiple of 2^-32 like the other sums, so the
// accumulated sum is exact while the sum of the terms' magnitudes stays below
// 2^21.
__device__ __forceinline__ void red_add_gram(const Dev& d, int par, int which, int q, float v) {
  atomicAdd(d.taa_acc + ((size_t)(par * 2 + which) * d.B * d.P + q) * kAccStride, quantize_partial(v));
}

// Bytes of the Anderson workspace: G and R by iteration parity, the Gram sums.
inline size_t taa_layout(int P, int64_t D, int B, size_t* o_r, size_t* o_acc, size_t* o_xe) {
  const size_t rows = align_up((size_t)2 * B * (P + 1) * D * sizeof(float), kAlign);
  *o_r = rows;
  *o_acc = 2 * rows;
  *o_xe = *o_acc + align_up((size_t)2 * 2 * B * P * kAccStride * sizeof(double), kAlign);
  return *o_xe + align_up((size_t)B * D * sizeof(float), kAlign);
}

// Grid-wide barrier of a launch whose CTAs are all resident at once (the
// fused step kernel, launched cooperatively). Thread 0 of each CTA publishes
// the CTA's writes (fence), adds one to the counter and waits until the count
// reaches the next multiple of the grid size: launches of one solver never
// overlap at the barrier (each starts its arrivals after the previous one
// completed), so the count before an arrival identifies the launch. The wait
// polls at most `limit` times; false = it ran out (the caller records
// PA_ERR_TIMEOUT and returns). Every thread of the CTA must call it.
__device__ __forceinline__ bool grid_sync(unsigned long long* ctr, unsigned long long n, uint32_t limit) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned long long old = atomicAdd(ctr, 1ull);
    const unsigned long long target = (old / n + 1ull) * n;
    int ok = 1;
    if (old + 1ull != target) {
      for (uint32_t polls = 0;; ++polls) {
        if (polls >= limit) {  // limit 0: every CTA but the last to arrive gives up at once
          ok = 0;
          break;
        }
        unsigned long long v;
        asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(ctr) : "memory");
        if (v >= target) break;
      }
    }
    s_ok = ok;  // the acquire load orders the CTA's later reads (after the barrier below)
  }
  __syncthreads();
  return s_ok != 0;
}

// Kernel launchers (k_solver.cu). Each returns the launch error. par = k mod 2
// for iteration k: the copy of the plan the kernel reads (and the accumulator
// set the update kernels add into).
cudaError_t launch_init(const Dev& d, cudaStream_t st);  // first plan, its batch, cleared sums
cudaError_t launch_gather(const Dev& d, int par, cudaStream_t st);
cudaError_t launch_update_plain(const Dev& d, const float* batch_eps, int par, cudaStream_t st);
// the decision after iteration k (par = k mod 2) and the gather of iteration k+1
cudaError_t launch_plan(const Dev& d, int par, cudaStream_t st, int* launches);
// k_update_bulk.cu
cudaError_t launch_update_bulk(const Dev& d, const float* batch_eps, int par, cudaStream_t st);
bool update_bulk_supported(const Dev& d, const float* batch_eps);
// k_update_lean.cu; shape: see launch_update_lean (cudaErrorNotSupported when
// the shape cannot hold the window)
cudaError_t launch_update_lean(const Dev& d, const float* batch_eps, int par, int shape, cudaStream_t st);
bool update_lean_supported(const Dev& d, const float* batch_eps);
// The fused step (k_update_lean.cu): the lean update, a grid barrier, the
// decision in every CTA and the next batch written from registers -- one
// kernel per iteration in place of the update and planning kernels. Only for
// grids that are resident in one wave; cudaErrorNotSupported otherwise.
cudaError_t launch_step_fused(const Dev& d, const float* batch_eps, int par, int shape, cudaStream_t st);
bool step_fused_supported(const Dev& d, const float* batch_eps, int shape);
// Triangular Anderson mixing (k_update_lean.cu, k_taa.cu): the lean update in
// its mixing form (G and R, Gram partials; the states are left to the mix
// kernel), then the mix kernel (X <- G - gamma_j (G - G'), the Eq. 2 and
// Eq. 4 partials). cudaErrorNotSupported when the lean form cannot run.
cudaError_t launch_update_taa(const Dev& d, const float* batch_eps, int par, cudaStream_t st);
cudaError_t launch_taa_mix(const Dev& d, int par, cudaStream_t st);
// An empty kernel with programmatic dependent launch (k_solver.cu)
cudaError_t launch_gap(cudaStream_t st);

}  // namespace pa
