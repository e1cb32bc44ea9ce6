// Solver-step kernels for sm_103a: first-iteration plan, miss gather (a4),
// plain-load Picard update (a6-a9, a11) and the planning kernel that takes
// the decision after an update (a10, a2, a3) and gathers the next batch (a4).
//
// Data layout (fp32, one row = one timestep's latent of D floats):
//   X    [B][P+1][D]  state ring, state i lives in slot i mod (P+1)
//   Xhat [B][P][D]    cache inputs  xhat_i  (Eq. 3), slot i mod P
//   Ehat [B][P][D]    cache outputs ehat_i  (Eq. 3), slot i mod P
//   batch_x [B*P][D]  gathered latents of the misses, rank order
#include <type_traits>

#include "pa_decide.cuh"
#include "pa_internal.h"

namespace pa {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ void set_status(Ctl* c, int code) {
  atomicCAS(&c->status, kDevOk, code);
}

// ---------------------------------------------------------------------------
// a4: batch_x[r] <- x_{miss[r]} for r < n_miss. A lazy state (i > e) reads
// state e, the value every new tail state was initialised to. Each thread
// moves kGatherUnroll vectors per row with all loads issued before the stores;
// 16 of them make a 4x64x64 row one CTA's work (100 planning CTAs at window
// 100: 25.9 against 26.3 us per iteration with quarter rows in 400 CTAs).
constexpr int kGatherThreads = 256;
constexpr int kGatherUnroll = 16;

template <int VEC>
__device__ __forceinline__ void copy_row(const Dev& d, int b, int src_state, int r) {
  using T = typename std::conditional<VEC == 4, float4, float>::type;
  const int64_t nvec = d.D / VEC;
  const int64_t stride = (int64_t)gridDim.x * kGatherThreads;
  const int64_t base = (int64_t)blockIdx.x * kGatherThreads + threadIdx.x;
  const T* from = reinterpret_cast<const T*>(d.X + ((int64_t)b * (d.P + 1) + src_state % (d.P + 1)) * d.D);
  T* to = reinterpret_cast<T*>(d.batch_x + (int64_t)r * d.D);
  for (int64_t v0 = base; v0 < nvec; v0 += stride * kGatherUnroll) {
    T buf[kGatherUnroll];
#pragma unroll
    for (int u = 0; u < kGatherUnroll; ++u) {
      const int64_t v = v0 + u * stride;
      if (v < nvec) buf[u] = __ldg(from + v);
    }
#pragma unroll
    for (int u = 0; u < kGatherUnroll; ++u) {
      const int64_t v = v0 + u * stride;
      if (v < nvec) to[v] = buf[u];
    }
  }
}

// The gather of a plan already in memory (copy par): after the first plan,
// and after the one-CTA planner.
template <int VEC>
__global__ void __launch_bounds__(kGatherThreads) k_gather(Dev d, int par) {
  pdl_wait();  // everything read here comes from the kernel that planned
  pdl_trigger();  // the successor may now run its prologue
  const int n = d.ctl->n_miss;
  const Traj* tr = d.traj + par * d.B;
  for (int r = blockIdx.y; r < n; r += gridDim.y) {
    const int b = d.miss_bt[2 * r], i = d.miss_bt[2 * r + 1];
    copy_row<VEC>(d, b, min(i, tr[b].e), r);
  }
}

// ---------------------------------------------------------------------------
// First iteration (after pa_init's copy of x_init into state 0): every
// timestep of every first window enters for the first time, hence is a miss
// (Sec. 2.2); states 1..p are lazy copies of state 0 = x_init, so the frontier
// e starts at 0 and batch row r = b p0 + j is state 0 of trajectory b. One
// launch on the planning kernel's grid: each CTA copies its part of its batch
// rows; all
// CTAs together write the ranks and the miss list and clear both sets of the
// reduction accumulators (the entries that are added into, every
// kAccStride-th) and the fused step's barrier counter; CTA (0, 0) writes the
// trajectories, counters and the plan's counter copy 0.
template <int VEC>
__global__ void __launch_bounds__(kGatherThreads) k_init(Dev d) {
  pdl_wait();  // x_init was copied into state 0 just before
  pdl_trigger();
  const int p0 = min(d.P, d.T);
  const int npair = d.B * d.P;
  const int64_t cta = (int64_t)blockIdx.y * gridDim.x + blockIdx.x;
  const int64_t step = (int64_t)gridDim.x * gridDim.y * kGatherThreads;
  for (int64_t q = cta * kGatherThreads + threadIdx.x; q < npair; q += step) {
    const int b = (int)(q / d.P), j = (int)(q % d.P);
    if (j < p0) {
      const int r = b * p0 + j;
      d.rank[q] = r;
      d.miss_bt[2 * r] = b;
      d.miss_bt[2 * r + 1] = j;
    } else {
      d.rank[q] = -1;
    }
  }
  for (int64_t q = cta * kGatherThreads + threadIdx.x; q < 4 * (int64_t)npair; q += step) {
    d.acc[q * kAccStride] = 0.0;  // [set][err, dist][B][P]
    if (d.taa) d.taa_acc[q * kAccStride] = 0.0;
  }
  if (cta == 0) {
    for (int b = threadIdx.x; b < d.B; b += blockDim.x) {
      Traj tr{};
      tr.t = 0; tr.p = p0; tr.e = 0; tr.done = 0; tr.m = p0; tr.h1 = 0;  // no entries yet: ne = nh = 0
      d.traj[b] = tr;  // copy 0: the plan of iteration 0
      if (d.adapt) d.tau[b] = d.cache_thresh;  // tau_cache starts at the configured value
    }
    if (threadIdx.x == 0) {
      *d.gbar = 0ull;
      Ctl c{};
      c.n_miss = d.B * p0;
      c.n_active = d.B;
      c.iter = 0;
      c.status = kDevOk;
      c.nfe = (long long)d.B * p0;
      c.hits = 0;
      *d.ctl = c;
      PlanCtr pc;
      pc.n_active = c.n_active;
      pc.iter = 0;
      pc.nfe = c.nfe;
      pc.hits = 0;
      d.pc[0] = pc;
    }
  }
  for (int r = blockIdx.y; r < d.B * p0; r += gridDim.y) copy_row<VEC>(d, r / p0, 0, r);
}

// ---------------------------------------------------------------------------
// Plain-load Picard update. One CTA = one column chunk of one trajectory;
// each thread owns VEC adjacent columns and walks the window sequentially,
// which makes the window-axis prefix sum (Eq. 1) a register recurrence.
// Per window position j (timestep i = t + j):
//   eps_i  = batch_eps[rank] (miss) or ehat_i (hit)              Eq. 6
//   miss:  ehat_i <- eps_i, xhat_i <- x_i                         Eq. 7
//   d_i    = (c_i - 1) x_i + e_i eps_i (+ sigma_i z_i)            drift
//   x'_{i+1} = x_t + sum_{l<=j} d_{t+l}  (compensated)            Eq. 1
//   err_j  partial of sum (x'_{i+1} - x_{i+1})^2                  Eq. 2
//   del_j  partial of sum |x'_{i+1} - xhat_{i+1}| (next iteration) Eq. 4
// Partials are reduced per CTA in a fixed order and added into the
// iteration's fp64 accumulators (red_add); the planning kernel reads the sums.
template <int VEC>
struct V;
template <>
struct V<1> {
  float a[1];
};
template <>
struct V<4> {
  float a[4];
};

template <int VEC>
__device__ __forceinline__ V<VEC> ldv(const float* p) {
  V<VEC> r;
  if constexpr (VEC == 4) {
    float4 q = *reinterpret_cast<const float4*>(p);
    r.a[0] = q.x; r.a[1] = q.y; r.a[2] = q.z; r.a[3] = q.w;
  } else {
    r.a[0] = *p;
  }
  return r;
}

template <int VEC>
__device__ __forceinline__ void stv(float* p, const V<VEC>& v) {
  if constexpr (VEC == 4) {
    *reinterpret_cast<float4*>(p) = make_float4(v.a[0], v.a[1], v.a[2], v.a[3]);
  } else {
    *p = v.a[0];
  }
}

// A cache entry row (xhat or ehat) at element offset `off`: fp32, or bfloat16 when CB.
template <int VEC, bool CB>
__device__ __forceinline__ V<VEC> ld_entry(const float* base, int64_t off) {
  if constexpr (CB) {
    V<VEC> r;
    Bf16Row<VEC>::load(reinterpret_cast<const uint16_t*>(base) + off, r.a);
    return r;
  } else {
    return ldv<VEC>(base + off);
  }
}
template <int VEC, bool CB>
__device__ __forceinline__ void st_entry(float* base, int64_t off, const V<VEC>& v) {
  if constexpr (CB) {
    Bf16Row<VEC>::store(reinterpret_cast<uint16_t*>(base) + off, v.a);
  } else {
    stv<VEC>(base + off, v);
  }
}
template <int VEC, bool CB>
__device__ __forceinline__ V<VEC> as_entry(const V<VEC>& v) {
  if constexpr (CB) {
    V<VEC> r;
#pragma unroll
    for (int k = 0; k < VEC; ++k) r.a[k] = __bfloat162float(__float2bfloat16_rn(v.a[k]));
    return r;
  } else {
    return v;
  }
}

constexpr int kPlainThreads = 128;

template <int VEC, bool CB>
__global__ void __launch_bounds__(kPlainThreads) k_update_plain(Dev d, const float* __restrict__ beps, int par) {
  extern __shared__ float red[];  // [2][nwarps][P]
  const int b = blockIdx.y;
  pdl_wait();
  pdl_trigger();  // the successor may now run its prologue
  const Traj tr = d.traj[par * d.B + b];
  if (tr.p == 0) return;
  const int t = tr.t, p = tr.p, e = tr.e, P = d.P;
  const int64_t D = d.D;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int nw = kPlainThreads / 32;
  const int64_t col = ((int64_t)blockIdx.x * kPlainThreads + threadIdx.x) * VEC;
  const bool live = col < D;
  float* Xb = d.X + (int64_t)b * (P + 1) * D + col;
  const int64_t cbase = (int64_t)b * P * D + col;  // element offset of this column in the cache rows
  const int32_t* rk = d.rank + b * P;
  const int n_miss = d.ctl->n_miss;

  V<VEC> xcur{}, acc{}, comp{}, xfill{};
  if (live) xcur = ldv<VEC>(Xb + (int64_t)(t % (P + 1)) * D);
  acc = xcur;
  xfill = xcur;  // state e when e == t
  for (int j = 0; j < p; ++j) {
    const int i = t + j;
    const int r = rk[j];
    if (r >= n_miss) set_status(d.ctl, kDevBadRank);
    const float cm1 = d.cm1[i], ec = d.ecoef[i];
    const float sg = d.noise ? d.sigma[i] : 0.f;
    const int slot = i % P;
    float ev = 0.f, dv = 0.f;
    if (live) {
      V<VEC> eps = (r >= 0) ? ldv<VEC>(beps + (int64_t)r * D + col)
                            : ld_entry<VEC, CB>(d.Ehat, cbase + (int64_t)slot * D);
      if (r >= 0) {
        st_entry<VEC, CB>(d.Ehat, cbase + (int64_t)slot * D, eps);
        st_entry<VEC, CB>(d.Xhat, cbase + (int64_t)slot * D, xcur);
      }
      V<VEC> xo;
      if (i + 1 <= e) {
        xo = ldv<VEC>(Xb + (int64_t)((i + 1) % (P + 1)) * D);
        if (i + 1 == e) xfill = xo;
      } else {
        xo = xfill;
      }
      V<VEC> zn{};
      if (d.noise) zn = ldv<VEC>(d.noise + ((int64_t)b * d.T + i) * D + col);  // the draw z_i
      V<VEC> xn;
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        const float dr = fmaf(sg, zn.a[v], cm1 * xcur.a[v] + ec * eps.a[v]);
        const float y = dr - comp.a[v];
        const float s = acc.a[v] + y;
        comp.a[v] = (s - acc.a[v]) - y;
        acc.a[v] = s;
        xn.a[v] = s;
        const float df = xn.a[v] - xo.a[v];
        ev += df * df;
      }
      stv<VEC>(Xb + (int64_t)((i + 1) % (P + 1)) * D, xn);
      if (j + 1 < p) {
        const int r1 = rk[j + 1];
        V<VEC> xh = (r1 >= 0) ? as_entry<VEC, CB>(xo) : ld_entry<VEC, CB>(d.Xhat, cbase + (int64_t)((i + 1) % P) * D);
#pragma unroll
        for (int v = 0; v < VEC; ++v) dv += fabsf(xn.a[v] - xh.a[v]);
      }
      xcur = xo;
    }
    ev = warp_sum(ev);
    dv = warp_sum(dv);
    if (lane == 0) {
      red[warp * P + j] = ev;
      red[(nw + warp) * P + j] = dv;
    }
  }
  __syncthreads();
  for (int j = threadIdx.x; j < p; j += kPlainThreads) {
    float se = 0.f, sd = 0.f;
#pragma unroll
    for (int w = 0; w < nw; ++w) {
      se += red[w * P + j];
      sd += red[(nw + w) * P + j];
    }
    red_add(d, par, 0, b * P + j, se);
    red_add(d, par, 1, b * P + j, sd);
  }
}

// ---------------------------------------------------------------------------
// Planning kernel (a10, a2, a3 after iteration k, then a4 of iteration k+1),
// one launch. The update kernel left complete fp64 sums of the Eq. 2 errors
// and Eq. 4 distances; every CTA reads them (B*P of each), divides by D and
// takes the whole decision in shared memory -- the same inputs and the same
// arithmetic give the same plan in every CTA -- then copies the column range
// blockIdx.x of batch rows blockIdx.y, blockIdx.y + gridDim.y, ... that hold
// a miss (one row per CTA unless the rows outnumber one wave of CTAs). CTA (0, 0)
// also publishes the plan (copy par ^ 1 of the trajectories and counters,
// ranks, miss list, iteration log, the reductions for the host) and clears
// the accumulator set of iteration k+1. Nobody waits for anybody: the other
// CTAs read copy par of the plan, which no CTA writes in this launch.
constexpr int kPlanThreads = 256;
constexpr int kPlanPerSm = 2;   // planning CTAs per SM (three: the launch bound makes the decision spill, slower)
constexpr int kFusedMaxPairs = 1024;  // B*P planned in every CTA at most; beyond, one CTA plans
// Beyond this many pairs one CTA plans and a separate gather follows unless
// tau_cache adapts (only the every-CTA planner forms the next tau): at the SD
// latent with 800 and 1000 pairs that measured 49.9 and 59.8 us per solver
// step against 51.7 and 62.8 us, at 300 and 400 pairs 28.6 and 34.9 against
// 27.9 and 34.4 us
constexpr int kFusedPreferPairs = 512;
static_assert(kFusedMaxPairs <= 32 * 32, "decide_par keeps one miss mask per 32-position chunk, 32 of them");

// The complete sums read from global memory (one-CTA planner).
struct RedSums {
  const double* e;
  const double* dl;
  double inv_d, tol_d, thr_d;
  __device__ double err(int q) const { return __ldcg(e + (size_t)q * kAccStride) * inv_d; }
  __device__ double del(int q) const { return __ldcg(dl + (size_t)q * kAccStride) * inv_d; }
  __device__ bool conv(int q) const { return sum_le(__ldcg(e + (size_t)q * kAccStride), tol_d); }
  __device__ bool near(int q) const { return sum_lt(__ldcg(dl + (size_t)q * kAccStride), thr_d); }
};

// The miss of batch row r < ds.total from the decision's chunk bits: chunk c
// holds ranks cbase[c] .. cbase[c] + popc(cmiss[c]) - 1, in bit order. Every
// lane of a warp calls it and gets the same answer; false if no chunk holds
// row r (never expected).
__device__ __forceinline__ bool row_miss(const DecideShared& ds, int B, int P, int r, int* b, int* i) {
  const int lane = threadIdx.x & 31;
  const int nchunk = (B * P + 31) / 32;  // <= 32 (kFusedMaxPairs)
  const unsigned mm = lane < nchunk ? ds.cmiss[lane] : 0u;
  const int base = lane < nchunk ? ds.cbase[lane] : 0;
  const unsigned held = __ballot_sync(0xffffffffu, lane < nchunk && r >= base && r < base + __popc(mm));
  if (held == 0u) return false;
  const int c = __ffs(held) - 1;
  const unsigned m = __shfl_sync(0xffffffffu, mm, c);
  const int n = r - __shfl_sync(0xffffffffu, base, c);  // row r is the n-th miss of chunk c
  const unsigned at = __ballot_sync(0xffffffffu, ((m >> lane) & 1u) && __popc(m & ((1u << lane) - 1u)) == n);
  if (at == 0u) return false;
  const int q = c * 32 + __ffs(at) - 1;
  if (q >= B * P) return false;
  *b = q / P;
  *i = ds.tn[*b] + (q - *b * P);
  return true;
}

template <int VEC>
__global__ void __launch_bounds__(kPlanThreads, kPlanPerSm) k_plan_gather(Dev d, int par) {
  __shared__ DecideShared ds;
  const bool publish = blockIdx.x == 0 && blockIdx.y == 0;
  decide_load<kPlanThreads>(d, ds, par);
  pdl_wait();  // the sums and the new states come from the update kernel
  pdl_trigger();  // the successor may now run its prologue
  stage_decision_bits(d, ds, par, publish ? 0 : -1, 1);
  __syncthreads();  // the decision's input bits and decide_load's state are staged
  const bool one_row = (int)gridDim.y >= d.B * d.P;  // every batch row has its own CTA
  decide_par(d, ds, par, publish ? 0 : -1, 1, one_row ? (int)blockIdx.y : -1);
  __syncthreads();  // the plan (the batch rows of this CTA) is known
  if (one_row) {
    if ((int)blockIdx.y < ds.total && ds.target_b >= 0) {
      const int b = ds.target_b;
      copy_row<VEC>(d, b, min(ds.target_i, ds.en[b]), blockIdx.y);
    }
    return;
  }
  for (int r = blockIdx.y; r < ds.total; r += gridDim.y) {
    int b = 0, i = 0;
    if (!row_miss(ds, d.B, d.P, r, &b, &i)) {
      if (threadIdx.x == 0) set_status(d.ctl, kDevBadRank);
      continue;
    }
    copy_row<VEC>(d, b, min(i, ds.en[b]), r);
  }
}

// One-CTA planner for B*P beyond kFusedPreferPairs (without adaptation) or
// kFusedMaxPairs: reads the sums from memory; a separate gather follows.
constexpr int kPlanOneThreads = 1024;

__global__ void __launch_bounds__(kPlanOneThreads) k_plan_one(Dev d, int par) {
  __shared__ DecideShared ds;
  const int npair = d.B * d.P;
  decide_load<kPlanOneThreads>(d, ds, par);
  pdl_wait();  // the sums come from the update kernel
  pdl_trigger();  // the successor may now run its prologue
  const double* acc_e = d.acc + (size_t)(par * 2 + 0) * npair * kAccStride;
  const double* acc_d = d.acc + (size_t)(par * 2 + 1) * npair * kAccStride;
  const RedSums red{acc_e, acc_d, d.inv_d, d.tol_d, d.thr_d};
  decide_run<kPlanOneThreads>(d, ds, red, par, true, -1);
  double* nxt = d.acc + (size_t)((par ^ 1) * 2) * npair * kAccStride;
  for (int q = threadIdx.x; q < npair; q += kPlanOneThreads) {
    d.red_err[q] = (float)red.err(q);
    d.red_del[q] = (float)red.del(q);
    nxt[(size_t)q * kAccStride] = 0.0;
    nxt[((size_t)npair + q) * kAccStride] = 0.0;
  }
}

}  // namespace

namespace {
// No work: waits for its predecessor and lets its successor start, like the
// library's other kernels (programmatic dependent launch).
__global__ void k_gap() {
  pdl_wait();
  pdl_trigger();
}
}  // namespace

cudaError_t launch_gap(cudaStream_t st) { return launch_ex(k_gap, dim3(1), dim3(32), 0, st, 0); }

namespace {
dim3 gather_grid(const Dev& d) {
  const int rows = min(d.B * d.P, 65535);
  const int vec = (d.D % 4 == 0) ? 4 : 1;
  const int64_t nvec = d.D / vec;
  const int64_t want = (nvec + kGatherThreads * kGatherUnroll - 1) / (kGatherThreads * kGatherUnroll);
  return dim3((int)(want < 64 ? want : 64), rows);
}
}  // namespace

cudaError_t launch_gather(const Dev& d, int par, cudaStream_t st) {
  const dim3 g = gather_grid(d);
  if (d.D % 4 == 0) return launch_ex(k_gather<4>, g, dim3(kGatherThreads), 0, st, 0, d, par);
  return launch_ex(k_gather<1>, g, dim3(kGatherThreads), 0, st, 0, d, par);
}

namespace {
// The grid of a kernel whose CTA (x, y) copies part x of batch row y: as many
// parts per row as keep the grid within per_sm CTAs per SM (one wave), each
// part at least 1024 float4 columns; with more rows than one wave holds, one
// wave of whole-row CTAs, CTA y taking rows y, y + gridDim.y, ... An error
// only if the SM count cannot be read.
cudaError_t split_grid(const Dev& d, int per_sm, dim3* out) {
  static int nsm[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && nsm[dev] == 0) {
    e = cudaDeviceGetAttribute(&nsm[dev], cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const int sms = (dev >= 0 && dev < 64 && nsm[dev] > 0) ? nsm[dev] : 148;
  dim3 g = gather_grid(d);
  const int64_t nvec = d.D / ((d.D % 4 == 0) ? 4 : 1);
  const int64_t cap = (nvec + kGatherThreads * 4 - 1) / (kGatherThreads * 4);
  int64_t gx = (int64_t)per_sm * sms / (int)g.y;
  if (gx > cap) gx = cap;
  if (gx > 64) gx = 64;
  g.x = gx < 1 ? 1 : (unsigned)gx;
  // more rows than one wave of CTAs: one wave, each CTA taking every
  // gridDim.y-th row (the planning kernel then plans once per CTA, not per row)
  if ((int64_t)g.y > (int64_t)per_sm * sms) g.y = (unsigned)(per_sm * sms);
  *out = g;
  return cudaSuccess;
}
}  // namespace

cudaError_t launch_init(const Dev& d, cudaStream_t st) {
  dim3 g;
  const cudaError_t e = split_grid(d, kPlanPerSm, &g);
  if (e != cudaSuccess) return e;
  if (d.D % 4 == 0) return launch_ex(k_init<4>, g, dim3(kGatherThreads), 0, st, 0, d);
  return launch_ex(k_init<1>, g, dim3(kGatherThreads), 0, st, 0, d);
}

cudaError_t launch_plan(const Dev& d, int par, cudaStream_t st, int* launches) {
  const int npair = d.B * d.P;
  if (npair <= kFusedPreferPairs || (d.adapt && npair <= kFusedMaxPairs)) {
    *launches = 1;
    // every CTA plans and copies a part of its batch row
    dim3 g;
    const cudaError_t e = split_grid(d, kPlanPerSm, &g);
    if (e != cudaSuccess) return e;
    if (d.D % 4 == 0) return launch_ex(k_plan_gather<4>, g, dim3(kPlanThreads), 0, st, 0, d, par);
    return launch_ex(k_plan_gather<1>, g, dim3(kPlanThreads), 0, st, 0, d, par);
  }
  *launches = 2;
  cudaError_t e = launch_ex(k_plan_one, dim3(1), dim3(kPlanOneThreads), 0, st, 0, d, par);
  if (e != cudaSuccess) return e;
  return launch_gather(d, par ^ 1, st);
}

cudaError_t launch_update_plain(const Dev& d, const float* batch_eps, int par, cudaStream_t st) {
  const size_t smem = (size_t)2 * (kPlainThreads / 32) * d.P * sizeof(float);
  // float4 rows need every row base 16-byte aligned: D % 4 == 0 and aligned
  // eps (and draws) pointers; the workspace arrays are 256-byte aligned
  const bool aligned = (reinterpret_cast<uintptr_t>(batch_eps) & 15) == 0 &&
                       (reinterpret_cast<uintptr_t>(d.noise) & 15) == 0;
  if (d.D % 4 == 0 && aligned) {
    const int nchunk = (int)((d.D + kPlainThreads * 4 - 1) / (kPlainThreads * 4));
    if (d.cache_bf16)
      return launch_ex(k_update_plain<4, true>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps, par);
    return launch_ex(k_update_plain<4, false>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps, par);
  }
  const int nchunk = (int)((d.D + kPlainThreads - 1) / kPlainThreads);
  if (d.cache_bf16)
    return launch_ex(k_update_plain<1, true>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps, par);
  return launch_ex(k_update_plain<1, false>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps, par);
}

}  // namespace pa
