// Solver-step kernels for sm_103a: first-iteration plan, miss gather (a4),
// plain-load Picard update (a6-a9, a11) and the decision kernel (a10, a2, a3).
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
// First iteration (after pa_init): every timestep of every first window enters
// for the first time, hence is a miss (Sec. 2.2). States 1..p are lazy copies
// of state 0 = x_init, so the frontier e starts at 0.
__global__ void k_init_plan(Dev d) {
  const int p0 = min(d.P, d.T);
  for (int b = threadIdx.x; b < d.B; b += blockDim.x) {
    Traj tr{};
    tr.t = 0; tr.p = p0; tr.e = 0; tr.done = 0; tr.m = p0; tr.h1 = 0;
    d.traj[b] = tr;
  }
  for (int q = threadIdx.x; q < d.B * d.P; q += blockDim.x) {
    const int b = q / d.P, j = q % d.P;
    if (j < p0) {
      const int r = b * p0 + j;
      d.rank[q] = r;
      d.miss_bt[2 * r] = b;
      d.miss_bt[2 * r + 1] = j;
    } else {
      d.rank[q] = -1;
    }
  }
  if (threadIdx.x == 0) {
    Ctl c{};
    c.n_miss = d.B * p0;
    c.n_active = d.B;
    c.iter = 0;
    c.status = kDevOk;
    c.nfe = (long long)d.B * p0;
    c.hits = 0;
    *d.ctl = c;
  }
}

// ---------------------------------------------------------------------------
// a4: batch_x[r] <- x_{miss[r]} for r < n_miss. A lazy state (i > e) reads
// state e, the value every new tail state was initialised to. Each thread
// moves kGatherUnroll vectors per row with all loads issued before the stores.
constexpr int kGatherThreads = 256;
constexpr int kGatherUnroll = 4;

template <int VEC>
__global__ void __launch_bounds__(kGatherThreads) k_gather(Dev d) {
  using T = typename std::conditional<VEC == 4, float4, float>::type;
  pdl_wait();  // everything read here comes from the decision kernel
  const int n = d.ctl->n_miss;
  const int64_t nvec = d.D / VEC;
  const int64_t stride = (int64_t)gridDim.x * kGatherThreads;
  const int64_t base = (int64_t)blockIdx.x * kGatherThreads + threadIdx.x;
  for (int r = blockIdx.y; r < n; r += gridDim.y) {
    const int b = d.miss_bt[2 * r], i = d.miss_bt[2 * r + 1];
    const int src = min(i, d.traj[b].e);
    const T* from = reinterpret_cast<const T*>(d.X + ((int64_t)b * (d.P + 1) + src % (d.P + 1)) * d.D);
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
// Partials are reduced per CTA in a fixed order and written to
// part_*[b][j][chunk]; the decision kernel finishes the reduction.
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

constexpr int kPlainThreads = 128;

template <int VEC>
__global__ void __launch_bounds__(kPlainThreads) k_update_plain(Dev d, const float* __restrict__ beps,
                                                             int nchunk) {
  extern __shared__ float red[];  // [2][nwarps][P]
  const int b = blockIdx.y;
  pdl_wait();
  const Traj tr = d.traj[b];
  if (tr.p == 0) return;
  const int t = tr.t, p = tr.p, e = tr.e, P = d.P;
  const int64_t D = d.D;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int nw = kPlainThreads / 32;
  const int64_t col = ((int64_t)blockIdx.x * kPlainThreads + threadIdx.x) * VEC;
  const bool live = col < D;
  float* Xb = d.X + (int64_t)b * (P + 1) * D + col;
  float* Xh = d.Xhat + (int64_t)b * P * D + col;
  float* Eh = d.Ehat + (int64_t)b * P * D + col;
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
      V<VEC> eps = (r >= 0) ? ldv<VEC>(beps + (int64_t)r * D + col) : ldv<VEC>(Eh + (int64_t)slot * D);
      if (r >= 0) {
        stv<VEC>(Eh + (int64_t)slot * D, eps);
        stv<VEC>(Xh + (int64_t)slot * D, xcur);
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
        V<VEC> xh = (r1 >= 0) ? xo : ldv<VEC>(Xh + (int64_t)((i + 1) % P) * D);
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
    const int64_t o = ((int64_t)b * P + j) * nchunk + blockIdx.x;
    d.part_err[o] = se;
    d.part_del[o] = sd;
  }
}

// ---------------------------------------------------------------------------
// Decision kernel for the update kernels that leave the reductions unfinished
// (plain-load and tile forms), one launch of many CTAs: every CTA finishes
// some of the reductions -- one warp per (quantity, b, j) sums the chunk
// partials of err[b][j] (Eq. 2) or of the distance of timestep t+j+1 (Eq. 4)
// in a fixed order (deterministic), to red_* -- and the CTA that finishes
// last (atomic ticket after a fence; nobody waits) runs decide_plan.
constexpr int kDecideThreads = 256;
constexpr int kDecideSmemPairs = 6144;  // (b, j) pairs whose reductions are staged in shared memory

__global__ void __launch_bounds__(kDecideThreads) k_decide(Dev d, int nchunk) {
  __shared__ int s_last;
  __shared__ DecideShared ds;
  extern __shared__ float s_red[];  // [2][B*P] when B*P <= kDecideSmemPairs
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int nwarps = kDecideThreads / 32;
  const int npair = d.B * d.P;

  // every CTA stages the trajectories and counters (written by the previous
  // decision, several kernels back) before the dependency wait: whichever
  // CTA finishes last then decides without another round trip to memory
  decide_load<kDecideThreads>(d, ds);
  pdl_wait();  // the partials come from the update kernel
  const int item = blockIdx.x * nwarps + warp;
  if (item < 2 * npair) {
    const int which = item / npair, pr = item % npair;
    const float* src = (which ? d.part_del : d.part_err) + (int64_t)pr * nchunk;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    int c = lane;
    for (; c + 96 < nchunk; c += 128) {
      acc[0] += src[c];
      acc[1] += src[c + 32];
      acc[2] += src[c + 64];
      acc[3] += src[c + 96];
    }
    for (; c < nchunk; c += 32) acc[0] += src[c];
    float v = (acc[0] + acc[1]) + (acc[2] + acc[3]);
    v = warp_sum(v);
    if (lane == 0) (which ? d.red_del : d.red_err)[pr] = v / (float)d.D;
  }
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const unsigned int k = atomicAdd(&d.ctl->ticket, 1u);
    s_last = (k == gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();  // the other CTAs' reductions are visible from here on
  if (tid == 0) d.ctl->ticket = 0u;  // ready for the next launch
  const bool in_smem = npair <= kDecideSmemPairs;
  if (in_smem) {
    for (int q = tid; q < npair; q += kDecideThreads) {
      s_red[q] = __ldcg(d.red_err + q);
      s_red[npair + q] = __ldcg(d.red_del + q);
    }
  }
  __syncthreads();
  decide_run<kDecideThreads>(d, ds, in_smem ? s_red : d.red_err, in_smem ? s_red + npair : d.red_del);
}

}  // namespace

cudaError_t launch_init_plan(const Dev& d, cudaStream_t st) {
  k_init_plan<<<1, 256, 0, st>>>(d);
  return cudaGetLastError();
}

cudaError_t launch_gather(const Dev& d, cudaStream_t st) {
  const int rows = min(d.B * d.P, 65535);
  const int vec = (d.D % 4 == 0) ? 4 : 1;
  const int64_t nvec = d.D / vec;
  const int64_t want = (nvec + kGatherThreads * kGatherUnroll - 1) / (kGatherThreads * kGatherUnroll);
  const int gx = (int)(want < 64 ? want : 64);
  if (vec == 4) return launch_ex(k_gather<4>, dim3(gx, rows), dim3(kGatherThreads), 0, st, 0, d);
  return launch_ex(k_gather<1>, dim3(gx, rows), dim3(kGatherThreads), 0, st, 0, d);
}

cudaError_t launch_update_plain(const Dev& d, const float* batch_eps, cudaStream_t st,
                                int* nchunk_out) {
  const size_t smem = (size_t)2 * (kPlainThreads / 32) * d.P * sizeof(float);
  // float4 rows need every row base 16-byte aligned: D % 4 == 0 and aligned
  // eps (and draws) pointers; the workspace arrays are 256-byte aligned
  const bool aligned = (reinterpret_cast<uintptr_t>(batch_eps) & 15) == 0 &&
                       (reinterpret_cast<uintptr_t>(d.noise) & 15) == 0;
  if (d.D % 4 == 0 && aligned) {
    const int nchunk = (int)((d.D + kPlainThreads * 4 - 1) / (kPlainThreads * 4));
    *nchunk_out = nchunk;
    return launch_ex(k_update_plain<4>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps,
                     nchunk);
  } else {
    const int nchunk = (int)((d.D + kPlainThreads - 1) / kPlainThreads);
    *nchunk_out = nchunk;
    return launch_ex(k_update_plain<1>, dim3(nchunk, d.B), dim3(kPlainThreads), smem, st, 0, d, batch_eps,
                     nchunk);
  }
  return cudaGetLastError();
}

cudaError_t launch_decide(const Dev& d, int nchunk, cudaStream_t st) {
  const int pairs = d.B * d.P;
  const size_t smem = pairs <= kDecideSmemPairs ? (size_t)2 * pairs * sizeof(float) : 0;
  const int nwarps = kDecideThreads / 32;
  const int grid = (2 * pairs + nwarps - 1) / nwarps;
  return launch_ex(k_decide, dim3(grid), dim3(kDecideThreads), smem, st, 0, d, nchunk);
  return cudaGetLastError();
}

}  // namespace pa
