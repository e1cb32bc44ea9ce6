// Triangular Anderson mixing of a Picard iteration (ParaTAA-style, sm_103a):
// the second half of an iteration whose first half is the lean update in its
// mixing form (k_update_lean.cu, TAA), which left, for every window state
// s = t + j + 1, the Picard map's value G_s (Eq. 1) and the residual
// R_s = G_s - X_s by iteration parity, and the Gram sums <dR, R>, <dR, dR> of
// every window position (dR = R_s - R'_s against the previous iteration).
//
// One CTA takes a column chunk of one window position j of one trajectory:
//   gamma_j = sum_{j' <= j} <dR, R> / sum_{j' <= j} <dR, dR>   (0 for a zero
//             denominator), the least-squares coefficient over the position
//             and the earlier ones (lower triangular in time); position 0 and
//             states without a history (state > e, not computed in the
//             previous iteration) are not mixed: gamma = 0;
//   X_s    <- G_s - gamma_j (G_s - G'_s);
// and, with the new state in registers, the Eq. 2 term (X_s - X_s old)^2 and
// the Eq. 4 term |X_s - xhat_s| of the next iteration (xhat_s: the entry of
// timestep s, which the update kernel has just set to the old state if
// position j+1 missed), summed over the CTA in a fixed order and added into
// the iteration's accumulators for the planning kernel's decision.
#include "pa_internal.h"

namespace pa {
namespace {

constexpr int kMixThreads = 256;
constexpr int kMixUnroll = 4;   // float4 vectors per thread: a CTA covers 4096 columns

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }

__global__ void __launch_bounds__(kMixThreads) k_taa_mix(Dev d, int par) {
  __shared__ double s_nu[32], s_de[32];
  __shared__ float s_red[2][kMixThreads / 32];
  __shared__ float s_gamma;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int j = blockIdx.y, b = blockIdx.z, P = d.P;
  const int64_t D = d.D;
  // written two or more kernels back: the plan and the next position's rank
  const Traj tr = d.traj[par * d.B + b];
  const int rank_next = j + 1 < P ? d.rank[b * P + j + 1] : -1;
  pdl_wait();     // G, R, the Gram sums and the cache entries come from the update kernel
  pdl_trigger();  // the successor may now run its prologue
  if (j >= tr.p) return;
  const int t = tr.t, p = tr.p, e = tr.e;
  const int s = t + j + 1;              // the state this CTA mixes
  const bool mix = j >= 1 && s <= e;    // it has a history and is not the window's first state
  if (warp == 0) {
    double nu = 0.0, de = 0.0;
    if (mix) {  // positions 0..j all have a history when j has one
      const double* acc_n = d.taa_acc + (size_t)(par * 2 + 0) * d.B * P * kAccStride;
      const double* acc_d = d.taa_acc + (size_t)(par * 2 + 1) * d.B * P * kAccStride;
      for (int q = lane; q <= j; q += 32) {
        nu += __ldcg(acc_n + (size_t)(b * P + q) * kAccStride);
        de += __ldcg(acc_d + (size_t)(b * P + q) * kAccStride);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      nu += __shfl_xor_sync(0xffffffffu, nu, o);
      de += __shfl_xor_sync(0xffffffffu, de, o);
    }
    if (lane == 0) s_gamma = (mix && de > 0.0) ? (float)(nu / de) : 0.f;
  }
  __syncthreads();
  const float gam = s_gamma;
  const int slot = s % (P + 1);
  const float* G = d.taa_g + ((int64_t)par * d.B + b) * (P + 1) * D + (int64_t)slot * D;
  const float* Gp = d.taa_g + ((int64_t)(par ^ 1) * d.B + b) * (P + 1) * D + (int64_t)slot * D;
  float* Xs = d.X + ((int64_t)b * (P + 1) + slot) * D;
  // the old state: its own slot, which only this CTA's columns write; a lazy
  // state (past e) is state e, whose slot the CTA of state e overwrites in
  // this launch, so it reads the copy the update kernel kept
  const float* Xo = s <= e ? d.X + ((int64_t)b * (P + 1) + slot) * D : d.taa_xe + (int64_t)b * D;
  const float* Xh = d.Xhat + ((int64_t)b * P + s % P) * D;  // entry of timestep s (used when j + 1 < p)
  const bool want_dl = j + 1 < p;
  const bool dl_from_old = rank_next >= 0;  // position j+1 missed: its entry is the old state
  const bool use_gp = mix && gam != 0.f;
  const int64_t nvec = D / 4;
  const int64_t v0 = (int64_t)blockIdx.x * kMixThreads * kMixUnroll + tid;
  float ev = 0.f, dv = 0.f;
  float4 g[kMixUnroll], gp[kMixUnroll], xo[kMixUnroll], xh[kMixUnroll];
#pragma unroll
  for (int u = 0; u < kMixUnroll; ++u) {
    const int64_t v = v0 + (int64_t)u * kMixThreads;
    if (v < nvec) {
      g[u] = ld4(G + 4 * v);
      xo[u] = ld4(Xo + 4 * v);
      if (use_gp) gp[u] = ld4(Gp + 4 * v);
      if (want_dl && !dl_from_old) xh[u] = ld4(Xh + 4 * v);
    }
  }
#pragma unroll
  for (int u = 0; u < kMixUnroll; ++u) {
    const int64_t v = v0 + (int64_t)u * kMixThreads;
    if (v >= nvec) break;
    float4 xn = g[u];
    if (use_gp) {
      xn.x = fmaf(-gam, g[u].x - gp[u].x, g[u].x);
      xn.y = fmaf(-gam, g[u].y - gp[u].y, g[u].y);
      xn.z = fmaf(-gam, g[u].z - gp[u].z, g[u].z);
      xn.w = fmaf(-gam, g[u].w - gp[u].w, g[u].w);
    }
    st4(Xs + 4 * v, xn);
    const float ax = xn.x - xo[u].x, ay = xn.y - xo[u].y, az = xn.z - xo[u].z, aw = xn.w - xo[u].w;
    ev += (ax * ax + ay * ay) + (az * az + aw * aw);
    if (want_dl) {
      const float4 r = dl_from_old ? xo[u] : xh[u];
      dv += (fabsf(xn.x - r.x) + fabsf(xn.y - r.y)) + (fabsf(xn.z - r.z) + fabsf(xn.w - r.w));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ev += __shfl_xor_sync(0xffffffffu, ev, o);
    dv += __shfl_xor_sync(0xffffffffu, dv, o);
  }
  if (lane == 0) {
    s_red[0][warp] = ev;
    s_red[1][warp] = dv;
  }
  __syncthreads();
  if (tid < 2) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kMixThreads / 32; ++w) sum += s_red[tid][w];
    red_add(d, par, tid, b * P + j, sum);
    if (blockIdx.x == 0)  // the next iteration adds its Gram sums into the other set
      d.taa_acc[((size_t)((par ^ 1) * 2 + tid) * d.B * P + b * P + j) * kAccStride] = 0.0;
  }
}

}  // namespace

cudaError_t launch_taa_mix(const Dev& d, int par, cudaStream_t st) {
  const int64_t nvec = d.D / 4;
  const int nchunk = (int)((nvec + kMixThreads * kMixUnroll - 1) / (kMixThreads * kMixUnroll));
  return launch_ex(k_taa_mix, dim3(nchunk, d.P, d.B), dim3(kMixThreads), 0, st, 0, d, par);
}

}  // namespace pa
