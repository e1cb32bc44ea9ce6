// The decision that ends one Picard iteration (a10, a2, a3), as a CTA-wide
// device function. Every CTA of the planning kernel runs it on the same
// inputs and reaches the same plan; one of them (publish) writes the plan to
// memory, the others keep what they need in shared memory (the batch row
// they gather).
#pragma once

#include "pa_internal.h"

namespace pa {

// Shared state of one decision (static shared memory of the calling kernel).
struct DecideShared {
  int t[kMaxBatch], p[kMaxBatch], e[kMaxBatch];
  int tn[kMaxBatch], pn[kMaxBatch], en[kMaxBatch], m[kMaxBatch], h1[kMaxBatch];
  int om[kMaxBatch], oh1[kMaxBatch];
  int warp_tot[32];
  unsigned cmiss[32], cwin[32];  // decide_par: miss / in-window bits of each 32-position chunk
  int cbase[32];                 // decide_par: misses before each chunk
  int pts;                       // decide_par: window positions planned
  int total, active, iter;
  long long nfe, hits;
  int target_b, target_i;  // the miss of the requested batch row, if any
};

// The plan of iteration k (copy par = k mod 2). It was written by the previous
// decision, several kernels back, so it may be read before the dependency
// wait. No barrier.
template <int NT>
__device__ void decide_load(const Dev& d, DecideShared& sh, int par) {
  const int tid = threadIdx.x;
  if (tid == 0) {
    const PlanCtr c = d.pc[par];
    sh.active = c.n_active;
    sh.iter = c.iter;
    sh.nfe = c.nfe;
    sh.hits = c.hits;
    sh.total = 0;
    sh.target_b = -1;
    sh.target_i = 0;
  }
  const Traj* tr0 = d.traj + par * d.B;
  for (int b = tid; b < d.B; b += NT) {
    const Traj tr = tr0[b];
    sh.t[b] = tr.t; sh.p[b] = tr.p; sh.e[b] = tr.e;
    sh.om[b] = tr.m; sh.oh1[b] = tr.h1;
    sh.m[b] = 0;
    sh.h1[b] = 0;
  }
}

// red_e[b*P + j]: Eq. 2 error of window position j of trajectory b (divided
// by D); red_d[b*P + j]: Eq. 4 distance of timestep t+j+1 (divided by D).
// Only positions j < p_b are read. With NT threads the CTA
//  1. per trajectory: stride = min(p, 1 + #leading err_j <= tol) (warp
//     ballots), advances t, shrinks p = min(P, T - t), sets the frontier
//     e = old t + p, done at t = T, and (publish) writes the iteration log;
//  2. plans the next iteration: a timestep of the new window with a cache
//     entry (i < e) hits iff delta < tau_cache (strict, Eq. 5), everything else
//     misses; misses are compacted trajectory-major with a block-wide prefix
//     sum; publish writes rank[b][j] (each miss's batch row) and miss_bt, and
//     every CTA notes the miss of batch row `target` (target_b, target_i);
//  3. publish writes the new trajectories and counters to copy par ^ 1 and
//     the host-visible counters.
// When no trajectory is active the plan is carried over unchanged. Starts
// with a barrier (after decide_load) and ends with one.
template <int NT, typename Red>
__device__ void decide_run(const Dev& d, DecideShared& sh, const Red& red, int par, bool publish, int target) {
  int* s_t = sh.t; int* s_p = sh.p; int* s_e = sh.e;
  int* s_tn = sh.tn; int* s_pn = sh.pn; int* s_m = sh.m; int* s_h1 = sh.h1;
  int* s_om = sh.om; int* s_oh1 = sh.oh1; int* s_warp = sh.warp_tot;
  constexpr int nwarps = NT / 32;
  static_assert(nwarps <= 32, "one warp scans the warp totals");
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int B = d.B, P = d.P, T = d.T;
  Traj* out_traj = d.traj + (par ^ 1) * B;
  __syncthreads();
  if (sh.active == 0) {  // finished: iterating further changes nothing
    if (publish) {
      const Traj* in_traj = d.traj + par * B;
      for (int b = tid; b < B; b += NT) out_traj[b] = in_traj[b];
      if (tid == 0) d.pc[par ^ 1] = d.pc[par];
    }
    for (int b = tid; b < B; b += NT) sh.en[b] = s_e[b];
    __syncthreads();
    return;
  }
  const int iter = sh.iter;

  // 1. window advance, one warp per trajectory
  for (int b = warp; b < B; b += nwarps) {
    const int t = s_t[b], p = s_p[b];
    if (p == 0) {
      if (lane == 0) {
        s_tn[b] = t; s_pn[b] = 0;
        if (publish) {
          int32_t* lg = d.iter_log + ((int64_t)iter * B + b) * kLogFields;
          for (int f = 0; f < kLogFields; ++f) lg[f] = 0;
          lg[0] = t;
        }
      }
      continue;
    }
    int lead = p;
    for (int j0 = 0; j0 < p; j0 += 32) {
      const int j = j0 + lane;
      const bool fail = (j < p) && !(red.err(b * P + j) <= d.tol);
      const unsigned m = __ballot_sync(0xffffffffu, fail);
      if (m) {
        lead = j0 + __ffs(m) - 1;
        break;
      }
    }
    if (lane == 0) {
      const int stride = min(p, 1 + lead);
      const int tn = t + stride;
      s_tn[b] = tn;
      s_pn[b] = min(P, T - tn);
      if (publish) {
        int32_t* lg = d.iter_log + ((int64_t)iter * B + b) * kLogFields;
        lg[0] = t; lg[1] = p; lg[2] = s_om[b]; lg[3] = stride;
        lg[4] = s_e[b]; lg[5] = s_oh1[b]; lg[6] = 0; lg[7] = 0;
      }
    }
  }
  __syncthreads();

  // 2. hit/miss plan of the next iteration and its compaction
  const int N = B * P;
  const int per = (N + NT - 1) / NT;
  const int q0 = tid * per, q1 = min(N, q0 + per);
  auto is_miss = [&](int q) -> int {
    const int b = q / P, j = q % P;
    if (j >= s_pn[b]) return 0;
    const int i = s_tn[b] + j;
    const int en = s_t[b] + s_p[b];  // new frontier
    if (i >= en) return 1;           // first entry
    const int jo = i - s_t[b] - 1;   // delta of timestep i was computed at old position jo
    return (red.del(b * P + jo) < d.cache_thresh) ? 0 : 1;
  };
  int cnt = 0;
  for (int q = q0; q < q1; ++q) cnt += is_miss(q);
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int w = lane < nwarps ? s_warp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += v;
    }
    if (lane < nwarps) s_warp[lane] = wi - w;  // exclusive
    if (lane == 31) sh.total = wi;
  }
  __syncthreads();
  int r = s_warp[warp] + incl - cnt;
  if (target >= r && target < r + cnt) {  // the requested batch row is one of this thread's misses
    int rr = r;
    for (int q = q0; q < q1; ++q) {
      if (!is_miss(q)) continue;
      if (rr == target) {
        sh.target_b = q / P;
        sh.target_i = s_tn[q / P] + q % P;
      }
      ++rr;
    }
  }
  if (publish) {
    for (int q = q0; q < q1; ++q) {
      const int b = q / P, j = q % P;
      if (is_miss(q)) {
        d.rank[q] = r;
        d.miss_bt[2 * r] = b;
        d.miss_bt[2 * r + 1] = s_tn[b] + j;
        atomicAdd(&s_m[b], 1);
        ++r;
      } else {
        d.rank[q] = -1;
        if (j >= 1 && j < s_pn[b]) atomicAdd(&s_h1[b], 1);
      }
    }
  }
  for (int b = tid; b < B; b += NT) sh.en[b] = (s_p[b] > 0) ? s_t[b] + s_p[b] : s_e[b];
  __syncthreads();

  // 3. trajectories and counters of the next iteration
  if (publish) {
    int pts = 0;
    for (int b = 0; b < B; ++b) pts += s_pn[b];
    for (int b = tid; b < B; b += NT) {
      Traj tr{};
      tr.t = s_tn[b];
      tr.p = s_pn[b];
      tr.e = sh.en[b];
      tr.done = (s_pn[b] == 0);
      tr.m = s_m[b];
      tr.h1 = s_h1[b];
      if (tr.t > T || tr.e < tr.t) atomicCAS(&d.ctl->status, kDevOk, kDevBadState);
      out_traj[b] = tr;
    }
    if (tid == 0) {
      int act = 0;
      for (int b = 0; b < B; ++b) act += (s_pn[b] > 0);
      const int n = sh.total;
      PlanCtr c;
      c.n_active = act;
      c.iter = iter + 1;
      c.nfe = sh.nfe + n;
      c.hits = sh.hits + (pts - n);
      d.pc[par ^ 1] = c;
      d.ctl->n_miss = n;
      d.ctl->n_active = act;
      d.ctl->iter = c.iter;
      d.ctl->nfe = c.nfe;
      d.ctl->hits = c.hits;
    }
  }
}

// The same decision with all warps of the CTA at work, for the planning
// kernel in which every CTA decides (B*P <= 32 * 32): warp w advances the
// windows of trajectories w, w + NW, ...; warp w tests the 32-position chunks
// w, w + NW, ... of the next windows; one warp turns the chunks' miss counts
// into each chunk's first rank; the chunks then place their misses. Gives the
// same plan, ranks and counters as decide_run. Every thread of
// the CTA calls it (it holds CTA barriers); the caller synchronises the CTA
// afterwards.
template <typename Red>
__device__ void decide_par(const Dev& d, DecideShared& sh, const Red& red, int par, bool publish, int target) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  const int B = d.B, P = d.P, T = d.T;
  Traj* out_traj = d.traj + (par ^ 1) * B;
  if (sh.active == 0) {  // finished: the plan carries over (uniform across the CTA)
    if (warp == 0) {
      if (publish) {
        const Traj* in_traj = d.traj + par * B;
        for (int b = lane; b < B; b += 32) out_traj[b] = in_traj[b];
        if (lane == 0) d.pc[par ^ 1] = d.pc[par];
      }
      for (int b = lane; b < B; b += 32) sh.en[b] = sh.e[b];
    }
    return;
  }
  const int iter = sh.iter;
  // 1. window advance, one warp per trajectory
  for (int b = warp; b < B; b += nw) {
    const int t = sh.t[b], p = sh.p[b];
    int stride = 0;
    if (p > 0) {
      int lead = p;
      for (int j0 = 0; j0 < p; j0 += 32) {
        const int j = j0 + lane;
        const unsigned m = __ballot_sync(0xffffffffu, (j < p) && !(red.err(b * P + j) <= d.tol));
        if (m) {
          lead = j0 + __ffs(m) - 1;
          break;
        }
      }
      stride = min(p, 1 + lead);
    }
    if (lane == 0) {
      const int tn = t + stride;
      sh.tn[b] = tn;
      sh.pn[b] = p > 0 ? min(P, T - tn) : 0;
      sh.en[b] = p > 0 ? t + p : sh.e[b];
      if (publish) {
        int32_t* lg = d.iter_log + ((int64_t)iter * B + b) * kLogFields;
        if (p > 0) {
          lg[0] = t; lg[1] = p; lg[2] = sh.om[b]; lg[3] = stride;
          lg[4] = sh.e[b]; lg[5] = sh.oh1[b]; lg[6] = 0; lg[7] = 0;
        } else {
          for (int f = 0; f < kLogFields; ++f) lg[f] = 0;
          lg[0] = t;
        }
      }
    }
  }
  __syncthreads();
  // 2. hit/miss tests of the next windows, one warp per 32-position chunk
  const int N = B * P, nchunk = (N + 31) / 32;
  for (int c = warp; c < nchunk; c += nw) {
    const int q = c * 32 + lane;
    int miss = 0, inwin = 0;
    if (q < N) {
      const int b = q / P, j = q % P;
      if (j < sh.pn[b]) {
        inwin = 1;
        const int i = sh.tn[b] + j;
        const int en = sh.t[b] + sh.p[b];  // new frontier
        if (i >= en) {
          miss = 1;                        // first entry
        } else {
          const int jo = i - sh.t[b] - 1;  // delta of timestep i was computed at old position jo
          miss = (red.del(b * P + jo) < d.cache_thresh) ? 0 : 1;
        }
      }
    }
    const unsigned mm = __ballot_sync(0xffffffffu, miss), wm = __ballot_sync(0xffffffffu, inwin);
    if (lane == 0) {
      sh.cmiss[c] = mm;
      sh.cwin[c] = wm;
    }
  }
  __syncthreads();
  // each chunk's first rank: an exclusive scan of the chunks' miss counts
  if (warp == 0) {
    const int cnt = lane < nchunk ? __popc(sh.cmiss[lane]) : 0;
    const int win = lane < nchunk ? __popc(sh.cwin[lane]) : 0;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane < nchunk) sh.cbase[lane] = incl - cnt;
    const int pts = __reduce_add_sync(0xffffffffu, win);
    if (lane == 31) sh.total = incl;
    if (lane == 0) sh.pts = pts;
  }
  __syncthreads();
  // 3. the misses' ranks (trajectory-major, ascending t), the requested row
  for (int c = warp; c < nchunk; c += nw) {
    const int q = c * 32 + lane;
    if (q >= N) continue;
    const unsigned mm = sh.cmiss[c];
    const int miss = (mm >> lane) & 1u;
    const int b = q / P, j = q % P;
    const int r = sh.cbase[c] + __popc(mm & ((1u << lane) - 1u));
    if (miss && r == target) {
      sh.target_b = b;
      sh.target_i = sh.tn[b] + j;
    }
    if (publish) {
      if (miss) {
        d.rank[q] = r;
        d.miss_bt[2 * r] = b;
        d.miss_bt[2 * r + 1] = sh.tn[b] + j;
        atomicAdd(&sh.m[b], 1);
      } else {
        d.rank[q] = -1;
        if (((sh.cwin[c] >> lane) & 1u) && j >= 1) atomicAdd(&sh.h1[b], 1);
      }
    }
  }
  if (publish) {
    __syncthreads();
    // 4. trajectories and counters of the next iteration
    for (int b = tid; b < B; b += blockDim.x) {
      Traj tr{};
      tr.t = sh.tn[b];
      tr.p = sh.pn[b];
      tr.e = sh.en[b];
      tr.done = (sh.pn[b] == 0);
      tr.m = sh.m[b];
      tr.h1 = sh.h1[b];
      if (tr.t > T || tr.e < tr.t) atomicCAS(&d.ctl->status, kDevOk, kDevBadState);
      out_traj[b] = tr;
    }
    if (tid == 0) {
      int act = 0;
      for (int b = 0; b < B; ++b) act += (sh.pn[b] > 0);
      const int base = sh.total;
      PlanCtr cc;
      cc.n_active = act;
      cc.iter = iter + 1;
      cc.nfe = sh.nfe + base;
      cc.hits = sh.hits + (sh.pts - base);
      d.pc[par ^ 1] = cc;
      d.ctl->n_miss = base;
      d.ctl->n_active = act;
      d.ctl->iter = cc.iter;
      d.ctl->nfe = cc.nfe;
      d.ctl->hits = cc.hits;
    }
  }
}

}  // namespace pa
