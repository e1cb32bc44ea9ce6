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
  int stride[kMaxBatch], nh[kMaxBatch];  // decide_par: window advance and next-window positions with an entry
  int one[kMaxBatch], onh[kMaxBatch];    // the planned iteration's positions with an entry, and hits among them
  double tau[kMaxBatch];                 // tau_cache per trajectory: of the planned iteration, then of the next
  double thr[kMaxBatch];                 // the next hit test's bound on the undivided sums, tau * D
  double del[32 * 32];                   // with adaptation: the Eq. 4 sums themselves
  int warp_tot[32];
  unsigned cmiss[32], cwin[32];  // decide_par: miss / in-window bits of each 32-position chunk
  unsigned conv[32], near[32];   // decide_par's inputs as bits: Eq. 2 error <= tol, Eq. 4 distance < tau_cache
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
    sh.one[b] = tr.ne; sh.onh[b] = tr.nh;
    sh.m[b] = 0;
    sh.h1[b] = 0;
    sh.tau[b] = d.adapt ? d.tau[par * d.B + b] : d.cache_thresh;
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
      const bool fail = (j < p) && !red.conv(b * P + j);
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
    return red.near(b * P + jo) ? 0 : 1;
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

// Set bits of the bit string w (bit q of the string = bit q & 31 of word
// q >> 5) in positions [lo, hi).
__device__ __forceinline__ int range_popc(const unsigned* w, int lo, int hi) {
  int n = 0;
  while (lo < hi) {
    const int c = lo >> 5, o = lo & 31;
    const int take = min(32 - o, hi - lo);
    const unsigned m = (take == 32 ? 0xffffffffu : ((1u << take) - 1u)) << o;
    n += __popc(w[c] & m);
    lo += take;
  }
  return n;
}

// Bits [pos, pos + 32) of a bit string of 32 words (bits past the last word read as 0).
__device__ __forceinline__ unsigned bits32(const unsigned* w, int pos) {
  const int c = pos >> 5, o = pos & 31;
  unsigned v = c < 32 ? w[c] >> o : 0u;
  if (o && c + 1 < 32) v |= w[c + 1] << (32 - o);
  return v;
}

// The decision that ends an iteration, for kernels in which every CTA decides
// (B*P <= 32 * 32), from the bit strings that stage_decision_bits left in
// sh.conv (bit b*P + j: the Eq. 2 error of window position j of trajectory b
// is <= tol) and sh.near (bit b*P + j: the Eq. 4 distance of timestep
// t_b + j + 1 is < tau_cache). Warp 0 alone takes it with bit operations:
//  1. lane b advances trajectory b: stride = min(p, 1 + leading ones of its
//     conv bits), t' = t + stride, p' = min(P, T - t'), frontier e' = t + p;
//     with adaptation on, lane b also forms trajectory b's tau_cache for the
//     next hit test from the planned iteration's hit rate and the stride;
//  2. the next windows' bits, one ballot per 32-position chunk: position j'
//     of trajectory b (timestep i = t' + j') is in the window for j' < p';
//     it has an entry iff i < t + p, i.e. j' < p - stride, and then hits iff
//     the distance computed at position j' + stride - 1 is below tau_cache
//     (Eq. 5, strict; the near bit, or the sum against tau * D when tau
//     adapts); all other window positions miss;
//  3. lane c turns the miss counts of 32-position chunk c into its first rank
//     (an exclusive scan): misses are ranked trajectory-major, ascending t.
// Then, after one CTA barrier, every warp handles chunks: the ranks and the
// miss list are written by publishing CTAs (chunk c by the CTA whose pub_id is
// c mod pub_count; pub_id < 0 writes nothing) and every CTA notes the miss of
// batch row `target` (target_b, target_i); the CTA with pub_id 0 also writes
// the trajectories, counters and iteration log. Gives the same plan, ranks and
// counters as decide_run. Every thread of the CTA calls it; the caller
// synchronises the CTA afterwards.
__device__ inline void decide_par(const Dev& d, DecideShared& sh, int par, int pub_id, int pub_count, int target) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  const int B = d.B, P = d.P, T = d.T;
  const int N = B * P, nchunk = (N + 31) / 32;
  Traj* out_traj = d.traj + (par ^ 1) * B;
  if (sh.active == 0) {  // finished: the plan carries over (uniform across the CTA)
    if (warp == 0) {
      if (pub_id == 0) {
        const Traj* in_traj = d.traj + par * B;
        for (int b = lane; b < B; b += 32) {
          out_traj[b] = in_traj[b];
          if (d.adapt) d.tau[(par ^ 1) * B + b] = d.tau[par * B + b];
        }
        if (lane == 0) d.pc[par ^ 1] = d.pc[par];
      }
      for (int b = lane; b < B; b += 32) sh.en[b] = sh.e[b];
    }
    return;
  }
  const int iter = sh.iter;
  if (warp == 0) {
    for (int b = lane; b < B; b += 32) {
      const int t = sh.t[b], p = sh.p[b];
      int stride = 0;
      if (p > 0) {
        int lead = 0;
        while (lead < p) {
          const unsigned w = bits32(sh.conv, b * P + lead);
          const int ones = w == 0xffffffffu ? 32 : __ffs(~w) - 1;
          lead += ones;
          if (ones < 32) break;
        }
        stride = min(p, 1 + min(lead, p));
      }
      const int tn = t + stride, pn = p > 0 ? min(P, T - tn) : 0;
      sh.tn[b] = tn;
      sh.pn[b] = pn;
      sh.en[b] = p > 0 ? t + p : sh.e[b];
      sh.stride[b] = stride;
      sh.nh[b] = p > 0 ? p - stride : 0;  // next-window positions with a cache entry
      if (d.adapt) {
        // tau_cache of the next hit test, from the planned iteration's hit
        // rate among positions with an entry and its stride: below the
        // target rate tau rises by (1 + rate) if the window advanced beyond
        // its first position, else holds; at or above it falls by (1 + rate);
        // kept within [tau_min, tau_max]; no entries: tau holds
        double tau = sh.tau[b];
        const int ne = sh.one[b], nh = sh.onh[b];
        if (p > 0 && ne > 0) {
          if ((double)nh / (double)ne < d.adapt_target) {
            if (stride > 1) tau = fmin(tau * d.adapt_up, d.tau_max);
          } else {
            tau = fmax(tau / d.adapt_up, d.tau_min);
          }
        }
        sh.tau[b] = tau;
        sh.thr[b] = tau * (double)d.D;
      }
      if (pub_id == 0) {
        int32_t* lg = d.iter_log + ((int64_t)iter * B + b) * kLogFields;
        if (p > 0) {
          lg[0] = t; lg[1] = p; lg[2] = sh.om[b]; lg[3] = stride;
          lg[4] = sh.e[b]; lg[5] = sh.oh1[b]; lg[6] = sh.one[b]; lg[7] = sh.onh[b];
        } else {
          for (int f = 0; f < kLogFields; ++f) lg[f] = 0;
          lg[0] = t;
        }
      }
    }
    __syncwarp();
    // the next windows' bits, one 32-position chunk per ballot: position j'
    // of trajectory b is in the window for j' < p', has an entry for
    // j' < nh (= p - stride) and then hits iff the Eq. 4 distance computed at
    // position j' + stride - 1 is below the bound (Eq. 5, strict)
    for (int c = 0; c < nchunk; ++c) {
      const int q = c * 32 + lane;
      bool win = false, miss = false;
      if (q < N) {
        const int b = q / P, jn = q - b * P;
        if (jn < sh.pn[b]) {
          win = true;
          bool hit = false;
          if (jn < sh.nh[b]) {
            const int qo = b * P + jn + sh.stride[b] - 1;
            hit = d.adapt ? sum_lt(sh.del[qo], sh.thr[b]) : ((sh.near[qo >> 5] >> (qo & 31)) & 1u);
          }
          miss = !hit;
        }
      }
      const unsigned wm = __ballot_sync(0xffffffffu, win), mm = __ballot_sync(0xffffffffu, miss);
      if (lane == 0) {
        sh.cwin[c] = wm;
        sh.cmiss[c] = mm;
      }
    }
    __syncwarp();
    const int cnt = lane < nchunk ? __popc(sh.cmiss[lane]) : 0;
    const int win = lane < nchunk ? __popc(sh.cwin[lane]) : 0;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    sh.cbase[lane] = incl - cnt;
    const int pts = __reduce_add_sync(0xffffffffu, win);
    if (lane == 31) sh.total = incl;
    if (lane == 0) sh.pts = pts;
  }
  __syncthreads();
  // the misses' ranks and miss list (trajectory-major, ascending t), the requested row
  for (int c = warp; c < nchunk; c += nw) {
    const bool writes = pub_id >= 0 && c % pub_count == pub_id;
    if (!writes && target < 0) continue;
    const int q = c * 32 + lane;
    if (q >= N) continue;
    const unsigned mm = sh.cmiss[c];
    const int miss = (mm >> lane) & 1u;
    const int b = q / P, j = q - b * P;
    const int r = sh.cbase[c] + __popc(mm & ((1u << lane) - 1u));
    if (miss && r == target) {
      sh.target_b = b;
      sh.target_i = sh.tn[b] + j;
    }
    if (writes) {
      if (miss) {
        d.rank[q] = r;
        d.miss_bt[2 * r] = b;
        d.miss_bt[2 * r + 1] = sh.tn[b] + j;
      } else {
        d.rank[q] = -1;
      }
    }
  }
  if (pub_id == 0) {
    // trajectories and counters of the next iteration; a trajectory's misses
    // and its hits at positions >= 1 come from the chunk bits
    for (int b = tid; b < B; b += blockDim.x) {
      Traj tr{};
      tr.t = sh.tn[b];
      tr.p = sh.pn[b];
      tr.e = sh.en[b];
      tr.done = (sh.pn[b] == 0);
      tr.m = range_popc(sh.cmiss, b * P, b * P + sh.pn[b]);
      tr.h1 = sh.pn[b] > 1 ? (sh.pn[b] - 1) - range_popc(sh.cmiss, b * P + 1, b * P + sh.pn[b]) : 0;
      tr.ne = sh.nh[b];
      tr.nh = sh.nh[b] - range_popc(sh.cmiss, b * P, b * P + sh.nh[b]);
      if (d.adapt) d.tau[(par ^ 1) * B + b] = sh.tau[b];
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

// The decision's inputs as bits in shared memory (sh.conv, sh.near), from the
// complete fp64 sums of iteration par (divided by D): every thread of the CTA
// takes positions tid, tid + blockDim.x, ... and each warp's ballot is the
// bit word of its 32 consecutive positions. When `keep` is set, the CTA also
// writes the reductions of positions q with q mod pub_count == pub_id for the
// host and clears them in the next iteration's accumulator set. The caller
// synchronises the CTA before reading the bits.
__device__ __forceinline__ void stage_decision_bits(const Dev& d, DecideShared& sh, int par, int pub_id,
                                                    int pub_count) {
  const int tid = threadIdx.x, lane = tid & 31;
  const int npair = d.B * d.P;
  const double* acc_e = d.acc + (size_t)(par * 2 + 0) * npair * kAccStride;
  const double* acc_d = d.acc + (size_t)(par * 2 + 1) * npair * kAccStride;
  double* nxt = d.acc + (size_t)((par ^ 1) * 2) * npair * kAccStride;  // iteration k+1 adds into these
  for (int base = 0; base < npair; base += blockDim.x) {  // blockDim.x is a multiple of 32
    const int q = base + tid;
    bool cv = false, nr = false;
    if (q < npair) {
      const size_t o = (size_t)q * kAccStride;
      const double se = __ldcg(acc_e + o), sd = __ldcg(acc_d + o);
      cv = sum_le(se, d.tol_d);
      nr = sum_lt(sd, d.thr_d);
      if (d.adapt) sh.del[q] = sd;  // the bound is known only once the windows have advanced
      if (pub_id >= 0 && q % pub_count == pub_id) {
        d.red_err[q] = (float)(se * d.inv_d);
        d.red_del[q] = (float)(sd * d.inv_d);
        nxt[o] = 0.0;
        nxt[(size_t)npair * kAccStride + o] = 0.0;
      }
    }
    const unsigned cm = __ballot_sync(0xffffffffu, cv), nm = __ballot_sync(0xffffffffu, nr);
    if (lane == 0 && q < npair) {
      sh.conv[q >> 5] = cm;
      sh.near[q >> 5] = nm;
    }
  }
}


}  // namespace pa
