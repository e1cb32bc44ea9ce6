// Picard update kernel, lean register form (sm_103a).
//
// The same step as the other update kernels (k_solver.cu, k_update_bulk.cu):
// for window position j (timestep i = t + j) Eq. 6 assembly, Eq. 7 cache
// update of a miss, the drift d_j = (c_i - 1) x_i + e_i eps_i (+ sigma_i z_i
// for stochastic steps) at the current latent, the window prefix sum of Eq. 1
// (x_{i+1} = x_t + sum_{q <= j} d_q), the Eq. 2 error term of state i+1 and the
// Eq. 4 distance term of timestep i+1 for the next iteration, with per-CTA
// sums added into the iteration's fp64 accumulators.
//
// Shaped for few instructions per element and many resident warps:
//  - a CTA owns a strip of 128 columns (4 per lane, 16-byte loads) of one
//    trajectory; its NW warps take contiguous runs of at most LMAX positions
//    (two passes joined by one CTA barrier: run totals, then the carry and
//    the new states);
//  - the step coefficients of every timestep are staged in shared memory
//    together with the ranks, before the plan is known, so the row loads
//    follow the plan load directly;
//  - hit/miss flags are warp-uniform bit masks; a lazy state (i > e) is read
//    from the row of state e, so no value selects; loops over a warp's
//    positions leave at its run length instead of predicating LMAX bodies;
//  - the window start x_t enters the run totals of warp 0, so later warps
//    need no copy of it;
//  - COMP carries every sum as an fp32 (hi, lo) pair (TwoSum); without it the
//    sums are plain fp32 (fewer instructions, rounding of a 100-term fp32 sum);
//  - CB stores the cache entries as bfloat16 (rounded to nearest even when
//    written, widened exactly when read).
// MINB CTAs per SM bound the registers: one CTA of 16 warps for windows up to
// 112 positions, two of 8 warps up to 64, three of 8 warps up to 32.
//
// TAA makes it the first half of a triangularly Anderson-mixed iteration
// (launch_update_taa): the prefix sum is the Picard map's output G of every
// window state; G and the residual R = G - X are stored by iteration parity
// (not the states: the mix kernel forms those), and each CTA adds its partials
// of <dR, R> and <dR, dR> (dR = R - R of the previous iteration, for states
// that have one) into the Gram sums instead of the Eq. 2 / Eq. 4 terms.
//
// FUSE makes it the whole solver step of one iteration (launch_step_fused):
// after the strip sums are added, a grid barrier (every CTA resident, a
// cooperative launch) makes the Eq. 2 / Eq. 4 sums complete; every CTA then
// reads them and takes the decision that ends the iteration (window advance,
// hit/miss plan and ranks of the next iteration, pa_decide.cuh) -- the same
// inputs and arithmetic give the same plan everywhere, CTA (0, 0) publishes it
// and writes its strip of the next batch (a4) straight from the new states
// still in its registers: the gather reads nothing. One kernel per iteration
// instead of the update and planning kernels.
#include "pa_decide.cuh"
#include "pa_internal.h"

namespace pa {
namespace {

struct Q {  // four adjacent columns as two packed fp32 pairs
  float2 l, h;
};

__device__ __forceinline__ Q ldq(const float* p) {
  const float4 v = *reinterpret_cast<const float4*>(p);
  return {make_float2(v.x, v.y), make_float2(v.z, v.w)};
}
__device__ __forceinline__ void stq(float* p, const Q& q) {
  *reinterpret_cast<float4*>(p) = make_float4(q.l.x, q.l.y, q.h.x, q.h.y);
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(-1.f, -1.f), a);  // -b exact, one rounding: a - b
}
__device__ __forceinline__ Q qadd(const Q& a, const Q& b) { return {__fadd2_rn(a.l, b.l), __fadd2_rn(a.h, b.h)}; }
__device__ __forceinline__ Q qsub(const Q& a, const Q& b) { return {sub2(a.l, b.l), sub2(a.h, b.h)}; }

// A cache entry row piece (xhat or ehat, four columns) as stored: fp32, or
// bfloat16 when CB (rounded to nearest even when written, widened exactly when
// read). The trajectory's rows start where its fp32 rows would; within them
// the row pitch is D entries.
template <bool CB>
__device__ __forceinline__ Q ld_ent(const float* traj_base, int off) {
  if constexpr (CB) {
    float a[4];
    Bf16Row<4>::load(reinterpret_cast<const uint16_t*>(traj_base) + off, a);
    return {make_float2(a[0], a[1]), make_float2(a[2], a[3])};
  } else {
    return ldq(traj_base + off);
  }
}
template <bool CB>
__device__ __forceinline__ void st_ent(float* traj_base, int off, const Q& q) {
  if constexpr (CB) {
    const float a[4] = {q.l.x, q.l.y, q.h.x, q.h.y};
    Bf16Row<4>::store(reinterpret_cast<uint16_t*>(traj_base) + off, a);
  } else {
    stq(traj_base + off, q);
  }
}
// The value an fp32 row piece takes once stored as an entry.
template <bool CB>
__device__ __forceinline__ Q as_ent(const Q& q) {
  if constexpr (CB) {
    auto r = [](float v) { return __bfloat162float(__float2bfloat16_rn(v)); };
    return {make_float2(r(q.l.x), r(q.l.y)), make_float2(r(q.h.x), r(q.h.y))};
  } else {
    return q;
  }
}

// (hi, lo) += v per component: s = fl(hi + v), s + err == hi + v exactly
// (Knuth's TwoSum), lo accumulates err.
__device__ __forceinline__ void two_sum2(float2& hi, float2& lo, float2 v) {
  const float2 s = __fadd2_rn(hi, v);
  const float2 bb = sub2(s, hi);
  const float2 err = __fadd2_rn(sub2(hi, sub2(s, bb)), sub2(v, bb));
  hi = s;
  lo = __fadd2_rn(lo, err);
}
// (hi, lo) += (h2, l2)
__device__ __forceinline__ void two_sum2p(float2& hi, float2& lo, float2 h2, float2 l2) {
  two_sum2(hi, lo, h2);
  lo = __fadd2_rn(lo, l2);
}

template <bool NOISE>
struct Coef;  // per timestep: c_i - 1, e_i (and sigma_i)
template <>
struct Coef<false> {
  using T = float2;
};
template <>
struct Coef<true> {
  using T = float4;
};

template <int NW, bool NOISE>
struct LeanShape {
  __host__ __device__ static size_t coef_bytes(int T) {
    return ((size_t)T * sizeof(typename Coef<NOISE>::T) + 127) / 128 * 128;
  }
  __host__ __device__ static size_t rank_bytes(int P) { return ((size_t)P * 4 + 127) / 128 * 128; }
  __host__ __device__ static size_t red_bytes(int P) { return ((size_t)2 * P * 33 * sizeof(float) + 127) / 128 * 128; }
  static constexpr size_t kTotBytes = (size_t)NW * 32 * 16;  // run totals, one float4 per lane and warp
  __host__ __device__ static size_t smem_bytes(int T, int P, bool comp) {
    return coef_bytes(T) + rank_bytes(P) + red_bytes(P) + kTotBytes * (comp ? 2 : 1);
  }
};

// The fused step after the update: grid barrier, the complete sums, the
// decision in every CTA, and the warp's share of the next batch from the new
// states in `xn` (states t + j0 + 1 .. t + j0 + nj of trajectory tr; NULL for a
// finished trajectory). Every thread of every CTA calls it.
template <int NW, int LMAX>
__device__ __forceinline__ void step_tail(const Dev& d, DecideShared& ds, int par, const Traj& tr, const Q* xn,
                                          int j0, int nj, int mycol, int D, bool live) {
  const int tid = threadIdx.x;
  const int P = d.P;
  const unsigned long long ncta = (unsigned long long)gridDim.x * gridDim.y;
  // the spin polls an L2 line (about half a microsecond each): 16 x the
  // mbarrier limit keeps the same order of time, about a second
  const uint32_t spin = d.wait_limit > (0xffffffffu >> 4) ? 0xffffffffu : d.wait_limit << 4;
  if (!grid_sync(d.gbar, ncta, spin)) {
    if (tid == 0) atomicCAS(&d.ctl->status, kDevOk, kDevTimeout);
    return;  // the plan is not published; the host reports PA_ERR_TIMEOUT
  }
  // every CTA publishes a share: CTA c writes the reductions and ranks of the
  // positions and chunks congruent to c, CTA 0 the trajectories and counters
  const int cta = blockIdx.y * gridDim.x + blockIdx.x;
  stage_decision_bits(d, ds, par, cta, (int)ncta);
  __syncthreads();
  decide_par(d, ds, par, cta, (int)ncta, -1);
  __syncthreads();  // the next plan (ds.tn, ds.pn, chunk masks and bases) is known
  if (xn == nullptr || !live || nj <= 0) return;
  // a4 of the next iteration: its timestep i (tn <= i < tn + pn) reads state
  // min(i, t + p) -- states past the frontier t + p are lazy copies of it --
  // which this warp holds if it is one of t + j0 + 1 .. t + j0 + nj
  const int b = blockIdx.y;
  const int tn = ds.tn[b], pn = ds.pn[b];
  const int s_end = tr.t + tr.p;  // the new frontier (last computed state)
  auto miss_rank = [&](int i) -> int {  // rank of next-window timestep i, -1 for a hit
    const int q = b * P + (i - tn);
    const unsigned mm = ds.cmiss[q >> 5];
    const unsigned bit = 1u << (q & 31);
    return (mm & bit) ? ds.cbase[q >> 5] + __popc(mm & (bit - 1u)) : -1;
  };
  Q last = xn[0];
#pragma unroll
  for (int g = 0; g < LMAX; ++g) {
    if (g >= nj) break;
    const int s = tr.t + j0 + g + 1;  // the state xn[g] holds
    last = xn[g];
    if (s < s_end && s >= tn && s < tn + pn) {
      const int r = miss_rank(s);
      if (r >= 0) stq(d.batch_x + (int64_t)r * D + mycol, xn[g]);
    }
  }
  if (j0 + nj == tr.p) {  // this warp holds the frontier state: it also serves the lazy timesteps
    for (int i = max(tn, s_end); i < tn + pn; ++i) {
      const int r = miss_rank(i);
      if (r >= 0) stq(d.batch_x + (int64_t)r * D + mycol, last);
    }
  }
}

template <int NW, int LMAX, int MINB, bool NOISE, bool COMP, bool CB = false, bool FUSE = false, bool TAA = false>
__global__ void __launch_bounds__(NW * 32, MINB) k_update_lean(Dev d, const float* __restrict__ beps, int par) {
  static_assert(!(FUSE && TAA), "the fused step and the Anderson mixing are separate forms");
  using Sh = LeanShape<NW, NOISE>;
  using CT = typename Coef<NOISE>::T;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int T = d.T, P = d.P, b = blockIdx.y;
  const int D = (int)d.D;  // (P + 1) * D and T * D fit in int32 (launcher)
  CT* s_coef = reinterpret_cast<CT*>(smem_raw);
  int32_t* s_rank = reinterpret_cast<int32_t*>(smem_raw + Sh::coef_bytes(T));
  float* s_red = reinterpret_cast<float*>(smem_raw + Sh::coef_bytes(T) + Sh::rank_bytes(P));  // [2][P][33]
  float4* s_tot = reinterpret_cast<float4*>(smem_raw + Sh::coef_bytes(T) + Sh::rank_bytes(P) + Sh::red_bytes(P));
  float4* s_lo = s_tot + NW * 32;  // COMP only
  __shared__ DecideShared ds;      // FUSE only (the compiler drops it otherwise)

  // Prologue: everything here was written two or more kernels back (plan,
  // ranks, n_miss by the planning kernel; coefficients at creation). None of
  // it depends on the plan, so all of it is in flight at once.
  const Traj tr = d.traj[par * d.B + b];
  const int n_miss = d.ctl->n_miss;
  if constexpr (FUSE) decide_load<NW * 32>(d, ds, par);  // the plan of every trajectory, for the decision
  for (int i = tid; i < T; i += NW * 32) {
    CT c;
    if constexpr (NOISE) {
      c = make_float4(d.cm1[i], d.ecoef[i], d.sigma[i], 0.f);
    } else {
      c = make_float2(d.cm1[i], d.ecoef[i]);
    }
    s_coef[i] = c;
  }
  for (int j = tid; j < P; j += NW * 32) {
    int r = d.rank[b * P + j];
    if (r >= n_miss) {  // never expected: keep every load in bounds and report it
      atomicCAS(&d.ctl->status, kDevOk, kDevBadRank);
      r = -1;
    }
    s_rank[j] = r;
  }
  if (tr.p == 0) {  // finished trajectory; every CTA passes the dependency wait before it exits
    pdl_wait();
    if constexpr (!FUSE) {
      return;
    } else {  // the fused step still meets the barrier and takes the decision
      pdl_trigger();
      step_tail<NW, LMAX>(d, ds, par, tr, nullptr, 0, 0, 0, 0, false);
      return;
    }
  }
  __syncthreads();

  const int t = tr.t, p = tr.p, e = tr.e;
  const int mycol = blockIdx.x * 128 + lane * 4;
  const bool live = mycol < D;
  const float* Xr = d.X + (int64_t)b * (P + 1) * D + mycol;  // this lane's column of each ring
  float* Xw = d.X + (int64_t)b * (P + 1) * D + mycol;
  float* Xh = d.Xhat + (int64_t)b * P * D;  // entries: column mycol of row slot s at s * D + mycol
  float* Eh = d.Ehat + (int64_t)b * P * D;
  const float* Zr = NOISE ? d.noise + (int64_t)b * T * D + mycol : nullptr;
  const float* Br = beps + mycol;
  // Anderson mixing: G and R of this iteration (parity par), R of the previous one
  float* Gw = TAA ? d.taa_g + ((int64_t)par * d.B + b) * (P + 1) * D + mycol : nullptr;
  float* Rw = TAA ? d.taa_r + ((int64_t)par * d.B + b) * (P + 1) * D + mycol : nullptr;
  const float* Rp = TAA ? d.taa_r + ((int64_t)(par ^ 1) * d.B + b) * (P + 1) * D + mycol : nullptr;
  const int L = (p + NW - 1) / NW;  // <= LMAX (launcher)
  const int j0 = warp * L;
  const int nj = min(j0 + L, p) - j0;  // positions of this warp (<= 0: none)

  // miss bits of positions j0 .. j0 + LMAX (bit g: position j0 + g is a miss;
  // positions past p count as misses so that they never select a cache input)
  uint32_t miss = 0;
#pragma unroll
  for (int g = 0; g <= LMAX; ++g) {
    const int j = j0 + g;
    if (g <= nj && (j >= p || s_rank[j] >= 0)) miss |= 1u << g;
  }
  const int sp0 = nj > 0 ? (t + j0) % P : 0;          // cache slot of position j0
  const int sx0 = nj > 0 ? (t + j0) % (P + 1) : 0;    // ring slot of state t + j0
  const int se = e % (P + 1);                         // ring slot of state e (lazy states read it)
  auto xslot = [&](int g) {  // ring slot of state t + j0 + g, lazy-resolved
    int s = sx0 + g;
    if (s > P) s -= P + 1;
    return t + j0 + g <= e ? s : se;
  };
  auto cslot = [&](int g) {  // cache slot of timestep t + j0 + g
    int s = sp0 + g;
    if (s >= P) s -= P;
    return s;
  };

  Q x[LMAX + 1], ep[LMAX], xh[LMAX], z[NOISE ? LMAX : 1];
  if (live && nj > 0) {
    // every row load issued before any is used: a lazy position reads the
    // row of state e by address (an L1 hit after the first). Copying the
    // first lazy load's registers to the later positions instead makes each
    // copy wait for its load, which serialises the loads (measured 44.4
    // against 36.6 us per update launch at 4x128x128, window 64)
#pragma unroll
    for (int g = 0; g <= LMAX; ++g) {
      if (g > nj) break;
      x[g] = ldq(Xr + xslot(g) * D);
    }
#pragma unroll
    for (int g = 0; g < LMAX; ++g) {
      if (g >= nj) break;
      if (!(miss >> g & 1)) ep[g] = ld_ent<CB>(Eh, cslot(g) * D + mycol);
      if constexpr (TAA) {
        // the previous iteration's residual of state t + j0 + g + 1, which it
        // has iff that state was computed then (state <= e)
        if (t + j0 + g + 1 <= e) {
          int sr = sx0 + g + 1;
          if (sr > P) sr -= P + 1;
          xh[g] = ldq(Rp + sr * D);
        }
      } else {
        if (!(miss >> (g + 1) & 1)) xh[g] = ld_ent<CB>(Xh, cslot(g + 1) * D + mycol);
      }
      if constexpr (NOISE) z[g] = ldq(Zr + (t + j0 + g) * D);
    }
  }
  pdl_wait();     // the batch eps rows come from the denoiser that ran just before
  pdl_trigger();  // the successor may now run its prologue
  if (live && nj > 0) {
#pragma unroll
    for (int g = 0; g < LMAX; ++g) {
      if (g >= nj) break;
      if (miss >> g & 1) ep[g] = ldq(Br + s_rank[j0 + g] * D);
    }
  }

  // Pass 1: Eq. 7 for the misses, the drifts (kept in ep) and the run total.
  Q tot = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)}, tlo = tot;
  if (live && nj > 0) {
    if constexpr (TAA) {
      // the frontier state's value before the iteration, for the mix kernel's
      // lazy states (the mix overwrites state e's slot): written by the one
      // warp whose run holds state e, the last warp when e = t + p
#pragma unroll
      for (int g = 0; g <= LMAX; ++g) {
        if (g > nj) break;
        if (t + j0 + g == e && (g < nj || j0 + nj == p)) stq(d.taa_xe + (int64_t)b * D + mycol, x[g]);
      }
    }
    if (warp == 0) tot = x[0];  // the window start x_t begins the sum
#pragma unroll
    for (int g = 0; g < LMAX; ++g) {
      if (g >= nj) break;
      if (miss >> g & 1) {
        const int o = cslot(g) * D + mycol;
        st_ent<CB>(Eh, o, ep[g]);
        st_ent<CB>(Xh, o, x[g]);
      }
      const CT c = s_coef[t + j0 + g];
      const float2 cm = make_float2(c.x, c.x), ec = make_float2(c.y, c.y);
      Q dr = {__ffma2_rn(cm, x[g].l, __fmul2_rn(ec, ep[g].l)), __ffma2_rn(cm, x[g].h, __fmul2_rn(ec, ep[g].h))};
      if constexpr (NOISE) {
        const float2 sg = make_float2(c.z, c.z);
        dr.l = __ffma2_rn(sg, z[g].l, dr.l);
        dr.h = __ffma2_rn(sg, z[g].h, dr.h);
      }
      ep[g] = dr;
      if constexpr (COMP) {
        two_sum2(tot.l, tlo.l, dr.l);
        two_sum2(tot.h, tlo.h, dr.h);
      } else {
        tot = qadd(tot, dr);
      }
    }
  }
  s_tot[warp * 32 + lane] = make_float4(tot.l.x, tot.l.y, tot.h.x, tot.h.y);
  if constexpr (COMP) s_lo[warp * 32 + lane] = make_float4(tlo.l.x, tlo.l.y, tlo.h.x, tlo.h.y);
  __syncthreads();

  // Pass 2: carry = x_t + totals of the earlier runs (fixed order), then the
  // new states, the Eq. 2 terms and the Eq. 4 terms of the next iteration.
  if (nj > 0) {
    Q c = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)}, cl = c;
    if (warp == 0) {
      c = x[0];
    } else {
      // earlier runs' totals in order, fetched four at a time so that the
      // shared-memory latency is paid once per group, not once per run
      for (int w0 = 0; w0 < warp; w0 += 4) {
        float4 v[4], u[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (w0 + q < warp) {
            v[q] = s_tot[(w0 + q) * 32 + lane];
            if constexpr (COMP) u[q] = s_lo[(w0 + q) * 32 + lane];
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (w0 + q < warp) {
            if constexpr (COMP) {
              two_sum2p(c.l, cl.l, make_float2(v[q].x, v[q].y), make_float2(u[q].x, u[q].y));
              two_sum2p(c.h, cl.h, make_float2(v[q].z, v[q].w), make_float2(u[q].z, u[q].w));
            } else {
              c = qadd(c, Q{make_float2(v[q].x, v[q].y), make_float2(v[q].z, v[q].w)});
            }
          }
        }
      }
    }
    int so = sx0 + 1;  // ring slot of the new state t + j0 + g + 1
    if (so > P) so -= P + 1;
#pragma unroll
    for (int g = 0; g < LMAX; ++g) {
      if (g >= nj) break;
      const int j = j0 + g;
      float ev = 0.f, dv = 0.f;
      if (live) {
        Q n;
        if constexpr (COMP) {
          two_sum2(c.l, cl.l, ep[g].l);
          two_sum2(c.h, cl.h, ep[g].h);
          n = qadd(c, cl);
        } else {
          c = qadd(c, ep[g]);
          n = c;
        }
        if constexpr (TAA) {
          // n is the Picard map's value G of state t + j + 1; R = G - X
          const Q rr = qsub(n, x[g + 1]);
          stq(Gw + so * D, n);
          stq(Rw + so * D, rr);
          if (t + j + 1 <= e) {  // a history: dR = R - R'
            const Q dr = qsub(rr, xh[g]);
            const float2 nr = __ffma2_rn(dr.h, rr.h, __fmul2_rn(dr.l, rr.l));
            const float2 dd = __ffma2_rn(dr.h, dr.h, __fmul2_rn(dr.l, dr.l));
            ev = nr.x + nr.y;
            dv = dd.x + dd.y;
          }
        } else {
          stq(Xw + so * D, n);
          Q df = qsub(n, x[g + 1]);  // against the old state i+1 (lazy-resolved)
          if constexpr (FUSE) ep[g] = n;  // the drift is spent: keep the new state for the next batch
          const float2 e2 = __ffma2_rn(df.h, df.h, __fmul2_rn(df.l, df.l));
          ev = e2.x + e2.y;
          if (j + 1 < p) {
            // the next timestep's cache input: its entry if it is a hit, else
            // the old state i+1, the entry it receives in this kernel
            if (!(miss >> (g + 1) & 1)) {
              df = qsub(n, xh[g]);
            } else if constexpr (CB) {
              df = qsub(n, as_ent<CB>(x[g + 1]));
            }
            dv = (fabsf(df.l.x) + fabsf(df.l.y)) + (fabsf(df.h.x) + fabsf(df.h.y));
          }
        }
      }
      s_red[j * 33 + lane] = ev;
      s_red[(P + j) * 33 + lane] = dv;
      if (++so > P) so = 0;
    }
  }
  __syncthreads();
  // strip partials: one thread per (quantity, position) sums its row of lanes
  for (int r = tid; r < 2 * p; r += NW * 32) {
    const int which = r >= p, j = which ? r - p : r;
    const float* row = s_red + (which * P + j) * 33;
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
    for (int k = 0; k < 32; k += 4) {
      a0 += row[k];
      a1 += row[k + 1];
      a2 += row[k + 2];
      a3 += row[k + 3];
    }
    if constexpr (TAA) {
      red_add_gram(d, par, which, b * P + j, (a0 + a1) + (a2 + a3));
    } else {
      red_add(d, par, which, b * P + j, (a0 + a1) + (a2 + a3));
    }
  }
  if constexpr (FUSE) step_tail<NW, LMAX>(d, ds, par, tr, ep, j0, nj, mycol, D, live);
}

template <int NW, int LMAX, int MINB, bool NOISE, bool COMP, bool CB = false, bool FUSE = false, bool TAA = false>
cudaError_t launch_lean(const Dev& d, const float* beps, int par, cudaStream_t st) {
  using Sh = LeanShape<NW, NOISE>;
  const int nstrip = (int)((d.D + 127) / 128);
  const size_t smem = Sh::smem_bytes(d.T, d.P, COMP);
  auto kern = k_update_lean<NW, LMAX, MINB, NOISE, COMP, CB, FUSE, TAA>;
  static size_t configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || smem > configured[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev] = smem;
  }
  return launch_ex(kern, dim3(nstrip, d.B, 1), dim3(NW * 32), smem, st, 0, d, beps, par);
}

constexpr size_t kLeanSmemMax = 200 * 1024;

// The fused step: launched cooperatively, so only when every CTA of the grid
// (a strip of 128 columns of each trajectory) can be resident at once;
// cudaErrorNotSupported otherwise (the caller then launches the update and
// planning kernels).
template <int NW, int LMAX, int MINB, bool NOISE, bool COMP, bool CB = false>
cudaError_t launch_fused(const Dev& d, const float* beps, int par, cudaStream_t st) {
  using Sh = LeanShape<NW, NOISE>;
  const int nstrip = (int)((d.D + 127) / 128);
  const size_t smem = Sh::smem_bytes(d.T, d.P, COMP);
  if (smem > kLeanSmemMax) return cudaErrorNotSupported;
  auto kern = k_update_lean<NW, LMAX, MINB, NOISE, COMP, CB, true>;
  // per device: the dynamic shared memory configured and the resident CTAs
  // the whole GPU holds at that size
  static size_t configured[64] = {};
  static size_t cap_smem[64] = {};
  static int capacity[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorNotSupported;
  if (smem > configured[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured[dev] = smem;
  }
  if (smem != cap_smem[dev]) {
    int per_sm = 0, nsm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NW * 32, smem);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    capacity[dev] = per_sm * nsm;
    cap_smem[dev] = smem;
  }
  if ((int64_t)nstrip * d.B > capacity[dev]) return cudaErrorNotSupported;
  return launch_ex_coop(kern, dim3(nstrip, d.B, 1), dim3(NW * 32), smem, st, 0, true, d, beps, par);
}

}  // namespace

// Lean launch shapes (shape % 10): 0 = by window (deterministic steps only),
// 1 = 16 warps x 7 positions (one CTA per SM), 2 = 12 x 9, 3 = 8 x 4 and
// 4 = 8 x 8 (two CTAs per SM), 5 = 8 x 4 (three CTAs per SM), 6 = 4 x 8 (four
// CTAs per SM); shape >= 10: compensated sums (shapes 1-4, deterministic steps
// only). Returns cudaErrorNotSupported when the shape cannot hold the window.
cudaError_t launch_update_lean(const Dev& d, const float* batch_eps, int par, int shape, cudaStream_t st) {
  const bool comp = shape >= 10;
  int s = shape % 10;
  if (s == 0) {
    // by window: as many CTAs per SM as the registers allow without spilling
    // (three of 8 x 4, two of 8 x 8), else 16 warps of at most 7 positions
    // (one CTA per SM). Stochastic steps keep the register-resident bulk form,
    // measured faster for them.
    if (d.noise) return cudaErrorNotSupported;
    s = d.P <= 32 ? (comp ? 3 : 5) : d.P <= 64 ? 4 : 1;
  }
  static const int kWarps[7] = {0, 16, 12, 8, 8, 8, 4};
  static const int kRun[7] = {0, 7, 9, 4, 8, 4, 8};
  if (s > 6 || d.P > kWarps[s] * kRun[s]) return cudaErrorNotSupported;
  if (d.cache_bf16) {  // bfloat16 entries: shapes 1, 4 and 5, plain sums, deterministic steps
    if (comp || d.noise) return cudaErrorNotSupported;
    if (s == 5) return launch_lean<8, 4, 3, false, false, true>(d, batch_eps, par, st);
    if (s == 4) return launch_lean<8, 8, 2, false, false, true>(d, batch_eps, par, st);
    if (s == 1) return launch_lean<16, 7, 1, false, false, true>(d, batch_eps, par, st);
    return cudaErrorNotSupported;
  }
  if (s >= 5 && (comp || d.noise)) return cudaErrorNotSupported;
  if (s == 5) return launch_lean<8, 4, 3, false, false>(d, batch_eps, par, st);
  if (s == 6) return launch_lean<4, 8, 4, false, false>(d, batch_eps, par, st);
  if (d.noise) {
    if (comp) return cudaErrorNotSupported;
    if (s == 1) return launch_lean<16, 7, 1, true, false>(d, batch_eps, par, st);
    if (s == 2) return launch_lean<12, 9, 1, true, false>(d, batch_eps, par, st);
    if (s == 3) return launch_lean<8, 4, 2, true, false>(d, batch_eps, par, st);
    return launch_lean<8, 8, 2, true, false>(d, batch_eps, par, st);
  }
  if (comp) {
    if (s == 1) return launch_lean<16, 7, 1, false, true>(d, batch_eps, par, st);
    if (s == 2) return launch_lean<12, 9, 1, false, true>(d, batch_eps, par, st);
    if (s == 3) return launch_lean<8, 4, 2, false, true>(d, batch_eps, par, st);
    return launch_lean<8, 8, 2, false, true>(d, batch_eps, par, st);
  }
  if (s == 1) return launch_lean<16, 7, 1, false, false>(d, batch_eps, par, st);
  if (s == 2) return launch_lean<12, 9, 1, false, false>(d, batch_eps, par, st);
  if (s == 3) return launch_lean<8, 4, 2, false, false>(d, batch_eps, par, st);
  return launch_lean<8, 8, 2, false, false>(d, batch_eps, par, st);
}

// Fused step shapes: as launch_update_lean's (0 = by window, also with
// stochastic steps); compensated sums are not offered.
cudaError_t launch_step_fused(const Dev& d, const float* batch_eps, int par, int shape, cudaStream_t st) {
  if (!step_fused_supported(d, batch_eps, shape)) return cudaErrorNotSupported;
  int s = shape % 10;
  // by window, as the lean form; with draws 16 x 7 above 32 positions (8 x 8
  // would spill)
  if (s == 0) s = d.P <= 32 ? (d.noise ? 3 : 5) : (d.P <= 64 && !d.noise) ? 4 : 1;
  static const int kWarps[7] = {0, 16, 12, 8, 8, 8, 4};
  static const int kRun[7] = {0, 7, 9, 4, 8, 4, 8};
  if (s > 6 || d.P > kWarps[s] * kRun[s]) return cudaErrorNotSupported;
  if (d.cache_bf16) {
    if (s == 5) return launch_fused<8, 4, 3, false, false, true>(d, batch_eps, par, st);
    if (s == 4) return launch_fused<8, 8, 2, false, false, true>(d, batch_eps, par, st);
    if (s == 1) return launch_fused<16, 7, 1, false, false, true>(d, batch_eps, par, st);
    return cudaErrorNotSupported;
  }
  if (d.noise) {
    if (s == 1) return launch_fused<16, 7, 1, true, false>(d, batch_eps, par, st);
    if (s == 3) return launch_fused<8, 4, 2, true, false>(d, batch_eps, par, st);
    if (s == 4) return launch_fused<8, 8, 2, true, false>(d, batch_eps, par, st);
    return cudaErrorNotSupported;
  }
  if (s == 1) return launch_fused<16, 7, 1, false, false>(d, batch_eps, par, st);
  if (s == 4) return launch_fused<8, 8, 2, false, false>(d, batch_eps, par, st);
  if (s == 5) return launch_fused<8, 4, 3, false, false>(d, batch_eps, par, st);
  return cudaErrorNotSupported;
}

// The mixing form of the lean update: by window like the lean form (16 x 7,
// 8 x 8 or 8 x 4 warps x positions; with draws 16 x 7 or 8 x 4 at two CTAs per
// SM), fp32 cache entries.
cudaError_t launch_update_taa(const Dev& d, const float* batch_eps, int par, cudaStream_t st) {
  if (!update_lean_supported(d, batch_eps) || d.cache_bf16 || !d.taa_g) return cudaErrorNotSupported;
  if (d.noise) {
    if (d.P <= 32) return launch_lean<8, 4, 2, true, false, false, false, true>(d, batch_eps, par, st);
    return launch_lean<16, 7, 1, true, false, false, false, true>(d, batch_eps, par, st);
  }
  if (d.P <= 32) return launch_lean<8, 4, 3, false, false, false, false, true>(d, batch_eps, par, st);
  if (d.P <= 64) return launch_lean<8, 8, 2, false, false, false, false, true>(d, batch_eps, par, st);
  return launch_lean<16, 7, 1, false, false, false, false, true>(d, batch_eps, par, st);
}

bool step_fused_supported(const Dev& d, const float* batch_eps, int shape) {
  // every CTA decides in shared memory from one miss mask per 32-position chunk
  if (shape >= 10 || (int64_t)d.B * d.P > 32 * 32) return false;
  return update_lean_supported(d, batch_eps);
}

bool update_lean_supported(const Dev& d, const float* batch_eps) {
  if (d.D % 4 != 0 || (d.cache_bf16 && d.noise)) return false;
  if ((reinterpret_cast<uintptr_t>(batch_eps) & 15) != 0) return false;
  if (d.noise && (reinterpret_cast<uintptr_t>(d.noise) & 15) != 0) return false;
  if (d.P > 16 * 7) return false;
  if ((int64_t)(d.P + 1) * d.D > INT32_MAX || (int64_t)d.T * d.D > INT32_MAX) return false;
  if ((int64_t)d.B * d.P * d.D > INT32_MAX) return false;  // batch rank * D
  const size_t smem = d.noise ? LeanShape<16, true>::smem_bytes(d.T, d.P, true)
                              : LeanShape<16, false>::smem_bytes(d.T, d.P, true);
  return smem <= kLeanSmemMax;
}

}  // namespace pa
