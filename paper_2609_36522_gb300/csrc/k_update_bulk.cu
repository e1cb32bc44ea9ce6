// Picard update kernels for sm_103a, three forms of the same arithmetic.
//
// Same mathematics as the plain-load kernel (k_solver.cu): per window position
// j (timestep i = t + j) Eq. 6 assembly, Eq. 7 cache update for misses, the
// drift d_j = (c_i - 1) x_i + e_i eps_i at the current latent, the window
// prefix sum of Eq. 1, the Eq. 2 error of state i+1 and the Eq. 4 distance of
// timestep i+1 for the next iteration. Every form reduces the per-lane Eq. 2
// and Eq. 4 terms over its CTA in a fixed order and adds the CTA's sums into
// the iteration's fp64 accumulators (red_add, pa_internal.h).
//
// Parallel structure. A CTA owns a strip of SEG = 32*V adjacent columns of one
// trajectory. The drifts of different positions are independent; only their
// prefix sum couples them. So warps take contiguous runs of positions, form
// their drifts and the runs' totals, and after one CTA barrier add the carry
// (the running sum from x_t plus the totals of the runs before theirs). All
// sums are carried as fp32 (hi, lo) pairs (TwoSum), so the blocked order loses
// nothing against a sequential compensated sum.
//
//   k_update_reg   each warp's run (at most LMAX positions) is loaded straight
//                  into registers; no staging, no waits (the bulk forms'
//                  choice for four columns per lane; the library's default
//                  with stochastic steps -- k_update_lean.cu has the default
//                  for deterministic steps)
//   k_update_seg   each warp's run is staged in shared memory by cp.async.bulk
//                  (TMA engine) onto the warp's mbarrier (whole window per CTA)
//   k_update_tile  the window walks in tiles of TW = NW*S positions through up
//                  to 16 shared-memory tile buffers (windows too large for the
//                  other two)
//
// Staging (seg, tile). Rows (per position: the eps row segment, from
// batch_eps for a miss or ehat_i for a hit; the old state x_{i+1} unless it is
// a lazy tail copy; xhat_{i+1} when timestep i+1 is a hit) are fetched with
// cp.async.bulk, one lane per row; completion is counted on mbarriers. Every
// mbarrier wait is bounded. A wait that runs out records kDevTimeout in the
// solver's status word and stops further issues; the CTA finishes its (now
// meaningless) arithmetic with in-bounds accesses only, drains the copies
// already issued with bounded waits, and returns.
#include <cooperative_groups.h>

#include "pa_bulk.cuh"
#include "pa_internal.h"

namespace pa {
namespace {

namespace cg = cooperative_groups;

// CTAs per thread-block cluster: the strips of a cluster combine their
// per-position partial sums through distributed shared memory.
constexpr int kCluster = 8;


// s = fl(a + b) and s + err == a + b exactly (Knuth's TwoSum).
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& err) {
  s = a + b;
  const float bb = s - a;
  err = (a - (s - bb)) + (b - bb);
}

// (hi, lo) += v
__device__ __forceinline__ void acc_add(float& hi, float& lo, float v) {
  float s, e;
  two_sum(hi, v, s, e);
  hi = s;
  lo += e;
}

// Two lanes of fp32 at once (sm_100 and later: one instruction for both,
// each rounded to nearest as the scalar operation would be).
__device__ __forceinline__ float2 x2_add(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 x2_sub(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(-1.f, -1.f), a);  // -b exact, one rounding: a - b
}
// (hi, lo) += v for two columns, the TwoSum above per component
__device__ __forceinline__ void acc_add_x2(float2& hi, float2& lo, float2 v) {
  const float2 s = x2_add(hi, v);
  const float2 bb = x2_sub(s, hi);
  const float2 err = x2_add(x2_sub(hi, x2_sub(s, bb)), x2_sub(v, bb));
  hi = s;
  lo = x2_add(lo, err);
}

// (hi, lo) += (h2, l2)
__device__ __forceinline__ void acc_add2(float& hi, float& lo, float h2, float l2) {
  float s, e;
  two_sum(hi, h2, s, e);
  hi = s;
  lo += e + l2;
}

template <int V>
struct Vec {
  float a[V];
};

template <int V>
__device__ __forceinline__ Vec<V> ldv(const float* p) {
  Vec<V> r;
  if constexpr (V == 4) {
    const float4 q = *reinterpret_cast<const float4*>(p);
    r.a[0] = q.x; r.a[1] = q.y; r.a[2] = q.z; r.a[3] = q.w;
  } else if constexpr (V == 2) {
    const float2 q = *reinterpret_cast<const float2*>(p);
    r.a[0] = q.x; r.a[1] = q.y;
  } else {
    r.a[0] = *p;
  }
  return r;
}

template <int V>
__device__ __forceinline__ void stv(float* p, const Vec<V>& v) {
  if constexpr (V == 4) {
    *reinterpret_cast<float4*>(p) = make_float4(v.a[0], v.a[1], v.a[2], v.a[3]);
  } else if constexpr (V == 2) {
    *reinterpret_cast<float2*>(p) = make_float2(v.a[0], v.a[1]);
  } else {
    *p = v.a[0];
  }
}

// A cache entry row (xhat or ehat) as stored: fp32, or bfloat16 when CB.
template <int V, bool CB>
__device__ __forceinline__ Vec<V> ld_entry(const float* base, int64_t off) {
  if constexpr (CB) {
    Vec<V> r;
    Bf16Row<V>::load(reinterpret_cast<const uint16_t*>(base) + off, r.a);
    return r;
  } else {
    return ldv<V>(base + off);
  }
}
template <int V, bool CB>
__device__ __forceinline__ void st_entry(float* base, int64_t off, const Vec<V>& v) {
  if constexpr (CB) {
    Bf16Row<V>::store(reinterpret_cast<uint16_t*>(base) + off, v.a);
  } else {
    stv<V>(base + off, v);
  }
}
// The value an entry holds once stored.
template <int V, bool CB>
__device__ __forceinline__ Vec<V> as_entry(const Vec<V>& v) {
  if constexpr (CB) {
    Vec<V> r;
#pragma unroll
    for (int k = 0; k < V; ++k) r.a[k] = __bfloat162float(__float2bfloat16_rn(v.a[k]));
    return r;
  } else {
    return v;
  }
}

template <int V, int NW, int S>
struct TileShape {
  static constexpr int SEG = 32 * V;                  // columns per strip
  static constexpr int TW = NW * S;                   // positions per tile
  static_assert(2 * TW <= NW * 32, "two reductions per position need 2*TW threads");
  static constexpr size_t kTileFloats = (size_t)TW * 3 * SEG;
  static constexpr size_t kTileBytes = kTileFloats * sizeof(float);
  static constexpr int kMaxBuf = 16;                  // mbarriers in the barrier area
  static constexpr size_t kBarBytes = 128;
  // per position: rank, c-1, e, cache slot, state-ring slot of the next state,
  // and this strip's two partial sums (err, distance)
  __host__ __device__ static size_t meta_bytes(int P) { return ((size_t)P * 28 + 127) / 128 * 128; }
  static constexpr size_t kTotBytes = (size_t)NW * SEG * 2 * sizeof(float);   // segment totals
  static constexpr size_t kCarBytes = kTotBytes;                              // carries into warps
  static constexpr size_t kRedBytes = ((size_t)2 * TW * 33 * sizeof(float) + 127) / 128 * 128;
  __host__ __device__ static size_t smem_bytes(int P, int nbuf) {
    return kBarBytes + meta_bytes(P) + kTotBytes + kCarBytes + kRedBytes + (size_t)nbuf * kTileBytes;
  }
};

// nbuf tile buffers (<= 16); when nbuf >= ceil(p / TW) every copy of the
// window is in flight right after the prologue. CLUSTER: combine the strip
// partials of kCluster CTAs through distributed shared memory (else one
// partial per strip). WAIT_ALL: every thread polls the tile's mbarrier (else
// warp 0 polls and the CTA barrier releases the others).
template <int V, int NW, int S, bool CLUSTER, bool WAIT_ALL>
__global__ void __launch_bounds__(NW * 32) k_update_tile(Dev d, const float* __restrict__ beps,
                                                         int nstrip, int nbuf, uint32_t wait_limit, int par) {
  using Sh = TileShape<V, NW, S>;
  constexpr int SEG = Sh::SEG, TW = Sh::TW;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = d.P;
  const int b = blockIdx.y;
  const int64_t D = d.D;

  // smem: barriers | per-position metadata | totals | carries | reductions | tiles
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem_raw);
  unsigned char* q = smem_raw + Sh::kBarBytes;
  int32_t* s_rank = reinterpret_cast<int32_t*>(q);
  float* s_cm1 = reinterpret_cast<float*>(q + (size_t)P * 4);
  float* s_ec = reinterpret_cast<float*>(q + (size_t)P * 8);
  int32_t* s_slot = reinterpret_cast<int32_t*>(q + (size_t)P * 12);  // (t+j) mod P
  int32_t* s_nxt = reinterpret_cast<int32_t*>(q + (size_t)P * 16);   // (t+j+1) mod (P+1)
  float* s_pos = reinterpret_cast<float*>(q + (size_t)P * 20);        // [2][P] strip partials
  q += Sh::meta_bytes(P);
  float* s_tot = reinterpret_cast<float*>(q);   // [NW][SEG][2]
  q += Sh::kTotBytes;
  float* s_car = reinterpret_cast<float*>(q);   // [NW][SEG][2]
  q += Sh::kCarBytes;
  float* s_red = reinterpret_cast<float*>(q);   // [2][TW][33]
  q += Sh::kRedBytes;
  float* s_tile = reinterpret_cast<float*>(q);  // 128-byte aligned: all offsets above are

  // round 1: independent loads of the bookkeeping and every rank of the window
  const Traj tr = d.traj[par * d.B + b];
  const int n_miss = d.ctl->n_miss;
  for (int j = tid; j < P; j += NW * 32) s_rank[j] = d.rank[b * P + j];
  if (tr.p == 0) {  // finished trajectory; every CTA passes the dependency wait before it exits
    pdl_wait();
    return;
  }
  const int t = tr.t, p = tr.p, e = tr.e;
  for (int j = tid; j < p; j += NW * 32) {
    s_slot[j] = (t + j) % P;
    s_nxt[j] = (t + j + 1) % (P + 1);
    s_cm1[j] = d.cm1[t + j];
    s_ec[j] = d.ecoef[t + j];
    s_pos[j] = 0.f;
    s_pos[P + j] = 0.f;
  }
  if (tid == 0) {
    for (int k = 0; k < nbuf; ++k) mbar_init(&bar[k], 1);
    fence_barrier_init();
  }
  __syncthreads();
  for (int j = tid; j < p; j += NW * 32) {
    if (s_rank[j] >= n_miss) {  // never expected: keep every copy in bounds and report it
      atomicCAS(&d.ctl->status, kDevOk, kDevBadRank);
      s_rank[j] = -1;
    }
  }
  __syncthreads();
  // Everything above came from the decision kernel and earlier; the eps rows
  // below come from the denoiser that ran just before this kernel.
  pdl_wait();
  pdl_trigger();  // the successor may now run its prologue

  const int strip = blockIdx.x;          // the grid is padded to whole clusters
  const bool active = strip < nstrip;
  const int64_t c0 = (int64_t)strip * SEG;
  const int64_t ncol = (D - c0) < SEG ? (D - c0) : SEG;
  const uint32_t seg_bytes = (uint32_t)ncol * sizeof(float);
  const int64_t mycol = c0 + (int64_t)lane * V;
  const bool live = mycol < D;
  float* Xb = d.X + (int64_t)b * (P + 1) * D;
  float* Xh = d.Xhat + (int64_t)b * P * D;
  float* Eh = d.Ehat + (int64_t)b * P * D;
  const int ntile = active ? (p + TW - 1) / TW : 0;

  // Warp 0 issues tile k into buffer k % nbuf; lane l fetches positions
  // k*TW + l, k*TW + l + 32, ... The whole tile's byte count is announced on
  // the buffer's mbarrier before any of its copies is issued.
  auto issue_tile = [&](int k) {
    float* buf = s_tile + (size_t)(k % nbuf) * Sh::kTileFloats;
    uint64_t* bk = &bar[k % nbuf];
    uint32_t total = 0;
    for (int qb = 0; qb < TW; qb += 32) {
      const int qi = qb + lane;
      const int j = k * TW + qi;
      if (qi < TW && j < p) {
        const uint32_t n = 1u + (((t + j + 1) <= e) ? 1u : 0u) +
                           (((j + 1 < p) && (s_rank[j + 1] < 0)) ? 1u : 0u);
        total += n * seg_bytes;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) total += __shfl_xor_sync(0xffffffffu, total, o);
    if (lane == 0) mbar_arrive_expect_tx(bk, total);
    __syncwarp();
    for (int qb = 0; qb < TW; qb += 32) {
      const int qi = qb + lane;
      const int j = k * TW + qi;
      if (qi < TW && j < p) {
        float* rowp = buf + (size_t)qi * 3 * SEG;
        const int r = s_rank[j];
        const float* src_eps = (r >= 0) ? beps + (int64_t)r * D + c0 : Eh + (int64_t)s_slot[j] * D + c0;
        bulk_g2s(rowp, src_eps, seg_bytes, bk);
        if (t + j + 1 <= e) bulk_g2s(rowp + SEG, Xb + (int64_t)s_nxt[j] * D + c0, seg_bytes, bk);
        if ((j + 1 < p) && (s_rank[j + 1] < 0))
          bulk_g2s(rowp + 2 * SEG, Xh + (int64_t)s_slot[j + 1] * D + c0, seg_bytes, bk);
      }
    }
  };

  // round 2: every tile that has a buffer goes out now; meanwhile every warp
  // loads the lazy fill value (old state e) and warp 0 the window start x_t
  const int pre = ntile < nbuf ? ntile : nbuf;
  if (warp == 0)
    for (int k = 0; k < pre; ++k) issue_tile(k);
  int issued = pre;  // tiles issued so far (same value in every thread)
  Vec<V> xfill{}, xlast{};
  if (live) {
    xfill = ldv<V>(Xb + (int64_t)(e % (P + 1)) * D + mycol);
    if (warp == 0) xlast = ldv<V>(Xb + (int64_t)(t % (P + 1)) * D + mycol);
  }
  // warp 0 keeps the running carry: x_t + every drift before the current tile
  float chi[V], clo[V];
#pragma unroll
  for (int v = 0; v < V; ++v) { chi[v] = xlast.a[v]; clo[v] = 0.f; }

  const int red_first = NW * 32 - 2 * TW;  // the last 2*TW threads finish the reductions
  int my_fail = 0;   // this thread's wait ran out
  int aborted = 0;   // some thread's wait ran out (CTA-uniform, from a barrier)
  for (int k = 0; k < ntile; ++k) {
    const int bi = k % nbuf;
    const uint32_t parity = (uint32_t)((k / nbuf) & 1);
    // warp 0 watches the tile's mbarrier; the other warps sleep at the CTA
    // barrier instead of polling (the barrier orders the landed data for them)
    if ((WAIT_ALL || warp == 0) && !my_fail && !aborted &&
        !mbar_wait_bounded(&bar[bi], parity, wait_limit)) {
      atomicCAS(&d.ctl->status, kDevOk, kDevTimeout);
      my_fail = 1;
    }
    if (!WAIT_ALL) __syncthreads();
    const float* buf = s_tile + (size_t)bi * Sh::kTileFloats;
    const int tb = k * TW;
    const int q0 = warp * S;

    // phase 1: drifts of this warp's S positions and their local prefix
    float phi[S][V], plo[S][V];
    Vec<V> xo_s[S];
    Vec<V> xc;
    if (q0 == 0) {
      xc = xlast;  // warp 0: old state at the tile's first position
    } else if (tb + q0 < p && t + tb + q0 <= e) {
      xc = ldv<V>(buf + (size_t)(q0 - 1) * 3 * SEG + SEG + lane * V);
    } else {
      xc = xfill;
    }
    float rh[V], rl[V];
#pragma unroll
    for (int v = 0; v < V; ++v) { rh[v] = 0.f; rl[v] = 0.f; }
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const int qi = q0 + s;
      const int j = tb + qi;
      const float* rowp = buf + (size_t)qi * 3 * SEG;
      Vec<V> xo = xfill;
      if (j < p && live) {
        const Vec<V> eps = ldv<V>(rowp + lane * V);
        if (s_rank[j] >= 0) {  // Eq. 7: the cache takes (x_i, eps_i) of a miss
          const int64_t o = (int64_t)s_slot[j] * D + mycol;
          stv<V>(Eh + o, eps);
          stv<V>(Xh + o, xc);
        }
        const float cm1 = s_cm1[j], ec = s_ec[j];
#pragma unroll
        for (int v = 0; v < V; ++v) acc_add(rh[v], rl[v], fmaf(cm1, xc.a[v], ec * eps.a[v]));
        if (t + j + 1 <= e) xo = ldv<V>(rowp + SEG + lane * V);
      }
#pragma unroll
      for (int v = 0; v < V; ++v) { phi[s][v] = rh[v]; plo[s][v] = rl[v]; }
      xo_s[s] = xo;
      xc = xo;
    }
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const size_t o = ((size_t)warp * SEG + lane * V + v) * 2;
      s_tot[o] = rh[v];
      s_tot[o + 1] = rl[v];
    }
    __syncthreads();  // A: totals published

    // warp 0: exclusive scan of the warp totals per column, on top of the
    // running carry, and the running carry of the next tile
    if (warp == 0) {
#pragma unroll
      for (int w = 0; w < NW; ++w) {
#pragma unroll
        for (int v = 0; v < V; ++v) {
          const size_t o = ((size_t)w * SEG + lane * V + v) * 2;
          s_car[o] = chi[v];
          s_car[o + 1] = clo[v];
          acc_add2(chi[v], clo[v], s_tot[o], s_tot[o + 1]);
        }
      }
    }
    __syncthreads();  // B: carries published

    // phase 2: new states, their Eq. 2 error and next-iteration Eq. 4 distance
    float ch[V], cl[V];
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const size_t o = ((size_t)warp * SEG + lane * V + v) * 2;
      ch[v] = s_car[o];
      cl[v] = s_car[o + 1];
    }
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const int qi = q0 + s;
      const int j = tb + qi;
      const float* rowp = buf + (size_t)qi * 3 * SEG;
      float ev = 0.f, dv = 0.f;
      if (j < p && live) {
        Vec<V> xn;
#pragma unroll
        for (int v = 0; v < V; ++v) {
          float h = ch[v], l = cl[v];
          acc_add2(h, l, phi[s][v], plo[s][v]);
          xn.a[v] = h + l;
          const float df = xn.a[v] - xo_s[s].a[v];
          ev = fmaf(df, df, ev);
        }
        stv<V>(Xb + (int64_t)s_nxt[j] * D + mycol, xn);
        if (j + 1 < p) {
          const Vec<V> xh = (s_rank[j + 1] < 0) ? ldv<V>(rowp + 2 * SEG + lane * V) : xo_s[s];
#pragma unroll
          for (int v = 0; v < V; ++v) dv += fabsf(xn.a[v] - xh.a[v]);
        }
      }
      s_red[(size_t)qi * 33 + lane] = ev;
      s_red[(size_t)(TW + qi) * 33 + lane] = dv;
    }
    // the next tile's first state, read by warp 0 before it refills the buffer
    if (warp == 0) {
      const int jl = tb + TW - 1;
      if (jl < p && live && t + jl + 1 <= e) {
        xlast = ldv<V>(buf + (size_t)(TW - 1) * 3 * SEG + SEG + lane * V);
      } else {
        xlast = xfill;
      }
    }
    // C: every warp is done with this buffer, the totals and the carries;
    // stop issuing after a timeout
    aborted = __syncthreads_or(my_fail);
    if (!aborted && k + nbuf < ntile) {
      if (warp == 0) issue_tile(k + nbuf);
      issued = k + nbuf + 1;
    }
    // per-position partials of this strip: one thread sums one row of lanes
    if (tid >= red_first) {
      const int r = tid - red_first;  // 0 .. 2*TW-1
      const int qi = r % TW;
      const int j = tb + qi;
      if (j < p) {
        const float* row = s_red + (size_t)r * 33;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
          acc[0] += row[c];
          acc[1] += row[c + 1];
          acc[2] += row[c + 2];
          acc[3] += row[c + 3];
        }
        s_pos[(r < TW ? 0 : P) + j] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
      }
    }
  }
  // after a timeout: wait (bounded) for the last issue of every buffer
  if (tid == 0 && aborted) {
    for (int k = (issued > nbuf ? issued - nbuf : 0); k < issued; ++k)
      mbar_wait_bounded(&bar[k % nbuf], (uint32_t)((k / nbuf) & 1), kDrainLimit);
  }
  if constexpr (CLUSTER) {
    // Combine the strips of this cluster: CTA rank q sums positions j = q mod
    // kCluster over the cluster's CTAs in rank order (distributed shared
    // memory) and adds it into the iteration's sums. The second cluster barrier keeps
    // every CTA's shared memory alive until its peers have read it.
    cg::cluster_group cluster = cg::this_cluster();
    cluster.sync();
    const int rank = (int)cluster.block_rank();
    for (int q2 = tid; q2 < 2 * p; q2 += NW * 32) {
      const int which = q2 / p, j = q2 % p;
      if (j % kCluster != rank) continue;
      float sum = 0.f;
#pragma unroll
      for (int r = 0; r < kCluster; ++r) sum += cluster.map_shared_rank(s_pos, r)[which * P + j];
      red_add(d, par, which, b * P + j, sum);
    }
    cluster.sync();
  } else {
    // one partial per strip and position, added into the iteration's sums
    __syncthreads();
    if (active) {
      for (int q2 = tid; q2 < 2 * p; q2 += NW * 32) {
        const int which = q2 / p, j = q2 % p;
        red_add(d, par, which, b * P + j, s_pos[which * P + j]);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Segment-per-warp Picard update: used when the whole window of a strip fits
// in shared memory. Warp w owns the contiguous window positions
// [w*L, min(p, (w+1)*L)), L = ceil(p / NW), and issues their bulk copies
// itself (one mbarrier per warp). Phase 1 forms the compensated sum of the
// segment's drifts; after one CTA barrier every warp builds its carry
// x_t + sum of the earlier segments' totals and walks its segment again,
// recomputing the drifts from shared memory, to produce the new states, the
// Eq. 2 errors and the next-iteration Eq. 4 distances. Per-lane err/distance
// values go through a transposed shared-memory buffer; after a second barrier
// one thread per (quantity, position) sums its row into the strip partial.
// Two CTA barriers per launch in all. With NOISE (stochastic steps) every
// position stages a fourth row, the draw z_i, and its drift gains sigma_i z_i.
template <int V, int NW, bool NOISE = false>
struct SegShape {
  static constexpr int SEG = 32 * V;
  static constexpr int NR = NOISE ? 4 : 3;  // staged rows per position
  __host__ __device__ static size_t meta_bytes(int P) { return ((size_t)P * 24 + 127) / 128 * 128; }
  __host__ __device__ static size_t rows_bytes(int P) { return (size_t)P * NR * SEG * sizeof(float); }
  __host__ __device__ static size_t red_bytes(int P) { return ((size_t)2 * P * 33 * sizeof(float) + 127) / 128 * 128; }
  static constexpr size_t kTotBytes = (size_t)NW * SEG * 2 * sizeof(float);
  static constexpr size_t kBarBytes = 128;  // NW <= 16 mbarriers
  __host__ __device__ static size_t smem_bytes(int P) {
    return kBarBytes + meta_bytes(P) + kTotBytes + red_bytes(P) + rows_bytes(P);
  }
};

template <int V, int NW, bool NOISE>
__global__ void __launch_bounds__(NW * 32) k_update_seg(Dev d, const float* __restrict__ beps,
                                                        uint32_t wait_limit, int par) {
  using Sh = SegShape<V, NW, NOISE>;
  constexpr int SEG = Sh::SEG;
  constexpr int NR = Sh::NR;
  static_assert(NW <= 16, "one mbarrier per warp in a 128-byte area");
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = d.P;
  const int b = blockIdx.y;
  const int64_t D = d.D;

  uint64_t* bar = reinterpret_cast<uint64_t*>(smem_raw);
  unsigned char* q = smem_raw + Sh::kBarBytes;
  int32_t* s_rank = reinterpret_cast<int32_t*>(q);
  float* s_cm1 = reinterpret_cast<float*>(q + (size_t)P * 4);
  float* s_ec = reinterpret_cast<float*>(q + (size_t)P * 8);
  int32_t* s_slot = reinterpret_cast<int32_t*>(q + (size_t)P * 12);  // (t+j) mod P
  int32_t* s_nxt = reinterpret_cast<int32_t*>(q + (size_t)P * 16);   // (t+j+1) mod (P+1)
  float* s_sig = reinterpret_cast<float*>(q + (size_t)P * 20);       // sigma_i (stochastic steps)
  q += Sh::meta_bytes(P);
  float* s_tot = reinterpret_cast<float*>(q);   // [NW][SEG][2]
  q += Sh::kTotBytes;
  float* s_red = reinterpret_cast<float*>(q);   // [2][P][33]
  q += Sh::red_bytes(P);
  float* s_rows = reinterpret_cast<float*>(q);  // [P][NR][SEG]: eps, old x_{i+1}, xhat_{i+1} (, z_i)

  // Everything read before pdl_wait() was written two or more kernels back
  // (the previous update and decision kernels); only the batch eps rows come
  // from the denoiser just before.
  const Traj tr = d.traj[par * d.B + b];
  const int n_miss = d.ctl->n_miss;
  if (tr.p == 0) {  // finished trajectory; every CTA passes the dependency wait before it exits
    pdl_wait();
    return;
  }
  const int t = tr.t, p = tr.p, e = tr.e;
  for (int j = tid; j < p; j += NW * 32) {
    int r = d.rank[b * P + j];
    if (r >= n_miss) {  // never expected: keep every copy in bounds and report it
      atomicCAS(&d.ctl->status, kDevOk, kDevBadRank);
      r = -1;
    }
    s_rank[j] = r;
    s_slot[j] = (t + j) % P;
    s_nxt[j] = (t + j + 1) % (P + 1);
  }
  if (tid == 0) {
    for (int k = 0; k < NW; ++k) mbar_init(&bar[k], 1);
    fence_barrier_init();
  }
  __syncthreads();

  const int strip = blockIdx.x;
  const int64_t c0 = (int64_t)strip * SEG;
  const int64_t ncol = (D - c0) < SEG ? (D - c0) : SEG;
  const uint32_t seg_bytes = (uint32_t)ncol * sizeof(float);
  const int64_t mycol = c0 + (int64_t)lane * V;
  const bool live = mycol < D;
  float* Xb = d.X + (int64_t)b * (P + 1) * D;
  float* Xh = d.Xhat + (int64_t)b * P * D;
  float* Eh = d.Ehat + (int64_t)b * P * D;
  const int L = (p + NW - 1) / NW;
  const int j0 = warp * L;
  const int j1 = (j0 + L) < p ? (j0 + L) : p;

  // this warp's copies: the whole byte count first, then one lane per
  // position; everything but the misses' batch eps rows goes out before
  // pdl_wait() and overlaps the denoiser's tail
  {
    uint32_t total = 0;
    for (int j = j0 + lane; j < j1; j += 32) {
      total += seg_bytes * ((NOISE ? 2u : 1u) + ((t + j + 1 <= e) ? 1u : 0u) +
                            (((j + 1 < p) && (s_rank[j + 1] < 0)) ? 1u : 0u));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) total += __shfl_xor_sync(0xffffffffu, total, o);
    if (lane == 0 && j0 < j1) mbar_arrive_expect_tx(&bar[warp], total);
    __syncwarp();
    for (int j = j0 + lane; j < j1; j += 32) {
      float* rowp = s_rows + (size_t)j * NR * SEG;
      if (s_rank[j] < 0) bulk_g2s(rowp, Eh + (int64_t)s_slot[j] * D + c0, seg_bytes, &bar[warp]);
      if (t + j + 1 <= e) bulk_g2s(rowp + SEG, Xb + (int64_t)s_nxt[j] * D + c0, seg_bytes, &bar[warp]);
      if ((j + 1 < p) && (s_rank[j + 1] < 0))
        bulk_g2s(rowp + 2 * SEG, Xh + (int64_t)s_slot[j + 1] * D + c0, seg_bytes, &bar[warp]);
      if (NOISE) bulk_g2s(rowp + 3 * SEG, d.noise + ((int64_t)b * d.T + t + j) * D + c0, seg_bytes, &bar[warp]);
    }
    pdl_wait();  // the batch eps rows come from the denoiser that ran just before
    pdl_trigger();  // the successor may now run its prologue
    for (int j = j0 + lane; j < j1; j += 32) {
      const int r = s_rank[j];
      if (r >= 0) bulk_g2s(s_rows + (size_t)j * NR * SEG, beps + (int64_t)r * D + c0, seg_bytes, &bar[warp]);
    }
  }
  // this warp's step coefficients (read by this warp only)
  for (int j = j0 + lane; j < j1; j += 32) {
    s_cm1[j] = d.cm1[t + j];
    s_ec[j] = d.ecoef[t + j];
    if (NOISE) s_sig[j] = d.sigma[t + j];
  }
  __syncwarp();
  Vec<V> xstart{}, xfill{};
  if (live) {
    xstart = ldv<V>(Xb + (int64_t)(t % (P + 1)) * D + mycol);
    xfill = ldv<V>(Xb + (int64_t)(e % (P + 1)) * D + mycol);
  }
  int my_fail = 0;
  if (j0 < j1 && !mbar_wait_bounded(&bar[warp], 0, wait_limit)) my_fail = 1;
  if (warp > 0 && j0 < j1 && !my_fail && !mbar_wait_bounded(&bar[warp - 1], 0, wait_limit)) my_fail = 1;
  if (my_fail) atomicCAS(&d.ctl->status, kDevOk, kDevTimeout);

  // old state at the segment's first position
  Vec<V> xc0 = xfill;
  if (j0 == 0) {
    xc0 = xstart;
  } else if (j0 < j1 && t + j0 <= e && live) {
    xc0 = ldv<V>(s_rows + (size_t)(j0 - 1) * NR * SEG + SEG + lane * V);
  }

  // phase 1: the drifts (written over the eps rows, for phase 2), the cache
  // update of the misses (Eq. 7), and the compensated sum of the segment
  float rh[V], rl[V];
#pragma unroll
  for (int v = 0; v < V; ++v) { rh[v] = 0.f; rl[v] = 0.f; }
  if (live) {
    Vec<V> xc = xc0;
    for (int j = j0; j < j1; ++j) {
      float* rowp = s_rows + (size_t)j * NR * SEG;
      const Vec<V> eps = ldv<V>(rowp + lane * V);
      if (s_rank[j] >= 0) {  // Eq. 7: the cache takes (x_i, eps_i) of a miss
        const int64_t o = (int64_t)s_slot[j] * D + mycol;
        stv<V>(Eh + o, eps);
        stv<V>(Xh + o, xc);
      }
      const float cm1 = s_cm1[j], ec = s_ec[j];
      Vec<V> zn{};
      if (NOISE) zn = ldv<V>(rowp + 3 * SEG + lane * V);
      Vec<V> dr;
#pragma unroll
      for (int v = 0; v < V; ++v) {
        dr.a[v] = fmaf(cm1, xc.a[v], ec * eps.a[v]);
        if (NOISE) dr.a[v] = fmaf(s_sig[j], zn.a[v], dr.a[v]);
        acc_add(rh[v], rl[v], dr.a[v]);
      }
      stv<V>(rowp + lane * V, dr);
      xc = (t + j + 1 <= e) ? ldv<V>(rowp + SEG + lane * V) : xfill;
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const size_t o = ((size_t)warp * SEG + lane * V + v) * 2;
    s_tot[o] = rh[v];
    s_tot[o + 1] = rl[v];
  }
  __syncthreads();

  // phase 2: carry into this segment, then the new states, errors, distances
  float ch[V], cl[V];
#pragma unroll
  for (int v = 0; v < V; ++v) { ch[v] = xstart.a[v]; cl[v] = 0.f; }
  for (int w = 0; w < warp; ++w) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const size_t o = ((size_t)w * SEG + lane * V + v) * 2;
      acc_add2(ch[v], cl[v], s_tot[o], s_tot[o + 1]);
    }
  }
  {
    for (int j = j0; j < j1; ++j) {
      const float* rowp = s_rows + (size_t)j * NR * SEG;
      float ev = 0.f, dv = 0.f;
      if (live) {
        const Vec<V> dr = ldv<V>(rowp + lane * V);  // the drift, from phase 1
        const Vec<V> xo = (t + j + 1 <= e) ? ldv<V>(rowp + SEG + lane * V) : xfill;
        Vec<V> xn;
#pragma unroll
        for (int v = 0; v < V; ++v) {
          acc_add(ch[v], cl[v], dr.a[v]);
          xn.a[v] = ch[v] + cl[v];
          const float df = xn.a[v] - xo.a[v];
          ev = fmaf(df, df, ev);
        }
        stv<V>(Xb + (int64_t)s_nxt[j] * D + mycol, xn);
        if (j + 1 < p) {
          const Vec<V> xh = (s_rank[j + 1] < 0) ? ldv<V>(rowp + 2 * SEG + lane * V) : xo;
#pragma unroll
          for (int v = 0; v < V; ++v) dv += fabsf(xn.a[v] - xh.a[v]);
        }
      }
      s_red[(size_t)j * 33 + lane] = ev;
      s_red[(size_t)(P + j) * 33 + lane] = dv;
    }
  }
  __syncthreads();
  // strip partials: one thread per (quantity, position) sums its row of lanes
  // and adds it into the iteration's sums
  for (int r = tid; r < 2 * p; r += NW * 32) {
    const int which = r / p, j = r % p;
    const float* row = s_red + (size_t)(which * P + j) * 33;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 32; c += 4) {
      acc[0] += row[c];
      acc[1] += row[c + 1];
      acc[2] += row[c + 2];
      acc[3] += row[c + 3];
    }
    red_add(d, par, which, b * P + j, (acc[0] + acc[1]) + (acc[2] + acc[3]));
  }
  // after a timeout, let this warp's copies land before the CTA exits
  if (my_fail && lane == 0 && j0 < j1) mbar_wait_bounded(&bar[warp], 0, kDrainLimit);
}

constexpr size_t kSegSmemMax = 200 * 1024;

template <int V, int NW, bool NOISE = false>
bool seg_fits(const Dev& d) {
  return SegShape<V, NW, NOISE>::smem_bytes(d.P) <= kSegSmemMax;
}

template <int V, int NW, bool NOISE = false>
cudaError_t launch_seg(const Dev& d, const float* beps, int par, cudaStream_t st) {
  using Sh = SegShape<V, NW, NOISE>;
  const int nstrip = (int)((d.D + Sh::SEG - 1) / Sh::SEG);
  const size_t smem = Sh::smem_bytes(d.P);
  auto kern = k_update_seg<V, NW, NOISE>;
  static size_t configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || smem > configured[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev] = smem;
  }
  return launch_ex(kern, dim3(nstrip, d.B, 1), dim3(NW * 32), smem, st, 0, d, beps, d.wait_limit, par);
}

// ---------------------------------------------------------------------------
// Register-resident segment update. The same segmentation and arithmetic as
// k_update_seg (warp w owns positions [w*L, min(p, (w+1)*L)), L = ceil(p/NW);
// two passes joined by one CTA barrier; per-lane err/distance terms reduced
// through a transposed shared-memory buffer), so its results are bit-identical
// to that kernel's. Rows are not staged in shared memory: every lane loads its
// V columns of each of its positions' rows (eps, old state, next cache input,
// draw) straight into registers with 16-byte loads, all issued before the
// first is used, and both passes run on registers. Each row crosses the SM's
// load/store path once (in) and the results once (out), against four times
// for the staged form (bulk copy in, a read in each pass, the drift written
// and read back). LMAX bounds the positions per warp (registers: about
// 3-4 rows x V x LMAX floats per thread). No waits of any kind.
template <int V, int NW>
struct RegShape {
  static constexpr int SEG = 32 * V;
  __host__ __device__ static size_t rank_bytes(int P) { return ((size_t)P * 4 + 127) / 128 * 128; }
  static constexpr size_t kTotBytes = (size_t)NW * SEG * 2 * sizeof(float);
  __host__ __device__ static size_t red_bytes(int P) { return ((size_t)2 * P * 33 * sizeof(float) + 127) / 128 * 128; }
  __host__ __device__ static size_t smem_bytes(int P) { return rank_bytes(P) + kTotBytes + red_bytes(P); }
};

template <int V, int NW, int LMAX, bool NOISE, bool CB = false>
__global__ void __launch_bounds__(NW * 32, 1) k_update_reg(Dev d, const float* __restrict__ beps, int par) {
  using Sh = RegShape<V, NW>;
  constexpr int SEG = Sh::SEG;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = d.P;
  const int b = blockIdx.y;
  const int64_t D = d.D;
  int32_t* s_rank = reinterpret_cast<int32_t*>(smem_raw);
  float* s_tot = reinterpret_cast<float*>(smem_raw + Sh::rank_bytes(P));              // [NW][SEG][2]
  float* s_red = reinterpret_cast<float*>(smem_raw + Sh::rank_bytes(P) + Sh::kTotBytes);  // [2][P][33]

  // Everything read before pdl_wait() was written two or more kernels back
  // (the previous update and decision kernels); only the batch eps rows come
  // from the denoiser just before. The ranks do not depend on the window, so
  // they are fetched together with it.
  const Traj tr = d.traj[par * d.B + b];
  const int n_miss = d.ctl->n_miss;
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
    return;
  }
  __syncthreads();
  const int t = tr.t, p = tr.p, e = tr.e;
  const int strip = blockIdx.x;
  const int64_t mycol = (int64_t)strip * SEG + (int64_t)lane * V;
  const bool live = mycol < D;
  float* Xb = d.X + (int64_t)b * (P + 1) * D;
  float* Xh = d.Xhat + (int64_t)b * P * D;
  float* Eh = d.Ehat + (int64_t)b * P * D;
  const int L = (p + NW - 1) / NW;  // <= LMAX (launcher)
  const int j0 = warp * L;
  const int nj = (j0 + L < p ? j0 + L : p) - j0;  // positions of this warp (may be <= 0)

  int rk[LMAX + 1];
#pragma unroll
  for (int g = 0; g <= LMAX; ++g) rk[g] = (g <= nj && j0 + g < p) ? s_rank[j0 + g] : -1;
  const int sl0 = nj > 0 ? (t + j0) % P : 0;        // cache slot of position j0
  const int nx0 = nj > 0 ? (t + j0 + 1) % (P + 1) : 0;  // state-ring slot of x_{t+j0+1}

  Vec<V> eps[LMAX], xo[LMAX], xh[LMAX], zn[LMAX];
  float cm1[LMAX], ec[LMAX], sg[LMAX];
  Vec<V> xstart{}, xfill{}, xc0{};
  if (live) {
    xstart = ldv<V>(Xb + (int64_t)(t % (P + 1)) * D + mycol);
    xfill = ldv<V>(Xb + (int64_t)(e % (P + 1)) * D + mycol);
    if (nj > 0 && j0 > 0 && t + j0 <= e) xc0 = ldv<V>(Xb + (int64_t)((t + j0) % (P + 1)) * D + mycol);
  }
#pragma unroll
  for (int g = 0; g < LMAX; ++g) {
    if (g < nj) {
      const int j = j0 + g;
      cm1[g] = d.cm1[t + j];
      ec[g] = d.ecoef[t + j];
      if (NOISE) sg[g] = d.sigma[t + j];
      if (live) {
        int sl = sl0 + g;
        if (sl >= P) sl -= P;
        int sl1 = sl + 1;
        if (sl1 >= P) sl1 -= P;
        int nx = nx0 + g;
        if (nx >= P + 1) nx -= P + 1;
        if (rk[g] < 0) eps[g] = ld_entry<V, CB>(Eh, (int64_t)sl * D + mycol);
        if (t + j + 1 <= e) xo[g] = ldv<V>(Xb + (int64_t)nx * D + mycol);
        if (j + 1 < p && rk[g + 1] < 0) xh[g] = ld_entry<V, CB>(Xh, (int64_t)sl1 * D + mycol);
        if (NOISE) zn[g] = ldv<V>(d.noise + ((int64_t)b * d.T + t + j) * D + mycol);
      }
    }
  }
  pdl_wait();  // the batch eps rows come from the denoiser that ran just before
  pdl_trigger();  // the successor may now run its prologue
  if (live) {
#pragma unroll
    for (int g = 0; g < LMAX; ++g)
      if (g < nj && rk[g] >= 0) eps[g] = ldv<V>(beps + (int64_t)rk[g] * D + mycol);
  }

  // phase 1: the drifts (kept in eps), the cache update of the misses
  // (Eq. 7), and the compensated sum of the segment
  float rh[V], rl[V];
#pragma unroll
  for (int v = 0; v < V; ++v) { rh[v] = 0.f; rl[v] = 0.f; }
  if (live) {
    Vec<V> xc = j0 == 0 ? xstart : ((t + j0 <= e) ? xc0 : xfill);
#pragma unroll
    for (int g = 0; g < LMAX; ++g) {
      if (g < nj) {
        const int j = j0 + g;
        if (rk[g] >= 0) {  // Eq. 7: the cache takes (x_i, eps_i) of a miss
          int sl = sl0 + g;
          if (sl >= P) sl -= P;
          const int64_t o = (int64_t)sl * D + mycol;
          st_entry<V, CB>(Eh, o, eps[g]);
          st_entry<V, CB>(Xh, o, xc);
        }
        const float2 cm2 = make_float2(cm1[g], cm1[g]), ec2 = make_float2(ec[g], ec[g]);
#pragma unroll
        for (int v = 0; v < V; v += 2) {  // two columns per instruction
          float2 dr = __ffma2_rn(cm2, make_float2(xc.a[v], xc.a[v + 1]),
                                 __fmul2_rn(ec2, make_float2(eps[g].a[v], eps[g].a[v + 1])));
          if (NOISE)
            dr = __ffma2_rn(make_float2(sg[g], sg[g]), make_float2(zn[g].a[v], zn[g].a[v + 1]), dr);
          float2 h = make_float2(rh[v], rh[v + 1]), l = make_float2(rl[v], rl[v + 1]);
          acc_add_x2(h, l, dr);
          rh[v] = h.x; rh[v + 1] = h.y;
          rl[v] = l.x; rl[v + 1] = l.y;
          eps[g].a[v] = dr.x;
          eps[g].a[v + 1] = dr.y;
        }
        xc = (t + j + 1 <= e) ? xo[g] : xfill;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const size_t o = ((size_t)warp * SEG + lane * V + v) * 2;
    s_tot[o] = rh[v];
    s_tot[o + 1] = rl[v];
  }
  __syncthreads();

  // phase 2: carry into this segment, then the new states, errors, distances
  float ch[V], cl[V];
#pragma unroll
  for (int v = 0; v < V; ++v) { ch[v] = xstart.a[v]; cl[v] = 0.f; }
  for (int w = 0; w < warp; ++w) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const size_t o = ((size_t)w * SEG + lane * V + v) * 2;
      acc_add2(ch[v], cl[v], s_tot[o], s_tot[o + 1]);
    }
  }
#pragma unroll
  for (int g = 0; g < LMAX; ++g) {
    if (g < nj) {
      const int j = j0 + g;
      float ev = 0.f, dv = 0.f;
      if (live) {
        const Vec<V> xold = (t + j + 1 <= e) ? xo[g] : xfill;
        Vec<V> xn;
#pragma unroll
        for (int v = 0; v < V; v += 2) {  // two columns per instruction
          float2 h = make_float2(ch[v], ch[v + 1]), l = make_float2(cl[v], cl[v + 1]);
          acc_add_x2(h, l, make_float2(eps[g].a[v], eps[g].a[v + 1]));
          ch[v] = h.x; ch[v + 1] = h.y;
          cl[v] = l.x; cl[v + 1] = l.y;
          const float2 n = x2_add(h, l);
          const float2 df = x2_sub(n, make_float2(xold.a[v], xold.a[v + 1]));
          xn.a[v] = n.x;
          xn.a[v + 1] = n.y;
          ev = fmaf(df.x, df.x, ev);  // the error terms keep their column order
          ev = fmaf(df.y, df.y, ev);
        }
        int nx = nx0 + g;
        if (nx >= P + 1) nx -= P + 1;
        stv<V>(Xb + (int64_t)nx * D + mycol, xn);
        if (j + 1 < p) {
          // the next timestep's cache input: its entry if it is a hit, else
          // this iteration's x_{i+1} (the entry it is about to receive)
          const Vec<V> xc1 = rk[g + 1] < 0 ? xh[g] : as_entry<V, CB>(xold);
#pragma unroll
          for (int v = 0; v < V; v += 2) {
            const float2 dd = x2_sub(make_float2(xn.a[v], xn.a[v + 1]), make_float2(xc1.a[v], xc1.a[v + 1]));
            dv += fabsf(dd.x);
            dv += fabsf(dd.y);
          }
        }
      }
      s_red[(size_t)j * 33 + lane] = ev;
      s_red[(size_t)(P + j) * 33 + lane] = dv;
    }
  }
  __syncthreads();
  // strip partials: one thread per (quantity, position) sums its row of lanes
  // and adds it into the iteration's sums
  for (int r = tid; r < 2 * p; r += NW * 32) {
    const int which = r / p, j = r % p;
    const float* row = s_red + (size_t)(which * P + j) * 33;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 32; c += 4) {
      acc[0] += row[c];
      acc[1] += row[c + 1];
      acc[2] += row[c + 2];
      acc[3] += row[c + 3];
    }
    red_add(d, par, which, b * P + j, (acc[0] + acc[1]) + (acc[2] + acc[3]));
  }
}

template <int V, int NW, int LMAX, bool NOISE, bool CB = false>
cudaError_t launch_reg(const Dev& d, const float* beps, int par, cudaStream_t st) {
  using Sh = RegShape<V, NW>;
  const int nstrip = (int)((d.D + Sh::SEG - 1) / Sh::SEG);
  const size_t smem = Sh::smem_bytes(d.P);
  auto kern = k_update_reg<V, NW, LMAX, NOISE, CB>;
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

// Positions per warp that the register-resident form holds for a window of P
// (8 warps): 0 when it does not apply.
constexpr int kRegMaxL = 13;       // deterministic steps: 3 rows x 4 x 13 floats per thread
constexpr int kRegMaxLNoise = 8;   // stochastic steps: 4 rows x 4 x 8
int reg_lmax(const Dev& d) {
  const int L = (d.P + 7) / 8;
  if (L <= 4) return 4;
  if (L <= 8) return 8;
  if (L <= kRegMaxL && !d.noise) return kRegMaxL;
  return 0;
}

cudaError_t launch_reg_auto(const Dev& d, const float* beps, int par, cudaStream_t st) {
  const int lm = reg_lmax(d);
  if (d.cache_bf16) {  // bfloat16 entries: deterministic steps only (update_bulk_supported)
    if (lm == 4) return launch_reg<4, 8, 4, false, true>(d, beps, par, st);
    if (lm == 8) return launch_reg<4, 8, 8, false, true>(d, beps, par, st);
    return launch_reg<4, 8, kRegMaxL, false, true>(d, beps, par, st);
  }
  if (d.noise) {
    if (lm == 4) return launch_reg<4, 8, 4, true>(d, beps, par, st);
    return launch_reg<4, 8, kRegMaxLNoise, true>(d, beps, par, st);
  }
  if (lm == 4) return launch_reg<4, 8, 4, false>(d, beps, par, st);
  if (lm == 8) return launch_reg<4, 8, 8, false>(d, beps, par, st);
  return launch_reg<4, 8, kRegMaxL, false>(d, beps, par, st);
}

// Shared memory budget per CTA for the tile buffers: enough for the whole
// window when it fits, so every copy is in flight from the start.
constexpr size_t kSmemBudget = 112 * 1024;

template <int V, int NW, int S, bool CLUSTER, bool WAIT_ALL>
cudaError_t launch_tile(const Dev& d, const float* beps, int par, cudaStream_t st) {
  using Sh = TileShape<V, NW, S>;
  const int nstrip = (int)((d.D + Sh::SEG - 1) / Sh::SEG);
  const int ntile_max = (d.P + Sh::TW - 1) / Sh::TW;
  const size_t fixed = Sh::smem_bytes(d.P, 0);
  int nbuf = ntile_max < Sh::kMaxBuf ? ntile_max : Sh::kMaxBuf;
  while (nbuf > 2 && fixed + (size_t)nbuf * Sh::kTileBytes > kSmemBudget) --nbuf;
  if (nbuf < 1) nbuf = 1;
  const size_t smem = Sh::smem_bytes(d.P, nbuf);
  auto kern = k_update_tile<V, NW, S, CLUSTER, WAIT_ALL>;
  // largest dynamic shared memory granted so far, per device and instantiation
  static size_t configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || smem > configured[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev] = smem;
  }
  const int gx = CLUSTER ? (nstrip + kCluster - 1) / kCluster * kCluster : nstrip;
  return launch_ex(kern, dim3(gx, d.B, 1), dim3(NW * 32), smem, st, CLUSTER ? kCluster : 0, d, beps, nstrip,
                   nbuf, d.wait_limit, par);
}

}  // namespace

bool update_bulk_supported(const Dev& d, const float* batch_eps) {
  // 16-byte granularity of bulk copies: every row segment must start on a
  // 16-byte boundary and be a multiple of 16 bytes long. Stochastic steps
  // stage the draws too, in the segment form only. bfloat16 cache entries:
  // the register form only, deterministic steps.
  const bool ok = d.D % 4 == 0 && (reinterpret_cast<uintptr_t>(batch_eps) & 15) == 0;
  if (d.cache_bf16) return ok && !d.noise && reg_lmax(d) > 0;
  if (!d.noise) return ok;
  return ok && (reinterpret_cast<uintptr_t>(d.noise) & 15) == 0 && seg_fits<2, 8, true>(d);
}

// Four columns per lane halve the per-element bookkeeping and the strip
// partials, but quadruple the shared memory of a strip; they pay off while the
// grid still fills the GPU in about one wave (window 100 at 4x64x64: 128 CTAs)
// or several CTAs fit per SM (window 32), not for multi-wave grids of one CTA
// per SM (window 64 at 4x128x128).
template <bool NOISE>
bool prefer_wide_strips(const Dev& d) {
  if (!seg_fits<4, 8, NOISE>(d)) return false;
  static int nsm[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (nsm[dev] == 0 && cudaDeviceGetAttribute(&nsm[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    nsm[dev] = 0;
    return false;
  }
  const size_t smem = SegShape<4, 8, NOISE>::smem_bytes(d.P) + 4096;  // + static shared memory and reserve
  const int per_sm = (int)((size_t)(228 * 1024) / smem);
  const int64_t grid = (int64_t)d.B * ((d.D + SegShape<4, 8>::SEG - 1) / SegShape<4, 8>::SEG);
  return per_sm >= 2 || grid <= nsm[dev];
}

cudaError_t launch_update_bulk(const Dev& d, const float* batch_eps, int par, cudaStream_t st) {
  if (d.cache_bf16) return launch_reg_auto(d, batch_eps, par, st);  // update_bulk_supported
  if (d.bulk_cfg == 12 && reg_lmax(d)) return launch_reg_auto(d, batch_eps, par, st);
  if (d.noise) {  // stochastic steps: the segment forms with the draws (update_bulk_supported)
    if (prefer_wide_strips<true>(d)) {
      if (d.bulk_cfg == 0 && reg_lmax(d)) return launch_reg_auto(d, batch_eps, par, st);
      return launch_seg<4, 8, true>(d, batch_eps, par, st);
    }
    return launch_seg<2, 8, true>(d, batch_eps, par, st);
  }
  switch (d.bulk_cfg) {
    case 0:  // four columns per lane in registers (or staged) when the grid suits
             // them, else the staged window in shared memory, else the tiled pipeline
      if (prefer_wide_strips<false>(d)) {
        if (reg_lmax(d)) return launch_reg_auto(d, batch_eps, par, st);
        return launch_seg<4, 8>(d, batch_eps, par, st);
      }
      if (seg_fits<2, 8>(d)) return launch_seg<2, 8>(d, batch_eps, par, st);
      return launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    case 1: return launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    case 2: return launch_tile<2, 8, 4, true, true>(d, batch_eps, par, st);
    case 3: return launch_tile<2, 4, 8, false, true>(d, batch_eps, par, st);
    case 4: return seg_fits<2, 8>(d) ? launch_seg<2, 8>(d, batch_eps, par, st)
                                     : launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    case 5: return seg_fits<2, 16>(d) ? launch_seg<2, 16>(d, batch_eps, par, st)
                                      : launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    case 6: return seg_fits<1, 8>(d) ? launch_seg<1, 8>(d, batch_eps, par, st)
                                     : launch_tile<1, 8, 4, false, true>(d, batch_eps, par, st);
    case 7: return seg_fits<1, 16>(d) ? launch_seg<1, 16>(d, batch_eps, par, st)
                                      : launch_tile<1, 8, 4, false, true>(d, batch_eps, par, st);
    case 8: return seg_fits<2, 4>(d) ? launch_seg<2, 4>(d, batch_eps, par, st)
                                     : launch_tile<2, 4, 8, false, true>(d, batch_eps, par, st);
    case 9: return launch_tile<2, 8, 2, false, true>(d, batch_eps, par, st);
    case 10: return seg_fits<4, 8>(d) ? launch_seg<4, 8>(d, batch_eps, par, st)
                                      : launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    case 11: return seg_fits<4, 4>(d) ? launch_seg<4, 4>(d, batch_eps, par, st)
                                      : launch_tile<2, 4, 8, false, true>(d, batch_eps, par, st);
    case 12: return reg_lmax(d) ? launch_reg_auto(d, batch_eps, par, st)
                                : launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
    default: return launch_tile<2, 8, 4, false, true>(d, batch_eps, par, st);
  }
}

}  // namespace pa
