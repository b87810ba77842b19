// Matrix-factorisation SGD on the version ring (Sec. 3.1 updates under the
// SSP / ESSP read schedule).  One clock is, for rows of 36..64 values (the
// work-list path):
//   user_copy_kernel    users without entries: row of version c-1 carried to
//                       version c, unless unchanged over the whole ring;
//   sgd_work16_kernel   every user with entries (its row of version c,
//                       written once) and every chunk of a very active one;
// and for other row widths:
//   sgd_chunks_kernel   entries of very active users, in chunks (if any);
//   sgd_users_kernel    every other user: its row of version c, written once
//                       (sgd_users32_kernel for rows of 68..128 values);
// then, for both:
//   heavy_merge_kernel  rows of the very active users (if any);
//   item_merge_kernel   the Clock() merge of the item rows.
// Item-row (and heavy-user) deltas are summed, unscaled, into zero-initialised
// replica rows so that popular rows spread their fp32 reductions over many
// L2 addresses; the merges apply eta, the hot-row scale and the sum of the
// replicas, then clear them for the next clock.
#include <algorithm>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"
#include "schedule.cuh"

namespace esspt {

namespace {

// Sum over the G lanes of a row group (G a power of two, <= 32).
template <int G>
__device__ __forceinline__ float group_sum(float x, unsigned mask) {
#pragma unroll
  for (int off = G / 2; off > 0; off >>= 1) x += __shfl_xor_sync(mask, x, off, G);
  return x;
}

template <int G>
__device__ __forceinline__ unsigned group_mask(int lane) {
  if constexpr (G == 32) {
    return 0xffffffffu;
  } else {
    return ((1u << G) - 1u) << (lane & ~(G - 1));
  }
}

__device__ __forceinline__ float4 f4_zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }

__device__ __forceinline__ float dot4(float4 a, float4 b) { return a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w; }

__device__ __forceinline__ float4 f4_axpy(float s, float4 x, float4 y) {  // y + s x
  return make_float4(y.x + s * x.x, y.y + s * x.y, y.z + s * x.z, y.w + s * x.w);
}

// Scale of a row's summed update under the hot-row step cap.
__device__ __forceinline__ float cap_scale(int32_t cap, int32_t n) {
  return (cap > 0 && n > cap) ? (float)cap / (float)n : 1.f;
}

// cap / n for a row past the cap, out of line: the rare case stays off the
// common path.
__device__ __noinline__ float capped_scale(int32_t cap, int32_t n) { return (float)cap / (float)n; }

// Ring slot of user u's read version: its worker's version, or in
// row-granular mode the slot its cached row was refreshed to this clock.
__device__ __forceinline__ int32_t user_slot(const SgdArgs& a, int64_t u) {
  return a.row_mode ? __ldg(a.user_slot + u) : __ldg(a.v + __ldg(a.worker + u)) % a.nslots;
}

// Entry t of the minibatch: item, value and the replica row its item update
// adds into; zeros past the end.
__device__ __forceinline__ void load_entry(const SgdArgs& a, int32_t t, int32_t& j, float& d, int32_t& dst) {
  if (t < a.n_b) {
    const uint64_t pol = policy_evict_first();
    j = ld_stream_i32(a.rec_j + t, pol);
    d = ld_stream_f32(a.rec_D + t, pol);
    dst = ld_stream_i32(a.rec_dst + t, pol);
  } else {
    j = 0;
    d = 0.f;
    dst = 0;
  }
}

// A group's sliding window over the minibatch entries: lane l holds entry
// W + l (cur) and W + G + l (nxt, prefetched).
template <int G>
struct Window {
  int32_t W;
  int32_t cj, cdst, nj, ndst;
  float cd, nd;

  __device__ __forceinline__ void reload(const SgdArgs& a, int32_t start, int glane) {
    W = start;
    load_entry(a, W + glane, cj, cd, cdst);
    load_entry(a, W + G + glane, nj, nd, ndst);
  }
  // Make entry t (>= W) part of cur.
  __device__ __forceinline__ void cover(const SgdArgs& a, int32_t t, int glane) {
    if (t < W + G) return;
    if (t < W + 2 * G) {
      W += G;
      cj = nj;
      cd = nd;
      cdst = ndst;
      load_entry(a, W + G + glane, nj, nd, ndst);
    } else {
      reload(a, t, glane);
    }
  }
};

// U entries (U = 1 or 2) of one row group, sitting in lanes i, i+1, ... of the
// window's cur part, all of one user whose read-version row is Lv.  For each:
// e = D - L.R at the read version; gL += e R (process_range adds the
// -lambda L terms once); the item update e L - lambda R goes (unscaled) into
// the entry's replica row of dR.  Rq and dRq already point at the lane's first
// slice (+glane); act[t] marks the slices inside the row (glane + t G < K4).
template <int G, int NV, int U>
__device__ __forceinline__ void process_entries(const SgdArgs& a, const Window<G>& win, int32_t i,
                                                const float4 (&Lv)[NV], float4 (&gL)[NV],
                                                const float4* __restrict__ Rq, float4* __restrict__ dRq,
                                                const bool (&act)[NV], unsigned gmask, int32_t K4, float& loss) {
  float4 R[U][NV];
  int32_t dst[U];
  float d[U], part[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const float4* row = Rq + __shfl_sync(gmask, win.cj, i + u, G) * K4;
#pragma unroll
    for (int t = 0; t < NV; ++t) R[u][t] = act[t] ? __ldg(row + t * G) : f4_zero();
  }
#pragma unroll
  for (int u = 0; u < U; ++u) {
    d[u] = __shfl_sync(gmask, win.cd, i + u, G);
    dst[u] = __shfl_sync(gmask, win.cdst, i + u, G);
    part[u] = 0.f;
#pragma unroll
    for (int t = 0; t < NV; ++t) part[u] += dot4(Lv[t], R[u][t]);
  }
#pragma unroll
  for (int off = G / 2; off > 0; off >>= 1) {
#pragma unroll
    for (int u = 0; u < U; ++u) part[u] += __shfl_xor_sync(gmask, part[u], off, G);
  }
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const float e = d[u] - part[u];
    loss += e * e;
    float4* out = dRq + dst[u] * a.dR_ld;
#pragma unroll
    for (int t = 0; t < NV; ++t) {
      const float4 r = R[u][t], l = Lv[t];
      gL[t].x += e * r.x;
      gL[t].y += e * r.y;
      gL[t].z += e * r.z;
      gL[t].w += e * r.w;
      red_add_v4_if(out + t * G,
                    make_float4(e * l.x - a.lambda * r.x, e * l.y - a.lambda * r.y, e * l.z - a.lambda * r.z,
                                e * l.w - a.lambda * r.w),
                    act[t]);
    }
  }
}

// All entries [beg, end) of one user (or chunk), two at a time:
// gL += sum_k (e_k R_j - lambda L_i).
template <int G, int NV>
__device__ __forceinline__ void process_range(const SgdArgs& a, Window<G>& win, int32_t beg, int32_t end,
                                              const float4 (&Lv)[NV], float4 (&gL)[NV],
                                              const float4* __restrict__ Rq, float4* __restrict__ dRq,
                                              const bool (&act)[NV], int glane, unsigned gmask, int32_t K4,
                                              float& loss) {
  int32_t t = beg;
  while (t < end) {
    win.cover(a, t, glane);
    const int32_t lim = min(end, win.W + G);
#ifdef ESSPT_STEP4
    for (; t + 4 <= lim; t += 4) process_entries<G, NV, 4>(a, win, t - win.W, Lv, gL, Rq, dRq, act, gmask, K4, loss);
#endif
    for (; t + 2 <= lim; t += 2) process_entries<G, NV, 2>(a, win, t - win.W, Lv, gL, Rq, dRq, act, gmask, K4, loss);
    if (t < lim) {
      process_entries<G, NV, 1>(a, win, t - win.W, Lv, gL, Rq, dRq, act, gmask, K4, loss);
      ++t;
    }
  }
  const float nl = -(float)(end - beg) * a.lambda;
#pragma unroll
  for (int t2 = 0; t2 < NV; ++t2) gL[t2] = f4_axpy(nl, Lv[t2], gL[t2]);
}

__device__ __forceinline__ float4 f4_add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

// Sum of n replica slices p[0], p[stride], ..., each cleared after reading;
// eight independent loads in flight per lane.
__device__ __forceinline__ float4 sum_and_clear(float4* p, int32_t n, int32_t stride) {
  float4 acc = f4_zero();
  int32_t r = 0;
  for (; r + 8 <= n; r += 8) {
    float4 x[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) x[k] = p[(int64_t)(r + k) * stride];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      p[(int64_t)(r + k) * stride] = f4_zero();
      acc = f4_add(acc, x[k]);
    }
  }
  for (; r < n; ++r) {
    acc = f4_add(acc, p[(int64_t)r * stride]);
    p[(int64_t)r * stride] = f4_zero();
  }
  return acc;
}

__device__ __forceinline__ void flush_loss(double* out, float v, int lane) {
  if (out == nullptr) return;
  double x = (double)v;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  if (lane == 0 && x != 0.0) atomicAdd(out, x);
}

}  // namespace

// Each warp takes 32 consecutive users (one coalesced metadata load); a row
// group of G lanes walks G of them in order, prefetching the next user's rows
// and the next window of entries while it computes the current user.
//   L_i^c = L_i^base + eta s_i sum_k (e_k R_j - lambda L_i)   (written once)
// Users with more than kHeavy entries are left to the chunk / heavy-merge path.
#ifndef ESSPT_USERS_MINB
#define ESSPT_USERS_MINB 3
#endif
template <int G, int NV>
__global__ void __launch_bounds__(256, ESSPT_USERS_MINB) sgd_users_kernel(SgdArgs a) {
  const int lane = threadIdx.x & 31;
  const int glane = lane & (G - 1);
  const int grp = lane / G;
  const unsigned gmask = group_mask<G>(lane);
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  // Per-lane base pointers: slice t of row r of a table is p[r * K4 + t * G].
  float4* ringq = reinterpret_cast<float4*>(a.ring) + glane;
  float4* outq = ringq + (int64_t)a.slot_out * slot4;
  const float4* baseq = ringq + (int64_t)a.slot_base * slot4;
  float4* dRq = reinterpret_cast<float4*>(a.dR) + glane;
  bool act[NV];
#pragma unroll
  for (int t = 0; t < NV; ++t) act[t] = glane + t * G < K4;
  const uint64_t pol = policy_evict_first();
  float loss = 0.f;
  const int64_t warp_id = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

  for (int64_t u0 = warp_id * 32; u0 < a.n_users; u0 += nwarps * 32) {
    const int64_t uu = u0 + lane;
    int32_t m_beg = 0, m_end = 0, m_vs = 0;
    if (uu < a.n_users) {
      m_beg = __ldg(a.uoff + uu);
      m_end = __ldg(a.uoff + uu + 1);
      m_vs = user_slot(a, uu);
    }
    const int64_t g0 = u0 + (int64_t)grp * G;
    const int32_t nusers = (int32_t)max((int64_t)0, min((int64_t)G, (int64_t)a.n_users - g0));
    if (nusers == 0) continue;

    Window<G> win;
    win.reload(a, __shfl_sync(gmask, m_beg, 0, G), glane);

    // rows of the group's first user
    int32_t nvs = __shfl_sync(gmask, m_vs, 0, G);
    int32_t nbeg = __shfl_sync(gmask, m_beg, 0, G);
    int32_t nend = __shfl_sync(gmask, m_end, 0, G);
    float4 Lvn[NV], Lbn[NV];
    bool nsame;
    {
      const int32_t n = nend - nbeg;
      nsame = (nvs == a.slot_base) && n > 0;
      const float4* pv = ringq + (int64_t)nvs * slot4 + g0 * K4;
      const float4* pb = baseq + g0 * K4;
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const bool in = act[t] && n <= kHeavy;
        Lvn[t] = ld_stream_if(pv + t * G, pol, in && n > 0);
        Lbn[t] = ld_stream_if(pb + t * G, pol, in && !nsame);
      }
    }

    for (int32_t t = 0; t < nusers; ++t) {
      const int64_t u = g0 + t;
      const int32_t vs = nvs, beg = nbeg, end = nend;
      const bool same = nsame;
      float4 Lv[NV], Lb[NV];
#pragma unroll
      for (int k = 0; k < NV; ++k) {
        Lv[k] = Lvn[k];
        Lb[k] = Lbn[k];
      }
      if (t + 1 < nusers) {  // prefetch the next user's rows
        nvs = __shfl_sync(gmask, m_vs, t + 1, G);
        nbeg = __shfl_sync(gmask, m_beg, t + 1, G);
        nend = __shfl_sync(gmask, m_end, t + 1, G);
        const int32_t n = nend - nbeg;
        nsame = (nvs == a.slot_base) && n > 0;
        const float4* pv = ringq + (int64_t)nvs * slot4 + (u + 1) * K4;
        const float4* pb = baseq + (u + 1) * K4;
#pragma unroll
        for (int k = 0; k < NV; ++k) {
          const bool in = act[k] && n <= kHeavy;
          Lvn[k] = ld_stream_if(pv + k * G, pol, in && n > 0);
          Lbn[k] = ld_stream_if(pb + k * G, pol, in && !nsame);
        }
      }
      const int32_t n = end - beg;
      if (n > kHeavy) continue;
      float4 gL[NV];
#pragma unroll
      for (int k = 0; k < NV; ++k) gL[k] = f4_zero();
      if (n > 0) {
        const float4* Rq = a.row_mode ? ringq : ringq + (int64_t)vs * slot4 + (int64_t)a.n_users * K4;
        process_range<G, NV>(a, win, beg, end, Lv, gL, Rq, dRq, act, glane, gmask, K4, loss);
      }
      const float sc = a.eta * cap_scale(a.cap, n);
      float4* po = outq + u * K4;
#pragma unroll
      for (int k = 0; k < NV; ++k) st_stream_if(po + k * G, f4_axpy(sc, gL[k], same ? Lv[k] : Lb[k]), pol, act[k]);
    }
  }
  flush_loss(a.sq_loss, glane == 0 ? loss : 0.f, lane);
}

#ifndef ESSPT_USERS32_MINB
#define ESSPT_USERS32_MINB 3
#endif
#ifndef ESSPT_U32_UNIT
#define ESSPT_U32_UNIT 16
#endif
#ifndef ESSPT_U32_USERCOST
#define ESSPT_U32_USERCOST 5
#endif
constexpr int kUnit = ESSPT_U32_UNIT;
constexpr int32_t kUserCost = ESSPT_U32_USERCOST;

// Rows of 68..128 values (17..32 float4 slices), one slice per lane: the
// whole warp holds one user's row (lane l owns slice l of L_i and of its
// update sum) and takes 4 of the user's entries per step, gathering each item
// row with one coalesced load.  The 4 partial dot products are reduced with
// a transposing butterfly (6 shuffles) that leaves entry q's dot product on
// lanes 8q .. 8q+7.  The user's rows at the read and base versions are staged
// in shared memory one user ahead by cp.async.
//
// Each warp takes one contiguous range of users, the ranges balanced by a
// cost of entries plus kUserCost per user (found by a 16-way search of the
// user offsets at the start), so that warps finish together whatever the
// spread of entries per user.  The range is walked in units of kUnit users:
// the metadata of the current unit sits in lanes [0, kUnit), that of the next
// in lanes [kUnit, 2 kUnit), so the row staging and the entry window run on
// across unit boundaries.
__global__ void __launch_bounds__(256, ESSPT_USERS32_MINB) sgd_users32_kernel(SgdArgs a) {
  __shared__ __align__(16) float4 stage[8][2][2][32];  // [warp][buffer][read row, base row][slice]
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int q = lane >> 3;  // the entry of a step whose dot product this lane ends up with
  const int32_t K4 = a.K >> 2;
  const bool on = lane < K4;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* outq = ring4 + (int64_t)a.slot_out * slot4;
  const float4* base4 = ring4 + (int64_t)a.slot_base * slot4;
  float4* dRq = reinterpret_cast<float4*>(a.dR) + lane;
  const uint64_t pol = policy_evict_first();
  float loss = 0.f;

  int32_t ua, ub;
  {
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int half = lane >> 4, hl = lane & 15;
    const int64_t total = (int64_t)a.n_b + (int64_t)kUserCost * a.n_users;
    const int64_t target = total * (w + half) / nw;
    int32_t lo = 0, hi = a.n_users;
    while (__any_sync(0xffffffffu, lo < hi)) {
      const int32_t step = (hi - lo + 15) / 16;
      const int32_t x = (int32_t)min((int64_t)lo + (int64_t)hl * step, (int64_t)hi);
      const bool ge = lo < hi && (int64_t)__ldg(a.uoff + x) + (int64_t)kUserCost * x >= target;
      const unsigned bits = (__ballot_sync(0xffffffffu, ge) >> (16 * half)) & 0xffffu;
      if (lo < hi) {
        if (bits == 0u) {
          lo = (int32_t)min((int64_t)lo + (int64_t)15 * step, (int64_t)hi) + 1;
        } else {
          const int f = __ffs(bits) - 1;
          const int32_t xf = (int32_t)min((int64_t)lo + (int64_t)f * step, (int64_t)hi);
          if (f == 0) {
            hi = lo;
          } else {
            lo = (int32_t)min((int64_t)lo + (int64_t)(f - 1) * step, (int64_t)hi) + 1;
            hi = xf;
          }
        }
      }
    }
    ua = __shfl_sync(0xffffffffu, lo, 0);
    ub = __shfl_sync(0xffffffffu, lo, 16);
  }

  int32_t m_beg = 0, m_end = 0, m_vs = 0;
  auto load_meta = [&](int64_t first, int lo) {
    if (lane >= lo && lane < lo + kUnit) {
      const int64_t uu = first + (lane - lo);
      m_beg = m_end = m_vs = 0;
      if (uu < ub) {
        m_beg = __ldg(a.uoff + uu);
        m_end = __ldg(a.uoff + uu + 1);
        m_vs = user_slot(a, uu);
      }
    }
  };
  auto stage_user = [&](int ml, int64_t u, int b) {
    const int32_t vs = __shfl_sync(0xffffffffu, m_vs, ml);
    const int32_t n = __shfl_sync(0xffffffffu, m_end, ml) - __shfl_sync(0xffffffffu, m_beg, ml);
    const bool same = vs == a.slot_base && n > 0;
    const bool in = on && n <= kHeavy;
    const float4* pv = ring4 + (int64_t)vs * slot4 + u * K4 + (on ? lane : 0);
    const float4* pb = base4 + u * K4 + (on ? lane : 0);
    cp_async16_hint(&stage[wib][b][0][lane], pv, in && n > 0, pol);
    cp_async16_hint(&stage[wib][b][1][lane], pb, in && !same, pol);
    cp_async_commit();
  };

  load_meta(ua, 0);
  load_meta((int64_t)ua + kUnit, kUnit);
  Window<32> win;
  if (ua < ub) {
    stage_user(0, ua, 0);
    win.reload(a, __shfl_sync(0xffffffffu, m_beg, 0), lane);
  }
  int b = 0;
  for (int64_t u0 = ua; u0 < ub; u0 += kUnit) {
    const int32_t nusers = (int32_t)min((int64_t)kUnit, (int64_t)ub - u0);
    for (int32_t t = 0; t < nusers; ++t, b ^= 1) {
      cp_async_wait_all();
      __syncwarp();
      if (t + 1 < nusers) {
        stage_user(t + 1, u0 + t + 1, b ^ 1);
      } else if (u0 + kUnit < ub) {
        stage_user(kUnit, u0 + kUnit, b ^ 1);
      }
      const int32_t vs = __shfl_sync(0xffffffffu, m_vs, t);
      const int32_t beg = __shfl_sync(0xffffffffu, m_beg, t);
      const int32_t end = __shfl_sync(0xffffffffu, m_end, t);
      const int32_t n = end - beg;
      if (n > kHeavy) continue;
      const float4 Lv = stage[wib][b][0][lane];
      // Lanes past the row end read slice 0 (their staged L is zero), so the
      // item-row loads need no row-end predicate.
      const float4* Rq =
          (a.row_mode ? ring4 : ring4 + (int64_t)vs * slot4 + (int64_t)a.n_users * K4) + (on ? lane : 0);
      float4 gL = f4_zero();
      // One step: entries tt .. tt+cnt-1 of the user.  It is compiled twice,
      // for full steps (cnt = 4, the common case), whose loads need no
      // predicate, and for the user's last, partial one, whose missing
      // entries load nothing, get e = 0 and add nothing.
      auto step = [&](auto full_tag, int32_t tt, int32_t cnt) {
        constexpr bool kFull = decltype(full_tag)::value;
        const int w0 = tt - win.W;
        float4 R[4];
        int32_t dst[4];
        float p[4];
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const int src = kFull ? w0 + e4 : min(w0 + e4, 31);
          const int32_t j = __shfl_sync(0xffffffffu, win.cj, src);
          dst[e4] = __shfl_sync(0xffffffffu, win.cdst, src);
          R[e4] = (kFull || e4 < cnt) ? __ldg(Rq + j * K4) : f4_zero();
          p[e4] = dot4(Lv, R[e4]);
        }
        // Transposing butterfly: lanes with bit 4 clear keep entries {0, 1},
        // the others {2, 3}; then bit 3 picks one of the pair; the last three
        // levels sum over the 8 lanes that share bits 3 and 4.
        const bool h4 = lane & 16, h3 = lane & 8;
        float k0 = h4 ? p[2] : p[0], k1 = h4 ? p[3] : p[1];
        k0 += __shfl_xor_sync(0xffffffffu, h4 ? p[0] : p[2], 16);
        k1 += __shfl_xor_sync(0xffffffffu, h4 ? p[1] : p[3], 16);
        float dot = h3 ? k1 : k0;
        dot += __shfl_xor_sync(0xffffffffu, h3 ? k0 : k1, 8);
        dot += __shfl_xor_sync(0xffffffffu, dot, 4);
        dot += __shfl_xor_sync(0xffffffffu, dot, 2);
        dot += __shfl_xor_sync(0xffffffffu, dot, 1);
        const float dq = __shfl_sync(0xffffffffu, win.cd, kFull ? w0 + q : min(w0 + q, 31));
        const float eq = (kFull || q < cnt) ? dq - dot : 0.f;
        if ((lane & 7) == 0) loss += eq * eq;
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const float e = __shfl_sync(0xffffffffu, eq, 8 * e4);
          const float4 r = R[e4];
          gL.x += e * r.x;
          gL.y += e * r.y;
          gL.z += e * r.z;
          gL.w += e * r.w;
          red_add_v4_if(dRq + dst[e4] * a.dR_ld,
                        make_float4(e * Lv.x - a.lambda * r.x, e * Lv.y - a.lambda * r.y,
                                    e * Lv.z - a.lambda * r.z, e * Lv.w - a.lambda * r.w),
                        on && (kFull || e4 < cnt));
        }
      };
      for (int32_t tt = beg; tt < end;) {
        win.cover(a, tt, lane);
        const int32_t cnt = min(4, min(end - tt, win.W + 32 - tt));
        if (cnt == 4) {
          step(std::true_type{}, tt, cnt);
        } else {
          step(std::false_type{}, tt, cnt);
        }
        tt += cnt;
      }
      const bool same = vs == a.slot_base && n > 0;
      const float4 lb = stage[wib][b][same ? 0 : 1][lane];
      float sc = a.eta;
      if (a.cap > 0 && n > a.cap) sc = a.eta * capped_scale(a.cap, n);
      const float4 g = f4_axpy(-(float)n * a.lambda, Lv, gL);
      st_stream_if(outq + (u0 + t) * K4 + lane, f4_axpy(sc, g, lb), pol, on);
    }
    m_beg = __shfl_down_sync(0xffffffffu, m_beg, kUnit);
    m_end = __shfl_down_sync(0xffffffffu, m_end, kUnit);
    m_vs = __shfl_down_sync(0xffffffffu, m_vs, kUnit);
    load_meta(u0 + 2 * kUnit, kUnit);
    __syncwarp();
  }
  flush_loss(a.sq_loss, loss, lane);
}

// Rows of 36..64 values (9..16 float4 slices) on the work-list path.
//
// sgd_work16_kernel: one half-warp per work item of minibatch b, the two
// halves of a warp on consecutive items in lockstep.  An item is either a
// user with 1..kHeavy entries (written once: L^c = L^base + eta s sum_k(e_k
// R_j - lambda L_i)) or a 64-entry chunk of a heavy user (its unscaled
// partial sum goes into the chunk's replica row of dL, merged by
// heavy_merge_kernel).  Lane l owns slice l mod 16 of its half's row L_i; a
// step takes 4 entries per half, so each gather instruction brings two item
// rows, and a transposing butterfly over the 16 lanes of a half (4 shuffles)
// leaves entry e's dot product on lanes 4e .. 4e+3.  Items are mostly users
// with a few entries, so pairing them keeps most gather slots busy and
// shares the per-item work (metadata, staging, the row store) between two
// items.  The items' rows at the read and base versions are staged in shared
// memory one pair ahead by cp.async, and each warp walks one contiguous range
// of items, balanced by entries plus kItemCost per item.
#ifndef ESSPT_WORK16_MINB
#define ESSPT_WORK16_MINB 4
#endif
#ifndef ESSPT_W16_ITEMCOST
#define ESSPT_W16_ITEMCOST 6
#endif
constexpr int32_t kItemCost = ESSPT_W16_ITEMCOST;
constexpr int kW16Unit = 16;      // items per metadata unit (8 pairs)
constexpr int32_t kNoItem = -2;   // metadata of a slot past the warp's range

__global__ void __launch_bounds__(256, ESSPT_WORK16_MINB) sgd_work16_kernel(ChunkArgs c) {
  const SgdArgs& a = c.a;
  __shared__ __align__(16) float4 stage[8][2][2][32];  // [warp][buffer][read row, base row][half * 16 + slice]
#if ESSPT_W16_HOT > 0
  // per warp and lane: the summed updates of the minibatch's hot items
  __shared__ __align__(16) float4 hacc[8][kHot][32];
#endif
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int h = lane >> 4;      // half: its own item
  const int hb = lane & 16;     // first lane of the half
  const int r = lane & 15;      // slice of the row this lane owns
  const int32_t K4 = a.K >> 2;
  const bool on = r < K4;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* outq = ring4 + (int64_t)a.slot_out * slot4;
  const float4* base4 = ring4 + (int64_t)a.slot_base * slot4;
  float4* dRq = reinterpret_cast<float4*>(a.dR) + (on ? r : 0);
  float4* dL4 = reinterpret_cast<float4*>(c.dL);
  const int32_t n_items = (int32_t)c.n_chunks;
  const uint64_t pol = policy_evict_first();
  float loss = 0.f;

  // Item x starts at entry chunk[x].y; the entries of consecutive items are
  // contiguous, so the cost of items [0, x) is chunk[x].y + kItemCost x.
  auto item_beg = [&](int32_t x) -> int64_t { return x < n_items ? (int64_t)__ldg(&c.chunk[x].y) : (int64_t)a.n_b; };
  int32_t ia, ib;
  {
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int half = lane >> 4, hl = lane & 15;
    const int64_t total = (int64_t)a.n_b + (int64_t)kItemCost * n_items;
    const int64_t target = total * (w + half) / nw;
    int32_t lo = 0, hi = n_items;
    while (__any_sync(0xffffffffu, lo < hi)) {
      const int32_t step = (hi - lo + 15) / 16;
      const int32_t x = (int32_t)min((int64_t)lo + (int64_t)hl * step, (int64_t)hi);
      const bool ge = lo < hi && item_beg(x) + (int64_t)kItemCost * x >= target;
      const unsigned bits = (__ballot_sync(0xffffffffu, ge) >> (16 * half)) & 0xffffu;
      if (lo < hi) {
        if (bits == 0u) {
          lo = (int32_t)min((int64_t)lo + (int64_t)15 * step, (int64_t)hi) + 1;
        } else {
          const int f = __ffs(bits) - 1;
          const int32_t xf = (int32_t)min((int64_t)lo + (int64_t)f * step, (int64_t)hi);
          if (f == 0) {
            hi = lo;
          } else {
            lo = (int32_t)min((int64_t)lo + (int64_t)(f - 1) * step, (int64_t)hi) + 1;
            hi = xf;
          }
        }
      }
    }
    ia = __shfl_sync(0xffffffffu, lo, 0);
    ib = __shfl_sync(0xffffffffu, lo, 16);
  }
  if (ia >= ib) {
    flush_loss(a.sq_loss, 0.f, lane);
    return;
  }
#if ESSPT_W16_HOT > 0
  for (int hs = 0; hs < kHot; ++hs) hacc[wib][hs][lane] = f4_zero();
#endif

  // Item metadata: the current unit in lanes [0, 16), the next in [16, 32).
  int4 m_it = make_int4(0, 0, 0, kNoItem);
  int32_t m_vs = 0;
  auto load_meta = [&](int64_t first, int lo) {
    if (lane >= lo && lane < lo + kW16Unit) {
      const int64_t x = first + (lane - lo);
      m_it = make_int4(0, 0, 0, kNoItem);
      m_vs = 0;
      if (x < ib) {
        m_it = __ldg(c.chunk + x);
        m_vs = user_slot(a, m_it.x);
      }
    }
  };
  // Stage the pair whose first item's metadata sits in lane ml: half h its
  // item's read-version row and, for a user item whose read version is not
  // the base, its base row.
  auto stage_pair = [&](int ml, int bb) {
    const int32_t u = __shfl_sync(0xffffffffu, m_it.x, ml + h);
    const int32_t dst = __shfl_sync(0xffffffffu, m_it.w, ml + h);
    const int32_t vs = __shfl_sync(0xffffffffu, m_vs, ml + h);
    const int64_t row = (int64_t)u * K4 + (on ? r : 0);
    cp_async16_hint(&stage[wib][bb][0][lane], ring4 + (int64_t)vs * slot4 + row, on && dst != kNoItem, pol);
    cp_async16_hint(&stage[wib][bb][1][lane], base4 + row, on && dst == -1 && vs != a.slot_base, pol);
    cp_async_commit();
  };

  load_meta(ia, 0);
  load_meta((int64_t)ia + kW16Unit, kW16Unit);
  stage_pair(0, 0);
  int bb = 0;
  // This half's window of 16 entries: lane hb + i holds entry W + i.
  int32_t W = 0, cj = 0, cdst = 0;
  float cd = 0.f;
  for (int64_t x0 = ia; x0 < ib; x0 += kW16Unit) {
    const int32_t nloc = (int32_t)min((int64_t)kW16Unit, (int64_t)ib - x0);
    for (int32_t t = 0; 2 * t < nloc; ++t, bb ^= 1) {
      cp_async_wait_all();
      __syncwarp();
      if (2 * t + 2 < nloc) {
        stage_pair(2 * t + 2, bb ^ 1);
      } else if (x0 + kW16Unit < ib) {
        stage_pair(kW16Unit, bb ^ 1);
      }
      const int src = 2 * t + h;
      const int32_t u = __shfl_sync(0xffffffffu, m_it.x, src);
      const int32_t beg = __shfl_sync(0xffffffffu, m_it.y, src);
      const int32_t dst = __shfl_sync(0xffffffffu, m_it.w, src);
      const int32_t z = __shfl_sync(0xffffffffu, m_it.z, src);  // every lane takes part in every shuffle
      const int32_t end = dst == kNoItem ? beg : z;
      const int32_t vs = __shfl_sync(0xffffffffu, m_vs, src);
      const int32_t n = end - beg;
      const float4 Lv = stage[wib][bb][0][lane];
      // Lanes past the row end read slice 0 of the item rows; their staged L is
      // zero, so they add nothing to the dot products.
      const float4* Rq =
          (a.row_mode ? ring4 : ring4 + (int64_t)vs * slot4 + (int64_t)a.n_users * K4) + (on ? r : 0);
      float4 gL = f4_zero();
      W = beg;
      load_entry(a, W + r, cj, cd, cdst);
      const int32_t nsteps = (n + 3) >> 2;
      const int32_t steps = max(nsteps, __shfl_xor_sync(0xffffffffu, nsteps, 16));
      // One step: entries tt .. tt+cnt-1 of this half's item (cnt <= 4, 0 once
      // the item is done while the other half's continues).  Compiled twice:
      // for steps where both halves have 4 entries, whose loads need no
      // predicate, and for the others.
      auto step = [&](auto full_tag, int32_t w0, int32_t cnt) {
        constexpr bool kFull = decltype(full_tag)::value;
        float4 R[4];
        int32_t dsts[4];
        float p[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int sl = hb + (kFull ? w0 + e : min(w0 + e, 15));
          const int32_t j = __shfl_sync(0xffffffffu, cj, sl);
          dsts[e] = __shfl_sync(0xffffffffu, cdst, sl);
          R[e] = (kFull || e < cnt) ? __ldg(Rq + j * K4) : f4_zero();
          p[e] = dot4(Lv, R[e]);
        }
        // Transposing butterfly over the 16 lanes of a half: bit 3 of the
        // lane keeps entries {0,1} or {2,3}, bit 2 one of the pair, bits 1
        // and 0 sum; lanes 4e .. 4e+3 end with entry e's dot product.
        const bool b3 = r & 8, b2 = r & 4;
        float k0 = b3 ? p[2] : p[0], k1 = b3 ? p[3] : p[1];
        k0 += __shfl_xor_sync(0xffffffffu, b3 ? p[0] : p[2], 8);
        k1 += __shfl_xor_sync(0xffffffffu, b3 ? p[1] : p[3], 8);
        float dot = b2 ? k1 : k0;
        dot += __shfl_xor_sync(0xffffffffu, b2 ? k0 : k1, 4);
        dot += __shfl_xor_sync(0xffffffffu, dot, 2);
        dot += __shfl_xor_sync(0xffffffffu, dot, 1);
        const int kq = r >> 2;  // the entry this lane's dot product belongs to
        const float dq = __shfl_sync(0xffffffffu, cd, hb + (kFull ? w0 + kq : min(w0 + kq, 15)));
        const float eq = (kFull || kq < cnt) ? dq - dot : 0.f;
        if ((r & 3) == 0) loss += eq * eq;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float ev = __shfl_sync(0xffffffffu, eq, hb + 4 * e);
          const float4 rr = R[e];
          gL.x += ev * rr.x;
          gL.y += ev * rr.y;
          gL.z += ev * rr.z;
          gL.w += ev * rr.w;
          const float4 dv = make_float4(ev * Lv.x - a.lambda * rr.x, ev * Lv.y - a.lambda * rr.y,
                                        ev * Lv.z - a.lambda * rr.z, ev * Lv.w - a.lambda * rr.w);
          const bool val = on && (kFull || e < cnt);
#if ESSPT_W16_HOT > 0
          const int32_t dd = dsts[e];
          red_add_v4_if(dRq + dd * a.dR_ld, dv, val && dd >= 0);
          if (val && dd < 0) hacc[wib][-1 - dd][lane] = f4_add(hacc[wib][-1 - dd][lane], dv);
#else
          red_add_v4_if(dRq + dsts[e] * a.dR_ld, dv, val);
#endif
        }
      };
      for (int32_t sidx = 0; sidx < steps; ++sidx) {
        const int32_t tt = beg + 4 * sidx;
        const int32_t cnt = max(0, min(4, end - tt));
        if (__any_sync(0xffffffffu, cnt > 0 && tt + cnt > W + 16)) {  // slide a half's window
          if (cnt > 0 && tt + cnt > W + 16) {
            W = tt;
            load_entry(a, W + r, cj, cd, cdst);
          }
        }
        if (__all_sync(0xffffffffu, cnt == 4)) {
          step(std::true_type{}, tt - W, 4);
        } else {
          step(std::false_type{}, tt - W, cnt);
        }
      }
      const float4 g = f4_axpy(-(float)n * a.lambda, Lv, gL);
      if (dst >= 0) {  // a heavy user's chunk: unscaled partial sum into its replica row
        if (on) red_add_v4(dL4 + (int64_t)dst * K4 + r, g);
      } else if (dst == -1) {
        const float4 lb = vs == a.slot_base ? Lv : stage[wib][bb][1][lane];
        float sc = a.eta;
        if (a.cap > 0 && n > a.cap) sc = a.eta * capped_scale(a.cap, n);
        st_stream_if(outq + (int64_t)u * K4 + r, f4_axpy(sc, g, lb), pol, on);
        if (r == 0 && a.chg != nullptr) a.chg[u] = a.clock;
      }
    }
    m_it.x = __shfl_down_sync(0xffffffffu, m_it.x, kW16Unit);
    m_it.y = __shfl_down_sync(0xffffffffu, m_it.y, kW16Unit);
    m_it.z = __shfl_down_sync(0xffffffffu, m_it.z, kW16Unit);
    m_it.w = __shfl_down_sync(0xffffffffu, m_it.w, kW16Unit);
    m_vs = __shfl_down_sync(0xffffffffu, m_vs, kW16Unit);
    load_meta(x0 + 2 * kW16Unit, kW16Unit);
    __syncwarp();
  }
  cp_async_wait_all();
#if ESSPT_W16_HOT > 0
  // Hot items: both halves' sums, added once into a replica row of the item
  // (the warp index picks among its replicas).
  __syncwarp();
  {
    const int64_t wg = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_items_all = a.n_rows - a.n_users;
    float4* dR4 = reinterpret_cast<float4*>(a.dR);
    for (int hs = 0; hs < kHot; ++hs) {
      const int32_t j = __ldg(a.hot_item + hs);
      const float4 v = f4_add(hacc[wib][hs][lane], hacc[wib][hs][lane ^ 16]);
      if (j >= 0 && h == 0 && on) {
        const int32_t e0 = __ldg(a.item_rep + j), e1 = __ldg(a.item_rep + j + 1);
        const int32_t rr = (int32_t)(wg & (int64_t)(e1 - e0));  // replicas are a power of two
        const int64_t row = rr == 0 ? (int64_t)j : n_items_all + e0 + rr - 1;
        red_add_v4(dR4 + row * a.dR_ld + r, v);
      }
    }
  }
#endif
  flush_loss(a.sq_loss, loss, lane);
}

// Forward copy of the users with no entry in minibatch b (version c-1 row to
// version c), on the work-list path.  One warp per 32 consecutive users: their
// entry counts come from two coalesced offset loads, and the warp copies the
// rows of the idle ones, all loads of a unit in flight before the stores.  A
// row unchanged over the last s+2 clocks is skipped: the ring slot of version
// c last held version c-(s+2), which is already its value.
#ifndef ESSPT_COPY_BATCH
#define ESSPT_COPY_BATCH 8
#endif
__global__ void __launch_bounds__(256, 4) user_copy_kernel(SgdArgs a) {
  const int lane = threadIdx.x & 31;
  const int h = lane >> 4, r = lane & 15;
  const int32_t K4 = a.K >> 2;
  const bool on = r < K4;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* outq = ring4 + (int64_t)a.slot_out * slot4;
  const float4* base4 = ring4 + (int64_t)a.slot_base * slot4;
  const uint64_t pol = policy_evict_first();
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const bool may_skip = a.chg != nullptr && a.clock > a.copy_all_until;
  for (int64_t u0 = warp * 32; u0 < a.n_users; u0 += nwarps * 32) {
    const int64_t u = u0 + lane;
    bool idle = false;
    if (u < a.n_users) {
      idle = __ldg(a.uoff + u + 1) == __ldg(a.uoff + u);
      // unchanged over the whole ring: the slot of version c already holds it
      if (idle && may_skip && a.clock - ld_stream_i32(a.chg + u, pol) >= a.nslots) idle = false;
    }
    const unsigned mask = __ballot_sync(0xffffffffu, idle);
    if (mask == 0u) continue;
    // rows 2q + h of the unit, q = 0..15, in batches
    const int64_t first = (u0 + h) * K4 + (on ? r : 0);
    const float4* src = base4 + first;
    float4* dst = outq + first;
    const unsigned mine = on ? (mask >> h) : 0u;  // bit q: row 2q + h is idle
#pragma unroll 1
    for (int q0 = 0; q0 < 16; q0 += ESSPT_COPY_BATCH) {
      float4 v[ESSPT_COPY_BATCH];
#pragma unroll
      for (int q = 0; q < ESSPT_COPY_BATCH; ++q)
        v[q] = ld_stream_if(src + (q0 + q) * 2 * K4, pol, (mine >> (2 * (q0 + q))) & 1u);
#pragma unroll
      for (int q = 0; q < ESSPT_COPY_BATCH; ++q)
        st_stream_if(dst + (q0 + q) * 2 * K4, v[q], pol, (mine >> (2 * (q0 + q))) & 1u);
    }
  }
}

// Row-granular SSP (Sec. 4 client cache, a clock c_param per cached row):
// thread x refreshes user x's row (if the user has entries) and entry x's
// item row in the cache of the reading worker.  All threads that refresh one
// (worker, row) in a clock write the same value, c-1, so the races are
// benign and every read of the row in the clock sees one version.
__global__ void __launch_bounds__(256) row_refresh_kernel(RowRefreshArgs a) {
  const int32_t lo = a.c - 1 - a.s;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t n = max((int64_t)a.n_users, (int64_t)a.n_b);
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < n; x += stride) {
    if (x < a.n_users) {
      int32_t* V = a.rowver + (int64_t)__ldg(a.worker + x) * a.n_rows + x;
      int32_t v = *V;
      if (__ldg(a.uoff + x + 1) > __ldg(a.uoff + x) && (v < 0 || v < lo)) {
        v = a.c - 1;
        *V = v;
      }
      a.user_slot[x] = v < 0 ? 0 : v % a.nslots;
    }
    if (x < a.n_b) {
      const int32_t j = __ldg(a.rec_j + x);
      const int64_t r = (int64_t)a.n_users + j;
      int32_t* V = a.rowver + (int64_t)__ldg(a.worker + __ldg(a.rec_u + x)) * a.n_rows + r;
      int32_t v = *V;
      if (v < 0 || v < lo) {
        v = a.c - 1;
        *V = v;
      }
      a.rec_row[x] = (int32_t)((int64_t)(v % a.nslots) * a.n_rows + r);
    }
  }
}

// Chunks of at most kChunk entries of users with more than kHeavy entries:
// the chunk's partial user update sum (e R - lambda L) goes, unscaled, into
// one of its user's replica rows of dL; item updates as in the user kernel.
template <int G, int NV>
__global__ void __launch_bounds__(256) sgd_chunks_kernel(ChunkArgs c) {
  const SgdArgs& a = c.a;
  const int lane = threadIdx.x & 31;
  const int glane = lane & (G - 1);
  const unsigned gmask = group_mask<G>(lane);
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  const float4* ring4 = reinterpret_cast<const float4*>(a.ring);
  float4* dR4 = reinterpret_cast<float4*>(a.dR);
  float4* dL4 = reinterpret_cast<float4*>(c.dL);
  bool act[NV];
#pragma unroll
  for (int t = 0; t < NV; ++t) act[t] = glane + t * G < K4;
  float loss = 0.f;
  const int64_t first = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * (32 / G);
  const int64_t step = (((int64_t)gridDim.x * blockDim.x) >> 5) * (32 / G);
  for (int64_t kb = first; kb < c.n_chunks; kb += step) {
    const int64_t k = kb + lane / G;
    if (k < c.n_chunks) {
      const int4 ch = c.chunk[k];
      const int32_t vs = user_slot(a, ch.x);
      const float4* Lrow = ring4 + (int64_t)vs * slot4 + (int64_t)ch.x * K4;
      float4 Lv[NV], gL[NV];
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        Lv[t] = q < K4 ? Lrow[q] : f4_zero();
        gL[t] = f4_zero();
      }
      Window<G> win;
      win.reload(a, ch.y, glane);
      const float4* Rq = (a.row_mode ? ring4 : ring4 + (int64_t)vs * slot4 + (int64_t)a.n_users * K4) + glane;
      process_range<G, NV>(a, win, ch.y, ch.z, Lv, gL, Rq, dR4 + glane, act, glane, gmask, K4, loss);
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        if (q < K4) red_add_v4(dL4 + (int64_t)ch.w * K4 + q, gL[t]);
      }
    }
  }
  flush_loss(a.sq_loss, glane == 0 ? loss : 0.f, lane);
}

// Heavy user rows: L^c = L^base + eta s sum of the user's replica rows (row u
// of dL, then rows hv.y .. hv.y + hv.z - 2); the replicas are cleared for the
// next clock.  One warp per heavy user.
__global__ void __launch_bounds__(256) heavy_merge_kernel(HeavyMergeArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* dL4 = reinterpret_cast<float4*>(a.dL);
  for (int64_t h = warp; h < a.n_heavy; h += nwarps) {
    const int4 hv = a.heavy[h];
    const float sc = a.eta * cap_scale(a.cap, hv.w);
    for (int32_t q = lane; q < K4; q += 32) {
      float4* p0 = dL4 + (int64_t)hv.x * K4 + q;
      float4 acc = *p0;
      *p0 = f4_zero();
      acc = f4_add(acc, sum_and_clear(dL4 + (int64_t)hv.y * K4 + q, hv.z - 1, K4));
      const float4 b = ring4[(int64_t)a.slot_base * slot4 + (int64_t)hv.x * K4 + q];
      ring4[(int64_t)a.slot_out * slot4 + (int64_t)hv.x * K4 + q] = f4_axpy(sc, acc, b);
    }
    if (lane == 0 && a.chg != nullptr) a.chg[hv.x] = a.clock;
  }
}

// Clock() merge of the item rows (Sec. 2.1 additive updates, Sec. 4 server
// clock): R^c_j = R^base_j + eta s_j sum of j's replica rows; replicas
// cleared.  Each thread merges U (item, float4 slice) pairs.  Replica 0 of
// item j is row j of dR, so the common single-replica item needs no index
// load before its data loads: every load of a thread is issued at once.  With do_schedule the
// first P threads also compute the next clock's read versions (the SGD
// kernels of this clock, the only readers of v, have finished).
template <int U>  // (item, slice) pairs per thread per round, the loads of all in flight
__global__ void __launch_bounds__(256) item_merge_kernel(ItemMergeArgs a) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t nth = (int64_t)gridDim.x * blockDim.x;
  if (a.do_schedule)
    for (int64_t p = tid; p < a.sched.P; p += nth) schedule_worker(a.sched, (int32_t)p);
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* dR4 = reinterpret_cast<float4*>(a.dR);
  // n_items * K/4 < 2^31 (checked at load), so the (item, slice) split is a
  // 32-bit division
  const int64_t total = (int64_t)a.n_items * K4;
  for (int64_t x0 = tid; x0 < total; x0 += U * nth) {
    float4 first[U], base[U];
    int32_t e0[U], e1[U], cnt[U];
    int64_t row[U], dofs[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int64_t x = min(x0 + k * nth, total - 1);
      const uint32_t j = (uint32_t)x / (uint32_t)K4;
      const int32_t q = (int32_t)((uint32_t)x - j * (uint32_t)K4);
      row[k] = ((int64_t)a.n_users + j) * K4 + q;
      dofs[k] = (int64_t)j * a.dR_ld + q;
      first[k] = dR4[dofs[k]];
      base[k] = ring4[(int64_t)a.slot_base * slot4 + row[k]];
      e0[k] = __ldg(a.item_rep + j);
      e1[k] = __ldg(a.item_rep + j + 1);
      cnt[k] = __ldg(a.item_cnt + j);
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      if (x0 + k * nth >= total) break;
      dR4[dofs[k]] = f4_zero();
      float4 acc = first[k];
      if (e1[k] > e0[k]) {
        const int32_t q = (int32_t)(dofs[k] % a.dR_ld);
        acc = f4_add(acc, sum_and_clear(dR4 + ((int64_t)a.n_items + e0[k]) * a.dR_ld + q, e1[k] - e0[k], a.dR_ld));
      }
      const float sc = a.eta * cap_scale(a.cap, cnt[k]);
      ring4[(int64_t)a.slot_out * slot4 + row[k]] = f4_axpy(sc, acc, base[k]);
    }
  }
}

namespace {

int sm_count() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 148;
  }
  return sms;
}

int grid_for(int64_t work_items, int64_t per_block, int max_per_sm) {
  const int64_t want = (work_items + per_block - 1) / per_block;
  return (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sm_count() * max_per_sm));
}

// One resident wave of sgd_users32_kernel; its warps balance the users among
// themselves.
#ifndef ESSPT_U32_CARVEOUT
#define ESSPT_U32_CARVEOUT 25
#endif
cudaError_t run_users32(const SgdArgs& a, cudaStream_t st) {
  static int per_sm = 0;
  if (per_sm == 0) {
    // Ask for the smallest shared-memory carveout that holds the resident
    // blocks' staging buffers (percent of the maximum), leaving the rest of
    // the SM's memory to L1, which caches the gathered item rows.
    if (ESSPT_U32_CARVEOUT >= 0)
      cudaFuncSetAttribute(sgd_users32_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, ESSPT_U32_CARVEOUT);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, sgd_users32_kernel, 256, 0) != cudaSuccess ||
        per_sm <= 0)
      per_sm = 1;
  }
  sgd_users32_kernel<<<grid_for((a.n_users + kUnit - 1) / kUnit, 8, per_sm), 256, 0, st>>>(a);
  return cudaGetLastError();
}

template <int G, int NV>
struct UsersF {
  static cudaError_t run(const SgdArgs& a, cudaStream_t st) {
    // 8 warps per block, 32 users per warp
    sgd_users_kernel<G, NV><<<grid_for(a.n_users, 256, 8), 256, 0, st>>>(a);
    return cudaGetLastError();
  }
};
template <int G, int NV>
struct ChunksF {
  static cudaError_t run(const ChunkArgs& c, cudaStream_t st) {
    if (c.n_chunks <= 0) return cudaSuccess;
    sgd_chunks_kernel<G, NV><<<grid_for(c.n_chunks, 256 / G, 8), 256, 0, st>>>(c);
    return cudaGetLastError();
  }
};

// Row-group shape for K: G lanes per row (power of two <= 32), NV float4 per
// lane.  K is a multiple of 4 in [4, 512].
template <template <int, int> class F, typename Arg>
cudaError_t dispatch_k(int32_t K, const Arg& a, cudaStream_t st) {
  const int32_t K4 = K / 4;
  if (K4 <= 1) return F<1, 1>::run(a, st);
  if (K4 <= 2) return F<2, 1>::run(a, st);
  if (K4 <= 4) return F<4, 1>::run(a, st);
  if (K4 <= 8) return F<8, 1>::run(a, st);
  if (K4 <= 16) return F<16, 1>::run(a, st);
  if (K4 <= 32) return F<32, 1>::run(a, st);
  if (K4 <= 64) return F<32, 2>::run(a, st);
  if (K4 <= 96) return F<32, 3>::run(a, st);
  return F<32, 4>::run(a, st);
}

}  // namespace

cudaError_t launch_sgd_users(const SgdArgs& a, cudaStream_t st) {
  if (a.K > 64 && a.K <= 128) return run_users32(a, st);
  return dispatch_k<UsersF>(a.K, a, st);
}
cudaError_t launch_sgd_chunks(const ChunkArgs& c, cudaStream_t st) { return dispatch_k<ChunksF>(c.a.K, c, st); }

// One resident wave of sgd_work16_kernel; its warps balance the items among
// themselves.
#ifndef ESSPT_W16_CARVEOUT
#define ESSPT_W16_CARVEOUT 50
#endif
cudaError_t launch_sgd_work16(const ChunkArgs& c, cudaStream_t st) {
  if (c.n_chunks <= 0) return cudaSuccess;
  static int per_sm = 0;
  if (per_sm == 0) {
    // The smallest shared-memory carveout that holds the resident blocks'
    // staging buffers (percent of the maximum): the rest of the SM's memory is
    // L1, which keeps the popular item rows.
    if (ESSPT_W16_CARVEOUT >= 0)
      cudaFuncSetAttribute(sgd_work16_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, ESSPT_W16_CARVEOUT);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, sgd_work16_kernel, 256, 0) != cudaSuccess ||
        per_sm <= 0)
      per_sm = 1;
  }
  sgd_work16_kernel<<<grid_for((c.n_chunks + kW16Unit - 1) / kW16Unit, 8, std::min(per_sm, kWorkBlocksPerSm)), 256,
                      0, st>>>(c);
  return cudaGetLastError();
}

cudaError_t launch_user_copy(const SgdArgs& a, cudaStream_t st) {
  if (a.n_users <= 0) return cudaSuccess;
  user_copy_kernel<<<grid_for((a.n_users + 31) / 32, 8, kCopyBlocksPerSm), 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_row_refresh(const RowRefreshArgs& a, cudaStream_t st) {
  const int64_t n = std::max<int64_t>(a.n_users, a.n_b);
  if (n <= 0) return cudaSuccess;
  row_refresh_kernel<<<grid_for(n, 256, 8), 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_heavy_merge(const HeavyMergeArgs& a, cudaStream_t st) {
  if (a.n_heavy <= 0) return cudaSuccess;
  heavy_merge_kernel<<<grid_for(a.n_heavy, 8, 8), 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_item_merge(const ItemMergeArgs& a, cudaStream_t st) {
  const int64_t work = std::max<int64_t>((int64_t)a.n_items * (a.K >> 2), a.do_schedule ? a.sched.P : 0);
  if (work <= 0) return cudaSuccess;
  // Every thread's loads are independent, so the whole merge is one set of
  // in-flight requests.  Eight (item, slice) pairs per thread: more loads in
  // flight per thread beat more threads with one each (0.019 against
  // 0.029 ms per clock on mid; 74 against 207 us on a 200k-item table).
  item_merge_kernel<8><<<(unsigned)std::min<int64_t>((work + 2047) / 2048, (int64_t)1 << 30), 256, 0, st>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Objective (Sec. 3.1, Sec. 5) over all entries: sum e^2 and
// sum [e^2 + lambda(|L_i|^2 + |R_j|^2)], fp32 residuals, fp64 sums.
// One warp per entry.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) objective_kernel(const float* __restrict__ slot, int64_t n_users, int32_t K,
                                                        const int32_t* __restrict__ rec_u,
                                                        const int32_t* __restrict__ rec_j,
                                                        const float* __restrict__ rec_D, int64_t n_obs, float lambda,
                                                        double* out2) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int32_t K4 = K >> 2;
  const float4* t4 = reinterpret_cast<const float4*>(slot);
  double s1 = 0.0, s2 = 0.0;
  for (int64_t k = warp; k < n_obs; k += nwarps) {
    const float4* L = t4 + (int64_t)rec_u[k] * K4;
    const float4* R = t4 + (n_users + rec_j[k]) * K4;
    float dot = 0.f, nl = 0.f, nr = 0.f;
    for (int32_t q = lane; q < K4; q += 32) {
      const float4 l = L[q], r = R[q];
      dot += dot4(l, r);
      nl += dot4(l, l);
      nr += dot4(r, r);
    }
    dot = group_sum<32>(dot, 0xffffffffu);
    nl = group_sum<32>(nl, 0xffffffffu);
    nr = group_sum<32>(nr, 0xffffffffu);
    if (lane == 0) {
      const double e = (double)(rec_D[k] - dot);
      s1 += e * e;
      s2 += e * e + (double)lambda * ((double)nl + (double)nr);
    }
  }
  __shared__ double sh[2][8];
  const int w = threadIdx.x >> 5;
  if (lane == 0) {
    sh[0][w] = s1;
    sh[1][w] = s2;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double x = 0.0, y = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
      x += sh[0][i];
      y += sh[1][i];
    }
    atomicAdd(out2, x);
    atomicAdd(out2 + 1, y);
  }
}

cudaError_t launch_objective(const float* slot, int64_t n_users, int32_t K, const int32_t* rec_u, const int32_t* rec_j,
                             const float* rec_D, int64_t n_obs, float lambda, double* out2, cudaStream_t st) {
  cudaError_t err = cudaMemsetAsync(out2, 0, 2 * sizeof(double), st);
  if (err != cudaSuccess || n_obs == 0) return err;
  objective_kernel<<<grid_for(n_obs, 8, 16), 256, 0, st>>>(slot, n_users, K, rec_u, rec_j, rec_D, n_obs, lambda, out2);
  return cudaGetLastError();
}

}  // namespace esspt
