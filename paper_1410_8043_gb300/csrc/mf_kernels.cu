// Matrix-factorisation SGD on the version ring (Sec. 3.1 updates under the
// SSP / ESSP read schedule): the fused per-clock kernel, the kernel for the
// entries of very active users, and the objective.
#include <cfloat>

#include "internal.h"
#include "ptx.cuh"

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

// Entries processed per batch of independent R-row gathers.
constexpr int kBatch = 4;

// Process entries [beg, end) of one user whose read-version row is Lv (lane
// slices of NV float4).  Accumulates the user's summed gradient term
// sum(e R_j - lambda L_i) into gL and issues every item row's scaled update
// eta s_j (e L_i - lambda R_j) into version c.  Returns the sum of e^2 on the
// group's lane 0.
template <int G, int NV>
__device__ __forceinline__ float process_entries(const SgdArgs& a, int32_t beg, int32_t end, const float4 (&Lv)[NV],
                                                 float4 (&gL)[NV], const float4* __restrict__ Rv_base,
                                                 float4* __restrict__ Rout_base, int glane, unsigned gmask,
                                                 int32_t K4) {
  float loss = 0.f;
  for (int32_t t0 = beg; t0 < end; t0 += G) {
    // Lane l of the group fetches entry t0 + l and its item's scale.
    const int32_t nb = min(G, end - t0);
    int32_t my_j = 0;
    float my_d = 0.f, my_s = 1.f;
    if (glane < nb) {
      my_j = a.rec_j[t0 + glane];
      my_d = a.rec_D[t0 + glane];
      if (a.cap > 0) {
        const int32_t cnt = a.item_cnt[my_j];
        if (cnt > a.cap) my_s = (float)a.cap / (float)cnt;
      }
    }
    for (int32_t b0 = 0; b0 < nb; b0 += kBatch) {
      int32_t jj[kBatch];
      float4 R[kBatch][NV];
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        jj[u] = __shfl_sync(gmask, my_j, b0 + u, G);
#pragma unroll
        for (int t = 0; t < NV; ++t) {
          const int32_t q = glane + t * G;
          R[u][t] = (b0 + u < nb && q < K4) ? Rv_base[(int64_t)jj[u] * K4 + q] : f4_zero();
        }
      }
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        const float d = __shfl_sync(gmask, my_d, b0 + u, G);
        const float sj = __shfl_sync(gmask, my_s, b0 + u, G);
        if (b0 + u >= nb) break;
        float part = 0.f;
#pragma unroll
        for (int t = 0; t < NV; ++t) part += dot4(Lv[t], R[u][t]);
        const float e = d - group_sum<G>(part, gmask);
        loss += e * e;
        const float ce = a.eta * sj * e, cl = a.eta * sj * a.lambda;
#pragma unroll
        for (int t = 0; t < NV; ++t) {
          const int32_t q = glane + t * G;
          if (q < K4) {
            const float4 r = R[u][t], l = Lv[t];
            gL[t].x += e * r.x - a.lambda * l.x;
            gL[t].y += e * r.y - a.lambda * l.y;
            gL[t].z += e * r.z - a.lambda * l.z;
            gL[t].w += e * r.w - a.lambda * l.w;
            red_add_v4(Rout_base + (int64_t)jj[u] * K4 + q,
                       make_float4(ce * l.x - cl * r.x, ce * l.y - cl * r.y, ce * l.z - cl * r.z,
                                   ce * l.w - cl * r.w));
          }
        }
      }
    }
  }
  return loss;
}

template <int G>
__device__ __forceinline__ void flush_loss(double* out, float v, int lane) {
  if (out == nullptr) return;
  double x = (double)v;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  if (lane == 0 && x != 0.0) atomicAdd(out, x);
}

}  // namespace

// One row group per user: L_i^c = L_i^{base} + eta s_i sum_k (e_k R_j - lambda L_i),
// written once (no atomics); every entry's item update goes to version c by
// a vector reduction at L2.  Users with more than kHeavy entries only get the
// copy here; their entries are handled by sgd_chunks_kernel afterwards.
template <int G, int NV>
__global__ void __launch_bounds__(256) sgd_users_kernel(SgdArgs a) {
  const int lane = threadIdx.x & 31;
  const int glane = lane & (G - 1);
  const unsigned gmask = group_mask<G>(lane);
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* out4 = ring4 + (int64_t)a.slot_out * slot4;
  const uint64_t pol = policy_evict_first();
  float loss = 0.f;
  // Groups of a warp stay together across the loop (uniform trip count).
  const int64_t warp_first = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * (32 / G);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t ubase = warp_first; ubase < a.n_users; ubase += nwarps * (32 / G)) {
    const int64_t u = ubase + lane / G;
    if (u < a.n_users) {
      const int32_t vs = a.v[a.worker[u]] % a.nslots;
      const int32_t beg = a.uoff[u], end = a.uoff[u + 1];
      const float4* Lv_row = ring4 + (int64_t)vs * slot4 + u * K4;
      const float4* Lb_row = ring4 + (int64_t)a.slot_base * slot4 + u * K4;
      float4 Lv[NV], Lb[NV], gL[NV];
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        Lv[t] = q < K4 ? ld_stream(Lv_row + q, pol) : f4_zero();
        gL[t] = f4_zero();
      }
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        Lb[t] = (vs == a.slot_base || q >= K4) ? Lv[t] : ld_stream(Lb_row + q, pol);
      }
      const int32_t n = end - beg;
      float scale = 0.f;
      if (n <= kHeavy) {
        const float4* Rv_base = ring4 + (int64_t)vs * slot4 + (int64_t)a.n_users * K4;
        float4* Rout_base = out4 + (int64_t)a.n_users * K4;
        loss += process_entries<G, NV>(a, beg, end, Lv, gL, Rv_base, Rout_base, glane, gmask, K4);
        scale = a.eta * ((a.cap > 0 && n > a.cap) ? (float)a.cap / (float)n : 1.f);
      }
      float4* Lo_row = out4 + u * K4;
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        if (q < K4) {
          const float4 b = Lb[t], g = gL[t];
          st_stream(Lo_row + q, make_float4(b.x + scale * g.x, b.y + scale * g.y, b.z + scale * g.z, b.w + scale * g.w),
                    pol);
        }
      }
    }
  }
  flush_loss<G>(a.sq_loss, glane == 0 ? loss : 0.f, lane);
}

// Entries of users with more than kHeavy entries in the minibatch, split in
// chunks of at most kChunk entries; each chunk adds its partial user update
// to version c by vector reductions (after sgd_users_kernel copied the row).
template <int G, int NV>
__global__ void __launch_bounds__(256) sgd_chunks_kernel(ChunkArgs c) {
  const SgdArgs& a = c.a;
  const int lane = threadIdx.x & 31;
  const int glane = lane & (G - 1);
  const unsigned gmask = group_mask<G>(lane);
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  float4* ring4 = reinterpret_cast<float4*>(a.ring);
  float4* out4 = ring4 + (int64_t)a.slot_out * slot4;
  float loss = 0.f;
  const int64_t warp_first = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * (32 / G);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t kbase = warp_first; kbase < c.n_chunks; kbase += nwarps * (32 / G)) {
    const int64_t k = kbase + lane / G;
    if (k < c.n_chunks) {
      const int32_t u = c.chunk_user[k];
      const int32_t vs = a.v[a.worker[u]] % a.nslots;
      const float4* Lv_row = ring4 + (int64_t)vs * slot4 + (int64_t)u * K4;
      float4 Lv[NV], gL[NV];
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        Lv[t] = q < K4 ? Lv_row[q] : f4_zero();
        gL[t] = f4_zero();
      }
      const float4* Rv_base = ring4 + (int64_t)vs * slot4 + (int64_t)a.n_users * K4;
      float4* Rout_base = out4 + (int64_t)a.n_users * K4;
      loss += process_entries<G, NV>(a, c.chunk_begin[k], c.chunk_end[k], Lv, gL, Rv_base, Rout_base, glane, gmask,
                                     K4);
      const int32_t n = a.uoff[u + 1] - a.uoff[u];
      const float scale = a.eta * ((a.cap > 0 && n > a.cap) ? (float)a.cap / (float)n : 1.f);
      float4* Lo_row = out4 + (int64_t)u * K4;
#pragma unroll
      for (int t = 0; t < NV; ++t) {
        const int32_t q = glane + t * G;
        if (q < K4) {
          const float4 g = gL[t];
          red_add_v4(Lo_row + q, make_float4(scale * g.x, scale * g.y, scale * g.z, scale * g.w));
        }
      }
    }
  }
  flush_loss<G>(a.sq_loss, glane == 0 ? loss : 0.f, lane);
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

template <int G, int NV>
cudaError_t launch_users_t(const SgdArgs& a, cudaStream_t st) {
  const int threads = 256;
  const int64_t groups_per_block = threads / G;
  const int64_t want = (a.n_users + groups_per_block - 1) / groups_per_block;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sm_count() * 8));
  sgd_users_kernel<G, NV><<<blocks, threads, 0, st>>>(a);
  return cudaGetLastError();
}

template <int G, int NV>
cudaError_t launch_chunks_t(const ChunkArgs& c, cudaStream_t st) {
  if (c.n_chunks <= 0) return cudaSuccess;
  const int threads = 256;
  const int64_t groups_per_block = threads / G;
  const int64_t want = (c.n_chunks + groups_per_block - 1) / groups_per_block;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sm_count() * 8));
  sgd_chunks_kernel<G, NV><<<blocks, threads, 0, st>>>(c);
  return cudaGetLastError();
}

// Row-group shape for K values: G lanes per row (power of two <= 32), NV
// float4 per lane.  K is a multiple of 4 in [4, 512].
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

template <int G, int NV>
struct UsersF {
  static cudaError_t run(const SgdArgs& a, cudaStream_t st) { return launch_users_t<G, NV>(a, st); }
};
template <int G, int NV>
struct ChunksF {
  static cudaError_t run(const ChunkArgs& a, cudaStream_t st) { return launch_chunks_t<G, NV>(a, st); }
};

}  // namespace

cudaError_t launch_sgd_users(const SgdArgs& a, cudaStream_t st) { return dispatch_k<UsersF>(a.K, a, st); }
cudaError_t launch_sgd_chunks(const ChunkArgs& c, cudaStream_t st) { return dispatch_k<ChunksF>(c.a.K, c, st); }

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
    double a = 0.0, b = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
      a += sh[0][i];
      b += sh[1][i];
    }
    atomicAdd(out2, a);
    atomicAdd(out2 + 1, b);
  }
}

cudaError_t launch_objective(const float* slot, int64_t n_users, int32_t K, const int32_t* rec_u, const int32_t* rec_j,
                             const float* rec_D, int64_t n_obs, float lambda, double* out2, cudaStream_t st) {
  cudaError_t err = cudaMemsetAsync(out2, 0, 2 * sizeof(double), st);
  if (err != cudaSuccess || n_obs == 0) return err;
  const int threads = 256;
  const int64_t want = (n_obs + 7) / 8;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sm_count() * 16));
  objective_kernel<<<blocks, threads, 0, st>>>(slot, n_users, K, rec_u, rec_j, rec_D, n_obs, lambda, out2);
  return cudaGetLastError();
}

}  // namespace esspt
