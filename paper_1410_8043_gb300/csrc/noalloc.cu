// Per-worker objective for callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocator): code that runs while
// a memory pool owned by someone else is the only source of device memory, a
// monitoring hook invoked from inside an application's hot loop where an
// allocation would synchronise the device or fragment the pool, or an
// embedded deployment with a fixed, pre-sized memory budget.  For them this
// file provides esspt_mf_worker_objective_noalloc(): the same per-entry
// objective as esspt_mf_objective(), summed per worker, whose accumulators
// live in a fixed array compiled into the library instead of in memory the
// caller hands over.
//
// Limits and behaviour:
//  - at most kNoAllocMaxWorkers workers (a 32 KB array, held by every GPU
//    that loads the library until the process exits); larger worker counts
//    are rejected with ESSPT_EINVAL before any work is queued;
//  - the first call on a device looks up the array's device address with the
//    device current (cudaGetSymbolAddress); make that first call outside any
//    stream capture;
//  - all calls share the one array and each call clears it first, so two
//    calls whose work overlaps on the GPU (different streams, no ordering
//    between them) race and may return mixed sums.
#include <mutex>

#include "internal.h"

namespace esspt {
namespace {

constexpr int32_t kNoAllocMaxWorkers = 2048;
constexpr int kMaxDevices = 64;

// Two fp64 sums per worker: sum e^2 at [p] and sum [e^2 + lambda(|L_i|^2+|R_j|^2)]
// at [kNoAllocMaxWorkers + p].
static __device__ __align__(256) double g_worker_sums[2 * kNoAllocMaxWorkers];

std::mutex g_mu;
double* g_sums_ptr[kMaxDevices] = {};

// One warp walks a contiguous span of the entries (sorted by minibatch and
// user, so runs of entries share a worker), keeps the running sums of the
// current worker on lane 0 and folds each run into the block's shared
// accumulators; the block then adds its accumulators to the global array.
__global__ void __launch_bounds__(256) worker_objective_kernel(const float* __restrict__ slot, int64_t n_users,
                                                               int32_t K, const int32_t* __restrict__ rec_u,
                                                               const int32_t* __restrict__ rec_j,
                                                               const float* __restrict__ rec_D,
                                                               const int32_t* __restrict__ worker, int64_t n_obs,
                                                               float lambda, int32_t P, double* sums) {
  __shared__ double sh[2 * kNoAllocMaxWorkers];  // [p] and [kNoAllocMaxWorkers + p]
  for (int i = threadIdx.x; i < 2 * kNoAllocMaxWorkers; i += blockDim.x) sh[i] = 0.0;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t span = (n_obs + nwarps - 1) / nwarps;
  const int64_t k0 = warp * span, k1 = min(n_obs, k0 + span);
  const int32_t K4 = K >> 2;
  const float4* t4 = reinterpret_cast<const float4*>(slot);
  int32_t cur = -1;
  double s1 = 0.0, s2 = 0.0;
  for (int64_t k = k0; k < k1; ++k) {
    const int32_t u = rec_u[k];
    const float4* L = t4 + (int64_t)u * K4;
    const float4* R = t4 + (n_users + rec_j[k]) * K4;
    float dot = 0.f, nl = 0.f, nr = 0.f;
    for (int32_t q = lane; q < K4; q += 32) {
      const float4 l = L[q], r = R[q];
      dot += l.x * r.x + l.y * r.y + l.z * r.z + l.w * r.w;
      nl += l.x * l.x + l.y * l.y + l.z * l.z + l.w * l.w;
      nr += r.x * r.x + r.y * r.y + r.z * r.z + r.w * r.w;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      dot += __shfl_xor_sync(0xffffffffu, dot, off);
      nl += __shfl_xor_sync(0xffffffffu, nl, off);
      nr += __shfl_xor_sync(0xffffffffu, nr, off);
    }
    if (lane == 0) {
      const int32_t p = worker[u];
      if (p != cur) {
        if (cur >= 0) {
          atomicAdd(&sh[cur], s1);
          atomicAdd(&sh[kNoAllocMaxWorkers + cur], s2);
        }
        cur = p;
        s1 = s2 = 0.0;
      }
      const double e = (double)(rec_D[k] - dot);
      s1 += e * e;
      s2 += e * e + (double)lambda * ((double)nl + (double)nr);
    }
  }
  if (lane == 0 && cur >= 0) {
    atomicAdd(&sh[cur], s1);
    atomicAdd(&sh[kNoAllocMaxWorkers + cur], s2);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < P; i += blockDim.x) {
    if (sh[i] != 0.0) atomicAdd(&sums[i], sh[i]);
    if (sh[kNoAllocMaxWorkers + i] != 0.0) atomicAdd(&sums[kNoAllocMaxWorkers + i], sh[kNoAllocMaxWorkers + i]);
  }
}

}  // namespace
}  // namespace esspt

extern "C" esspt_status esspt_mf_worker_objective_noalloc(esspt_ctx* ctx, int32_t version, float lambda,
                                                          double* h_sq, double* h_pen) {
  using namespace esspt;
  if (!ctx) return ESSPT_EINVAL;
  const float* slot = nullptr;
  const int32_t *rec_u = nullptr, *rec_j = nullptr, *worker = nullptr;
  const float* rec_D = nullptr;
  int64_t n_users = 0, n_obs = 0;
  int32_t K = 0, P = 0;
  cudaStream_t st = nullptr;
  esspt_status s = mf_view(ctx, version, &slot, &n_users, &K, &rec_u, &rec_j, &rec_D, &worker, &n_obs, &P, &st);
  if (s != ESSPT_OK) return s;
  if (!h_sq || !h_pen) return mf_fail(ctx, ESSPT_EINVAL, "null output");
  if (P > kNoAllocMaxWorkers)
    return mf_fail(ctx, ESSPT_EINVAL,
                               "esspt_mf_worker_objective_noalloc: more than 2048 workers do not fit its fixed "
                               "accumulator array; use esspt_mf_objective");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return mf_fail(ctx, ESSPT_ECUDA, cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return mf_fail(ctx, ESSPT_EINVAL, "device ordinal too large");
  double* sums = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_sums_ptr[dev]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_worker_sums);
      if (e != cudaSuccess) return mf_fail(ctx, ESSPT_ECUDA, cudaGetErrorString(e));
      g_sums_ptr[dev] = static_cast<double*>(p);
    }
    sums = g_sums_ptr[dev];
  }
  // Every call starts from zero: the array keeps the previous call's sums.
  e = cudaMemsetAsync(sums, 0, sizeof(double) * 2 * kNoAllocMaxWorkers, st);
  if (e == cudaSuccess && n_obs > 0) {
    int sms = 148;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (n_obs + 255) / 256;
    const int blocks = (int)(want < (int64_t)sms * 4 ? (want > 0 ? want : 1) : (int64_t)sms * 4);
    worker_objective_kernel<<<blocks, 256, 0, st>>>(slot, n_users, K, rec_u, rec_j, rec_D, worker, n_obs, lambda, P,
                                                    sums);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(h_sq, sums, sizeof(double) * P, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h_pen, sums + kNoAllocMaxWorkers, sizeof(double) * P, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return mf_fail(ctx, ESSPT_ECUDA, cudaGetErrorString(e));
  return ESSPT_OK;
}
