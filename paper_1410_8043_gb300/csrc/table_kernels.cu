// Table kernels: the read-version schedule, the Clock() copy-forward of the
// version ring, and the generic GET / INC row kernels.
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"
#include "schedule.cuh"

namespace esspt {

// ---------------------------------------------------------------------------
// Schedule: v_p(c) for every worker p; one thread per worker (the rule is in
// schedule.cuh).  The MF clock computes the next schedule inside its item
// merge kernel instead of launching this one.
// ---------------------------------------------------------------------------
__global__ void schedule_kernel(ScheduleArgs a) {
  for (int32_t p = blockIdx.x * blockDim.x + threadIdx.x; p < a.P; p += gridDim.x * blockDim.x)
    schedule_worker(a, p);
}

cudaError_t launch_schedule(const ScheduleArgs& a, cudaStream_t st) {
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((a.P + threads - 1) / threads, 1024);
  schedule_kernel<<<blocks, threads, 0, st>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Copy-forward: slot(c) <- slot(c-1) for a range of rows, so that the
// deltas of clock c can land in place (Clock() merge, Sec. 2.1 / Sec. 4).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) copy_rows_kernel(float4* __restrict__ dst, const float4* __restrict__ src,
                                                        int64_t n4) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; k + 3 * stride < n4; k += 4 * stride) {
    const float4 a = src[k], b = src[k + stride], c = src[k + 2 * stride], d = src[k + 3 * stride];
    dst[k] = a;
    dst[k + stride] = b;
    dst[k + 2 * stride] = c;
    dst[k + 3 * stride] = d;
  }
  for (; k < n4; k += stride) dst[k] = src[k];
}

cudaError_t launch_copy_rows(float* dst, const float* src, int64_t n_floats, cudaStream_t st) {
  const int64_t n4 = n_floats / 4;
  if (n4 == 0) return cudaSuccess;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int threads = 256;
  const int64_t want = (n4 + threads * 4 - 1) / (threads * 4);
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sms * 8));
  copy_rows_kernel<<<blocks, threads, 0, st>>>(reinterpret_cast<float4*>(dst), reinterpret_cast<const float4*>(src),
                                               n4);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// GET: rows of worker p's read version.  One warp per requested row.
// ---------------------------------------------------------------------------
__global__ void get_rows_kernel(const float* __restrict__ ring, int64_t n_rows, int32_t K, int32_t nslots,
                                const int32_t* __restrict__ v, int32_t worker, const int32_t* __restrict__ ids,
                                int64_t n, float* __restrict__ out, uint32_t* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int32_t slot = v[worker] % nslots;
  const int32_t K4 = K >> 2;
  const float4* base = reinterpret_cast<const float4*>(ring + (int64_t)slot * n_rows * K);
  for (int64_t k = warp; k < n; k += nwarps) {
    const int32_t r = ids[k];
    float4* o = reinterpret_cast<float4*>(out + k * K);
    if (r < 0 || r >= n_rows) {
      if (lane == 0) atomicOr(status, kErrRowRange);
      continue;
    }
    const float4* src = base + (int64_t)r * K4;
    for (int32_t q = lane; q < K4; q += 32) o[q] = src[q];
  }
}

cudaError_t launch_get(const float* ring, int64_t n_rows, int32_t K, int32_t nslots, const int32_t* v, int32_t worker,
                       const int32_t* ids, int64_t n, float* out, uint32_t* status, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((n * 32 + threads - 1) / threads, 4096);
  get_rows_kernel<<<blocks, threads, 0, st>>>(ring, n_rows, K, nslots, v, worker, ids, n, out, status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// INC: additive updates into the version being written (Sec. 2.1, Sec. 4).
// ---------------------------------------------------------------------------
__global__ void inc_rows_kernel(float* __restrict__ slot, int64_t n_rows, int32_t K, const int32_t* __restrict__ ids,
                                const float* __restrict__ d, int64_t n, uint32_t* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int32_t K4 = K >> 2;
  for (int64_t k = warp; k < n; k += nwarps) {
    const int32_t r = ids[k];
    if (r < 0 || r >= n_rows) {
      if (lane == 0) atomicOr(status, kErrRowRange);
      continue;
    }
    float4* dst = reinterpret_cast<float4*>(slot) + (int64_t)r * K4;
    const float4* src = reinterpret_cast<const float4*>(d + k * K);
    for (int32_t q = lane; q < K4; q += 32) red_add_v4(dst + q, src[q]);
  }
}

cudaError_t launch_inc(float* slot, int64_t n_rows, int32_t K, const int32_t* ids, const float* d, int64_t n,
                       uint32_t* status, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((n * 32 + threads - 1) / threads, 4096);
  inc_rows_kernel<<<blocks, threads, 0, st>>>(slot, n_rows, K, ids, d, n, status);
  return cudaGetLastError();
}

}  // namespace esspt
