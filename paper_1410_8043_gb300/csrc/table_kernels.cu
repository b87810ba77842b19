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
// VAP in-transit norms (Sec. 2.1): for k = 1..kmax, the max over the table of
// |X[c-1] - X[c-1-k]|, folded per block and combined with an integer atomic
// max on the bits of the non-negative fp32 value (which orders like the
// value).  Candidates are taken 8 at a time so that each pass reads X[c-1]
// once for 8 older versions.
// ---------------------------------------------------------------------------
constexpr int kVapBatch = 8;

__device__ __forceinline__ float vap_absdiff_max(float m, float4 a, float4 b) {
  const float d0 = fabsf(a.x - b.x), d1 = fabsf(a.y - b.y), d2 = fabsf(a.z - b.z), d3 = fabsf(a.w - b.w);
  // fmaxf drops NaN; a NaN difference must fail the bound, so it becomes +inf.
  const bool nan = (d0 != d0) || (d1 != d1) || (d2 != d2) || (d3 != d3);
  return nan ? __int_as_float(0x7f800000) : fmaxf(fmaxf(m, fmaxf(d0, d1)), fmaxf(d2, d3));
}

__global__ void __launch_bounds__(256) vap_norms_kernel(const float4* __restrict__ ring, int64_t slot4, int32_t nslots,
                                                        int32_t c, int32_t k0, int32_t nk, uint32_t* __restrict__ norm) {
  __shared__ float red[kVapBatch][8];
  float m[kVapBatch];
#pragma unroll
  for (int t = 0; t < kVapBatch; ++t) m[t] = 0.f;
  const float4* cur = ring + (int64_t)((c - 1) % nslots) * slot4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < slot4; q += stride) {
    const float4 x = cur[q];
#pragma unroll
    for (int t = 0; t < kVapBatch; ++t) {
      if (t < nk) {
        const int32_t ver = c - 1 - (k0 + t);
        m[t] = vap_absdiff_max(m[t], x, ring[(int64_t)(ver % nslots) * slot4 + q]);
      }
    }
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int t = 0; t < kVapBatch; ++t) {
    float v = m[t];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
    if (lane == 0) red[t][wid] = v;
  }
  __syncthreads();
  if (threadIdx.x < kVapBatch && (int)threadIdx.x < nk) {
    float v = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) v = fmaxf(v, red[threadIdx.x][w]);
    if (v > 0.f) atomicMax(norm + k0 + threadIdx.x, __float_as_uint(v));
  }
}

cudaError_t launch_vap_norms(const float* ring, int64_t slot_floats, int32_t nslots, int32_t c, int32_t kmax,
                             uint32_t* norm, cudaStream_t st) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t slot4 = slot_floats / 4;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>((slot4 + 255) / 256, (int64_t)sms * 8));
  for (int32_t k0 = 1; k0 <= kmax; k0 += kVapBatch) {
    const int32_t nk = std::min(kVapBatch, kmax - k0 + 1);
    vap_norms_kernel<<<blocks, 256, 0, st>>>(reinterpret_cast<const float4*>(ring), slot4, nslots, c, k0, nk, norm);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
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
                                int64_t n, float* __restrict__ out, uint32_t* status, int32_t* rowver, int32_t c,
                                int32_t s, int32_t* vmin) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int32_t K4 = K >> 2;
  const int64_t slot4 = n_rows * K4;
  const int32_t wslot = rowver ? 0 : v[worker] % nslots;
  for (int64_t k = warp; k < n; k += nwarps) {
    const int32_t r = ids[k];
    float4* o = reinterpret_cast<float4*>(out + k * K);
    if (r < 0 || r >= n_rows) {
      if (lane == 0) atomicOr(status, kErrRowRange);
      continue;
    }
    int32_t slot = wslot;
    if (rowver) {
      // Row-granular cache: refresh the row to c-1 if it is missing or too
      // stale (every refresh of it in this clock writes the same value).
      int32_t ver = 0;
      if (lane == 0) {
        int32_t* V = rowver + (int64_t)worker * n_rows + r;
        ver = *V;
        if (ver < 0 || ver < c - 1 - s) {
          ver = c - 1;
          *V = ver;
        }
        atomicMin(vmin, ver);
      }
      slot = __shfl_sync(0xffffffffu, ver, 0) % nslots;
    }
    const float4* src = reinterpret_cast<const float4*>(ring) + (int64_t)slot * slot4 + (int64_t)r * K4;
    for (int32_t q = lane; q < K4; q += 32) o[q] = src[q];
  }
}

cudaError_t launch_get(const float* ring, int64_t n_rows, int32_t K, int32_t nslots, const int32_t* v, int32_t worker,
                       const int32_t* ids, int64_t n, float* out, uint32_t* status, int32_t* rowver, int32_t c,
                       int32_t s, int32_t* vmin, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((n * 32 + threads - 1) / threads, 4096);
  get_rows_kernel<<<blocks, threads, 0, st>>>(ring, n_rows, K, nslots, v, worker, ids, n, out, status, rowver, c, s,
                                              vmin);
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
