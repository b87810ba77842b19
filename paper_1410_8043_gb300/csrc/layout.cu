// Setup (once per data set, not per clock): lay the observed entries out by
// minibatch and user so that a clock streams one contiguous, user-sorted
// segment (Sec. 3.1: D_obs partitioned over workers; Sec. 5: a fixed
// minibatch per Clock()).  The radix sort is stable, so entries of a user
// keep their input order and every run sees the same layout.
#include <algorithm>

#include <cub/device/device_radix_sort.cuh>
#include <cub/device/device_scan.cuh>

#include "internal.h"

namespace esspt {

namespace {

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__global__ void validate_kernel(const int32_t* __restrict__ i, const int32_t* __restrict__ j,
                                const uint8_t* __restrict__ mb, int64_t n_obs, const int32_t* __restrict__ worker,
                                int64_t n_users, int64_t n_items, int32_t F, int32_t P, uint32_t* status) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  bool bad = false;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n_obs; k += stride)
    bad |= i[k] < 0 || i[k] >= n_users || j[k] < 0 || j[k] >= n_items || mb[k] >= F;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n_users; u += stride)
    bad |= worker[u] < 0 || worker[u] >= P;
  if (bad) atomicOr(status, kErrInput);
}

__global__ void keys_kernel(const int32_t* __restrict__ i, const int32_t* __restrict__ j,
                            const uint8_t* __restrict__ mb, int64_t n_obs, int64_t n_users, int64_t n_items,
                            uint32_t* __restrict__ key, uint32_t* __restrict__ val, int32_t* __restrict__ cnt,
                            int32_t* __restrict__ item_cnt) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n_obs; k += stride) {
    const uint32_t x = (uint32_t)((int64_t)mb[k] * n_users + i[k]);
    key[k] = x;
    val[k] = (uint32_t)k;
    atomicAdd(cnt + x, 1);
    atomicAdd(item_cnt + (int64_t)mb[k] * n_items + j[k], 1);
  }
}

__global__ void gather_kernel(const uint32_t* __restrict__ perm, int64_t n_obs, const int32_t* __restrict__ i,
                              const int32_t* __restrict__ j, const float* __restrict__ D, int32_t* __restrict__ ru,
                              int32_t* __restrict__ rj, float* __restrict__ rD) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n_obs; k += stride) {
    const uint32_t s = perm[k];
    ru[k] = i[s];
    rj[k] = j[s];
    rD[k] = D[s];
  }
}

// uoff[b][u] = off[b*N+u] - off[b*N] for u in [0, N]; mb_base[b] = off[b*N].
__global__ void offsets_kernel(const int64_t* __restrict__ off, int64_t n_users, int32_t F, int32_t* __restrict__ uoff,
                               int64_t* __restrict__ mb_base, const int32_t* __restrict__ cnt,
                               int32_t* __restrict__ nchunks) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t total = (int64_t)F * (n_users + 1);
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total; x += stride) {
    const int64_t b = x / (n_users + 1), u = x % (n_users + 1);
    const int64_t base = off[b * n_users];
    uoff[x] = (int32_t)(off[b * n_users + u] - base);
    if (u == 0) mb_base[b] = base;
    if (u < n_users) {
      const int32_t n = cnt[b * n_users + u];
      nchunks[b * n_users + u] = n > kHeavy ? (n + kChunk - 1) / kChunk : 0;
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) mb_base[F] = off[(int64_t)F * n_users];
}

__global__ void chunks_kernel(const int64_t* __restrict__ choff, const int32_t* __restrict__ nchunks,
                              const int32_t* __restrict__ uoff, int64_t n_users, int32_t F,
                              int32_t* __restrict__ cu, int32_t* __restrict__ cb, int32_t* __restrict__ ce,
                              int64_t* __restrict__ chunk_base, int64_t max_chunks, uint32_t* status) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t total = (int64_t)F * n_users;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total; x += stride) {
    const int32_t nc = nchunks[x];
    if (nc == 0) continue;
    const int64_t b = x / n_users, u = x % n_users;
    const int32_t beg = uoff[b * (n_users + 1) + u], end = uoff[b * (n_users + 1) + u + 1];
    for (int32_t t = 0; t < nc; ++t) {
      const int64_t k = choff[x] + t;
      if (k >= max_chunks) {  // cannot happen: sum of ceil(n/kChunk) over n > kHeavy is < 2 n_obs / kChunk
        atomicOr(status, kErrInput);
        break;
      }
      cu[k] = (int32_t)u;
      cb[k] = beg + t * kChunk;
      ce[k] = min(end, beg + (t + 1) * kChunk);
    }
  }
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b <= F; b += stride)
    chunk_base[b] = choff[b * n_users];
}

int blocks_for(int64_t n) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return (int)std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, (int64_t)sms * 16));
}

struct ScratchPlan {
  size_t key_in, key_out, val_in, val_out, cnt, off, nchunks, choff, cub, total;
  size_t cub_bytes;
};

ScratchPlan plan(int64_t n_obs, int64_t n_users, int32_t F) {
  ScratchPlan p{};
  const int64_t keys = (int64_t)F * n_users;
  size_t sort_bytes = 0, scan_bytes = 0, scan2_bytes = 0;
  cub::DeviceRadixSort::SortPairs(nullptr, sort_bytes, (const uint32_t*)nullptr, (uint32_t*)nullptr,
                                  (const uint32_t*)nullptr, (uint32_t*)nullptr, (int)std::max<int64_t>(n_obs, 1), 0,
                                  32);
  cub::DeviceScan::ExclusiveSum(nullptr, scan_bytes, (const int32_t*)nullptr, (int64_t*)nullptr,
                                (int)(keys + 1));
  cub::DeviceScan::ExclusiveSum(nullptr, scan2_bytes, (const int32_t*)nullptr, (int64_t*)nullptr,
                                (int)(keys + 1));
  p.cub_bytes = std::max(sort_bytes, std::max(scan_bytes, scan2_bytes));
  size_t o = 0;
  p.key_in = o; o += align256(sizeof(uint32_t) * n_obs);
  p.key_out = o; o += align256(sizeof(uint32_t) * n_obs);
  p.val_in = o; o += align256(sizeof(uint32_t) * n_obs);
  p.val_out = o; o += align256(sizeof(uint32_t) * n_obs);
  p.cnt = o; o += align256(sizeof(int32_t) * (keys + 1));
  p.off = o; o += align256(sizeof(int64_t) * (keys + 1));
  p.nchunks = o; o += align256(sizeof(int32_t) * (keys + 1));
  p.choff = o; o += align256(sizeof(int64_t) * (keys + 1));
  p.cub = o; o += align256(p.cub_bytes);
  p.total = o;
  return p;
}

int bits_for(uint64_t max_key) {
  int b = 1;
  while (b < 32 && (max_key >> b) != 0) ++b;
  return b;
}

}  // namespace

size_t layout_scratch_bytes(int64_t n_obs, int64_t n_users, int32_t F) { return plan(n_obs, n_users, F).total; }

int64_t layout_max_chunks(int64_t n_obs, int32_t F) {
  // A heavy segment has n > kHeavy >= kChunk entries and ceil(n/kChunk) <= 2n/kChunk chunks.
  return 2 * n_obs / kChunk + F + 1;
}

cudaError_t build_layout(const LayoutBuild& b, cudaStream_t st) {
  const ScratchPlan p = plan(b.n_obs, b.n_users, b.F);
  if (b.scratch_bytes < p.total) return cudaErrorInvalidValue;
  char* s = static_cast<char*>(b.scratch);
  uint32_t* key_in = reinterpret_cast<uint32_t*>(s + p.key_in);
  uint32_t* key_out = reinterpret_cast<uint32_t*>(s + p.key_out);
  uint32_t* val_in = reinterpret_cast<uint32_t*>(s + p.val_in);
  uint32_t* val_out = reinterpret_cast<uint32_t*>(s + p.val_out);
  int32_t* cnt = reinterpret_cast<int32_t*>(s + p.cnt);
  int64_t* off = reinterpret_cast<int64_t*>(s + p.off);
  int32_t* nch = reinterpret_cast<int32_t*>(s + p.nchunks);
  int64_t* choff = reinterpret_cast<int64_t*>(s + p.choff);
  void* cub_tmp = s + p.cub;
  const int64_t keys = (int64_t)b.F * b.n_users;
  cudaError_t e;

  if ((e = cudaMemsetAsync(cnt, 0, sizeof(int32_t) * (keys + 1), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(nch, 0, sizeof(int32_t) * (keys + 1), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(b.item_cnt, 0, sizeof(int32_t) * b.F * b.n_items, st)) != cudaSuccess) return e;
  keys_kernel<<<blocks_for(b.n_obs), 256, 0, st>>>(b.i, b.j, b.mb, b.n_obs, b.n_users, b.n_items, key_in, val_in, cnt,
                                                  b.item_cnt);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (b.n_obs > 0) {
    size_t tb = p.cub_bytes;
    e = cub::DeviceRadixSort::SortPairs(cub_tmp, tb, key_in, key_out, val_in, val_out, (int)b.n_obs, 0,
                                        bits_for((uint64_t)keys), st);
    if (e != cudaSuccess) return e;
    gather_kernel<<<blocks_for(b.n_obs), 256, 0, st>>>(val_out, b.n_obs, b.i, b.j, b.D, b.rec_u, b.rec_j, b.rec_D);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  size_t tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, cnt, off, (int)(keys + 1), st)) != cudaSuccess) return e;
  offsets_kernel<<<blocks_for((int64_t)b.F * (b.n_users + 1)), 256, 0, st>>>(off, b.n_users, b.F, b.uoff, b.mb_base,
                                                                            cnt, nch);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, nch, choff, (int)(keys + 1), st)) != cudaSuccess) return e;
  chunks_kernel<<<blocks_for(keys + 1), 256, 0, st>>>(choff, nch, b.uoff, b.n_users, b.F, b.chunk_user, b.chunk_begin,
                                                      b.chunk_end, b.chunk_base, b.max_chunks, b.status);
  return cudaGetLastError();
}

cudaError_t launch_validate(const LayoutBuild& b, cudaStream_t st) {
  validate_kernel<<<blocks_for(std::max(b.n_obs, b.n_users)), 256, 0, st>>>(b.i, b.j, b.mb, b.n_obs, b.worker,
                                                                           b.n_users, b.n_items, b.F, b.P, b.status);
  return cudaGetLastError();
}

}  // namespace esspt
