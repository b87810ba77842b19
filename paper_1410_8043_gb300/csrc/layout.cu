// Setup (once per data set, not per clock): lay the observed entries out by
// minibatch and user so that a clock streams one contiguous, user-sorted
// segment (Sec. 3.1: D_obs partitioned over workers; Sec. 5: a fixed
// minibatch per Clock()).  The radix sort is stable, so entries of a user
// keep their input order and every run sees the same layout.  Also builds
// the chunk and heavy-user lists and the replica rows of popular items and
// heavy users.
#include <algorithm>
#include <vector>

#include <cub/device/device_radix_sort.cuh>
#include <cub/device/device_scan.cuh>

#include "internal.h"

namespace esspt {

namespace {

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__host__ __device__ inline int32_t next_pow2(int32_t x) {
  int32_t p = 1;
  while (p < x) p <<= 1;
  return p;
}

// Replicas of a heavy user with nch chunks: one per kUserRep chunks, rounded
// up to a power of two (never more than nch), at most kMaxRep.
__host__ __device__ inline int32_t user_reps(int32_t nch) {
  const int32_t r = next_pow2((nch + kUserRep - 1) / kUserRep);
  return r < kMaxRep ? r : kMaxRep;
}

// Replicas of an item whose largest minibatch count is mx, at most kMaxRep.
__host__ __device__ inline int32_t item_reps(int32_t mx) {
  const int32_t want = (mx + kItemRep - 1) / kItemRep;
  const int32_t r = next_pow2(want > 1 ? want : 1);
  return r < kMaxRep ? r : kMaxRep;
}

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

// uoff[b][u] = off[b*N+u] - off[b*N] for u in [0, N]; mb_base[b] = off[b*N];
// per (b, u): chunks, heavy flag and extra replica rows.
__global__ void offsets_kernel(const int64_t* __restrict__ off, int64_t n_users, int32_t F, int32_t* __restrict__ uoff,
                               int64_t* __restrict__ mb_base, const int32_t* __restrict__ cnt,
                               int32_t* __restrict__ nch, int32_t* __restrict__ hflag, int32_t* __restrict__ hextra,
                               bool light_items) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t total = (int64_t)F * (n_users + 1);
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total; x += stride) {
    const int64_t b = x / (n_users + 1), u = x % (n_users + 1);
    const int64_t base = off[b * n_users];
    uoff[x] = (int32_t)(off[b * n_users + u] - base);
    if (u == 0) mb_base[b] = base;
    if (u < n_users) {
      const int32_t n = cnt[b * n_users + u];
      const int32_t c = n > kHeavy ? (n + kChunk - 1) / kChunk : 0;
      nch[b * n_users + u] = c + (light_items && n > 0 && c == 0 ? 1 : 0);
      hflag[b * n_users + u] = c > 0 ? 1 : 0;
      hextra[b * n_users + u] = c > 0 ? user_reps(c) - 1 : 0;
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) mb_base[F] = off[(int64_t)F * n_users];
}

// Chunk descriptors (user, begin, end, replica row) and heavy-user
// descriptors (user, first extra replica row, replicas, entries).  Replica 0
// of heavy user u is row u of dL; replicas 1.. are rows n_users + hext[...].
__global__ void heavy_kernel(const int64_t* __restrict__ choff, const int32_t* __restrict__ nch,
                             const int64_t* __restrict__ hoff, const int64_t* __restrict__ hext,
                             const int32_t* __restrict__ uoff, int64_t n_users, int32_t F, int4* __restrict__ chunk,
                             int64_t* __restrict__ chunk_base, int64_t max_chunks, int4* __restrict__ heavy,
                             int64_t* __restrict__ heavy_base, int64_t max_heavy, int64_t max_user_reps,
                             uint32_t* status) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t total = (int64_t)F * n_users;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total; x += stride) {
    const int32_t nc = nch[x];
    if (nc == 0) continue;
    const int64_t b = x / n_users, u = x % n_users;
    const int32_t beg = uoff[b * (n_users + 1) + u], end = uoff[b * (n_users + 1) + u + 1];
    if (end - beg <= kHeavy) {  // a light user: one work item, written directly
      if (choff[x] >= max_chunks) {
        atomicOr(status, kErrInput);
        continue;
      }
      chunk[choff[x]] = make_int4((int32_t)u, beg, end, -1);
      continue;
    }
    const int32_t reps = user_reps(nc);
    const int64_t extra0 = n_users + hext[x];
    // The bounds below hold by construction; the checks keep every store in range.
    if (hoff[x] >= max_heavy || choff[x] + nc > max_chunks || hext[x] + reps - 1 > max_user_reps) {
      atomicOr(status, kErrInput);
      continue;
    }
    heavy[hoff[x]] = make_int4((int32_t)u, (int32_t)extra0, reps, end - beg);
    for (int32_t t = 0; t < nc; ++t) {
      const int32_t r = t & (reps - 1);
      const int32_t dst = r == 0 ? (int32_t)u : (int32_t)(extra0 + r - 1);
      chunk[choff[x] + t] = make_int4((int32_t)u, beg + t * kChunk, min(end, beg + (t + 1) * kChunk), dst);
    }
  }
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b <= F; b += stride) {
    chunk_base[b] = choff[b * n_users];
    heavy_base[b] = hoff[b * n_users];
  }
}

// Extra replica rows of every item (replicas - 1) from its largest minibatch
// count.  Replica 0 of item j is row j of dR; the extra ones follow all items.
__global__ void item_reps_kernel(const int32_t* __restrict__ item_cnt, int64_t n_items, int32_t F,
                                 int32_t* __restrict__ reps) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j <= n_items; j += stride) {
    if (j == n_items) {
      reps[j] = 0;
      continue;
    }
    int32_t mx = 0;
    for (int32_t b = 0; b < F; ++b) mx = max(mx, item_cnt[(int64_t)b * n_items + j]);
    reps[j] = item_reps(mx) - 1;
  }
}

// Replica row of every entry's item update: entry t (position within its
// minibatch) of item j adds into replica (t mod replicas of j): replica 0 is
// row j, replica r > 0 row n_items + item_rep[j] + r - 1.
// With hot_item (work-list path, kHot > 0) an entry of hot slot h of its
// minibatch gets -1 - h instead.
__global__ void dst_kernel(const uint32_t* __restrict__ key, const int64_t* __restrict__ mb_base,
                           const int32_t* __restrict__ rec_j, const int32_t* __restrict__ item_rep, int64_t n_obs,
                           int64_t n_users, int64_t n_items, const int32_t* __restrict__ hot_item,
                           int32_t* __restrict__ rec_dst) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n_obs; k += stride) {
    const int64_t b = (int64_t)key[k] / n_users;
    const int64_t t = k - mb_base[b];
    const int32_t j = rec_j[k];
    const int32_t e0 = item_rep[j], e1 = item_rep[j + 1];  // extra replicas of j: e1 - e0 (reps - 1)
    const int32_t r = (int32_t)(t & (int64_t)(e1 - e0));    // reps is a power of two
    int32_t d = r == 0 ? j : (int32_t)(n_items + e0 + r - 1);
    if (hot_item != nullptr)
      for (int h = 0; h < kHot; ++h)
        if (hot_item[b * kHot + h] == j) d = -1 - h;
    rec_dst[k] = d;
  }
}

// The kHot items with the most entries of each minibatch (at least 2), most
// popular first, ties by id; -1 for unused slots.  Host side, at setup.
cudaError_t build_hot(const LayoutBuild& b, cudaStream_t st) {
  if (kHot <= 0 || b.hot_item == nullptr) return cudaSuccess;
  const size_t FM = (size_t)b.F * (size_t)b.n_items;
  std::vector<int32_t> cnt(FM), hot((size_t)b.F * kHot, -1), idx((size_t)b.n_items);
  cudaError_t e = cudaMemcpyAsync(cnt.data(), b.item_cnt, sizeof(int32_t) * FM, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return e;
  for (int32_t mb = 0; mb < b.F; ++mb) {
    const int32_t* c = cnt.data() + (size_t)mb * b.n_items;
    for (int64_t j = 0; j < b.n_items; ++j) idx[j] = (int32_t)j;
    const int64_t h = std::min<int64_t>(kHot, b.n_items);
    std::partial_sort(idx.begin(), idx.begin() + h, idx.end(),
                      [c](int32_t x, int32_t y) { return c[x] != c[y] ? c[x] > c[y] : x < y; });
    for (int64_t r = 0; r < h && c[idx[r]] >= 2; ++r) hot[(size_t)mb * kHot + r] = idx[r];
  }
  e = cudaMemcpyAsync(b.hot_item, hot.data(), sizeof(int32_t) * hot.size(), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  return e;
}

// A staged minibatch against the loaded one: every user id, item id and
// user offset must be equal; any difference latches kErrInput.
__global__ void stage_check_kernel(const int32_t* __restrict__ su, const int32_t* __restrict__ sj,
                                   const int32_t* __restrict__ suoff, const int32_t* __restrict__ ru,
                                   const int32_t* __restrict__ rj, const int32_t* __restrict__ ruoff, int64_t n,
                                   int64_t n_off, uint32_t* status) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  bool bad = false;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n; k += stride)
    bad |= su[k] != ru[k] || sj[k] != rj[k];
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n_off; u += stride)
    bad |= suoff[u] != ruoff[u];
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(status, kErrInput);
}

int blocks_for(int64_t n) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return (int)std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, (int64_t)sms * 16));
}

struct ScratchPlan {
  size_t key_in, key_out, val_in, val_out, cnt, off, nch, choff, hflag, hoff, hextra, hext, ireps, cub, total;
  size_t cub_bytes;
};

ScratchPlan plan(int64_t n_obs, int64_t n_users, int64_t n_items, int32_t F) {
  ScratchPlan p{};
  const int64_t keys = (int64_t)F * n_users;
  size_t sort_bytes = 0, scan_bytes = 0, scan2_bytes = 0;
  cub::DeviceRadixSort::SortPairs(nullptr, sort_bytes, (const uint32_t*)nullptr, (uint32_t*)nullptr,
                                  (const uint32_t*)nullptr, (uint32_t*)nullptr, (int)std::max<int64_t>(n_obs, 1), 0,
                                  32);
  cub::DeviceScan::ExclusiveSum(nullptr, scan_bytes, (const int32_t*)nullptr, (int64_t*)nullptr, (int)(keys + 1));
  cub::DeviceScan::ExclusiveSum(nullptr, scan2_bytes, (const int32_t*)nullptr, (int32_t*)nullptr,
                                (int)(n_items + 1));
  p.cub_bytes = std::max(sort_bytes, std::max(scan_bytes, scan2_bytes));
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    const size_t at = o;
    o += align256(bytes);
    return at;
  };
  p.key_in = take(sizeof(uint32_t) * n_obs);
  p.key_out = take(sizeof(uint32_t) * n_obs);
  p.val_in = take(sizeof(uint32_t) * n_obs);
  p.val_out = take(sizeof(uint32_t) * n_obs);
  p.cnt = take(sizeof(int32_t) * (keys + 1));
  p.off = take(sizeof(int64_t) * (keys + 1));
  p.nch = take(sizeof(int32_t) * (keys + 1));
  p.choff = take(sizeof(int64_t) * (keys + 1));
  p.hflag = take(sizeof(int32_t) * (keys + 1));
  p.hoff = take(sizeof(int64_t) * (keys + 1));
  p.hextra = take(sizeof(int32_t) * (keys + 1));
  p.hext = take(sizeof(int64_t) * (keys + 1));
  p.ireps = take(sizeof(int32_t) * (n_items + 1));
  p.cub = take(p.cub_bytes);
  p.total = o;
  return p;
}

int bits_for(uint64_t max_key) {
  int b = 1;
  while (b < 32 && (max_key >> b) != 0) ++b;
  return b;
}

}  // namespace

size_t layout_scratch_bytes(int64_t n_obs, int64_t n_users, int64_t n_items, int32_t F) {
  return plan(n_obs, n_users, n_items, F).total;
}

// A heavy segment has n > kHeavy >= kChunk entries and ceil(n/kChunk) < 2n/kChunk chunks.
// On the work-list path every user with entries in a minibatch adds one more item.
int64_t layout_max_chunks(int64_t n_obs, int32_t F, int64_t n_users, bool light_items) {
  return 2 * n_obs / kChunk + F + 1 + (light_items ? std::min(n_obs, (int64_t)F * n_users) : 0);
}

int64_t layout_max_heavy(int64_t n_obs, int32_t F) { return n_obs / (kHeavy + 1) + F + 1; }

// Replica rows: one per item plus the extra ones, sum (reps - 1) with reps - 1 < 3 mx / (2 kItemRep).
int64_t layout_max_item_reps(int64_t n_obs, int64_t n_items) { return n_items + 3 * n_obs / (2 * kItemRep) + 2; }

// Extra replica rows of heavy users: reps - 1 < 3 nch / (2 kUserRep), sum nch < 2 n_obs / kChunk.
int64_t layout_max_user_reps(int64_t n_obs) { return 3 * n_obs / (kChunk * kUserRep) + 2; }

cudaError_t build_layout(const LayoutBuild& b, cudaStream_t st) {
  const ScratchPlan p = plan(b.n_obs, b.n_users, b.n_items, b.F);
  if (b.scratch_bytes < p.total) return cudaErrorInvalidValue;
  char* s = static_cast<char*>(b.scratch);
  uint32_t* key_in = reinterpret_cast<uint32_t*>(s + p.key_in);
  uint32_t* key_out = reinterpret_cast<uint32_t*>(s + p.key_out);
  uint32_t* val_in = reinterpret_cast<uint32_t*>(s + p.val_in);
  uint32_t* val_out = reinterpret_cast<uint32_t*>(s + p.val_out);
  int32_t* cnt = reinterpret_cast<int32_t*>(s + p.cnt);
  int64_t* off = reinterpret_cast<int64_t*>(s + p.off);
  int32_t* nch = reinterpret_cast<int32_t*>(s + p.nch);
  int64_t* choff = reinterpret_cast<int64_t*>(s + p.choff);
  int32_t* hflag = reinterpret_cast<int32_t*>(s + p.hflag);
  int64_t* hoff = reinterpret_cast<int64_t*>(s + p.hoff);
  int32_t* hextra = reinterpret_cast<int32_t*>(s + p.hextra);
  int64_t* hext = reinterpret_cast<int64_t*>(s + p.hext);
  int32_t* ireps = reinterpret_cast<int32_t*>(s + p.ireps);
  void* cub_tmp = s + p.cub;
  const int64_t keys = (int64_t)b.F * b.n_users;
  cudaError_t e;

  for (void* z : {(void*)cnt, (void*)nch, (void*)hflag, (void*)hextra})
    if ((e = cudaMemsetAsync(z, 0, sizeof(int32_t) * (keys + 1), st)) != cudaSuccess) return e;
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
                                                                            cnt, nch, hflag, hextra,
                                                                            b.light_items);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, nch, choff, (int)(keys + 1), st)) != cudaSuccess) return e;
  tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, hflag, hoff, (int)(keys + 1), st)) != cudaSuccess) return e;
  tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, hextra, hext, (int)(keys + 1), st)) != cudaSuccess) return e;
  heavy_kernel<<<blocks_for(keys + 1), 256, 0, st>>>(choff, nch, hoff, hext, b.uoff, b.n_users, b.F, b.chunk,
                                                     b.chunk_base, b.max_chunks, b.heavy, b.heavy_base, b.max_heavy,
                                                     layout_max_user_reps(b.n_obs), b.status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  item_reps_kernel<<<blocks_for(b.n_items + 1), 256, 0, st>>>(b.item_cnt, b.n_items, b.F, ireps);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  tb = p.cub_bytes;
  if ((e = cub::DeviceScan::ExclusiveSum(cub_tmp, tb, ireps, b.item_rep, (int)(b.n_items + 1), st)) != cudaSuccess)
    return e;
  if (b.n_obs == 0) return cudaSuccess;
  if ((e = build_hot(b, st)) != cudaSuccess) return e;
  dst_kernel<<<blocks_for(b.n_obs), 256, 0, st>>>(key_out, b.mb_base, b.rec_j, b.item_rep, b.n_obs, b.n_users,
                                                  b.n_items, kHot > 0 ? b.hot_item : nullptr, b.rec_dst);
  return cudaGetLastError();
}

cudaError_t launch_stage_check(const int32_t* su, const int32_t* sj, const int32_t* suoff, const int32_t* ru,
                               const int32_t* rj, const int32_t* ruoff, int64_t n, int64_t n_off, uint32_t* status,
                               cudaStream_t st) {
  stage_check_kernel<<<blocks_for(std::max(n, n_off)), 256, 0, st>>>(su, sj, suoff, ru, rj, ruoff, n, n_off, status);
  return cudaGetLastError();
}

cudaError_t launch_validate(const LayoutBuild& b, cudaStream_t st) {
  validate_kernel<<<blocks_for(std::max(b.n_obs, b.n_users)), 256, 0, st>>>(b.i, b.j, b.mb, b.n_obs, b.worker,
                                                                           b.n_users, b.n_items, b.F, b.P, b.status);
  return cudaGetLastError();
}

}  // namespace esspt
