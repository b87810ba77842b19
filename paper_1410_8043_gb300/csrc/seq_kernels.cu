// Sequential (read-my-writes) MF-SGD of one clock: each worker walks its own
// entries in order and reads L_i and R_j from its read version plus its own
// updates of this clock so far, as the per-entry SGD of Sec. 3.1 runs inside
// a worker (Sec. 5); the workers' summed changes then join the Clock() merge.
// Within a clock the entries of one worker form one dependent chain, so the
// parallelism is one warp per worker: this is a semantic variant, not the
// data-parallel hot path.
#include <algorithm>

#include "internal.h"

namespace esspt {

namespace {

constexpr int kSeqNV = 4;  // float4 slices per lane: rows of up to 512 values

__device__ __forceinline__ float seq_cap_scale(int32_t cap, int32_t n) {
  return (cap > 0 && n > cap) ? (float)cap / (float)n : 1.f;
}

// One warp per worker p.  The warp scans the users 32 at a time and walks
// those of worker p in ascending id, a user's entries in layout (input)
// order.  Lane l holds slices l, l+32, ... of the user's local row and of its
// summed update; the worker's own item updates of the clock live in
// mine[p][j] (zero on entry), so a later entry of item j sees them.
__global__ void __launch_bounds__(256) seq_users_kernel(SeqArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t p = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (p >= a.P) return;
  const int32_t K4 = a.K >> 2;
  const int64_t slot4 = a.n_rows * K4;
  const float4* ring4 = reinterpret_cast<const float4*>(a.ring);
  const float4* X = ring4 + (int64_t)(__ldg(a.v + p) % a.nslots) * slot4;
  const float4* base = ring4 + (int64_t)a.slot_base * slot4;
  float4* out = reinterpret_cast<float4*>(a.ring) + (int64_t)a.slot_out * slot4;
  float4* mine = reinterpret_cast<float4*>(a.mine) + p * a.n_items * K4;
  bool act[kSeqNV];
#pragma unroll
  for (int t = 0; t < kSeqNV; ++t) act[t] = lane + 32 * t < K4;
  float loss = 0.f;
  for (int64_t u0 = 0; u0 < a.n_users; u0 += 32) {
    const bool here = u0 + lane < a.n_users && __ldg(a.worker + u0 + lane) == (int32_t)p;
    unsigned todo = __ballot_sync(0xffffffffu, here);
    while (todo) {
      const int64_t u = u0 + __ffs(todo) - 1;
      todo &= todo - 1;
      const int32_t beg = __ldg(a.uoff + u), end = __ldg(a.uoff + u + 1);
      float4 L[kSeqNV], dL[kSeqNV];
#pragma unroll
      for (int t = 0; t < kSeqNV; ++t) {
        const int64_t q = lane + 32 * t;
        L[t] = act[t] ? X[u * K4 + q] : make_float4(0.f, 0.f, 0.f, 0.f);
        dL[t] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
      for (int32_t k = beg; k < end; ++k) {
        const int32_t j = __ldg(a.rec_j + k);
        const float d = __ldg(a.rec_D + k);
        const float4* Rx = X + ((int64_t)a.n_users + j) * K4;
        float4* Rm = mine + (int64_t)j * K4;
        float4 R[kSeqNV];
        float part = 0.f;
#pragma unroll
        for (int t = 0; t < kSeqNV; ++t) {
          const int64_t q = lane + 32 * t;
          if (act[t]) {
            const float4 x = Rx[q], m = Rm[q];
            R[t] = make_float4(x.x + m.x, x.y + m.y, x.z + m.z, x.w + m.w);
          } else {
            R[t] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
          part += L[t].x * R[t].x + L[t].y * R[t].y + L[t].z * R[t].z + L[t].w * R[t].w;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        const float e = d - part;
        if (lane == 0) loss += e * e;
#pragma unroll
        for (int t = 0; t < kSeqNV; ++t) {
          if (!act[t]) continue;
          const float4 l = L[t], r = R[t];
          const float4 gl = make_float4(a.eta * (e * r.x - a.lambda * l.x), a.eta * (e * r.y - a.lambda * l.y),
                                        a.eta * (e * r.z - a.lambda * l.z), a.eta * (e * r.w - a.lambda * l.w));
          const float4 gr = make_float4(a.eta * (e * l.x - a.lambda * r.x), a.eta * (e * l.y - a.lambda * r.y),
                                        a.eta * (e * l.z - a.lambda * r.z), a.eta * (e * l.w - a.lambda * r.w));
          L[t] = make_float4(l.x + gl.x, l.y + gl.y, l.z + gl.z, l.w + gl.w);
          dL[t] = make_float4(dL[t].x + gl.x, dL[t].y + gl.y, dL[t].z + gl.z, dL[t].w + gl.w);
          const int64_t q = lane + 32 * t;
          const float4 m = Rm[q];
          Rm[q] = make_float4(m.x + gr.x, m.y + gr.y, m.z + gr.z, m.w + gr.w);
        }
      }
      // L_i^c = L_i^base + scale * (the user's summed change).
      const float sc = seq_cap_scale(a.cap, end - beg);
#pragma unroll
      for (int t = 0; t < kSeqNV; ++t) {
        if (!act[t]) continue;
        const int64_t q = u * K4 + lane + 32 * t;
        const float4 b = base[q];
        out[q] = make_float4(b.x + sc * dL[t].x, b.y + sc * dL[t].y, b.z + sc * dL[t].z, b.w + sc * dL[t].w);
      }
    }
  }
  if (a.sq_loss != nullptr) {
    double x = (double)loss;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
    if (lane == 0 && x != 0.0) atomicAdd(a.sq_loss, x);
  }
}

// Clock() merge of the item rows: R_j^c = R_j^base + scale_j * sum over
// workers (in worker order) of their changes to R_j.  One thread per
// (item, float4 slice).
__global__ void __launch_bounds__(256) seq_item_merge_kernel(SeqArgs a) {
  const int32_t K4 = a.K >> 2;
  const int64_t n = (int64_t)a.n_items * K4;
  const int64_t slot4 = a.n_rows * K4;
  const float4* base = reinterpret_cast<const float4*>(a.ring) + (int64_t)a.slot_base * slot4 +
                       (int64_t)a.n_users * K4;
  float4* out = reinterpret_cast<float4*>(a.ring) + (int64_t)a.slot_out * slot4 + (int64_t)a.n_users * K4;
  const float4* mine = reinterpret_cast<const float4*>(a.mine);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < n; x += stride) {
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int32_t p = 0; p < a.P; ++p) {
      const float4 m = mine[(int64_t)p * n + x];
      s = make_float4(s.x + m.x, s.y + m.y, s.z + m.z, s.w + m.w);
    }
    const float sc = seq_cap_scale(a.cap, __ldg(a.item_cnt + x / K4));
    const float4 b = base[x];
    out[x] = make_float4(b.x + sc * s.x, b.y + sc * s.y, b.z + sc * s.z, b.w + sc * s.w);
  }
}

}  // namespace

cudaError_t launch_seq_clock(const SeqArgs& a, cudaStream_t st) {
  if ((a.K >> 2) > 32 * kSeqNV) return cudaErrorInvalidValue;
  const int blocks = (int)((a.P * 32 + 255) / 256);
  seq_users_kernel<<<blocks, 256, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t n = (int64_t)a.n_items * (a.K >> 2);
  if (n > 0) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int mb = (int)std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, (int64_t)sms * 8));
    seq_item_merge_kernel<<<mb, 256, 0, st>>>(a);
    e = cudaGetLastError();
  }
  return e;
}

}  // namespace esspt
