// Small inline-PTX helpers: vector loads/stores with L2 eviction hints and
// vector fp32 reductions into global memory (sm_90 and later).
#pragma once

#include <stdint.h>

namespace esspt {

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// Streaming load: skip L1, mark the L2 lines for early eviction.
__device__ __forceinline__ float4 ld_stream(const float4* p, uint64_t pol) {
  float4 r;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
               : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
               : "l"(p), "l"(pol));
  return r;
}

// Load that keeps the line in L2 (hot, reused rows).
__device__ __forceinline__ float4 ld_keep(const float4* p, uint64_t pol) {
  float4 r;
  asm volatile("ld.global.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
               : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
               : "l"(p), "l"(pol));
  return r;
}

__device__ __forceinline__ void st_stream(float4* p, float4 v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1,%2,%3,%4}, %5;"
               :
               : "l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
               : "memory");
}

// Predicated forms: the access happens only when `pred` is true, without a
// branch around the asm (loads give zeros when it is false).
__device__ __forceinline__ float4 ld_stream_if(const float4* p, uint64_t pol, bool pred) {
  float4 r;
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %5, 0;\n mov.f32 %0, 0f00000000;\n mov.f32 %1, 0f00000000;\n"
      " mov.f32 %2, 0f00000000;\n mov.f32 %3, 0f00000000;\n"
      " @q ld.global.L1::no_allocate.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %6;\n}"
      : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
      : "l"(p), "r"((int)pred), "l"(pol));
  return r;
}

__device__ __forceinline__ void st_stream_if(float4* p, float4 v, uint64_t pol, bool pred) {
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %5, 0;\n"
      " @q st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1,%2,%3,%4}, %6;\n}"
      :
      : "l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"((int)pred), "l"(pol)
      : "memory");
}

// out[0..3] += v when `pred`, performed at L2 (vector reduction, sm_90 and
// later), predicated inside the asm so that no branch surrounds it.
__device__ __forceinline__ void red_add_v4_if(float4* p, float4 v, bool pred) {
  asm volatile("{\n .reg .pred q;\n setp.ne.b32 q, %5, 0;\n @q red.global.add.v4.f32 [%0], {%1,%2,%3,%4};\n}" ::"l"(p),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"((int)pred)
               : "memory");
}

// 16-byte asynchronous global -> shared copy (bypassing L1); when `pred` is
// false the 16 shared bytes are zero-filled and nothing is read.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool pred) {
  const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gmem), "r"(pred ? 16 : 0) : "memory");
}
// The same with an L2 eviction-priority policy for the source lines.
__device__ __forceinline__ void cp_async16_hint(void* smem, const void* gmem, bool pred, uint64_t pol) {
  const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2, %3;" ::"r"(s), "l"(gmem),
               "r"(pred ? 16 : 0), "l"(pol)
               : "memory");
}

// Streaming 32-bit loads (entries read once per clock): skip L1, evict-first in L2.
__device__ __forceinline__ int32_t ld_stream_i32(const int32_t* p, uint64_t pol) {
  int32_t r;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.b32 %0, [%1], %2;" : "=r"(r) : "l"(p), "l"(pol));
  return r;
}
__device__ __forceinline__ float ld_stream_f32(const float* p, uint64_t pol) {
  float r;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(r) : "l"(p), "l"(pol));
  return r;
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// out[0..3] += v, performed at L2 (no return value).
__device__ __forceinline__ void red_add_v4(float4* p, float4 v) { atomicAdd(p, v); }

// SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): output n of the sequence
// whose state starts at s0 is mix64(s0 + n * 0x9E3779B97F4A7C15).
__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Draw `index` of stream `stream` under `seed`: output index+1 of SplitMix64
// started at state mix64(seed) ^ mix64(stream).
__host__ __device__ __forceinline__ uint64_t ctr_u64(uint64_t seed, uint64_t stream, uint64_t index) {
  const uint64_t s0 = mix64(seed) ^ mix64(stream);
  return mix64(s0 + (index + 1ull) * 0x9E3779B97F4A7C15ull);
}

}  // namespace esspt
