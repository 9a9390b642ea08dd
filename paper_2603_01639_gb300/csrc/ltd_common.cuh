// Device helpers shared by the LTD kernels: ordered 64-bit keys for
// (value desc, index asc) selection, warp-distributed top-k lists, warp and
// block reductions, the splitmix64-keyed uniforms, and vector loads.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>

#include "ltd.h"

namespace ltd {

constexpr int kWarp = 32;
constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

// ---------------------------------------------------------------- keys
// Monotone map of a float to uint32 (larger float -> larger code); -0 and +0
// map to the same code so that equal values tie exactly as in the oracle.
__device__ __forceinline__ uint32_t float_order_bits(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float order_bits_float(uint32_t o) {
  const uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(u);
}

// Larger key = better: value descending, then index ascending.  Every real
// key is > 0, so 0 serves as the empty slot.
__device__ __forceinline__ uint64_t make_key(float v, uint32_t idx) {
  return (static_cast<uint64_t>(float_order_bits(v)) << 32) |
         static_cast<uint64_t>(0xFFFFFFFFu - idx);
}
__device__ __forceinline__ uint32_t key_index(uint64_t k) {
  return 0xFFFFFFFFu - static_cast<uint32_t>(k);
}
__device__ __forceinline__ float key_value(uint64_t k) {
  return order_bits_float(static_cast<uint32_t>(k >> 32));
}

// Warp bitonic sort of one key per lane, descending (lane 0 = largest).
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, v, stride);
      const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0);
      v = keep_max ? (v > o ? v : o) : (v < o ? v : o);
    }
  }
  return v;
}

// The 32 largest of two descending lane-sorted lists, descending: the
// element-wise max of a and reversed b is bitonic and holds the 32 largest;
// five half-cleaner steps sort it.
__device__ __forceinline__ uint64_t warp_merge_desc(uint64_t a, uint64_t b) {
  const int lane = threadIdx.x & 31;
  const uint64_t br = __shfl_sync(0xFFFFFFFFu, b, 31 - lane);
  uint64_t v = a > br ? a : br;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, v, stride);
    v = ((lane & stride) == 0) ? (v > o ? v : o) : (v < o ? v : o);
  }
  return v;
}

// Warp-distributed top list: lane i holds the i-th largest key seen so far
// (descending; 0 = empty); the first k lanes are the top-k (k <= 32).  All
// lanes of the warp must call its members.
struct WarpTopK {
  uint64_t v;
  __device__ __forceinline__ void init() { v = 0ull; }
  // one unsorted key per lane; skipped when no key beats the k-th
  __device__ __forceinline__ void offer(uint64_t key, int k) {
    const uint64_t kth = __shfl_sync(0xFFFFFFFFu, v, k - 1);
    if (__any_sync(0xFFFFFFFFu, key > kth)) v = warp_merge_desc(v, warp_sort_desc(key));
  }
};

// -------------------------------------------------------------- reductions
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t y = __shfl_xor_sync(0xFFFFFFFFu, x, o);
    x = (y > x) ? y : x;
  }
  return x;
}

__device__ __forceinline__ float warp_max_f(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xFFFFFFFFu, x, o));
  return x;
}

__device__ __forceinline__ float warp_sum_f(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  return x;
}

// (max, sum of exp(x - max)) pairs: the merge of two partial softmax
// normalisers.  An empty side has max = -inf and sum = 0.
__device__ __forceinline__ void ms_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -CUDART_INF_F) return;
  if (m == -CUDART_INF_F) {
    m = m2;
    s = s2;
    return;
  }
  const float mm = fmaxf(m, m2);
  s = s * __expf(m - mm) + s2 * __expf(m2 - mm);
  m = mm;
}

__device__ __forceinline__ void warp_ms(float& m, float& s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o);
    const float s2 = __shfl_xor_sync(0xFFFFFFFFu, s, o);
    ms_merge(m, s, m2, s2);
  }
}

template <int NT>
__device__ __forceinline__ uint64_t block_max_u64(uint64_t x, uint64_t* red) {
  constexpr int NW = NT / kWarp;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  x = warp_max_u64(x);
  __syncthreads();
  if (lane == 0) red[warp] = x;
  __syncthreads();
  uint64_t t = 0;
  for (int w = 0; w < NW; ++w) t = red[w] > t ? red[w] : t;
  return t;
}

// -------------------------------------------------------- counter uniforms
// splitmix64 output finaliser (Steele, Lea & Flood 2014).
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// h_0 = seed; h_{j+1} = mix64(h_j + gamma (j+1) + w_j), for words w_0..w_{n-1}
// starting at position j0 (so a prefix hash can be extended later).
__device__ __forceinline__ uint64_t hash_step(uint64_t h, int j, uint64_t w) {
  return mix64(h + kGamma * static_cast<uint64_t>(j + 1) + w);
}

constexpr uint64_t kStreamRatio = 0;
constexpr uint64_t kStreamBonus = 1;

// Prefix (seed, b, cycle, stream, slot) -> 4 hash steps.
__device__ __forceinline__ uint64_t hash_prefix(uint64_t seed, uint64_t b, uint64_t cycle,
                                                uint64_t stream, uint64_t slot) {
  uint64_t h = seed;
  h = hash_step(h, 0, b);
  h = hash_step(h, 1, cycle);
  h = hash_step(h, 2, stream);
  h = hash_step(h, 3, slot);
  return h;
}

// Top 24 bits times 2^-24: exact in fp32.
__device__ __forceinline__ float uniform_ratio(uint64_t prefix, uint64_t i) {
  const uint64_t h = hash_step(prefix, 4, i);
  return static_cast<float>(h >> 40) * 5.9604644775390625e-8f;
}
// (2 (h >> 41) + 1) 2^-24, in (0, 1), exact in fp32.
__device__ __forceinline__ float uniform_gumbel(uint64_t prefix, uint64_t t) {
  const uint64_t h = hash_step(prefix, 4, t);
  return static_cast<float>(2ull * (h >> 41) + 1ull) * 5.9604644775390625e-8f;
}

// -------------------------------------------------------------- loads
template <typename T>
__device__ __forceinline__ float to_f(T x);
template <>
__device__ __forceinline__ float to_f<float>(float x) {
  return x;
}
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

// Element j of a 16-byte vector of T, as float (j a compile-time constant).
template <typename T>
__device__ __forceinline__ float elem(const uint4& r, int j);
template <>
__device__ __forceinline__ float elem<float>(const uint4& r, int j) {
  const uint32_t w = j == 0 ? r.x : (j == 1 ? r.y : (j == 2 ? r.z : r.w));
  return __uint_as_float(w);
}
template <>
__device__ __forceinline__ float elem<__nv_bfloat16>(const uint4& r, int j) {
  const int q = j >> 1;
  const uint32_t w = q == 0 ? r.x : (q == 1 ? r.y : (q == 2 ? r.z : r.w));
  return __uint_as_float((j & 1) ? (w & 0xFFFF0000u) : (w << 16));
}
// A streaming 16-byte load that the compiler may neither repeat nor move.
__device__ __forceinline__ uint4 ld_stream16_once(const void* p) {
  uint4 r;
  asm volatile("ld.global.cs.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void flag_error(uint32_t* err, uint32_t bits) {
  if (err) atomicOr(err, bits);
}

// Programmatic dependent launch.  Every kernel of this library is launched
// so that it may start while the previous kernel on the stream finishes;
// grid_wait() returns once that kernel has completed and its writes are
// visible (at once when there is none), and must come before any read of
// data another kernel wrote.  trigger_dependents() lets the next kernel on
// the stream start its own prologue.
__device__ __forceinline__ void grid_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void trigger_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

}  // namespace ltd
