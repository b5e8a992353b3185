// tv_device.cuh -- device helpers shared by the verification kernels.
//
// Numerics of the GPU path (float32 throughout):
//   M_b(x|X^i) = exp2((l_i(x) - m_i) * c) / s_i  with  c = log2(e) / T,
// where m_i is the row's largest logit and s_i = sum_x exp2((l_i(x) - m_i) c)
// (the softmax of l / T written in base 2, §3.1's target distributions).
// The difference l - m is exact for bf16 inputs, so the exponent carries only
// the rounding of one multiply; exp2 is the hardware ex2.approx instruction.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace tvk {

constexpr int kChunk = 8;            // elements per thread per step (16 B of bf16)
#define TV_NEG_INF (__int_as_float(0xff800000u))

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two bf16 values packed in one 32-bit word -> float (bf16 is the upper half
// of an IEEE float32, so widening is a shift or a mask).
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ uint4 ld_nc16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Logit element types.
struct Bf16Logits {
  using elem = uint16_t;
  static constexpr int kBytes = 2;
  __device__ static __forceinline__ float at(const elem* row, int x) {
    return __uint_as_float(static_cast<uint32_t>(row[x]) << 16);
  }
  // 8 consecutive elements starting at x0 (x0 % 8 == 0, row 16-byte aligned)
  __device__ static __forceinline__ void chunk_vec(const elem* row, int x0, float v[8]) {
    uint4 u = ld_nc16(row + x0);
    v[0] = bf16_lo(u.x); v[1] = bf16_hi(u.x);
    v[2] = bf16_lo(u.y); v[3] = bf16_hi(u.y);
    v[4] = bf16_lo(u.z); v[5] = bf16_hi(u.z);
    v[6] = bf16_lo(u.w); v[7] = bf16_hi(u.w);
  }
};

struct F32Logits {
  using elem = float;
  static constexpr int kBytes = 4;
  __device__ static __forceinline__ float at(const elem* row, int x) { return __ldg(row + x); }
  __device__ static __forceinline__ void chunk_vec(const elem* row, int x0, float v[8]) {
    uint4 a = ld_nc16(row + x0);
    uint4 b = ld_nc16(row + x0 + 4);
    v[0] = __uint_as_float(a.x); v[1] = __uint_as_float(a.y);
    v[2] = __uint_as_float(a.z); v[3] = __uint_as_float(a.w);
    v[4] = __uint_as_float(b.x); v[5] = __uint_as_float(b.y);
    v[6] = __uint_as_float(b.z); v[7] = __uint_as_float(b.w);
  }
};

// Chunk of 8 logits; elements past the end of the row read as -inf.
template <typename L, bool VEC>
__device__ __forceinline__ void load_logits(const typename L::elem* row, int x0, int V, float v[8]) {
  if (VEC) {
    L::chunk_vec(row, x0, v);
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = (x0 + k < V) ? L::at(row, x0 + k) : TV_NEG_INF;
  }
}

// Chunk of 8 draft probabilities; elements past the end read as 0.
template <bool VEC>
__device__ __forceinline__ void load_probs(const float* row, int x0, int V, float q[8]) {
  if (VEC) {
    uint4 a = ld_nc16(row + x0);
    uint4 b = ld_nc16(row + x0 + 4);
    q[0] = __uint_as_float(a.x); q[1] = __uint_as_float(a.y);
    q[2] = __uint_as_float(a.z); q[3] = __uint_as_float(a.w);
    q[4] = __uint_as_float(b.x); q[5] = __uint_as_float(b.y);
    q[6] = __uint_as_float(b.z); q[7] = __uint_as_float(b.w);
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) q[k] = (x0 + k < V) ? __ldg(row + x0 + k) : 0.f;
  }
}

// Pairwise sum of 8 values (three levels).
__device__ __forceinline__ float sum8(const float t[8]) {
  return ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
}

// Compensated (Kahan-Babuska / Neumaier) accumulation of chunk sums.
struct Comp {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float v) {
    float t = s + v;
    c += (fabsf(s) >= fabsf(v)) ? ((s - t) + v) : ((v - t) + s);
    s = t;
  }
  __device__ __forceinline__ float value() const { return s + c; }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Merge two (max, sum-of-exp2 relative to that max) pairs.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2, float c) {
  float M = fmaxf(m, m2);
  if (M == TV_NEG_INF) { m = M; s = 0.f; return; }
  float a = (m == TV_NEG_INF) ? 0.f : s * ex2((m - M) * c);
  float b = (m2 == TV_NEG_INF) ? 0.f : s2 * ex2((m2 - M) * c);
  m = M;
  s = a + b;
}

__device__ __forceinline__ void warp_lse(float& m, float& s, float c) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2, c);
  }
}

}  // namespace tvk
