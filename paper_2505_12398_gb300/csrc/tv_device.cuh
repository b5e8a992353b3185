// tv_device.cuh -- device helpers shared by the verification kernels.
//
// Numerics of the GPU path:
//   M_b(x|X^i) = e_i(x) / s_i,  e_i(x) = 2^((l_i(x) - m_i) c),  c = log2(e) / T,
// where m_i is the row's largest logit and s_i = sum_x e_i(x) (the softmax of
// l / T written in base 2; the target distributions of §3.1).  Vocabulary-wide
// work is float32; the serial control of the traversal is float64.
//
// e(x) is computed so that its relative error stays near one float32 ulp:
// the exponent E = (l - m) c is formed as an unevaluated sum E_hi + E_lo
// (c split into c_hi + c_lo, the product error recovered with an FMA), split
// into an integer n and a fraction f in [-1/2, 1/2] with f carrying E_lo,
// and 2^f is taken from the ex2.approx instruction on that small argument;
// 2^n is applied by adding n to the exponent field.  Rounding the exponent of
// a large |E| to float32 first would leave a relative error of up to
// |E| 2^-24 ln 2 in every e(x), with a systematic sign; the rejection sum
// S = sum_x [p M_b(x) - M_s(x)]_+ amplifies such errors when it cancels.
#pragma once

#include <cuda_bf16.h>
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

// 2^E for E = d c with c = c_hi + c_lo and d = d_hi + d_lo (see above).
__device__ __forceinline__ float exp2_split(float d, float d_lo, float c_hi, float c_lo) {
  d = fmaxf(d, -1.0e4f);                      // -inf / NaN logits -> weight ~0
  const float e_hi = d * c_hi;
  float e_lo = fmaf(d, c_hi, -e_hi);          // exact error of the product
  e_lo = fmaf(d, c_lo, e_lo);
  e_lo = fmaf(d_lo, c_hi, e_lo);
  const float t = e_hi + 12582912.f;          // 1.5 * 2^23: round to integer
  const float nf = t - 12582912.f;
  int ni = __float_as_int(t) - 0x4B400000;
  const float f = (e_hi - nf) + e_lo;         // e_hi - nf is exact
  const float r = ex2(f);
  // below the normal range the weight is taken as exactly 0 (this also makes
  // padding elements, read as -inf, contribute nothing)
  return (ni < -125) ? 0.f : __int_as_float(__float_as_int(r) + (ni << 23));
}

// 2^E for E = d c, by a first-order correction of ex2.approx(E_hi) with the
// exact product error E_lo: 2^(E_hi + E_lo) = 2^E_hi (1 + E_lo ln 2 + O(E_lo^2)),
// |E_lo| <= 2^-24 |E|.  Measured on GB300 over bf16-exact d in [-60, 0]: max
// relative error 1.7e-7, mean -5.0e-8 (ex2.approx's own bias on full-range
// arguments), i.e. five fewer FP32 operations than exp2_split for a slightly
// larger, uniform bias.  Used where a uniform relative bias cancels
// (numerator and normaliser of the same distribution) or only decides
// near-ties (the bonus draw).
__device__ __forceinline__ float exp2_corrected(float d, float c_hi, float c_lo) {
  d = fmaxf(d, -1.0e4f);
  const float e_hi = d * c_hi;
  float e_lo = fmaf(d, c_hi, -e_hi);
  e_lo = fmaf(d, c_lo, e_lo);
  const float r = ex2(e_hi);
  return fmaf(r, e_lo * 0.6931471805599453f, r);
}

// ---- packed-pair (float2) forms for the bf16 hot loops (sm_100+ f32x2) ----

// Eight bf16 logits from one 16-byte word, clamped below at -9984 (so -inf and
// NaN become a finite number whose weight is 0 or below 2^-125) and widened
// to four (even, odd) float pairs.
__device__ __forceinline__ void bf16x8_pairs(uint4 w, float2 out[4]) {
  const uint32_t lo_clamp = 0xC61CC61Cu;   // two bf16 -9984
  uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&ws[k]);
    h = __hmax2(h, *reinterpret_cast<const __nv_bfloat162*>(&lo_clamp));
    const uint32_t c = *reinterpret_cast<uint32_t*>(&h);
    out[k] = make_float2(__uint_as_float(c << 16), __uint_as_float(c & 0xffff0000u));
  }
}

// exp2_corrected on a pair (d already clamped below).
__device__ __forceinline__ float2 exp2_corrected_x2(float2 d, float2 c_hi, float2 c_lo) {
  const float2 e_hi = __fmul2_rn(d, c_hi);
  float2 e_lo = __ffma2_rn(d, c_hi, make_float2(-e_hi.x, -e_hi.y));
  e_lo = __ffma2_rn(d, c_lo, e_lo);
  const float2 r = make_float2(ex2(e_hi.x), ex2(e_hi.y));
  const float2 t = __fmul2_rn(e_lo, make_float2(0.6931471805599453f, 0.6931471805599453f));
  return __ffma2_rn(r, t, r);
}

// exp2_split on a pair (d already clamped below).  Results below 2^-125 are
// returned as a value under 2^-124 instead of the exact tiny number.
__device__ __forceinline__ float2 exp2_split_x2(float2 d, float2 c_hi, float2 c_lo) {
  const float2 e_hi = __fmul2_rn(d, c_hi);
  float2 e_lo = __ffma2_rn(d, c_hi, make_float2(-e_hi.x, -e_hi.y));
  e_lo = __ffma2_rn(d, c_lo, e_lo);
  const float2 t = __fadd2_rn(e_hi, make_float2(12582912.f, 12582912.f));
  const float2 nf = __fadd2_rn(t, make_float2(-12582912.f, -12582912.f));
  const float2 f = __fadd2_rn(__fadd2_rn(e_hi, make_float2(-nf.x, -nf.y)), e_lo);
  const int tb0 = max(__float_as_int(t.x), 0x4B400000 - 125);
  const int tb1 = max(__float_as_int(t.y), 0x4B400000 - 125);
  const float r0 = ex2(f.x), r1 = ex2(f.y);
  // bits(r) + n * 2^23, n = bits(t) - bits(1.5 * 2^23), in modular arithmetic
  const int k = (int)(0u - (0x4B400000u << 23));
  return make_float2(__int_as_float(__float_as_int(r0) + (tb0 << 23) + k),
                     __int_as_float(__float_as_int(r1) + (tb1 << 23) + k));
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
  // 2^((v - m) c): v - m is exact for two bf16 values
  __device__ static __forceinline__ float exp_rel(float v, float m, float c_hi, float c_lo) {
    return exp2_split(v - m, 0.f, c_hi, c_lo);
  }
  // cheaper form for the per-element work of rejection passes and bonus draws
  __device__ static __forceinline__ float exp_pass(float v, float m, float c_hi, float c_lo) {
    return exp2_corrected(v - m, c_hi, c_lo);
  }
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
  // 2^((v - m) c) with the rounding error of v - m carried along (two-sum)
  __device__ static __forceinline__ float exp_rel(float v, float m, float c_hi, float c_lo) {
    v = fmaxf(v, m - 1.0e4f);                 // -inf / NaN: finite, weight ~0
    const float d = v - m;
    const float bb = d - v;
    const float d_lo = (v - (d - bb)) + (-m - bb);
    return exp2_split(d, d_lo, c_hi, c_lo);
  }
  __device__ static __forceinline__ float exp_pass(float v, float m, float c_hi, float c_lo) {
    return exp_rel(v, m, c_hi, c_lo);
  }
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

// The smallest |eta - p| over the tree's tests: every node with a positive
// recorded rate (dbgp, the rate at its test; removals at rate 0 record 0 and
// untested nodes NaN) was tested with its own uniform u[i].  +inf without a
// test.  One thread; only for the debug output.
__device__ inline float test_margin_serial(const float* dbgp, const float* u, int R) {
  float m = __int_as_float(0x7f800000);
  for (int i = 1; i < R; ++i) {
    const float p = dbgp[i];
    if (p > 0.f) m = fminf(m, (float)fabs((double)u[i] - (double)p));
  }
  return m;
}

}  // namespace tvk
