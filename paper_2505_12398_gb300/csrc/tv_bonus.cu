// tv_bonus.cu -- the bonus draw at an accepted original leaf, as a kernel of
// its own (the second phase of tv_verify_batch_host).
//
// When the accepted node X^tau of a tree is an original leaf of the drafted
// tree, Algorithm 3 draws the extra token Y from that leaf's target
// distribution M_b(.|X^tau) = softmax(l / T) (Definition 2; the last step of
// §3.1).  Of all leaf rows of a batch only those of accepted leaves are ever
// needed, at most one per tree, so the host entry point first verifies with
// the rows of nodes that have children only, then copies the accepted
// leaves' rows and draws their Y here.
//
// One CTA per pending tree: the row's maximum m, the sums of
// e(x) = 2^((l(x) - m) log2(e) / T) over 256-token tiles (float32, shared
// memory), a float64 prefix over the tiles to find the one where u W falls,
// then a float64 prefix over that tile's tokens: Y is the smallest token with
// u W < CDF(Y), in ascending token order.  No waits, no loops beyond the row.
#include <cuda_runtime.h>
#include <stdint.h>

#include "tv_device.cuh"
#include "tv_launch.h"

namespace tvk {
namespace {

constexpr int kBonusThreads = 256;
constexpr int kBonusTile = 256;   // one warp x 8 elements

__device__ __forceinline__ double warp_scan_incl(double v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double w = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += w;
  }
  return v;
}

// e(x) of 8 consecutive tokens from x0 (0 past the end of the row).
template <typename L, bool VEC>
__device__ __forceinline__ void tile_weights(const typename L::elem* row, int x0, int V, float m,
                                             float c_hi, float c_lo, float w8[8]) {
  if (x0 < V) {
    float v[8];
    load_logits<L, VEC>(row, x0, V, v);
#pragma unroll
    for (int e = 0; e < 8; ++e)
      w8[e] = (v[e] == TV_NEG_INF) ? 0.f : L::exp_rel(v[e], m, c_hi, c_lo);
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) w8[e] = 0.f;
  }
}

template <typename L, bool VEC>
__global__ void __launch_bounds__(kBonusThreads)
    tv_leaf_bonus_kernel(const void* logits_v, const float* uniforms, const int2* pending,
                         int B, int R, int V, float c_hi, float c_lo, int32_t* out_bonus) {
  extern __shared__ float tile_sum[];
  __shared__ float red[kBonusThreads / 32];
  __shared__ int found_tile;
  __shared__ double found_base, found_target;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int2 job = pending[blockIdx.x];
  const int b = job.x, node = job.y;
  if (b < 0 || b >= B || node < 0 || node >= R) return;
  const typename L::elem* row =
      reinterpret_cast<const typename L::elem*>(logits_v) + ((size_t)b * R + node) * (size_t)V;
  const int nt = (V + kBonusTile - 1) / kBonusTile;

  // ---- the row's maximum ----
  float lm = TV_NEG_INF;
  for (int x0 = tid * kChunk; x0 < V; x0 += kBonusThreads * kChunk) {
    float v[8];
    load_logits<L, VEC>(row, x0, V, v);
#pragma unroll
    for (int e = 0; e < 8; ++e) lm = fmaxf(lm, v[e]);
  }
  lm = warp_max(lm);
  if (lane == 0) red[wid] = lm;
  __syncthreads();
  float m = red[0];
  for (int w = 1; w < kBonusThreads / 32; ++w) m = fmaxf(m, red[w]);
  if (!(m > TV_NEG_INF)) {   // no finite logit: nothing to draw from
    if (tid == 0) out_bonus[b] = -1;
    return;
  }

  // ---- tile sums of e(x), one warp per tile ----
  for (int t = wid; t < nt; t += kBonusThreads / 32) {
    float w8[8];
    tile_weights<L, VEC>(row, t * kBonusTile + lane * kChunk, V, m, c_hi, c_lo, w8);
    const float ts = warp_sum(sum8(w8));
    if (lane == 0) tile_sum[t] = ts;
  }
  __syncthreads();

  // ---- warp 0: total, crossing tile (float64 prefix) ----
  if (wid == 0) {
    double tot = 0.0;
    for (int t = lane; t < nt; t += 32) tot += (double)tile_sum[t];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    const double target = (double)uniforms[(size_t)b * (R + 1) + R] * tot;
    int tile = -1, last = -1;
    double base = 0.0, tbase = 0.0, last_base = 0.0;
    for (int k0 = 0; k0 < nt && tile < 0; k0 += 32) {
      const double own = (k0 + lane < nt) ? (double)tile_sum[k0 + lane] : 0.0;
      const double incl = warp_scan_incl(own, lane);
      const unsigned hit = __ballot_sync(0xffffffffu, (k0 + lane < nt) && target < base + incl);
      const unsigned pos = __ballot_sync(0xffffffffu, own > 0.0);
      if (pos) {
        const int l = 31 - __clz(pos);
        last = k0 + l;
        last_base = base + __shfl_sync(0xffffffffu, incl - own, l);
      }
      if (hit) {
        const int l = __ffs(hit) - 1;
        tile = k0 + l;
        tbase = base + __shfl_sync(0xffffffffu, incl - own, l);
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (tile < 0) {   // rounding put u W at or past the total: last tile with weight
      tile = (last >= 0) ? last : 0;
      tbase = (last >= 0) ? last_base : 0.0;
    }
    if (lane == 0) {
      found_tile = tile;
      found_base = tbase;
      found_target = target;
    }
  }
  __syncthreads();

  // ---- warp 0: the token inside the crossing tile ----
  if (wid == 0) {
    const int tile = found_tile;
    const double target = found_target;
    const int x0 = tile * kBonusTile + lane * kChunk;
    float w8[8];
    tile_weights<L, VEC>(row, x0, V, m, c_hi, c_lo, w8);
    double pre[8];
    double run = 0.0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      run += (double)w8[e];
      pre[e] = run;
    }
    const double incl = warp_scan_incl(run, lane);
    const double lbase = found_base + (incl - run);
    int found = 8;
#pragma unroll
    for (int e = 7; e >= 0; --e)
      if (target < lbase + pre[e]) found = e;
    const unsigned hit = __ballot_sync(0xffffffffu, found < 8);
    int y;
    if (hit) {
      const int l = __ffs(hit) - 1;
      y = tile * kBonusTile + l * kChunk + __shfl_sync(0xffffffffu, found, l);
    } else {   // rounding: the last token of the tile with weight
      int lastx = -1;
#pragma unroll
      for (int e = 0; e < 8; ++e)
        if (w8[e] > 0.f) lastx = x0 + e;
      const unsigned any = __ballot_sync(0xffffffffu, lastx >= 0);
      y = any ? __shfl_sync(0xffffffffu, lastx, 31 - __clz(any)) : min(V - 1, x0);
    }
    if (lane == 0) out_bonus[b] = y;
  }
}

}  // namespace
}  // namespace tvk

size_t tv_leaf_bonus_smem_bytes(int V) {
  return (size_t)((V + tvk::kBonusTile - 1) / tvk::kBonusTile) * sizeof(float);
}

int tv_launch_leaf_bonus(const void* logits, int logit_is_bf16, const float* uniforms,
                         const int2* pending, int n_pending, int B, int R, int V, float c_hi,
                         float c_lo, int32_t* out_bonus, cudaStream_t stream) {
  if (n_pending <= 0) return 0;
  if (n_pending > B) return -1;
  const size_t smem = tv_leaf_bonus_smem_bytes(V);
  if (smem > 48 * 1024) return -3;
  const bool vec = (V % 8) == 0 && (reinterpret_cast<uintptr_t>(logits) & 15u) == 0;
  const dim3 grid(n_pending), block(tvk::kBonusThreads);
  if (logit_is_bf16) {
    if (vec)
      tvk::tv_leaf_bonus_kernel<tvk::Bf16Logits, true><<<grid, block, smem, stream>>>(
          logits, uniforms, pending, B, R, V, c_hi, c_lo, out_bonus);
    else
      tvk::tv_leaf_bonus_kernel<tvk::Bf16Logits, false><<<grid, block, smem, stream>>>(
          logits, uniforms, pending, B, R, V, c_hi, c_lo, out_bonus);
  } else {
    if (vec)
      tvk::tv_leaf_bonus_kernel<tvk::F32Logits, true><<<grid, block, smem, stream>>>(
          logits, uniforms, pending, B, R, V, c_hi, c_lo, out_bonus);
    else
      tvk::tv_leaf_bonus_kernel<tvk::F32Logits, false><<<grid, block, smem, stream>>>(
          logits, uniforms, pending, B, R, V, c_hi, c_lo, out_bonus);
  }
  if (cudaGetLastError() != cudaSuccess) return -5;
  return 0;
}
