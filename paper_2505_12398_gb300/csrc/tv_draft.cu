// tv_draft.cu -- drafting a token tree's children without replacement
// (Definition 1) from the draft rows (sm_103a).
//
// Every child c of node i takes the pre-drawn uniform u[c] and is drawn by
// inverse CDF, in ascending token order, from M_s(.|X^i) with the tokens of
// i's earlier children removed: the smallest y with u[c] W < CDF'(y), where
// CDF' and W = CDF'(V - 1) are the cumulative sums of the row with those
// tokens zeroed.  Siblings are drawn in child-index order, the order in which
// the verification tests them.
//
// One CTA per (tree, row); rows without children return at once.  The CTA
// streams its row once: each warp reduces 256-token tiles (8 tokens a lane,
// four tiles in flight) to float32 tile sums, and one warp turns the tile
// sums into a float64 inclusive prefix.  Each child then
//   * finds the first tile whose prefix, less the masses of the earlier
//     siblings' tokens up to that tile, exceeds u W (all threads, a few tiles
//     each), and
//   * scans that tile in float64 (one warp: lane sums, a shuffle scan, then
//     the lane that crosses u W walks its 8 tokens); the tile is in L1/L2.
// The row is read from HBM once; a child costs one tile re-read.
//
// The cumulative sums are float64 over float32 tile sums, so a draw whose
// u W lies within about 1e-6 W of a step of the exact CDF may land on the
// neighbouring token.  If rounding leaves u W past the scanned tile (or past
// the whole row), the last token of positive mass there is taken.  No mass
// left for a child (more children than tokens of positive draft probability,
// or a row that does not sum to a positive finite value) gives -1 for it and
// its later siblings and raises TV_STATUS_DRAFT_EXHAUSTED.
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tv.h"
#include "tv_launch.h"

namespace tvk {
namespace draft {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kTile = 256;   // tokens per tile: 32 lanes x 8

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ double warp_exclusive_scan(double v, int lane) {
  double x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  return x - v;
}

// The 8 draft probabilities of tokens x0 .. x0+7 (0 past the end).
template <bool kVec>
__device__ __forceinline__ void load8(const float* __restrict__ q, int x0, int V, float* v) {
  if (kVec && x0 + 8 <= V) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(q + x0));
    const float4 b = __ldg(reinterpret_cast<const float4*>(q + x0 + 4));
    v[0] = a.x, v[1] = a.y, v[2] = a.z, v[3] = a.w;
    v[4] = b.x, v[5] = b.y, v[6] = b.z, v[7] = b.w;
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = x0 + k < V ? __ldg(q + x0 + k) : 0.f;
  }
}

// Tree blockIdx.x, row blockIdx.y.  Dynamic shared memory (draft_smem_bytes):
// pre[n_tiles] f64, rem_q[R] f64, tsum[n_tiles] f32, par[R], kids[R],
// rem_tok[R] int32.
template <bool kVec>
__global__ void __launch_bounds__(kThreads)
    tv_draft_kernel(const int32_t* __restrict__ parents, const float* __restrict__ drafts,
                    const float* __restrict__ uniforms, int32_t* __restrict__ tokens, int N,
                    int V, uint32_t* __restrict__ status) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int n_kids, found;
  const int R = N + 1, b = blockIdx.x, i = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_tiles = (V + kTile - 1) / kTile;
  double* pre = reinterpret_cast<double*>(smem);
  double* rem_q = pre + n_tiles;
  float* tsum = reinterpret_cast<float*>(rem_q + R);
  int* par = reinterpret_cast<int*>(tsum + n_tiles);
  int* kids = par + R;
  int* rem_tok = kids + R;
  const int32_t* pb = parents + (size_t)b * R;
  int32_t* tb = tokens + (size_t)b * R;

  // ---- the tree's parents: valid (parents[0] = -1, parents[c] in [0, c))?
  int badl = 0;
  for (int c = tid; c < R; c += kThreads) {
    const int p = pb[c];
    par[c] = p;
    if (c == 0 ? p != -1 : (p < 0 || p >= c)) badl = 1;
  }
  if (__syncthreads_or(badl)) {
    if (i == 0) {   // one CTA of the tree reports it
      for (int c = tid; c < R; c += kThreads) tb[c] = c == 0 ? 0 : -1;
      if (tid == 0) atomicOr(status, (uint32_t)TV_STATUS_BAD_TREE);
    }
    return;
  }
  if (i == 0 && tid == 0) tb[0] = 0;

  // ---- the children of row i, in index order (warp 0, 32 candidates a step)
  if (warp == 0) {
    int n = 0;
    for (int c0 = i + 1; c0 < R; c0 += 32) {
      const int c = c0 + lane;
      const bool is_kid = c < R && par[c] == i;
      const unsigned m = __ballot_sync(0xffffffffu, is_kid);
      if (is_kid) kids[n + __popc(m & ((1u << lane) - 1u))] = c;
      n += __popc(m);
    }
    if (lane == 0) n_kids = n;
  }
  __syncthreads();
  const int nk = n_kids;
  if (nk == 0) return;

  // ---- stream the row once: float32 sums of 256-token tiles
  const float* q = drafts + ((size_t)b * R + i) * (size_t)V;
  // four tiles a warp per step with 16-byte loads (loads past the end read as
  // zeros), so that enough bytes are in flight to stream at the copy bandwidth
  constexpr int kU = kVec ? 4 : 1;
  for (int t = warp; t < n_tiles; t += kU * kWarps) {
    float v[kU][8];
#pragma unroll
    for (int k = 0; k < kU; ++k) load8<kVec>(q, (t + k * kWarps) * kTile + lane * 8, V, v[k]);
#pragma unroll
    for (int k = 0; k < kU; ++k) {
      const float s = ((v[k][0] + v[k][1]) + (v[k][2] + v[k][3])) +
                      ((v[k][4] + v[k][5]) + (v[k][6] + v[k][7]));
      const float ts = warp_sum_f(s);
      if (lane == 0 && t + k * kWarps < n_tiles) tsum[t + k * kWarps] = ts;
    }
  }
  __syncthreads();
  // float64 inclusive prefix of the tile sums (warp 0: a run of tiles a lane)
  if (warp == 0) {
    const int per = (n_tiles + 31) / 32;
    const int t0 = min(n_tiles, lane * per), t1 = min(n_tiles, t0 + per);
    double acc = 0.0;
    for (int t = t0; t < t1; ++t) acc += (double)tsum[t];
    double run = warp_exclusive_scan(acc, lane);
    for (int t = t0; t < t1; ++t) {
      run += (double)tsum[t];
      pre[t] = run;
    }
  }
  __syncthreads();
  const double total = pre[n_tiles - 1];

  // ---- the children, in order
  for (int j = 0; j < nk; ++j) {
    const int c = kids[j];
    double rsum = 0.0;
    for (int r = 0; r < j; ++r) rsum += rem_q[r];
    const double W = total - rsum;
    if (!(W > 0.0) || !isfinite(W)) {   // the same decision in every thread
      for (int r = j + tid; r < nk; r += kThreads) tb[kids[r]] = -1;
      if (tid == 0) atomicOr(status, (uint32_t)TV_STATUS_DRAFT_EXHAUSTED);
      return;
    }
    const double target = (double)__ldg(uniforms + (size_t)b * R + c) * W;
    // the first tile whose prefix, less the earlier siblings' masses up to it,
    // exceeds u W (n_tiles: none, u W is at or past the end by rounding)
    if (tid == 0) found = n_tiles;
    __syncthreads();
    for (int t = tid; t < n_tiles; t += kThreads) {
      double adj = pre[t];
      for (int r = 0; r < j; ++r)
        if (rem_tok[r] / kTile <= t) adj -= rem_q[r];
      if (target < adj) {
        atomicMin(&found, t);
        break;   // this thread's tiles increase
      }
    }
    __syncthreads();
    const int ts = found;
    if (warp == 0) {
      int y = -1;
      bool take_last = ts == n_tiles;
      if (!take_last) {
        double base = ts > 0 ? pre[ts - 1] : 0.0;
        for (int r = 0; r < j; ++r)
          if (rem_tok[r] / kTile < ts) base -= rem_q[r];
        const int x0 = ts * kTile + lane * 8;
        float v[8];
        load8<kVec>(q, x0, V, v);
        double d[8], ls = 0.0;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          bool rm = false;
          for (int r = 0; r < j; ++r) rm |= rem_tok[r] == x0 + k;
          d[k] = rm ? 0.0 : (double)v[k];
          ls += d[k];
        }
        const double ex = warp_exclusive_scan(ls, lane);
        const unsigned m = __ballot_sync(0xffffffffu, target < base + ex + ls);
        if (m) {
          const int first = __ffs(m) - 1;
          if (lane == first) {
            double run = base + ex;
            int last = -1;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              if (d[k] > 0.0) last = x0 + k;
              run += d[k];
              if (y < 0 && target < run) y = x0 + k;
            }
            if (y < 0) y = last;   // the lane's sum crossed u W, its running sum did not
          }
          y = __shfl_sync(0xffffffffu, y, first);
        } else {
          take_last = true;   // rounding left u W past this tile
        }
      }
      if (take_last) {
        // the last token of positive mass at or before the tile
        for (int t = ts == n_tiles ? n_tiles - 1 : ts; t >= 0 && y < 0; --t) {
          const int x0 = t * kTile + lane * 8;
          float v[8];
          load8<kVec>(q, x0, V, v);
          int last = -1;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            bool rm = false;
            for (int r = 0; r < j; ++r) rm |= rem_tok[r] == x0 + k;
            if (!rm && v[k] > 0.f) last = x0 + k;
          }
          const unsigned m = __ballot_sync(0xffffffffu, last >= 0);
          if (m) y = __shfl_sync(0xffffffffu, last, 31 - __clz(m));
        }
      }
      if (lane == 0) {
        tb[c] = y;
        rem_tok[j] = y;
        rem_q[j] = y >= 0 ? (double)__ldg(q + y) : 0.0;
        if (y < 0) atomicOr(status, (uint32_t)TV_STATUS_DRAFT_EXHAUSTED);
      }
    }
    __syncthreads();
  }
}

}  // namespace draft
}  // namespace tvk

size_t tv_draft_smem_bytes(int N, int V) {
  const size_t R = (size_t)N + 1, tiles = ((size_t)V + tvk::draft::kTile - 1) / tvk::draft::kTile;
  return tiles * 8 + R * 8 + tiles * 4 + R * 12;
}

int tv_launch_draft(const int32_t* parents, const float* drafts, const float* uniforms,
                    int32_t* tokens, int B, int N, int V, uint32_t* status, cudaStream_t stream) {
  using namespace tvk::draft;
  if (B <= 0) return 0;
  const size_t smem = tv_draft_smem_bytes(N, V);
  const dim3 grid((unsigned)B, (unsigned)(N + 1));
  const bool vec = (V % 4) == 0 && (reinterpret_cast<uintptr_t>(drafts) & 15u) == 0;
  if (vec)
    tv_draft_kernel<true><<<grid, kThreads, smem, stream>>>(parents, drafts, uniforms, tokens, N,
                                                            V, status);
  else
    tv_draft_kernel<false><<<grid, kThreads, smem, stream>>>(parents, drafts, uniforms, tokens,
                                                             N, V, status);
  return cudaGetLastError() == cudaSuccess ? 0 : -5;
}
