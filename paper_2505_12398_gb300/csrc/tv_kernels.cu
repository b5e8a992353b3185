// tv_kernels.cu -- CUDA kernels of batched Traversal Verification (sm_103a).
//
// One call verifies B independent trees in three launches on one stream:
//
//   tv_prep_kernel       one warp per tree: structural checks of the parent
//                        array and the token range, then appends the tree's
//                        internal rows (rows with >= 1 child) to a work list.
//   tv_row_stats_kernel  the row normaliser of every internal row, fully
//                        parallel over B x |I| rows: one streaming pass with an
//                        online max / sum of exp2((l - m) log2(e) / T).  These
//                        are the target distributions M_b(.|X^i) Algorithm 3
//                        initialises its acceptance rates from (§3.1).
//   tv_traverse_kernel   one CTA per tree: thread 0 runs the serial post-order
//                        traversal of Algorithm 3 (Appendix E order) on chip;
//                        every rejection's vocabulary-wide reduction
//                        S = sum_x [p M_b(x) - M_s(x)]_+ of Eqs. (1)/(3), and the
//                        final inverse-CDF draw of Y, are streamed by the whole
//                        CTA.
//
// The mutable distributions of Algorithm 3 are never materialised.  After k
// rejections at node i (children tokens t_0..t_{k-1} removed) they are, for
// every token x not yet removed,
//     M_b^(k)(x) = [a_k M_b^(0)(x) - b_k M_s^(0)(x)]_+,   M_s^(k)(x) = M_s^(0)(x) / Z_k,
// with a_0 = 1, b_0 = 0, Z_0 = 1 and, at the rejection with rate p and sum S,
//     a_{k+1} = p a_k / S,   b_{k+1} = (p b_k + 1/Z_k) / S,   Z_{k+1} = Z_k - M_s^(0)(t_k),
// which is Eq. (1) and Eq. (2) applied to that form.  A removed token t keeps
// M_s = 0 and M_b(t) = m_t, stored per removed child and rescaled by p / S at
// each later rejection.  Each rejection therefore streams the ORIGINAL target
// and draft rows of the parent once, with two scalars and the short sorted
// list of removed tokens.
#include <cuda_runtime.h>
#include <stdint.h>

#include "tv_device.cuh"
#include "tv_launch.h"

namespace tvk {

// ------------------------------------------------------------------ prep --

__global__ void __launch_bounds__(256) tv_prep_kernel(const int32_t* __restrict__ parents,
                                                      const int32_t* __restrict__ tokens,
                                                      int B, int R, int V,
                                                      int32_t* __restrict__ row_list,
                                                      int32_t* __restrict__ n_rows) {
  __shared__ uint32_t s_has[8][32];   // one bit per row (R <= 1024), per warp
  const int wl = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tree = blockIdx.x * 8 + wl;
  s_has[wl][lane] = 0u;
  __syncwarp();
  if (tree >= B) return;
  const int32_t* par = parents + (size_t)tree * R;
  const int32_t* tok = tokens + (size_t)tree * R;
  bool bad = false;
  for (int i = lane; i < R; i += 32) {
    int p = par[i];
    if (i == 0) {
      bad |= (p != -1);
    } else {
      int t = tok[i];
      bad |= (t < 0 || t >= V);
      if (p < 0 || p >= i) bad = true;
      else atomicOr(&s_has[wl][p >> 5], 1u << (p & 31));
    }
  }
  bad = __any_sync(0xffffffffu, bad);
  __syncwarp();
  if (bad) return;   // the traversal kernel reports it; no row work queued
  uint32_t word = s_has[wl][lane];
  int cnt = __popc(word);
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  int total = __shfl_sync(0xffffffffu, incl, 31);
  int base = 0;
  if (lane == 31) base = atomicAdd(n_rows, total);
  base = __shfl_sync(0xffffffffu, base, 31);
  int pos = base + incl - cnt;
  while (word) {
    int bit = __ffs(word) - 1;
    word &= word - 1;
    row_list[pos++] = tree * R + lane * 32 + bit;
  }
}

// ------------------------------------------------------------- row stats --

constexpr int kStatsThreads = 256;
constexpr int kStatsUnroll = 4;

template <typename L, bool VEC>
__global__ void __launch_bounds__(kStatsThreads) tv_row_stats_kernel(
    const typename L::elem* __restrict__ logits, int V, float c_hi, float c_lo,
    const int32_t* __restrict__ row_list, const int32_t* __restrict__ n_rows,
    float2* __restrict__ stats) {
  __shared__ float s_red[kStatsThreads / 32];
  __shared__ float s_max;
  const int n = *n_rows;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int r = blockIdx.x; r < n; r += gridDim.x) {
    const int g = row_list[r];
    const typename L::elem* row = logits + (size_t)g * V;
    // phase 1: per-thread online max / sum relative to that max
    float m = TV_NEG_INF;
    Comp acc;
    const int step = kStatsThreads * kChunk;
    int x0 = threadIdx.x * kChunk;
    for (; x0 + (kStatsUnroll - 1) * step < V; x0 += kStatsUnroll * step) {
      float v[kStatsUnroll][8];
#pragma unroll
      for (int u = 0; u < kStatsUnroll; ++u) load_logits<L, VEC>(row, x0 + u * step, V, v[u]);
#pragma unroll
      for (int u = 0; u < kStatsUnroll; ++u) {
        float cm = fmaxf(fmaxf(fmaxf(v[u][0], v[u][1]), fmaxf(v[u][2], v[u][3])),
                         fmaxf(fmaxf(v[u][4], v[u][5]), fmaxf(v[u][6], v[u][7])));
        if (cm > m) {
          if (m != TV_NEG_INF) {
            const float sc = L::exp_rel(m, cm, c_hi, c_lo);
            acc.s *= sc;
            acc.c *= sc;
          }
          m = cm;
        }
        if (m != TV_NEG_INF) {
          float t[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) t[e] = L::exp_rel(v[u][e], m, c_hi, c_lo);
          acc.add(sum8(t));
        }
      }
    }
    for (; x0 < V; x0 += step) {
      float v[8];
      load_logits<L, VEC>(row, x0, V, v);
      float cm = v[0];
#pragma unroll
      for (int e = 1; e < 8; ++e) cm = fmaxf(cm, v[e]);
      if (cm > m) {
        if (m != TV_NEG_INF) {
          const float sc = L::exp_rel(m, cm, c_hi, c_lo);
          acc.s *= sc;
          acc.c *= sc;
        }
        m = cm;
      }
      if (m != TV_NEG_INF) {
        float t[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) t[e] = L::exp_rel(v[e], m, c_hi, c_lo);
        acc.add(sum8(t));
      }
    }
    // phase 2: the row max, then every partial rescaled once to it and summed
    float bm = warp_max(m);
    if (lane == 0) s_red[wid] = bm;
    __syncthreads();
    if (wid == 0) {
      float x = (lane < kStatsThreads / 32) ? s_red[lane] : TV_NEG_INF;
      x = warp_max(x);
      if (lane == 0) s_max = x;
    }
    __syncthreads();
    const float M = s_max;
    float part = (m == TV_NEG_INF) ? 0.f : acc.value() * L::exp_rel(m, M, c_hi, c_lo);
    part = warp_sum(part);
    __syncthreads();
    if (lane == 0) s_red[wid] = part;
    __syncthreads();
    if (wid == 0) {
      float x = (lane < kStatsThreads / 32) ? s_red[lane] : 0.f;
      x = warp_sum(x);
      if (lane == 0) stats[g] = make_float2(M, x);
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------- traversal --

constexpr int kTravThreads = 512;
constexpr int kTravWarps = kTravThreads / 32;
constexpr int kTile = 32 * kChunk;   // elements of one warp-tile in the bonus draw

enum : uint8_t { kAlive = 0, kRejected = 1, kPruned = 2 };
enum : int { kCmdPass = 0, kCmdDone = 1 };

struct Ctl {
  int cmd;
  int pass_node;      // node whose rows the next pass streams
  int nmask;          // removed tokens to skip in that pass
  float alpha1;       // coefficient of e(x) = 2^((l - m) c) in the pass
  float beta;         // coefficient of M_s^(0)(x) in the pass
  float S;            // pass result (removed tokens excluded)
  int accepted;       // accepted node, -1 if the tree is invalid
  uint32_t bad;       // TV_STATUS_* bits found for this tree
  float bonus_a;      // residual bonus weights: bonus_a e(x) - bonus_b q(x)
  float bonus_b;
  float rowmax;
  int bonus_y;
  float bmargin;      // margin of the bonus draw (out_margin[b][1])
};

// Per-tree shared state.  The serial control keeps its scalars in float64.
struct TravSmem {
  double *p, *a, *b, *Z, *invZ, *m;
  int32_t *par, *tok, *first, *next, *npass, *mask_tok;
  float *gl, *gq, *rowm, *rows, *dbgp, *mask_val, *tsum, *tmax;
  uint8_t* state;
};

__device__ __forceinline__ TravSmem carve(char* base, int R, int V) {
  TravSmem s;
  double* dp = reinterpret_cast<double*>(base);
  s.p = dp; dp += R;
  s.a = dp; dp += R;
  s.b = dp; dp += R;
  s.Z = dp; dp += R;
  s.invZ = dp; dp += R;
  s.m = dp; dp += R;
  int32_t* ip = reinterpret_cast<int32_t*>(dp);
  s.par = ip; ip += R;
  s.tok = ip; ip += R;
  s.first = ip; ip += R;
  s.next = ip; ip += R;
  s.npass = ip; ip += R;
  s.mask_tok = ip; ip += R;
  float* fp = reinterpret_cast<float*>(ip);
  s.gl = fp; fp += R;
  s.gq = fp; fp += R;
  s.rowm = fp; fp += R;
  s.rows = fp; fp += R;
  s.dbgp = fp; fp += R;
  s.mask_val = fp; fp += R;
  const int nt = (V + kTile - 1) / kTile;
  s.tsum = fp; fp += nt;
  s.tmax = fp; fp += nt;
  s.state = reinterpret_cast<uint8_t*>(fp);
  return s;
}

struct Control {
  // serial state of the traversal, owned by thread 0
  int node = 0;
  int pending = -1;       // child whose rejection the running pass serves
  double masked_sum = 0;  // sum of m over the removed tokens of that pass
  int n_tests = 0, n_passes = 0;
};

__device__ __forceinline__ int first_alive_child(const TravSmem& s, int i) {
  int j = s.first[i];
  while (j >= 0 && s.state[j] != kAlive) j = s.next[j];
  return j;
}

// M_b^(0)(x_c | X^i) of child c's token.  The numerator is evaluated in
// float64: a residual a M_b(x) - b M_s(x) formed from it can cancel by orders
// of magnitude, and a single float32 exponential (unlike the row sum, which
// averages many) would carry its full rounding into the child's rate.
__device__ __forceinline__ double mb0_of(const TravSmem& s, int i, int c, double cd) {
  return exp2(((double)s.gl[c] - (double)s.rowm[i]) * cd) / (double)s.rows[i];
}

// Rate of child c of node i from i's current state:
// min(p_i M_b(x_c) / M_s(x_c), 1).  Returns false if M_s(x_c) == 0.
__device__ __forceinline__ bool child_rate(const TravSmem& s, int i, int c, double cd, double* out) {
  const double q = (double)s.gq[c];
  const double mb = fmax(s.a[i] * mb0_of(s, i, c, cd) - s.b[i] * q, 0.0);
  const double ms = q * s.invZ[i];
  if (!(ms > 0.0)) return false;
  *out = fmin(s.p[i] * mb / ms, 1.0);
  return true;
}

__device__ void start_pass(const TravSmem& s, Ctl& ctl, Control& st, int i, int c) {
  st.pending = c;
  const double p = s.p[i];
  ctl.alpha1 = (float)(p * s.a[i] / (double)s.rows[i]);
  ctl.beta = (float)(p * s.b[i] + s.invZ[i]);
  int n = 0;
  double msum = 0.0;
  for (int j = s.first[i]; j >= 0; j = s.next[j]) {
    if (j == c || s.state[j] == kAlive) continue;
    // removed tokens in increasing order
    const int t = s.tok[j];
    int k = n;
    while (k > 0 && s.mask_tok[k - 1] > t) {
      s.mask_tok[k] = s.mask_tok[k - 1];
      --k;
    }
    s.mask_tok[k] = t;
    msum += s.m[j];
    ++n;
  }
  ctl.nmask = n;
  st.masked_sum = msum;
  ctl.pass_node = i;
  ctl.cmd = kCmdPass;
  st.n_passes++;
  s.npass[i]++;
}

// Eqs. (1)-(3) at node i after removing child c, in the (a, b, Z) form.
__device__ void apply_rejection(const TravSmem& s, Ctl& ctl, Control& st, int i, int c, double cd) {
  const double p = s.p[i], a = s.a[i], b = s.b[i];
  const double S = (double)ctl.S + p * st.masked_sum;
  const double alpha = p * a;
  const double beta = p * b + s.invZ[i];
  const double mb0 = mb0_of(s, i, c, cd);
  const double q0 = (double)s.gq[c];
  if (S > 0.0) {
    const double na = alpha / S, nb = beta / S, scale = p / S;
    for (int j = s.first[i]; j >= 0; j = s.next[j])
      if (j != c && s.state[j] != kAlive) s.m[j] *= scale;
    s.m[c] = fmax(na * mb0 - nb * q0, 0.0);
    s.a[i] = na;
    s.b[i] = nb;
    s.p[i] = S / (S + (1.0 - p));
  } else {
    // 0/0 in Eqs. (1)/(3): the node keeps its target distribution; its rate
    // becomes 0 (it can no longer be accepted) unless it was 1.
    ctl.bad |= 16u;
    s.m[c] = fmax(a * mb0 - b * q0, 0.0);
    s.p[i] = (p == 1.0) ? 1.0 : 0.0;
  }
  const double Z = s.Z[i] - q0;
  s.Z[i] = Z;
  s.invZ[i] = (Z > 0.0) ? 1.0 / Z : 0.0;
}

// Runs the serial traversal until a vocabulary pass is needed or it ends.
__device__ void control_step(const TravSmem& s, Ctl& ctl, Control& st, const float* __restrict__ u,
                             double cd) {
  if (st.pending >= 0) {
    const int c = st.pending, i = s.par[c];
    apply_rejection(s, ctl, st, i, c, cd);
    st.pending = -1;
    st.node = i;
    if (i != 0 && s.p[i] == 0.0) {   // rate 0: remove i with what is left below it
      s.state[i] = kPruned;
      s.dbgp[i] = 0.f;
      start_pass(s, ctl, st, s.par[i], i);
      return;
    }
  }
  for (;;) {
    const int node = st.node;
    const int c = first_alive_child(s, node);
    if (c < 0) {
      if (node == 0) { ctl.accepted = 0; ctl.cmd = kCmdDone; return; }
      st.n_tests++;
      s.dbgp[node] = (float)s.p[node];
      if ((double)u[node] < s.p[node]) { ctl.accepted = node; ctl.cmd = kCmdDone; return; }
      s.state[node] = kRejected;
      start_pass(s, ctl, st, s.par[node], node);
      return;
    }
    double pc;
    if (!child_rate(s, node, c, cd, &pc)) {
      ctl.bad |= 8u;
      ctl.accepted = -1;
      ctl.cmd = kCmdDone;
      return;
    }
    if (pc == 0.0) {
      s.state[c] = kPruned;
      s.dbgp[c] = 0.f;
      start_pass(s, ctl, st, node, c);
      return;
    }
    s.p[c] = pc;
    st.node = c;
  }
}

template <typename L, bool VEC>
__global__ void __launch_bounds__(kTravThreads, 1) tv_traverse_kernel(TravArgs args) {
  extern __shared__ __align__(16) char smem_raw[];
  __shared__ Ctl ctl;
  __shared__ float red[kTravWarps];
  const int R = args.N + 1, V = args.V;
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const float c_hi = args.c_hi, c_lo = args.c_lo;
  TravSmem s = carve(smem_raw, R, V);
  const typename L::elem* logits = reinterpret_cast<const typename L::elem*>(args.logits);
  const size_t tree_row0 = (size_t)b * R;

  if (tid == 0) {
    ctl.bad = 0u;
    ctl.accepted = -1;
    ctl.cmd = kCmdPass;
  }
  for (int i = tid; i < R; i += kTravThreads) {
    s.par[i] = args.parents[tree_row0 + i];
    s.tok[i] = args.tokens[tree_row0 + i];
    s.first[i] = 0x7fffffff;
    s.npass[i] = 0;
    s.state[i] = kAlive;
    s.a[i] = 1.0;
    s.b[i] = 0.0;
    s.Z[i] = 1.0;
    s.invZ[i] = 1.0;
    s.m[i] = 0.0;
    s.p[i] = 0.0;
    s.dbgp[i] = __int_as_float(0x7fc00000);
  }
  __syncthreads();
  // structure: parents precede children, tokens in range, first child of each node
  {
    uint32_t bad = 0u;
    for (int i = tid; i < R; i += kTravThreads) {
      const int p = s.par[i];
      if (i == 0) {
        if (p != -1) bad |= 1u;
      } else {
        if (p < 0 || p >= i) bad |= 1u;
        else atomicMin(&s.first[p], i);
        const int t = s.tok[i];
        if (t < 0 || t >= V) bad |= 2u;
      }
    }
    if (bad) atomicOr(&ctl.bad, bad);
  }
  __syncthreads();
  if (ctl.bad == 0u) {
    uint32_t bad = 0u;
    for (int i = tid; i < R; i += kTravThreads) {
      if (s.first[i] == 0x7fffffff) s.first[i] = -1;
      int nx = -1;
      if (i > 0) {
        const int p = s.par[i], t = s.tok[i];
        for (int j = i + 1; j < R; ++j) {
          if (s.par[j] != p) continue;
          if (nx < 0) nx = j;
          if (s.tok[j] == t) bad |= 4u;
        }
        // gathers of the child's token in its parent's rows
        const size_t prow = (tree_row0 + p) * (size_t)V;
        s.gl[i] = L::at(logits + prow, t);
        s.gq[i] = __ldg(args.draft_probs + prow + t);
        if (!(s.gq[i] > 0.f)) bad |= 8u;
      }
      s.next[i] = nx;
    }
    if (bad) atomicOr(&ctl.bad, bad);
  }
  __syncthreads();
  bool ok = (ctl.bad == 0u);
  if (ok) {
    for (int i = tid; i < R; i += kTravThreads) {
      if (s.first[i] >= 0) {
        const float2 st2 = args.stats[tree_row0 + i];
        s.rowm[i] = st2.x;
        s.rows[i] = st2.y;
        if (!(st2.y > 0.f)) atomicOr(&ctl.bad, 64u);   // no finite logit in the row
      }
    }
    if (tid == 0) s.p[0] = 1.0;
  }
  __syncthreads();

  Control st;
  const float* u = args.uniforms + (size_t)b * (R + 1);
  if (ok && (ctl.bad & 64u)) ok = false;
  if (ok) {
    for (;;) {
      if (tid == 0) control_step(s, ctl, st, u, args.c);
      __syncthreads();
      if (ctl.cmd == kCmdDone) break;
      // ---- S = sum over tokens not removed of [alpha1 e(x) - beta q(x)]_+ ----
      const int i = ctl.pass_node;
      const typename L::elem* lrow = logits + (tree_row0 + i) * (size_t)V;
      const float* qrow = args.draft_probs + (tree_row0 + i) * (size_t)V;
      const float m = s.rowm[i], al = ctl.alpha1, be = ctl.beta;
      const int nmask = ctl.nmask;
      Comp acc;
      int mp = 0;
      for (int x0 = tid * kChunk; x0 < V; x0 += kTravThreads * kChunk) {
        float v[8], q[8], t[8];
        load_logits<L, VEC>(lrow, x0, V, v);
        load_probs<VEC>(qrow, x0, V, q);
#pragma unroll
        for (int k = 0; k < 8; ++k)
          t[k] = fmaxf(fmaf(al, L::exp_rel(v[k], m, c_hi, c_lo), -be * q[k]), 0.f);
        while (mp < nmask && s.mask_tok[mp] < x0) ++mp;
        for (int mq = mp; mq < nmask && s.mask_tok[mq] < x0 + kChunk; ++mq) {
          const int off = s.mask_tok[mq] - x0;
#pragma unroll
          for (int k = 0; k < 8; ++k) if (k == off) t[k] = 0.f;
        }
        acc.add(sum8(t));
      }
      float tot = warp_sum(acc.value());
      if (lane == 0) red[wid] = tot;
      __syncthreads();
      if (wid == 0) {
        float v = (lane < kTravWarps) ? red[lane] : 0.f;
        v = warp_sum(v);
        if (lane == 0) ctl.S = v;
      }
      __syncthreads();
    }
  }

  // ---- bonus token: inverse CDF of the accepted node's current M_b ----
  const int acc_node = ok ? ctl.accepted : -1;
  int y = -1;
  if (acc_node >= 0) {
    const int a = acc_node;
    const bool leaf = s.first[a] < 0;
    const typename L::elem* lrow = logits + (tree_row0 + a) * (size_t)V;
    const float* qrow = args.draft_probs + (tree_row0 + a) * (size_t)V;
    // removed tokens of the accepted node (all its children) with their M_b
    if (tid == 0) {
      int n = 0;
      if (!leaf) {
        for (int j = s.first[a]; j >= 0; j = s.next[j]) {
          const int t = s.tok[j];
          int k = n;
          while (k > 0 && s.mask_tok[k - 1] > t) {
            s.mask_tok[k] = s.mask_tok[k - 1];
            s.mask_val[k] = s.mask_val[k - 1];
            --k;
          }
          s.mask_tok[k] = t;
          s.mask_val[k] = (float)s.m[j];
          ++n;
        }
        ctl.bonus_a = (float)(s.a[a] / (double)s.rows[a]);
        ctl.bonus_b = (float)s.b[a];
        ctl.rowmax = s.rowm[a];
      }
      ctl.nmask = n;
    }
    __syncthreads();
    const int nt = (V + kTile - 1) / kTile;
    const int nmask = ctl.nmask;
    const float ba = ctl.bonus_a, bb = ctl.bonus_b, rm = ctl.rowmax;
    // pass 1: per warp-tile sums (leaf: relative to the tile's own max)
    int mp = 0;
    for (int k = wid; k < nt; k += kTravWarps) {
      const int x0 = k * kTile + lane * kChunk;
      float w[8];
      if (leaf) {
        float v[8];
        if (x0 < V) load_logits<L, VEC>(lrow, x0, V, v);
        else {
#pragma unroll
          for (int e = 0; e < 8; ++e) v[e] = TV_NEG_INF;
        }
        float lm = v[0];
#pragma unroll
        for (int e = 1; e < 8; ++e) lm = fmaxf(lm, v[e]);
        const float tm = warp_max(lm);
#pragma unroll
        for (int e = 0; e < 8; ++e)
          w[e] = (v[e] == TV_NEG_INF) ? 0.f : L::exp_rel(v[e], tm, c_hi, c_lo);
        const float ts = warp_sum(sum8(w));
        if (lane == 0) { s.tsum[k] = ts; s.tmax[k] = tm; }
      } else {
        float v[8], q[8];
        if (x0 < V) {
          load_logits<L, VEC>(lrow, x0, V, v);
          load_probs<VEC>(qrow, x0, V, q);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) { v[e] = TV_NEG_INF; q[e] = 0.f; }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
          w[e] = (v[e] == TV_NEG_INF) ? 0.f
                                      : fmaxf(fmaf(ba, L::exp_rel(v[e], rm, c_hi, c_lo), -bb * q[e]), 0.f);
        while (mp < nmask && s.mask_tok[mp] < x0) ++mp;
        for (int mq = mp; mq < nmask && s.mask_tok[mq] < x0 + kChunk; ++mq) {
          const int off = s.mask_tok[mq] - x0;
          const float mv = s.mask_val[mq];
#pragma unroll
          for (int e = 0; e < 8; ++e) if (e == off) w[e] = mv;
        }
        const float ts = warp_sum(sum8(w));
        if (lane == 0) s.tsum[k] = ts;
      }
    }
    __syncthreads();
    // scan of the tile sums in token order (warp 0), then the crossing tile
    if (wid == 0) {
      float M = 0.f;
      if (leaf) {
        float lm = TV_NEG_INF;
        for (int k = lane; k < nt; k += 32) lm = fmaxf(lm, s.tmax[k]);
        M = warp_max(lm);
        for (int k = lane; k < nt; k += 32)
          s.tsum[k] = (s.tmax[k] == TV_NEG_INF) ? 0.f : s.tsum[k] * L::exp_rel(s.tmax[k], M, c_hi, c_lo);
        __syncwarp();
      }
      float base = 0.f;
      for (int k0 = 0; k0 < nt; k0 += 32) {
        float v = (k0 + lane < nt) ? s.tsum[k0 + lane] : 0.f;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          float w2 = __shfl_up_sync(0xffffffffu, v, o);
          if (lane >= o) v += w2;
        }
        base += __shfl_sync(0xffffffffu, v, 31);
      }
      const float W = base;
      const float target = u[R] * W;
      int tile = -1;
      float tbase = 0.f;
      base = 0.f;
      for (int k0 = 0; k0 < nt && tile < 0; k0 += 32) {
        float v = (k0 + lane < nt) ? s.tsum[k0 + lane] : 0.f;
        const float own = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          float w2 = __shfl_up_sync(0xffffffffu, v, o);
          if (lane >= o) v += w2;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, (k0 + lane < nt) && (target < base + v));
        if (hit) {
          const int l = __ffs(hit) - 1;
          tile = k0 + l;
          tbase = base + __shfl_sync(0xffffffffu, v - own, l);
        }
        base += __shfl_sync(0xffffffffu, v, 31);
      }
      if (tile < 0) {   // rounding left u W at or past the total: last tile with weight
        tile = nt - 1;
        while (tile > 0 && !(s.tsum[tile] > 0.f)) --tile;
        float acc0 = 0.f;
        for (int k = 0; k < tile; ++k) acc0 += s.tsum[k];
        tbase = acc0;
      }
      // rescan the crossing tile element by element
      const int x0 = tile * kTile + lane * kChunk;
      float w[8];
      if (leaf) {
        float v[8];
        if (x0 < V) load_logits<L, VEC>(lrow, x0, V, v);
        else {
#pragma unroll
          for (int e = 0; e < 8; ++e) v[e] = TV_NEG_INF;
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
          w[e] = (v[e] == TV_NEG_INF) ? 0.f : L::exp_rel(v[e], M, c_hi, c_lo);
      } else {
        float v[8], q[8];
        if (x0 < V) {
          load_logits<L, VEC>(lrow, x0, V, v);
          load_probs<VEC>(qrow, x0, V, q);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) { v[e] = TV_NEG_INF; q[e] = 0.f; }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
          w[e] = (v[e] == TV_NEG_INF) ? 0.f
                                      : fmaxf(fmaf(ba, L::exp_rel(v[e], rm, c_hi, c_lo), -bb * q[e]), 0.f);
        for (int mq = 0; mq < nmask; ++mq) {
          const int off = s.mask_tok[mq] - x0;
          const float mv = s.mask_val[mq];
#pragma unroll
          for (int e = 0; e < 8; ++e) if (e == off) w[e] = mv;
        }
      }
      float pre[8];
      float run = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) { run += w[e]; pre[e] = run; }
      float v = run;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        float w2 = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += w2;
      }
      const float lbase = tbase + (v - run);
      int found = 8;
#pragma unroll
      for (int e = 7; e >= 0; --e) if (target < lbase + pre[e]) found = e;
      const unsigned hit = __ballot_sync(0xffffffffu, found < 8);
      // the draw's margin: distance of u W to the nearer end of the chosen
      // token's CDF interval (kernel sums), relative to W
      float clo = lbase, chi = lbase;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        if (e == found) chi = lbase + pre[e];
        if (e + 1 == found) clo = lbase + pre[e];
      }
      const float my_margin = fminf(target - clo, chi - target) / W;
      int yy;
      if (hit) {
        const int l = __ffs(hit) - 1;
        yy = tile * kTile + l * kChunk + __shfl_sync(0xffffffffu, found, l);
        const float bm = __shfl_sync(0xffffffffu, my_margin, l);
        if (lane == 0) ctl.bmargin = bm;
      } else {
        if (lane == 0) ctl.bmargin = 0.f;
        // rounding: take the last token of the tile with positive weight
        int last = -1;
#pragma unroll
        for (int e = 0; e < 8; ++e) if (w[e] > 0.f) last = x0 + e;
        const unsigned any = __ballot_sync(0xffffffffu, last >= 0);
        if (any) {
          const int l = 31 - __clz(any);
          yy = __shfl_sync(0xffffffffu, last, l);
        } else {
          yy = V - 1;
        }
      }
      if (lane == 0) ctl.bonus_y = yy;
    }
    __syncthreads();
    y = ctl.bonus_y;
  }

  // ---- outputs ----
  const int N = args.N;
  for (int k = tid; k < N; k += kTravThreads) args.out_path[(size_t)b * N + k] = -1;
  if (args.out_node_p) {
    for (int i = tid; i < R; i += kTravThreads)
      args.out_node_p[tree_row0 + i] = ok ? s.dbgp[i] : __int_as_float(0x7fc00000);
  }
  __syncthreads();
  if (tid == 0) {
    if (acc_node >= 0) {
      int depth = 0;
      for (int j = acc_node; j != 0; j = s.par[j]) ++depth;
      int k = depth - 1;
      for (int j = acc_node; j != 0; j = s.par[j]) args.out_path[(size_t)b * N + (k--)] = j;
      args.out_accept_len[b] = depth;
      args.out_bonus[b] = y;
    } else {
      args.out_accept_len[b] = -1;
      args.out_bonus[b] = -1;
    }
    if (args.out_stats) {
      int distinct = 0;
      for (int i = 0; i < R; ++i) distinct += (s.npass[i] > 0);
      int internal = 0;
      for (int i = 0; i < R; ++i) internal += (s.first[i] >= 0);
      int32_t* o = args.out_stats + (size_t)b * 5;
      o[0] = ok ? st.n_tests : 0;
      o[1] = ok ? st.n_passes : 0;
      o[2] = ok ? distinct : 0;
      o[3] = (acc_node >= 0 && s.first[acc_node] < 0) ? 1 : 0;
      o[4] = ok ? internal : 0;
    }
    if (args.out_margin) {
      const float nan = __int_as_float(0x7fc00000);
      args.out_margin[2 * (size_t)b] = acc_node >= 0 ? test_margin_serial(s.dbgp, u, R) : nan;
      args.out_margin[2 * (size_t)b + 1] = acc_node >= 0 ? ctl.bmargin : nan;
    }
    if (ctl.bad) atomicOr(args.status, ctl.bad);
  }
}

}  // namespace tvk

// --------------------------------------------------------------- launchers --

namespace {
int launch_error() {
  return (cudaGetLastError() == cudaSuccess) ? 0 : -5;
}
}  // namespace

size_t tv_traverse_smem_bytes(int R, int V) {
  const int nt = (V + tvk::kTile - 1) / tvk::kTile;
  return (size_t)R * (6 * 8 + 6 * 4 + 6 * 4 + 1) + (size_t)nt * 8 + 64;
}

namespace {

template <typename L, bool VEC>
int launch_typed(const TravArgs& a, int* row_list, int* n_rows, int stats_grid,
                 cudaStream_t stream, cudaEvent_t* ev) {
  const int R = a.N + 1;
  const size_t smem = tv_traverse_smem_bytes(R, a.V);
  const auto* lg = reinterpret_cast<const typename L::elem*>(a.logits);
  if (ev && cudaEventRecord(ev[0], stream) != cudaSuccess) return -5;
  if (cudaMemsetAsync(n_rows, 0, sizeof(int), stream) != cudaSuccess) return -5;
  tvk::tv_prep_kernel<<<(a.B + 7) / 8, 256, 0, stream>>>(a.parents, a.tokens, a.B, R, a.V,
                                                          row_list, n_rows);
  if (launch_error()) return -5;
  if (ev && cudaEventRecord(ev[1], stream) != cudaSuccess) return -5;
  tvk::tv_row_stats_kernel<L, VEC><<<stats_grid, tvk::kStatsThreads, 0, stream>>>(
      lg, a.V, a.c_hi, a.c_lo, row_list, n_rows, a.stats);
  if (launch_error()) return -5;
  if (ev && cudaEventRecord(ev[2], stream) != cudaSuccess) return -5;
  if (cudaFuncSetAttribute(tvk::tv_traverse_kernel<L, VEC>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return -5;
  tvk::tv_traverse_kernel<L, VEC><<<a.B, tvk::kTravThreads, smem, stream>>>(a);
  if (launch_error()) return -5;
  if (ev && cudaEventRecord(ev[3], stream) != cudaSuccess) return -5;
  return 0;
}

}  // namespace

int tv_launch_all(const TravArgs& a, int logit_is_bf16, int* row_list, int* n_rows,
                  int stats_grid, cudaStream_t stream, cudaEvent_t* events) {
  const bool vec = (a.V % 8) == 0;
  if (logit_is_bf16) {
    return vec ? launch_typed<tvk::Bf16Logits, true>(a, row_list, n_rows, stats_grid, stream, events)
               : launch_typed<tvk::Bf16Logits, false>(a, row_list, n_rows, stats_grid, stream, events);
  }
  return vec ? launch_typed<tvk::F32Logits, true>(a, row_list, n_rows, stats_grid, stream, events)
             : launch_typed<tvk::F32Logits, false>(a, row_list, n_rows, stats_grid, stream, events);
}
