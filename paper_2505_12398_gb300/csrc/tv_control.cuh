// tv_control.cuh -- per-tree state and the serial control of Algorithm 3
// (§3.1), shared by the fused kernels.
//
// The tree's state lives in the shared memory of the CTA that owns it; thread
// 0 advances the traversal (control_step) until it needs vocabulary-wide work
// and describes that work as a Job: normalisers of a list of rows, one
// rejection pass (Eqs. (1)/(3)), or the bonus draw.  Scalars are float64 (see
// children_mb0 and the parity notes of the repository's design document).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tv_device.cuh"

namespace tvk {
namespace fused {

// A CTA of the cluster kernel has NCW consumer warps (4 or 8) and one producer
// warp; its ring stages hold 3 * NCW KB: a target + draft slice of 512 * NCW
// tokens (bf16), or a target-only slice of 1536 * NCW tokens.  (The
// persistent kernel sizes its stages itself, tv_flow.cu.)
constexpr int kMaxStages = 8;
constexpr int kMaxCluster = 8;
constexpr int kTileElems = 256;       // one warp x 8 elements
__host__ __device__ constexpr int stage_bytes(int ncw) { return 3072 * ncw; }

enum : int { kJobStats = 1, kJobPass = 2, kJobBonusLeaf = 3, kJobBonusRes = 4, kJobDone = 5 };
enum : uint8_t { kAlive = 0, kRejected = 1, kPruned = 2 };

struct Job {
  int kind;
  int n_rows;        // rows listed in job_rows (kJobStats), else 1
  int node;          // row of kJobPass / bonus jobs
  int nmask;         // removed tokens of that row (sorted in mask_tok / mask_val)
  float alpha1;      // kJobPass: coefficient of e(x); bonus residual: a / s
  float beta;        // kJobPass: coefficient of q(x); bonus residual: b
  float rowmax;      // row max used by e(x)
};

struct Ctl {
  Job job;
  uint32_t bad;        // TV_STATUS_* bits
  int accepted;        // accepted node (-1: invalid tree)
  float S;             // result of the last pass
  int bonus_y;
  float bmargin;       // margin of the bonus draw (out_margin[b][1])
  // serial control state (thread 0)
  int node;
  int pending;         // child whose rejection the running pass serves
  double masked_sum;
  int n_tests, n_passes;
  int stage, phase;    // consumer ring position
  uint32_t xphase;     // parity of the cluster-exchange barrier
  int xbuf;            // double-buffer index of the exchange slots
};

struct TreeSmem {
  double *p, *a, *b, *Z, *invZ, *m, *mb0, *invq, *invs;
  int32_t *par, *tok, *first, *next, *npass, *mask_tok, *job_rows;
  float *gl, *gq, *rowm, *rows, *dbgp, *mask_val, *tsum, *tmax;
  uint8_t* state;
};

__host__ __device__ inline int slice_len(int V, int C) {
  int per = (V + C - 1) / C;
  return (per + kChunk - 1) / kChunk * kChunk;
}

__host__ __device__ inline int n_tiles(int V, int C) {
  return (slice_len(V, C) + kTileElems - 1) / kTileElems;
}

// Shared memory of one tree's state with `nt` bonus tiles.
__host__ __device__ inline size_t tree_smem_bytes_nt(int R, int nt) {
  return (size_t)R * (9 * 8 + 7 * 4 + 6 * 4 + 1) + (size_t)nt * 8 + 64;
}

__host__ __device__ inline size_t tree_smem_bytes(int R, int V, int C) {
  return tree_smem_bytes_nt(R, n_tiles(V, C));
}

__device__ __forceinline__ TreeSmem carve_tree_nt(char* base, int R, int nt) {
  TreeSmem s;
  double* dp = reinterpret_cast<double*>(base);
  s.p = dp; dp += R;
  s.a = dp; dp += R;
  s.b = dp; dp += R;
  s.Z = dp; dp += R;
  s.invZ = dp; dp += R;
  s.m = dp; dp += R;
  s.mb0 = dp; dp += R;
  s.invq = dp; dp += R;
  s.invs = dp; dp += R;
  int32_t* ip = reinterpret_cast<int32_t*>(dp);
  s.par = ip; ip += R;
  s.tok = ip; ip += R;
  s.first = ip; ip += R;
  s.next = ip; ip += R;
  s.npass = ip; ip += R;
  s.mask_tok = ip; ip += R;
  s.job_rows = ip; ip += R;
  float* fp = reinterpret_cast<float*>(ip);
  s.gl = fp; fp += R;
  s.gq = fp; fp += R;
  s.rowm = fp; fp += R;
  s.rows = fp; fp += R;
  s.dbgp = fp; fp += R;
  s.mask_val = fp; fp += R;
  s.tsum = fp; fp += nt;
  s.tmax = fp; fp += nt;
  s.state = reinterpret_cast<uint8_t*>(fp);
  return s;
}

__device__ __forceinline__ TreeSmem carve_tree(char* base, int R, int V, int C) {
  return carve_tree_nt(base, R, n_tiles(V, C));
}

// ------------------------------------------------------------ control ----

__device__ __forceinline__ int first_alive_child(const TreeSmem& s, int i) {
  int j = s.first[i];
  while (j >= 0 && s.state[j] != kAlive) j = s.next[j];
  return j;
}

// M_b^(0)(x_c | X^i) of every child c of node i, in float64, computed by the
// consumer warps as soon as row i's normaliser is known (a residual
// a M_b(x) - b M_s(x) of a sibling can cancel by orders of magnitude, so this
// single value must not carry a float32 rounding).  Kept in s.mb0[c].
__device__ __forceinline__ void children_mb0(const TreeSmem& s, int i, double cd, int lane) {
  int j = s.first[i];
  for (int k = 0; j >= 0; ++k, j = s.next[j])
    if ((k & 31) == lane)
      s.mb0[j] = exp2(((double)s.gl[j] - (double)s.rowm[i]) * cd) * s.invs[i];
}

// min(p_i M_b(x_c) / M_s(x_c), 1) from i's current state, with
// M_s(x_c) = q_c / Z_i; false if it is zero.
__device__ __forceinline__ bool child_rate(const TreeSmem& s, int i, int c, double* out) {
  const double q = (double)s.gq[c];
  const double mb = fmax(s.a[i] * s.mb0[c] - s.b[i] * q, 0.0);
  if (!(s.invZ[i] > 0.0)) return false;
  *out = fmin(s.p[i] * mb * s.Z[i] * s.invq[c], 1.0);
  return true;
}

__device__ inline void post_pass(const TreeSmem& s, Ctl& ctl, int i, int c) {
  ctl.pending = c;
  const double p = s.p[i];
  ctl.job.kind = kJobPass;
  ctl.job.n_rows = 1;
  ctl.job.node = i;
  ctl.job.alpha1 = (float)(p * s.a[i] * s.invs[i]);
  ctl.job.beta = (float)(p * s.b[i] + s.invZ[i]);
  ctl.job.rowmax = s.rowm[i];
  int n = 0;
  double msum = 0.0;
  for (int j = s.first[i]; j >= 0; j = s.next[j]) {
    if (j == c || s.state[j] == kAlive) continue;
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
  ctl.job.nmask = n;
  ctl.masked_sum = msum;
  ctl.n_passes++;
  s.npass[i]++;
}

__device__ inline void apply_rejection(const TreeSmem& s, Ctl& ctl, int i, int c) {
  const double p = s.p[i], a = s.a[i], b = s.b[i];
  const double S = (double)ctl.S + p * ctl.masked_sum;
  const double alpha = p * a;
  const double beta = p * b + s.invZ[i];
  const double mb0 = s.mb0[c];
  const double q0 = (double)s.gq[c];
  if (S > 0.0) {
    const double invS = 1.0 / S;
    const double na = alpha * invS, nb = beta * invS, scale = p * invS;
    for (int j = s.first[i]; j >= 0; j = s.next[j])
      if (j != c && s.state[j] != kAlive) s.m[j] *= scale;
    s.m[c] = fmax(na * mb0 - nb * q0, 0.0);
    s.a[i] = na;
    s.b[i] = nb;
    s.p[i] = S / (S + (1.0 - p));
  } else {
    ctl.bad |= 16u;
    s.m[c] = fmax(a * mb0 - b * q0, 0.0);
    s.p[i] = (p == 1.0) ? 1.0 : 0.0;
  }
  const double Z = s.Z[i] - q0;
  s.Z[i] = Z;
  s.invZ[i] = (Z > 0.0) ? 1.0 / Z : 0.0;
}

// Lists the not-yet-normalised internal nodes of the chain that starts at
// `node` (following first remaining children); returns how many.
__device__ inline int chain_needing_stats(const TreeSmem& s, int node) {
  int n = 0;
  for (int i = node; i >= 0; i = first_alive_child(s, i)) {
    if (s.first[i] < 0) break;            // a leaf: no row statistics needed
    if (!(s.rows[i] > 0.f)) s.job_rows[n++] = i;
  }
  return n;
}

__device__ inline void post_bonus(const TreeSmem& s, Ctl& ctl, int a) {
  ctl.accepted = a;
  ctl.job.node = a;
  ctl.job.n_rows = 1;
  if (s.first[a] < 0) {
    ctl.job.kind = kJobBonusLeaf;
    ctl.job.nmask = 0;
    return;
  }
  ctl.job.kind = kJobBonusRes;
  ctl.job.alpha1 = (float)(s.a[a] * s.invs[a]);
  ctl.job.beta = (float)s.b[a];
  ctl.job.rowmax = s.rowm[a];
  int n = 0;
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
  ctl.job.nmask = n;
}

// ---------------------------------------------------- deciding ahead ----
//
// While the pass that rejects child c of node i runs, most of the next step is
// already fixed.  In the common case -- the next remaining child c2 of i is a
// leaf -- that step is the test of c2, and with
//   D = S + (1 - p_i),   X = [alpha M_b0(c2) - beta q(c2)]_+ Z' / q(c2),
//   alpha = p_i a_i,  beta = p_i b_i + 1/Z_i,  Z' = Z_i - q(c),
// Eqs. (1)-(3) give c2's rate min(X / D, 1), so c2 is accepted iff u D < X, and
// the pass that rejects c2 uses alpha1 = alpha / (s_i D), beta' = beta / D + 1/Z'.
// Only D depends on the pass's S, so the next job can be posted right after
// S arrives and the state update (control_step_ahead) done afterwards.
// The other common case -- i has no remaining child -- is the test of i
// itself with its new rate S / D: i is rejected iff u D >= S, and the pass
// that then rejects i at its parent g depends only on g's state.
struct Ahead {
  int ok;          // 1: the next step is decided from D alone (see mode)
  int mode;        // 1: test of leaf c2 of i; 2: test of i itself (then a pass at g)
  int i, c, c2, g, nmask;
  double omp;      // 1 - p_i
  double X, ainvs, beta, invZn;
  float alpha1_g, beta_g, rowmax_g;   // mode 2: the pass at g that rejects i
};

// S-independent part of the next step, after posting the pass for ctl.pending;
// the next pass's removed tokens (ascending) go to mtok2.
__device__ inline void prepare_ahead(const TreeSmem& s, const Ctl& ctl, Ahead& ah,
                                     int* mtok2) {
  ah.ok = 0;
  if (ctl.job.kind != kJobPass) return;
  const int c = ctl.pending, i = s.par[c];
  const int c2 = first_alive_child(s, i);
  if (c2 < 0) {
    if (i == 0) return;   // the root: the bonus draw follows
    const int g = s.par[i];
    // the pass post_pass(s, ctl, g, i) would post (g's state does not change)
    const double pg = s.p[g];
    ah.alpha1_g = (float)(pg * s.a[g] * s.invs[g]);
    ah.beta_g = (float)(pg * s.b[g] + s.invZ[g]);
    ah.rowmax_g = s.rowm[g];
    int n = 0;
    for (int j = s.first[g]; j >= 0; j = s.next[j]) {
      if (j == i || s.state[j] == kAlive) continue;
      const int t = s.tok[j];
      int k = n;
      while (k > 0 && mtok2[k - 1] > t) {
        mtok2[k] = mtok2[k - 1];
        --k;
      }
      mtok2[k] = t;
      ++n;
    }
    ah.mode = 2;
    ah.i = i;
    ah.c = c;
    ah.c2 = -1;
    ah.g = g;
    ah.nmask = n;
    ah.omp = 1.0 - s.p[i];
    ah.ok = 1;
    return;
  }
  if (s.first[c2] >= 0 || !(s.rows[i] > 0.f)) return;
  const double p = s.p[i], a = s.a[i], b = s.b[i];
  const double Zn = s.Z[i] - (double)s.gq[c];
  if (!(Zn > 0.0)) return;
  const double alpha = p * a, beta = p * b + s.invZ[i];
  const double X = fmax(alpha * s.mb0[c2] - beta * (double)s.gq[c2], 0.0) * Zn * s.invq[c2];
  if (!(X > 0.0)) return;
  int n = 0;
  for (int j = s.first[i]; j >= 0; j = s.next[j]) {
    if (j == c2 || s.state[j] == kAlive) continue;
    const int t = s.tok[j];
    int k = n;
    while (k > 0 && mtok2[k - 1] > t) {
      mtok2[k] = mtok2[k - 1];
      --k;
    }
    mtok2[k] = t;
    ++n;
  }
  ah.i = i;
  ah.c = c;
  ah.c2 = c2;
  ah.nmask = n;
  ah.omp = 1.0 - p;
  ah.X = X;
  ah.ainvs = alpha * s.invs[i];
  ah.beta = beta;
  ah.invZn = 1.0 / Zn;
  ah.mode = 1;
  ah.g = -1;
  ah.ok = 1;
}

// control_step for the pass described by `ah`, with the test of ah.c2 going
// the way `accept` says (the decision taken ahead, so that the state follows
// the job already posted).
__device__ inline void control_step_ahead(const TreeSmem& s, Ctl& ctl, const Ahead& ah,
                                          bool accept) {
  apply_rejection(s, ctl, ah.i, ah.c);
  ctl.pending = -1;
  if (ah.mode == 2) {
    ctl.node = ah.i;
    ctl.n_tests++;
    s.dbgp[ah.i] = (float)s.p[ah.i];
    if (accept) {
      post_bonus(s, ctl, ah.i);
      return;
    }
    s.state[ah.i] = kRejected;
    post_pass(s, ctl, ah.g, ah.i);
    return;
  }
  double pc = 0.0;
  child_rate(s, ah.i, ah.c2, &pc);
  s.p[ah.c2] = pc;
  ctl.node = ah.c2;
  ctl.n_tests++;
  s.dbgp[ah.c2] = (float)pc;
  if (accept) {
    post_bonus(s, ctl, ah.c2);
    return;
  }
  s.state[ah.c2] = kRejected;
  post_pass(s, ctl, ah.i, ah.c2);
}

// Advances the serial traversal until it needs vocabulary work; posts it.
__device__ inline void control_step(const TreeSmem& s, Ctl& ctl, const float* __restrict__ u) {
  if (ctl.job.kind == kJobPass) {
    const int c = ctl.pending, i = s.par[c];
    apply_rejection(s, ctl, i, c);
    ctl.pending = -1;
    ctl.node = i;
    if (i != 0 && s.p[i] == 0.0) {   // rate 0: remove i with what is left below it
      s.state[i] = kPruned;
      s.dbgp[i] = 0.f;
      post_pass(s, ctl, s.par[i], i);
      return;
    }
  }
  for (;;) {
    const int node = ctl.node;
    const int c = first_alive_child(s, node);
    if (c < 0) {
      if (node == 0) { post_bonus(s, ctl, 0); return; }
      ctl.n_tests++;
      s.dbgp[node] = (float)s.p[node];
      if ((double)u[node] < s.p[node]) { post_bonus(s, ctl, node); return; }
      s.state[node] = kRejected;
      post_pass(s, ctl, s.par[node], node);
      return;
    }
    if (!(s.rows[node] > 0.f)) {
      ctl.job.kind = kJobStats;
      ctl.job.n_rows = chain_needing_stats(s, node);
      return;
    }
    double pc;
    if (!child_rate(s, node, c, &pc)) {
      ctl.bad |= 8u;
      ctl.accepted = -1;
      ctl.job.kind = kJobDone;
      return;
    }
    if (pc == 0.0) {
      s.state[c] = kPruned;
      s.dbgp[c] = 0.f;
      post_pass(s, ctl, node, c);
      return;
    }
    s.p[c] = pc;
    ctl.node = c;
  }
}

// ------------------------------------------- token-level verification ----
//
// The top-down verifier Traversal Verification is compared with (§2.2, "Tok.V"
// of §4): at the current node ctl.node its children are tried in order by
// Recursive Rejection Sampling without replacement (Algorithm 2).  That is
// Eqs. (1)-(3) with the node's rate held at 1: min(M_b'(x_c) / M_s'(x_c), 1) is
// child_rate at p = 1, and the residual update [M_b' - M_s']_+ / S with x_c
// removed from M_s' is apply_rejection at p = 1, which leaves p = 1.  An
// accepted child becomes the current node with its own rows (a = 1, b = 0,
// Z = 1 from the tree set-up); the bonus token comes from an accepted leaf's
// own row, or from the current node's residual once all its children are
// rejected.  Only the current node's row is normalised.  A child of rate 0
// is rejected without counting as a test (its uniform cannot accept it).
__device__ inline void control_step_token(const TreeSmem& s, Ctl& ctl,
                                          const float* __restrict__ u) {
  if (ctl.job.kind == kJobPass) {
    const int c = ctl.pending, i = s.par[c];
    apply_rejection(s, ctl, i, c);
    ctl.pending = -1;
    ctl.node = i;
  }
  for (;;) {
    const int node = ctl.node;
    if (s.first[node] < 0) {   // an accepted leaf (or a root without children)
      post_bonus(s, ctl, node);
      return;
    }
    if (!(s.rows[node] > 0.f)) {
      ctl.job.kind = kJobStats;
      ctl.job.n_rows = 1;
      s.job_rows[0] = node;
      return;
    }
    const int c = first_alive_child(s, node);
    if (c < 0) {               // every child rejected: the residual at node
      post_bonus(s, ctl, node);
      return;
    }
    double pc;
    if (!child_rate(s, node, c, &pc)) {
      ctl.bad |= 8u;
      ctl.accepted = -1;
      ctl.job.kind = kJobDone;
      return;
    }
    s.dbgp[c] = (float)pc;
    if (pc > 0.0) {
      ctl.n_tests++;
      if ((double)u[c] < pc) {   // accepted: c becomes the current node
        s.p[c] = 1.0;
        ctl.node = c;
        continue;
      }
    }
    s.state[c] = kRejected;
    post_pass(s, ctl, node, c);
    return;
  }
}

// One step of the tree's verification method until it needs vocabulary work.
__device__ inline void advance(const TreeSmem& s, Ctl& ctl, const float* __restrict__ u,
                               bool token_level) {
  if (token_level) control_step_token(s, ctl, u);
  else control_step(s, ctl, u);
}

}  // namespace fused
}  // namespace tvk
