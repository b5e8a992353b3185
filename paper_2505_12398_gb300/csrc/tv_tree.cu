// tv_tree.cu -- fused, lazy, TMA-pipelined Traversal Verification (sm_103a).
//
// One kernel does all of Algorithm 3 (§3.1) for a batch of trees.  Each tree
// is owned by a thread-block cluster of C CTAs (C = 1, 2 or 4): CTA r streams
// the vocabulary slice [v0_r, v1_r) of every row the tree needs, and every CTA
// runs the same serial control on identical data, so their decisions agree
// without being broadcast; only per-row partial results cross the cluster
// (distributed shared memory + a remote mbarrier arrive).
//
// Inside a CTA, warp 8 is a producer: one lane issues 1-D bulk copies
// (cp.async.bulk, TMA) of row slices into a ring of shared-memory stages,
// completion counted on per-stage mbarriers; warps 0-7 consume the stages
// (128-bit shared loads) and arrive on per-stage "empty" mbarriers.
//
// Rows are read lazily.  The target row of a node is streamed (for its
// normaliser) only when the traversal first descends through the node --
// the rates of a node's children are needed only then -- so sub-trees the
// traversal never enters cost nothing.  The whole not-yet-normalised part of
// the chain being entered is requested as one job.  Each rejection streams the
// parent's ORIGINAL target and draft rows once (the (a, b, Z) closed form of
// Eqs. (1)-(2), see tv_kernels.cu); the bonus draw streams one row (pair).
#include <cuda_runtime.h>
#include <stdint.h>

#include "tv_control.cuh"
#include "tv_device.cuh"
#include "tv_launch.h"
#include "tv_ptx.cuh"

namespace tvk {
namespace fused {

// ----------------------------------------------------- cluster exchange ---

// Publishes this CTA's partial (x, y) for the current row to every CTA of the
// cluster and waits for all of them; returns false on timeout.  Called by
// thread 0 only.  Slots are double-buffered so that a fast CTA's next
// exchange cannot overwrite a slot a slow CTA has not read yet.
__device__ bool exchange(float2 (*slots)[kMaxCluster], uint64_t* xbar, Ctl& ctl, int C,
                         uint32_t rank, float x, float y) {
  const int buf = ctl.xbuf;
  for (int r = 0; r < C; ++r) {
    st_cluster_v2(map_shared(&slots[buf][rank], r), x, y);
    mbar_arrive_remote(map_shared(xbar, r));
  }
  const bool ok = mbar_wait_cluster(xbar, ctl.xphase);
  ctl.xphase ^= 1u;
  ctl.xbuf ^= 1;
  return ok;
}

// ------------------------------------------------------------- kernel -----

struct ConsumerCtx {
  int stage, phase;
};

template <typename L, int NCW>
__global__ void __launch_bounds__(NCW * 32 + 32, 16 / NCW) tv_tree_kernel(TravArgs args, int C,
                                                                      int n_stages) {
  constexpr int kConsumerWarps = NCW;
  constexpr int kConsumers = NCW * 32;
  constexpr int kThreads = kConsumers + 32;
  constexpr int kStageBytes = stage_bytes(NCW);
  constexpr int kSweep = kConsumers * kChunk;   // tokens one pass of all consumers covers
  extern __shared__ __align__(128) char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t xbar;
  __shared__ float2 xslots[2][kMaxCluster];
  __shared__ Ctl ctl;
  __shared__ float red_a[kConsumerWarps], red_b[kConsumerWarps];

  using E = typename L::elem;
  constexpr int kLB = L::kBytes;
  constexpr int kPairElems = kStageBytes / (kLB + 4) / kTileElems * kTileElems;  // target + draft
  constexpr int kRowElems = kStageBytes / kLB;               // target only per stage

  const int R = args.N + 1, V = args.V;
  const uint32_t rank = (C > 1) ? cluster_rank() : 0u;
  const int b = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const bool producer = (wid == kConsumerWarps);
  const float c_hi = args.c_hi, c_lo = args.c_lo;
  const int SL = slice_len(V, C);
  const int v0 = min((int)rank * SL, V);
  const int v1 = min(v0 + SL, V);
  const int nt = n_tiles(V, C);

  char* ring = smem_raw;
  TreeSmem s = carve_tree(smem_raw + (size_t)n_stages * kStageBytes, R, V, C);
  const E* logits = reinterpret_cast<const E*>(args.logits);
  const size_t tree_row0 = (size_t)b * R;
  const float* u = args.uniforms + (size_t)b * (R + 1);

  // ---- set-up: barriers, tree structure, validation, gathers ----
  if (tid == 0) {
    for (int k = 0; k < n_stages; ++k) {
      mbar_init(&full_bar[k], 1);
      mbar_init(&empty_bar[k], kConsumerWarps);
    }
    mbar_init(&xbar, C);
    fence_mbar_init();
    ctl.bad = 0u;
    ctl.accepted = -1;
    ctl.node = 0;
    ctl.pending = -1;
    ctl.masked_sum = 0.0;
    ctl.n_tests = ctl.n_passes = 0;
    ctl.xphase = 0u;
    ctl.xbuf = 0;
    ctl.job.kind = 0;
    ctl.bonus_y = -1;
  }
  for (int i = tid; i < R; i += kThreads) {
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
    s.rows[i] = 0.f;
    s.dbgp[i] = __int_as_float(0x7fc00000);
  }
  __syncthreads();
  {
    uint32_t bad = 0u;
    for (int i = tid; i < R; i += kThreads) {
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
    for (int i = tid; i < R; i += kThreads) {
      if (s.first[i] == 0x7fffffff) s.first[i] = -1;
      int nx = -1;
      if (i > 0) {
        const int p = s.par[i], t = s.tok[i];
        for (int j = i + 1; j < R; ++j) {
          if (s.par[j] != p) continue;
          if (nx < 0) nx = j;
          if (s.tok[j] == t) bad |= 4u;
        }
        const size_t prow = (tree_row0 + p) * (size_t)V;
        s.gl[i] = L::at(logits + prow, t);
        s.gq[i] = __ldg(args.draft_probs + prow + t);
        if (!(s.gq[i] > 0.f)) bad |= 8u;
        s.invq[i] = 1.0 / (double)s.gq[i];
      }
      s.next[i] = nx;
    }
    if (bad) atomicOr(&ctl.bad, bad);
  }
  __syncthreads();
  if (tid == 0) {
    if (ctl.bad == 0u) s.p[0] = 1.0;
    else ctl.job.kind = kJobDone;
  }
  if (C > 1) cluster_sync_all();   // peers' barriers initialised before any remote arrive
  else __syncthreads();

  uint32_t timeout = 0u;

  if (producer) {
    // =================== producer warp: TMA bulk copies ===================
    // One named barrier per job on every path (the consumers do the same).
    int stage = 0, phase = 0;
    for (;;) {
      named_sync(1, kThreads);             // the next job is posted
      const Job job = ctl.job;
      if (job.kind == kJobDone) break;
      if (timeout) continue;
      const bool pair = (job.kind == kJobPass || job.kind == kJobBonusRes);
      const int per = pair ? kPairElems : kRowElems;
      const int nrows = (job.kind == kJobStats) ? job.n_rows : 1;
      if (lane == 0) {
        for (int r = 0; r < nrows && !timeout; ++r) {
          const int node = (job.kind == kJobStats) ? s.job_rows[r] : job.node;
          const size_t row = (tree_row0 + node) * (size_t)V;
          for (int x = v0; x < v1; x += per) {
            const int n = min(per, v1 - x);
            if (!mbar_wait(&empty_bar[stage], phase ^ 1)) { timeout = 1u; break; }
            char* dst = ring + (size_t)stage * kStageBytes;
            const uint32_t lbytes = (uint32_t)n * kLB;
            const uint32_t qbytes = pair ? (uint32_t)n * 4u : 0u;
            mbar_arrive_expect_tx(&full_bar[stage], lbytes + qbytes);
            tma_load_1d(dst, logits + row + x, lbytes, &full_bar[stage]);
            if (pair)
              tma_load_1d(dst + (size_t)kPairElems * kLB, args.draft_probs + row + x, qbytes,
                          &full_bar[stage]);
            if (++stage == n_stages) { stage = 0; phase ^= 1; }
          }
        }
        if (timeout) atomicOr(&ctl.bad, 32u);
      }
      timeout = __shfl_sync(0xffffffffu, timeout, 0);
      stage = __shfl_sync(0xffffffffu, stage, 0);
      phase = __shfl_sync(0xffffffffu, phase, 0);
    }
  } else {
    // =================== consumer warps ===================
    int stage = 0, phase = 0;
    volatile uint32_t* vbad = &ctl.bad;
    for (;;) {
      if (tid == 0) {
        if (*vbad & (32u | 64u)) ctl.job.kind = kJobDone;         // timeout / unusable row
        else if (ctl.job.kind != kJobDone) advance(s, ctl, u, args.token_level != 0);
      }
      named_sync(1, kThreads);
      const Job job = ctl.job;
      if (job.kind == kJobDone) break;
      const bool pair = (job.kind == kJobPass || job.kind == kJobBonusRes);
      const int per = pair ? kPairElems : kRowElems;
      const int nrows = (job.kind == kJobStats) ? job.n_rows : 1;
      for (int r = 0; r < nrows; ++r) {
        const int node = (job.kind == kJobStats) ? s.job_rows[r] : job.node;
        float m_run = TV_NEG_INF;   // stats / leaf: running max
        Comp acc;
        int mp = 0;
        for (int x = v0; x < v1; x += per) {
          const int n = min(per, v1 - x);
          if ((*vbad & 32u) || !mbar_wait(&full_bar[stage], phase)) {
            atomicOr(&ctl.bad, 32u);
            break;
          }
          const char* buf = ring + (size_t)stage * kStageBytes;
          const E* lb = reinterpret_cast<const E*>(buf);
          const float* qb = reinterpret_cast<const float*>(buf + (size_t)kPairElems * kLB);
          // warp-uniform iteration over 256-element tiles (warp shuffles below)
          for (int t0 = wid * kTileElems; t0 < n; t0 += kSweep) {
            const int e0 = t0 + lane * kChunk;
            const bool valid = e0 < n;
            const int xg = x + e0;   // global token index of the lane's first element
            if constexpr (kLB == 2) {
              // ---------------- bf16 logits: packed-pair arithmetic ----------------
              float2 vp[4];
              if (valid) {
                bf16x8_pairs(lds128(lb + e0), vp);
              } else {
#pragma unroll
                for (int k2 = 0; k2 < 4; ++k2) vp[k2] = make_float2(-9984.f, -9984.f);
              }
              const float2 ch = make_float2(c_hi, c_hi), cl = make_float2(c_lo, c_lo);
              if (job.kind == kJobStats) {
                if (valid) {
                  const float cm = fmaxf(fmaxf(fmaxf(vp[0].x, vp[0].y), fmaxf(vp[1].x, vp[1].y)),
                                         fmaxf(fmaxf(vp[2].x, vp[2].y), fmaxf(vp[3].x, vp[3].y)));
                  if (cm > m_run) {
                    if (m_run != TV_NEG_INF) {
                      const float sc = L::exp_rel(m_run, cm, c_hi, c_lo);
                      acc.s *= sc;
                      acc.c *= sc;
                    }
                    m_run = cm;
                  }
                  const float2 mm = make_float2(-m_run, -m_run);
                  float2 e[4];
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2) e[k2] = exp2_split_x2(__fadd2_rn(vp[k2], mm), ch, cl);
                  const float2 s2 = __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3]));
                  acc.add(s2.x + s2.y);
                }
              } else if (job.kind == kJobBonusLeaf) {
                const float lm = fmaxf(fmaxf(fmaxf(vp[0].x, vp[0].y), fmaxf(vp[1].x, vp[1].y)),
                                       fmaxf(fmaxf(vp[2].x, vp[2].y), fmaxf(vp[3].x, vp[3].y)));
                const float tm = warp_max(lm);
                const float2 mm = make_float2(-tm, -tm);
                float2 e[4];
#pragma unroll
                for (int k2 = 0; k2 < 4; ++k2) e[k2] = exp2_corrected_x2(__fadd2_rn(vp[k2], mm), ch, cl);
                const float2 s2 = __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3]));
                const float ts = warp_sum(valid ? s2.x + s2.y : 0.f);
                if (lane == 0) {
                  const int tile = (x + t0 - v0) / kTileElems;
                  s.tsum[tile] = ts;
                  s.tmax[tile] = tm;
                }
              } else {
                float2 qp[4];
                if (valid) {
                  const uint4 qa = lds128(qb + e0);
                  const uint4 qc = lds128(qb + e0 + 4);
                  qp[0] = make_float2(__uint_as_float(qa.x), __uint_as_float(qa.y));
                  qp[1] = make_float2(__uint_as_float(qa.z), __uint_as_float(qa.w));
                  qp[2] = make_float2(__uint_as_float(qc.x), __uint_as_float(qc.y));
                  qp[3] = make_float2(__uint_as_float(qc.z), __uint_as_float(qc.w));
                } else {
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2) qp[k2] = make_float2(0.f, 0.f);
                }
                const float2 mm = make_float2(-job.rowmax, -job.rowmax);
                const float2 al2 = make_float2(job.alpha1, job.alpha1);
                const float2 nb2 = make_float2(-job.beta, -job.beta);
                float t[8];
#pragma unroll
                for (int k2 = 0; k2 < 4; ++k2) {
                  const float2 e = exp2_corrected_x2(__fadd2_rn(vp[k2], mm), ch, cl);
                  const float2 xx = __ffma2_rn(al2, e, __fmul2_rn(nb2, qp[k2]));
                  t[2 * k2] = fmaxf(xx.x, 0.f);
                  t[2 * k2 + 1] = fmaxf(xx.y, 0.f);
                }
                while (mp < job.nmask && s.mask_tok[mp] < xg) ++mp;
                for (int mq = mp; mq < job.nmask && s.mask_tok[mq] < xg + kChunk; ++mq) {
                  const int off = s.mask_tok[mq] - xg;
                  const float mv = (job.kind == kJobPass) ? 0.f : s.mask_val[mq];
#pragma unroll
                  for (int k2 = 0; k2 < 8; ++k2) if (k2 == off) t[k2] = mv;
                }
                if (job.kind == kJobPass) {
                  if (valid) acc.add(sum8(t));
                } else {
                  const float ts = warp_sum(valid ? sum8(t) : 0.f);
                  if (lane == 0) s.tsum[(x + t0 - v0) / kTileElems] = ts;
                }
              }
            } else {
            float v[8];
            if (!valid) {
#pragma unroll
              for (int k2 = 0; k2 < 8; ++k2) v[k2] = TV_NEG_INF;
            } else {
              const uint4 a4 = lds128(lb + e0);
              const uint4 b4 = lds128(lb + e0 + 4);
              v[0] = __uint_as_float(a4.x); v[1] = __uint_as_float(a4.y);
              v[2] = __uint_as_float(a4.z); v[3] = __uint_as_float(a4.w);
              v[4] = __uint_as_float(b4.x); v[5] = __uint_as_float(b4.y);
              v[6] = __uint_as_float(b4.z); v[7] = __uint_as_float(b4.w);
            }
            if (job.kind == kJobStats) {
              float cm = fmaxf(fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3])),
                               fmaxf(fmaxf(v[4], v[5]), fmaxf(v[6], v[7])));
              if (cm > m_run) {
                if (m_run != TV_NEG_INF) {
                  const float sc = L::exp_rel(m_run, cm, c_hi, c_lo);
                  acc.s *= sc;
                  acc.c *= sc;
                }
                m_run = cm;
              }
              float t[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) t[k] = L::exp_rel(v[k], m_run, c_hi, c_lo);
              acc.add(sum8(t));
            } else if (job.kind == kJobBonusLeaf) {
              float lm = fmaxf(fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3])),
                               fmaxf(fmaxf(v[4], v[5]), fmaxf(v[6], v[7])));
              const float tm = warp_max(lm);
              float t[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) t[k] = L::exp_pass(v[k], tm, c_hi, c_lo);
              const float ts = warp_sum(sum8(t));
              if (lane == 0) {
                const int tile = (x + t0 - v0) / kTileElems;
                s.tsum[tile] = ts;
                s.tmax[tile] = tm;
              }
            } else {
              float q[8];
              if (valid) {
                const uint4 qa = lds128(qb + e0);
                const uint4 qc = lds128(qb + e0 + 4);
                q[0] = __uint_as_float(qa.x); q[1] = __uint_as_float(qa.y);
                q[2] = __uint_as_float(qa.z); q[3] = __uint_as_float(qa.w);
                q[4] = __uint_as_float(qc.x); q[5] = __uint_as_float(qc.y);
                q[6] = __uint_as_float(qc.z); q[7] = __uint_as_float(qc.w);
              } else {
#pragma unroll
                for (int k2 = 0; k2 < 8; ++k2) q[k2] = 0.f;
              }
              const float al = job.alpha1, be = job.beta, rm = job.rowmax;
              float t[8];
#pragma unroll
              for (int k = 0; k < 8; ++k)
                t[k] = fmaxf(fmaf(al, L::exp_pass(v[k], rm, c_hi, c_lo), -be * q[k]), 0.f);
              while (mp < job.nmask && s.mask_tok[mp] < xg) ++mp;
              for (int mq = mp; mq < job.nmask && s.mask_tok[mq] < xg + kChunk; ++mq) {
                const int off = s.mask_tok[mq] - xg;
                const float mv = (job.kind == kJobPass) ? 0.f : s.mask_val[mq];
#pragma unroll
                for (int k = 0; k < 8; ++k) if (k == off) t[k] = mv;
              }
              if (job.kind == kJobPass) {
                acc.add(sum8(t));
              } else {
                const float ts = warp_sum(sum8(t));
                if (lane == 0) s.tsum[(x + t0 - v0) / kTileElems] = ts;
              }
            }
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&empty_bar[stage]);
          if (++stage == n_stages) { stage = 0; phase ^= 1; }
        }
        // ---- per-row reduction over the consumers, then over the cluster ----
        if (job.kind == kJobStats) {
          const float wm = warp_max(m_run);
          if (lane == 0) red_a[wid] = wm;
          named_sync(2, kConsumers);
          float M = red_a[0];
#pragma unroll
          for (int w = 1; w < kConsumerWarps; ++w) M = fmaxf(M, red_a[w]);
          float part = (m_run == TV_NEG_INF) ? 0.f : acc.value() * L::exp_rel(m_run, M, c_hi, c_lo);
          part = warp_sum(part);
          named_sync(2, kConsumers);
          if (lane == 0) red_b[wid] = part;
          named_sync(2, kConsumers);
          if (tid == 0) {
            float S = 0.f;
            for (int w = 0; w < kConsumerWarps; ++w) S += red_b[w];
            if (C > 1) {
              if (!exchange(xslots, &xbar, ctl, C, rank, M, S)) atomicOr(&ctl.bad, 32u);
              const int bb = ctl.xbuf ^ 1;
              float Mg = xslots[bb][0].x;
              for (int rr = 1; rr < C; ++rr) Mg = fmaxf(Mg, xslots[bb][rr].x);
              float Sg = 0.f;
              for (int rr = 0; rr < C; ++rr) {
                const float mr = xslots[bb][rr].x;
                if (mr != TV_NEG_INF) Sg += xslots[bb][rr].y * L::exp_rel(mr, Mg, c_hi, c_lo);
              }
              M = Mg;
              S = Sg;
            }
            s.rowm[node] = M;
            s.rows[node] = S;
            s.invs[node] = 1.0 / (double)S;
            if (!(S > 0.f)) ctl.bad |= 64u;   // no finite logit in the row
          }
          __syncwarp();
          if (wid == 0) {
            children_mb0(s, node, args.c, lane);
            __syncwarp();
          }
        } else if (job.kind == kJobPass) {
          const float ws = warp_sum(acc.value());
          if (lane == 0) red_a[wid] = ws;
          named_sync(2, kConsumers);
          if (tid == 0) {
            float S = 0.f;
            for (int w = 0; w < kConsumerWarps; ++w) S += red_a[w];
            if (C > 1) {
              if (!exchange(xslots, &xbar, ctl, C, rank, S, 0.f)) atomicOr(&ctl.bad, 32u);
              const int bb = ctl.xbuf ^ 1;
              float Sg = 0.f;
              for (int rr = 0; rr < C; ++rr) Sg += xslots[bb][rr].x;
              S = Sg;
            }
            ctl.S = S;
          }
        } else {
          // ---- bonus draw: slice totals, crossing slice, crossing tile, token ----
          named_sync(2, kConsumers);
          if (wid == 0) {
            const bool leaf = (job.kind == kJobBonusLeaf);
            const int ntl = (v1 - v0 + kTileElems - 1) / kTileElems;
            float Mc = 0.f;
            if (leaf) {
              float lm = TV_NEG_INF;
              for (int k = lane; k < ntl; k += 32) lm = fmaxf(lm, s.tmax[k]);
              Mc = warp_max(lm);
              for (int k = lane; k < ntl; k += 32)
                s.tsum[k] = (s.tmax[k] == TV_NEG_INF) ? 0.f : s.tsum[k] * L::exp_rel(s.tmax[k], Mc, c_hi, c_lo);
              __syncwarp();
            }
            float Wc = 0.f;
            for (int k0 = 0; k0 < ntl; k0 += 32) {
              const float v = (k0 + lane < ntl) ? s.tsum[k0 + lane] : 0.f;
              Wc += warp_sum(v);
            }
            // cluster: every CTA learns every slice's (max, total)
            float scale = 1.f, target = 0.f, before = 0.f, Wtot = 0.f;
            int owner = 0;
            if (lane == 0) {
              float Mg = Mc, W = Wc;
              if (C > 1) {
                if (!exchange(xslots, &xbar, ctl, C, rank, Mc, Wc)) atomicOr(&ctl.bad, 32u);
                const int bb = ctl.xbuf ^ 1;
                Mg = xslots[bb][0].x;
                if (leaf) for (int rr = 1; rr < C; ++rr) Mg = fmaxf(Mg, xslots[bb][rr].x);
                W = 0.f;
                float sc[kMaxCluster];
                for (int rr = 0; rr < C; ++rr) {
                  sc[rr] = leaf ? ((xslots[bb][rr].x == TV_NEG_INF) ? 0.f
                                       : L::exp_rel(xslots[bb][rr].x, Mg, c_hi, c_lo))
                                : 1.f;
                  W += xslots[bb][rr].y * sc[rr];
                }
                target = u[R] * W;
                float acc0 = 0.f;
                owner = -1;
                for (int rr = 0; rr < C; ++rr) {
                  const float wr = xslots[bb][rr].y * sc[rr];
                  if (owner < 0 && target < acc0 + wr) { owner = rr; before = acc0; }
                  acc0 += wr;
                }
                if (owner < 0) {   // rounding: the last slice with weight
                  owner = C - 1;
                  while (owner > 0 && !(xslots[bb][owner].y > 0.f)) --owner;
                  before = 0.f;
                  for (int rr = 0; rr < owner; ++rr) before += xslots[bb][rr].y * sc[rr];
                }
                scale = sc[rank];
              } else {
                target = u[R] * W;
              }
              (void)Mg;
              Wtot = W;
            }
            owner = __shfl_sync(0xffffffffu, owner, 0);
            if ((uint32_t)owner == rank) {
              target = __shfl_sync(0xffffffffu, target, 0);
              before = __shfl_sync(0xffffffffu, before, 0);
              scale = __shfl_sync(0xffffffffu, scale, 0);
              Wtot = __shfl_sync(0xffffffffu, Wtot, 0);
              // local target in this slice's units
              const float lt = (scale > 0.f) ? (target - before) / scale : 0.f;
              int tile = -1;
              float tbase = 0.f, base = 0.f;
              for (int k0 = 0; k0 < ntl && tile < 0; k0 += 32) {
                float v = (k0 + lane < ntl) ? s.tsum[k0 + lane] : 0.f;
                const float own = v;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                  const float w2 = __shfl_up_sync(0xffffffffu, v, o);
                  if (lane >= o) v += w2;
                }
                const unsigned hit = __ballot_sync(0xffffffffu, (k0 + lane < ntl) && (lt < base + v));
                if (hit) {
                  const int l = __ffs(hit) - 1;
                  tile = k0 + l;
                  tbase = base + __shfl_sync(0xffffffffu, v - own, l);
                }
                base += __shfl_sync(0xffffffffu, v, 31);
              }
              if (tile < 0) {
                tile = ntl - 1;
                while (tile > 0 && !(s.tsum[tile] > 0.f)) --tile;
                float a0 = 0.f;
                for (int k = 0; k < tile; ++k) a0 += s.tsum[k];
                tbase = a0;
              }
              // element-level rescan of the crossing tile (global loads, L2-hot)
              const int x0 = v0 + tile * kTileElems + lane * kChunk;
              const size_t row = (tree_row0 + node) * (size_t)V;
              float w[8];
              if (leaf) {
                float v[8];
                if (x0 < v1) load_logits<L, true>(logits + row, x0, V, v);
                else {
#pragma unroll
                  for (int e = 0; e < 8; ++e) v[e] = TV_NEG_INF;
                }
#pragma unroll
                for (int e = 0; e < 8; ++e)
                  w[e] = (v[e] == TV_NEG_INF) ? 0.f : L::exp_pass(v[e], Mc, c_hi, c_lo);
              } else {
                float v[8], q[8];
                if (x0 < v1) {
                  load_logits<L, true>(logits + row, x0, V, v);
                  load_probs<true>(args.draft_probs + row, x0, V, q);
                } else {
#pragma unroll
                  for (int e = 0; e < 8; ++e) { v[e] = TV_NEG_INF; q[e] = 0.f; }
                }
#pragma unroll
                for (int e = 0; e < 8; ++e)
                  w[e] = (v[e] == TV_NEG_INF) ? 0.f
                         : fmaxf(fmaf(job.alpha1, L::exp_pass(v[e], job.rowmax, c_hi, c_lo), -job.beta * q[e]), 0.f);
                for (int mq = 0; mq < job.nmask; ++mq) {
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
                const float w2 = __shfl_up_sync(0xffffffffu, v, o);
                if (lane >= o) v += w2;
              }
              const float lbase = tbase + (v - run);
              int found = 8;
#pragma unroll
              for (int e = 7; e >= 0; --e) if (lt < lbase + pre[e]) found = e;
              const unsigned hit = __ballot_sync(0xffffffffu, found < 8);
              // the draw's margin (kernel sums), in this slice's units, then
              // relative to the total
              float clo = lbase, chi = lbase;
#pragma unroll
              for (int e = 0; e < 8; ++e) {
                if (e == found) chi = lbase + pre[e];
                if (e + 1 == found) clo = lbase + pre[e];
              }
              const float my_margin = fminf(lt - clo, chi - lt) * scale / Wtot;
              int yy;
              float bm = 0.f;
              if (hit) {
                const int l = __ffs(hit) - 1;
                yy = x0 - lane * kChunk + l * kChunk + __shfl_sync(0xffffffffu, found, l);
                bm = __shfl_sync(0xffffffffu, my_margin, l);
              } else {
                int last = -1;
#pragma unroll
                for (int e = 0; e < 8; ++e) if (w[e] > 0.f) last = x0 + e;
                const unsigned any = __ballot_sync(0xffffffffu, last >= 0);
                yy = any ? __shfl_sync(0xffffffffu, last, 31 - __clz(any)) : v1 - 1;
              }
              if (lane == 0) {
                args.out_bonus[b] = yy;
                if (args.out_margin) args.out_margin[2 * (size_t)b + 1] = bm;
              }
            }
          }
          if (tid == 0) ctl.job.kind = kJobDone;   // the bonus ends the traversal
        }
      }
    }
    // ---- outputs (rank 0) ----
    named_sync(2, kConsumers);
    if (rank == 0) {
      const bool ok = (ctl.bad & (15u | 32u | 64u)) == 0u;
      const int N = args.N;
      for (int k = tid; k < N; k += kConsumers) args.out_path[(size_t)b * N + k] = -1;
      if (args.out_node_p)
        for (int i = tid; i < R; i += kConsumers)
          args.out_node_p[tree_row0 + i] = ok ? s.dbgp[i] : __int_as_float(0x7fc00000);
      named_sync(2, kConsumers);
      if (tid == 0) {
        const int acc_node = ok ? ctl.accepted : -1;
        if (acc_node >= 0) {
          int depth = 0;
          for (int j = acc_node; j != 0; j = s.par[j]) ++depth;
          int k = depth - 1;
          for (int j = acc_node; j != 0; j = s.par[j]) args.out_path[(size_t)b * N + (k--)] = j;
          args.out_accept_len[b] = depth;
        } else {
          args.out_accept_len[b] = -1;
          args.out_bonus[b] = -1;
        }
        if (args.out_stats) {
          int distinct = 0;
          for (int i = 0; i < R; ++i) distinct += (s.npass[i] > 0);
          int normalised = 0;
          for (int i = 0; i < R; ++i) normalised += (s.rows[i] > 0.f);
          int32_t* o = args.out_stats + (size_t)b * 5;
          o[0] = ok ? ctl.n_tests : 0;
          o[1] = ok ? ctl.n_passes : 0;
          o[2] = ok ? distinct : 0;
          o[3] = (acc_node >= 0 && s.first[acc_node] < 0) ? 1 : 0;
          o[4] = ok ? normalised : 0;
        }
        if (args.out_margin) {
          // the bonus margin was written by the CTA that drew the bonus
          const float nan = __int_as_float(0x7fc00000);
          args.out_margin[2 * (size_t)b] = acc_node >= 0 ? test_margin_serial(s.dbgp, u, R) : nan;
          if (acc_node < 0) args.out_margin[2 * (size_t)b + 1] = nan;
        }
        if (ctl.bad) atomicOr(args.status, ctl.bad);
      }
    }
  }
  if (C > 1) cluster_sync_all();   // no CTA leaves while a peer may still write to it
}

}  // namespace fused
}  // namespace tvk

// --------------------------------------------------------------- launcher --

namespace {

// Ring stages that fit when `per_sm` CTAs share an SM's shared memory.
int stages_for(int ncw, int per_sm, size_t tree, int smem_per_sm, int smem_per_block) {
  using namespace tvk::fused;
  const long reserve = 1024 + 512;   // per-CTA system reserve and static shared memory
  long per_cta = (long)smem_per_sm / per_sm - reserve;
  if (per_cta > smem_per_block) per_cta = smem_per_block;
  const long st = (per_cta - (long)tree) / stage_bytes(ncw);
  return (int)(st > kMaxStages ? kMaxStages : st);
}

}  // namespace

FusedPlan tv_fused_plan(int B, int R, int V, int sm_count, int smem_per_sm, int smem_per_block,
                        int force_ncw, int force_c, int force_stages) {
  using namespace tvk::fused;
  FusedPlan p;
  // Large batches fill the GPU with one CTA of 8 consumer warps per tree; smaller
  // ones use CTAs of 4 consumer warps (four per SM) and clusters that split a
  // tree's vocabulary across up to 8 SMs, as many as fit in one wave, keeping
  // every CTA's slice at least 2048 tokens.
  int ncw = (B >= 2 * sm_count) ? 8 : 4;
  if (force_ncw == 4 || force_ncw == 8) ncw = force_ncw;
  int per_sm = 16 / ncw;
  int C = 1;
  while (C < kMaxCluster && (long)B * (2 * C) <= (long)sm_count * per_sm &&
         V / (2 * C) >= 2048)
    C *= 2;
  if (force_c == 1 || force_c == 2 || force_c == 4 || force_c == 8) C = force_c;
  const size_t tree = tree_smem_bytes(R, V, C);
  int stages = stages_for(ncw, per_sm, tree, smem_per_sm, smem_per_block);
  while (stages < 3 && per_sm > 1) {
    --per_sm;
    stages = stages_for(ncw, per_sm, tree, smem_per_sm, smem_per_block);
  }
  if (force_stages >= 2 && force_stages <= kMaxStages && force_stages < stages) stages = force_stages;
  p.ncw = ncw;
  p.C = C;
  p.stages = stages;
  p.smem = (size_t)stages * stage_bytes(ncw) + tree;
  p.ok = stages >= 2 && p.smem <= (size_t)smem_per_block;
  return p;
}

namespace {

template <typename L, int NCW>
cudaError_t launch_one(const TravArgs& a, const FusedPlan& plan, cudaStream_t stream) {
  auto k = tvk::fused::tv_tree_kernel<L, NCW>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(a.B * plan.C), 1, 1);
  cfg.blockDim = dim3(NCW * 32 + 32, 1, 1);
  cfg.dynamicSmemBytes = plan.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)plan.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = (plan.C > 1) ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k, a, plan.C, plan.stages);
}

}  // namespace

int tv_launch_fused(const TravArgs& a, int logit_is_bf16, const FusedPlan& plan,
                    cudaStream_t stream, cudaEvent_t* ev) {
  if (!plan.ok) return -3;
  if (ev) {
    for (int k = 0; k < 3; ++k)
      if (cudaEventRecord(ev[k], stream) != cudaSuccess) return -5;
  }
  cudaError_t e;
  if (logit_is_bf16)
    e = plan.ncw == 8 ? launch_one<tvk::Bf16Logits, 8>(a, plan, stream)
                      : launch_one<tvk::Bf16Logits, 4>(a, plan, stream);
  else
    e = plan.ncw == 8 ? launch_one<tvk::F32Logits, 8>(a, plan, stream)
                      : launch_one<tvk::F32Logits, 4>(a, plan, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return -5;
  }
  if (ev && cudaEventRecord(ev[3], stream) != cudaSuccess) return -5;
  return 0;
}
