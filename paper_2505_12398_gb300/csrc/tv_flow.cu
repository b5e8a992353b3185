// tv_flow.cu -- persistent, load-balanced Traversal Verification (sm_103a).
//
// The per-tree traversal of Algorithm 3 (§3.1) is serial, and trees differ a
// lot in how many vocabulary passes they need, so a fixed assignment of SMs to
// trees leaves most of the GPU idle while the slowest trees finish.  Here
// every tree has an owner CTA that keeps the tree's state in shared memory
// and runs its serial control (tv_control.cuh), but the vocabulary work of
// each job -- row normalisers, a rejection pass, the bonus draw -- is cut into
// slices that are published to a global work queue and processed by whichever
// CTA holds the slot's ticket.  The owner combines the slices' partial results
// in a fixed order (results do not depend on which CTA did what) and advances
// its tree.  The kernel's time is then set by the slowest tree's chain of
// jobs, each taking a few microseconds, instead of by its total bytes.
//
// One cooperative launch keeps all CTAs resident, so CTAs may wait on work
// published by others; every wait is bounded, and a global abort flag ends
// the kernel cleanly if one ever gives up.  Inside a CTA, a producer warp
// streams a slice into a shared-memory ring with 1-D bulk copies (TMA) and
// four consumer warps reduce it.
//
// Queue protocol: a poster reserves a range of slots with one atomicAdd on
// the tail, writes the slots' bodies, fences, then stores each slot's tag
// (call epoch, slot number).  A CTA takes a ticket -- the next slot number,
// one atomicAdd on the head -- and processes that slot once its tag appears,
// doing its own tree's work meanwhile.  Slots are never reused within a call
// (the queue holds every item the call can post), so a ticket past the last
// item just waits for the end of the call.  Polls are relaxed loads issued
// together; a positive poll is followed by one acquire fence.
#include <cuda_runtime.h>
#include <stdint.h>

#include "tv_control.cuh"
#include "tv_device.cuh"
#include "tv_launch.h"
#include "tv_ptx.cuh"

namespace tvk {
namespace flow {

using namespace tvk::fused;

constexpr int kMaxNCW = 8;
constexpr int kPBuf = 256;          // partials of a job kept in shared memory by the poll
constexpr unsigned long long kNoPart = ~0ull;   // a partial slot not written yet
constexpr unsigned kNoTicket = 0xffffffffu;
constexpr unsigned long long kExitTag = 0x80000000ull;   // tag bit: no more items, exit
constexpr int kMaxGrid = 4096;      // tickets taken past the last item: one per CTA at most
constexpr unsigned long long kIdleNs = 2000000000ull;   // 2 s without progress: abort

enum : int { kActIdle = 0, kActItem = 1, kActCombine = 2, kActNewTree = 3, kActExit = 4 };
enum : int {
  kCtrTail = 0, kCtrHead = 1, kCtrDone = 2, kCtrNextTree = 3, kCtrAbort = 4, kCtrExit = 5,
  kNumCtr = 6
};

struct Shared {
  int act;
  int my_tree;          // tree owned by this CTA (-1: none)
  int outstanding;      // items of the own tree's current job (0: none)
  unsigned ticket;      // queue slot this CTA processes next (kNoTicket: none)
  int jkind, jrows, jK, jslice;   // own tree's current job, for the combine
  int4 it[3];           // body of the item being processed
  int trees_left;       // the next-tree counter may still be below B
  Ctl ctl;              // serial control state of the own tree
  float red_a[kMaxNCW], red_b[kMaxNCW];
  float out_x, out_y;   // partial result of the item
  float2 pbuf[kPBuf];   // the own job's partials, as read by the poll
};

__device__ __forceinline__ unsigned ld_relaxed_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_relaxed_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned long long pack_part(float x, float y) {
  unsigned long long v = ((unsigned long long)__float_as_uint(y) << 32) | __float_as_uint(x);
  return (v == kNoPart) ? (v & 0x7fffffffffffffffull) : v;   // never the "not yet" pattern
}

__device__ __forceinline__ float2 unpack_part(unsigned long long v) {
  return make_float2(__uint_as_float((unsigned)v), __uint_as_float((unsigned)(v >> 32)));
}

__device__ __forceinline__ void fence_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Ends the whole kernel cleanly: every CTA sees the flag at its next decision.
__device__ __forceinline__ void raise_abort(const TravArgs& a, const FlowArgs& f) {
  atomicOr(a.status, 32u);
  atomicExch(&f.ctr[kCtrAbort], 1u);
}

// --------------------------------------------------------------- posting --

// Publishes the own tree's current job (ctl.job) as slice items; warp 0.
__device__ void post_job(const TreeSmem& s, Shared& sh, const TravArgs& a, const FlowArgs& f,
                         int b, int V, int lane) {
  const Job& j = sh.ctl.job;
  const bool stats = (j.kind == kJobStats);
  const int n_rows = stats ? j.n_rows : 1;
  const int slice = stats ? f.slice_stats : f.slice_pass;
  const int K = (V + slice - 1) / slice;
  const int nmask = (j.kind == kJobPass || j.kind == kJobBonusRes) ? j.nmask : 0;
  const int n = n_rows * K;
  const size_t R = (size_t)f.R;
  for (int q = lane; q < nmask; q += 32) {
    f.job_mtok[b * R + q] = s.mask_tok[q];
    f.job_mval[b * R + q] = s.mask_val[q];
  }
  unsigned base = 0u;
  if (lane == 0) base = atomicAdd(&f.ctr[kCtrTail], (unsigned)n);
  base = __shfl_sync(0xffffffffu, base, 0);
  // the last kMaxGrid slots are kept for exit tags; a correctly sized queue
  // never reaches them
  if ((size_t)base + n + kMaxGrid > (size_t)f.cap) {
    if (lane == 0) raise_abort(a, f);
    return;
  }
  // the job's partial slots start as "not yet"
  for (int q = lane; q < n; q += 32) {
    const int r = q / K;
    __stcg(f.part + ((size_t)b * R + r) * f.Kmax + (q - r * K), kNoPart);
  }
  const int4 w1 = make_int4(j.kind, slice, nmask, 0);
  const int4 w2 = make_int4(__float_as_int(j.alpha1), __float_as_int(j.beta),
                            __float_as_int(j.rowmax), 0);
  for (int q = lane; q < n; q += 32) {
    const int r = q / K;
    int4* w = reinterpret_cast<int4*>(f.items + base + q);
    __stcg(w, make_int4(b, stats ? s.job_rows[r] : j.node, r, q - r * K));
    __stcg(w + 1, w1);
    __stcg(w + 2, w2);
  }
  fence_gpu();   // bodies, masks and partial resets before tags
  __syncwarp();
  for (int q = lane; q < n; q += 32)
    st_relaxed_u64(&f.items[base + q].tag, (f.epoch << 32) | (unsigned long long)(base + q));
  if (lane == 0) {
    sh.outstanding = n;
    sh.jkind = j.kind;
    sh.jrows = n_rows;
    sh.jK = K;
    sh.jslice = slice;
  }
}

// ------------------------------------------------------------- the kernel --

template <typename L, int kNCW>
__global__ void __launch_bounds__(kNCW * 32 + 32, 16 / kNCW)
    tv_flow_kernel(TravArgs args, FlowArgs f, int n_stages) {
  extern __shared__ __align__(128) char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ Shared sh;

  using E = typename L::elem;
  constexpr int kConsumers = kNCW * 32;
  constexpr int kThreads = kConsumers + 32;
  constexpr int kWarps = kThreads / 32;
  constexpr int kStageBytes = stage_bytes(kNCW);
  constexpr int kSweep = kConsumers * kChunk;
  constexpr int kLB = L::kBytes;
  constexpr int kPairElems = kStageBytes / (kLB + 4) / kTileElems * kTileElems;
  constexpr int kRowElems = kStageBytes / kLB;

  const int R = args.N + 1, V = args.V, B = args.B;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const bool producer = (wid == kNCW);
  const float c_hi = args.c_hi, c_lo = args.c_lo;
  char* ring = smem_raw;
  TreeSmem s = carve_tree_nt(smem_raw + (size_t)n_stages * kStageBytes, R, 0);
  int* it_mtok = reinterpret_cast<int*>(smem_raw + (size_t)n_stages * kStageBytes +
                                        ((tree_smem_bytes_nt(R, 0) + 15) & ~(size_t)15));
  float* it_mval = reinterpret_cast<float*>(it_mtok + R);
  const E* logits = reinterpret_cast<const E*>(args.logits);
  // with fewer trees than half the CTAs, owners leave the slices to CTAs
  // without a tree so that their own combines are never delayed
  const bool owners_serve = 2 * B >= (int)gridDim.x;

  if (tid == 0) {
    for (int k = 0; k < n_stages; ++k) {
      mbar_init(&full_bar[k], 1);
      mbar_init(&empty_bar[k], kNCW);
    }
    fence_mbar_init();
    sh.my_tree = -1;
    sh.outstanding = 0;
    sh.ticket = kNoTicket;
    sh.trees_left = 1;
  }
  __syncthreads();

  int stage = 0, phase = 0;   // ring position (producer and consumers alike)
  unsigned long long idle_since = 0ull;
  unsigned polls = 0u, nap = 32u;
  for (;;) {
    // ---------------- warp 0 decides what this CTA does next ----------------
    if (wid == 0) {
      const int mt = sh.my_tree;
      // the own job is finished when none of its partial slots is "not yet";
      // the lanes poll them, keeping what they read for the combine
      bool job_done = false;
      const int nout = sh.outstanding;
      if (mt >= 0 && nout > 0) {
        const int K = sh.jK;
        bool all = true;
        for (int q = lane; q < nout; q += 32) {
          const int r = q / K;
          const unsigned long long v =
              ld_relaxed_u64(f.part + ((size_t)mt * R + r) * f.Kmax + (q - r * K));
          if (v == kNoPart) all = false;
          else if (q < kPBuf) sh.pbuf[q] = unpack_part(v);
        }
        job_done = __all_sync(0xffffffffu, all);
      }
      if (lane == 0) {
        // Polls touch only this CTA's ticket slot and its own tree's partials;
        // the shared abort flag is read every 32nd round, the shared counters
        // only when about to take a new tree or ticket.
        int act = kActIdle;
        const unsigned h = sh.ticket;
        const unsigned long long want = (f.epoch << 32) | (unsigned long long)h;
        const unsigned long long tag =
            (h < (unsigned)f.cap) ? ld_relaxed_u64(&f.items[h].tag) : 0ull;
        const unsigned abort_f = ((++polls & 31u) == 0u) ? ld_relaxed_u32(&f.ctr[kCtrAbort]) : 0u;
        if (abort_f) {
          act = kActExit;
        } else if (job_done) {
          // the bonus draw reads tiles written before its partials
          if (sh.jkind == kJobBonusLeaf || sh.jkind == kJobBonusRes) fence_gpu();
          act = kActCombine;
        } else if (h < (unsigned)f.cap && tag == want) {
          fence_gpu();
          const int4* bp = reinterpret_cast<const int4*>(f.items + h);
          sh.it[0] = __ldcg(bp);
          sh.it[1] = __ldcg(bp + 1);
          sh.it[2] = __ldcg(bp + 2);
          sh.ticket = kNoTicket;
          act = kActItem;
        } else if (h < (unsigned)f.cap && tag == (want | kExitTag)) {
          act = kActExit;   // every tree is done
        } else {
          if (mt < 0 && sh.trees_left) {
            if (ld_relaxed_u32(&f.ctr[kCtrNextTree]) < (unsigned)B) {
              const unsigned t = atomicAdd(&f.ctr[kCtrNextTree], 1u);
              if (t < (unsigned)B) {
                sh.my_tree = (int)t;
                act = kActNewTree;
              } else {
                sh.trees_left = 0;
              }
            } else {
              sh.trees_left = 0;
            }
          }
          if (act == kActIdle && h == kNoTicket && (mt < 0 || owners_serve)) {
            if (ld_relaxed_u32(&f.ctr[kCtrDone]) >= (unsigned)B)
              act = kActExit;   // nothing will be posted any more
            else
              sh.ticket = atomicAdd(&f.ctr[kCtrHead], 1u);   // polled from the next round on
          }
        }
        if (act == kActIdle) {
          const unsigned long long now = global_ns();
          if (idle_since == 0ull) {
            idle_since = now;
          } else if (now - idle_since > kIdleNs) {   // no progress for seconds: give up cleanly
            raise_abort(args, f);
            act = kActExit;
          }
          if (act == kActIdle) {
            __nanosleep(nap);
            if (nap < 256u) nap <<= 1;
          }
        } else {
          idle_since = 0ull;
          nap = 32u;
        }
        sh.act = act;
      }
    }
    named_sync(1, kThreads);
    const int act = sh.act;
    if (act == kActExit) break;
    if (act == kActIdle) continue;

    if (act == kActItem) {
      // ---------------- one slice of some tree's job ----------------
      const int b = sh.it[0].x, node = sh.it[0].y, item_row = sh.it[0].z, item_slice = sh.it[0].w;
      const int kind = sh.it[1].x, slice_len = sh.it[1].y, nmask = sh.it[1].z;
      const float alpha1 = __int_as_float(sh.it[2].x);
      const float beta = __int_as_float(sh.it[2].y);
      const float rowmax = __int_as_float(sh.it[2].z);
      const int x0 = item_slice * slice_len;
      const int x1 = min(V, x0 + slice_len);
      const size_t row = ((size_t)b * R + node) * (size_t)V;
      const bool pair = (kind == kJobPass || kind == kJobBonusRes);
      const int per = pair ? kPairElems : kRowElems;
      for (int q = tid; q < nmask; q += kThreads) {
        it_mtok[q] = __ldcg(f.job_mtok + (size_t)b * R + q);
        it_mval[q] = __ldcg(f.job_mval + (size_t)b * R + q);
      }
      __syncthreads();
      if (producer) {
        if (lane == 0) {
          for (int x = x0; x < x1; x += per) {
            const int n = min(per, x1 - x);
            if (!mbar_wait(&empty_bar[stage], phase ^ 1)) {
              raise_abort(args, f);
              break;
            }
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
        stage = __shfl_sync(0xffffffffu, stage, 0);
        phase = __shfl_sync(0xffffffffu, phase, 0);
      } else {
        float m_run = TV_NEG_INF;
        Comp acc;
        int mp = 0;
        const float2 ch = make_float2(c_hi, c_hi), cl = make_float2(c_lo, c_lo);
        bool fail = false;
        for (int x = x0; x < x1; x += per) {
          const int n = min(per, x1 - x);
          // every issued copy is waited for (bounded), even after a failure
          if (!mbar_wait(&full_bar[stage], phase)) fail = true;
          if (!fail) {
            const char* buf = ring + (size_t)stage * kStageBytes;
            const E* lb = reinterpret_cast<const E*>(buf);
            const float* qb = reinterpret_cast<const float*>(buf + (size_t)kPairElems * kLB);
            for (int t0 = wid * kTileElems; t0 < n; t0 += kSweep) {
              const int e0 = t0 + lane * kChunk;
              const bool valid = e0 < n;
              const int xg = x + e0;
              float v[8];
              float2 vp[4];
              if constexpr (kLB == 2) {
                if (valid) bf16x8_pairs(lds128(lb + e0), vp);
                else {
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2) vp[k2] = make_float2(-9984.f, -9984.f);
                }
#pragma unroll
                for (int k2 = 0; k2 < 4; ++k2) { v[2 * k2] = vp[k2].x; v[2 * k2 + 1] = vp[k2].y; }
              } else {
                if (valid) {
                  const uint4 a4 = lds128(lb + e0);
                  const uint4 b4 = lds128(lb + e0 + 4);
                  v[0] = __uint_as_float(a4.x); v[1] = __uint_as_float(a4.y);
                  v[2] = __uint_as_float(a4.z); v[3] = __uint_as_float(a4.w);
                  v[4] = __uint_as_float(b4.x); v[5] = __uint_as_float(b4.y);
                  v[6] = __uint_as_float(b4.z); v[7] = __uint_as_float(b4.w);
                } else {
#pragma unroll
                  for (int k2 = 0; k2 < 8; ++k2) v[k2] = TV_NEG_INF;
                }
              }
              if (kind == kJobStats) {
                if (valid) {
                  float cm = v[0];
#pragma unroll
                  for (int k2 = 1; k2 < 8; ++k2) cm = fmaxf(cm, v[k2]);
                  if (cm > m_run) {
                    if (m_run != TV_NEG_INF) {
                      const float sc = L::exp_rel(m_run, cm, c_hi, c_lo);
                      acc.s *= sc;
                      acc.c *= sc;
                    }
                    m_run = cm;
                  }
                  float sum;
                  if constexpr (kLB == 2) {
                    const float2 mm = make_float2(-m_run, -m_run);
                    float2 e[4];
#pragma unroll
                    for (int k2 = 0; k2 < 4; ++k2) e[k2] = exp2_split_x2(__fadd2_rn(vp[k2], mm), ch, cl);
                    const float2 s2 = __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3]));
                    sum = s2.x + s2.y;
                  } else {
                    float t[8];
#pragma unroll
                    for (int k2 = 0; k2 < 8; ++k2) t[k2] = L::exp_rel(v[k2], m_run, c_hi, c_lo);
                    sum = sum8(t);
                  }
                  acc.add(sum);
                }
              } else if (kind == kJobBonusLeaf) {
                float lm = v[0];
#pragma unroll
                for (int k2 = 1; k2 < 8; ++k2) lm = fmaxf(lm, v[k2]);
                const float tm = warp_max(lm);
                float t[8];
#pragma unroll
                for (int k2 = 0; k2 < 8; ++k2) t[k2] = L::exp_pass(v[k2], tm, c_hi, c_lo);
                const float ts = warp_sum(valid ? sum8(t) : 0.f);
                if (lane == 0)
                  __stcg(f.tiles + (size_t)b * f.ntiles + (x + t0) / kTileElems,
                         make_float2(ts, tm));
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
                float t[8];
                if constexpr (kLB == 2) {
                  const float2 mm = make_float2(-rowmax, -rowmax);
                  const float2 al2 = make_float2(alpha1, alpha1);
                  const float2 nb2 = make_float2(-beta, -beta);
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2) {
                    const float2 e = exp2_corrected_x2(__fadd2_rn(vp[k2], mm), ch, cl);
                    const float2 xx = __ffma2_rn(al2, e, __fmul2_rn(nb2, make_float2(q[2 * k2], q[2 * k2 + 1])));
                    t[2 * k2] = fmaxf(xx.x, 0.f);
                    t[2 * k2 + 1] = fmaxf(xx.y, 0.f);
                  }
                } else {
#pragma unroll
                  for (int k2 = 0; k2 < 8; ++k2)
                    t[k2] = fmaxf(fmaf(alpha1, L::exp_pass(v[k2], rowmax, c_hi, c_lo),
                                       -beta * q[k2]), 0.f);
                }
                while (mp < nmask && it_mtok[mp] < xg) ++mp;
                for (int mq = mp; mq < nmask && it_mtok[mq] < xg + kChunk; ++mq) {
                  const int off = it_mtok[mq] - xg;
                  const float mv = (kind == kJobPass) ? 0.f : it_mval[mq];
#pragma unroll
                  for (int k2 = 0; k2 < 8; ++k2) if (k2 == off) t[k2] = mv;
                }
                if (kind == kJobPass) {
                  if (valid) acc.add(sum8(t));
                } else {
                  const float ts = warp_sum(valid ? sum8(t) : 0.f);
                  if (lane == 0)
                    __stcg(f.tiles + (size_t)b * f.ntiles + (x + t0) / kTileElems,
                           make_float2(ts, 0.f));
                }
              }
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&empty_bar[stage]);
          if (++stage == n_stages) { stage = 0; phase ^= 1; }
        }
        if (fail) raise_abort(args, f);
        // ---- the slice's partial result ----
        if (kind == kJobStats) {
          const float wm = warp_max(m_run);
          if (lane == 0) sh.red_a[wid] = wm;
          named_sync(2, kConsumers);
          float M = sh.red_a[0];
#pragma unroll
          for (int w = 1; w < kNCW; ++w) M = fmaxf(M, sh.red_a[w]);
          float part = (m_run == TV_NEG_INF) ? 0.f : acc.value() * L::exp_rel(m_run, M, c_hi, c_lo);
          part = warp_sum(part);
          if (lane == 0) sh.red_b[wid] = part;
          named_sync(2, kConsumers);
          if (tid == 0) {
            float S = 0.f;
            for (int w = 0; w < kNCW; ++w) S += sh.red_b[w];
            sh.out_x = M;
            sh.out_y = S;
          }
        } else if (kind == kJobPass) {
          const float ws = warp_sum(acc.value());
          if (lane == 0) sh.red_a[wid] = ws;
          named_sync(2, kConsumers);
          if (tid == 0) {
            float S = 0.f;
            for (int w = 0; w < kNCW; ++w) S += sh.red_a[w];
            sh.out_x = S;
            sh.out_y = 0.f;
          }
        } else {
          // bonus: the slice's total (leaf: relative to the slice's own max),
          // from the tiles this CTA just wrote
          fence_gpu();
          named_sync(2, kConsumers);
          if (wid == 0) {
            const int t_lo = x0 / kTileElems, t_hi = (x1 + kTileElems - 1) / kTileElems;
            const float2* tl = f.tiles + (size_t)b * f.ntiles;
            float Mc = 0.f;
            if (kind == kJobBonusLeaf) {
              float lm = TV_NEG_INF;
              for (int k2 = t_lo + lane; k2 < t_hi; k2 += 32) lm = fmaxf(lm, __ldcg(tl + k2).y);
              Mc = warp_max(lm);
            }
            float W = 0.f;
            for (int k2 = t_lo + lane; k2 < t_hi; k2 += 32) {
              const float2 tv = __ldcg(tl + k2);
              W += (kind == kJobBonusLeaf)
                       ? ((tv.y == TV_NEG_INF) ? 0.f : tv.x * L::exp_rel(tv.y, Mc, c_hi, c_lo))
                       : tv.x;
            }
            W = warp_sum(W);
            if (lane == 0) {
              sh.out_x = Mc;
              sh.out_y = W;
            }
          }
        }
      }
      named_sync(1, kThreads);
      if (tid == 0)   // the partial is its own completion flag
        st_relaxed_u64(f.part + ((size_t)b * R + item_row) * f.Kmax + item_slice,
                       pack_part(sh.out_x, sh.out_y));
      continue;
    }

    const int b = sh.my_tree;
    const size_t row0 = (size_t)b * R;
    if (act == kActNewTree) {
      // ---------------- a new tree: structure, validation, gathers ----------------
      if (tid == 0) {
        sh.outstanding = 0;
        Ctl& c = sh.ctl;
        c.bad = 0u;
        c.accepted = -1;
        c.node = 0;
        c.pending = -1;
        c.masked_sum = 0.0;
        c.n_tests = c.n_passes = 0;
        c.job.kind = 0;
      }
      for (int i = tid; i < R; i += kThreads) {
        s.par[i] = args.parents[row0 + i];
        s.tok[i] = args.tokens[row0 + i];
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
        if (bad) atomicOr(&sh.ctl.bad, bad);
      }
      __syncthreads();
      if (sh.ctl.bad == 0u) {
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
            const size_t prow = (row0 + p) * (size_t)V;
            s.gl[i] = L::at(logits + prow, t);
            s.gq[i] = __ldg(args.draft_probs + prow + t);
            if (!(s.gq[i] > 0.f)) bad |= 8u;
            s.invq[i] = 1.0 / (double)s.gq[i];
          }
          s.next[i] = nx;
        }
        if (bad) atomicOr(&sh.ctl.bad, bad);
      }
      __syncthreads();
      if (tid == 0) {
        if (sh.ctl.bad == 0u) {
          s.p[0] = 1.0;
          control_step(s, sh.ctl, args.uniforms + row0 + b);
        } else {
          sh.ctl.job.kind = kJobDone;
        }
      }
    } else {
      // ---------------- kActCombine: own tree's job finished; combine, advance ----------------
      const int K = sh.jK;
      const bool in_smem = sh.outstanding <= kPBuf;
      auto part_of = [&](int r, int k) -> float2 {
        return in_smem ? sh.pbuf[r * K + k]
                       : unpack_part(__ldcg(f.part + (row0 + r) * f.Kmax + k));
      };
      if (sh.jkind == kJobStats) {
        // one warp per row: normaliser from the slices, then the children's M_b0
        for (int r = wid; r < sh.jrows; r += kWarps) {
          float M = TV_NEG_INF;
          for (int k2 = lane; k2 < K; k2 += 32) M = fmaxf(M, part_of(r, k2).x);
          M = warp_max(M);
          float S = 0.f;
          for (int k2 = lane; k2 < K; k2 += 32) {
            const float2 pk = part_of(r, k2);
            if (pk.x != TV_NEG_INF) S += pk.y * L::exp_rel(pk.x, M, c_hi, c_lo);
          }
          S = warp_sum(S);
          const int node = s.job_rows[r];
          if (lane == 0) {
            s.rowm[node] = M;
            s.rows[node] = S;
            s.invs[node] = 1.0 / (double)S;
            if (!(S > 0.f)) atomicOr(&sh.ctl.bad, 64u);
          }
          __syncwarp();
          children_mb0(s, node, args.c, lane);
        }
      } else if (sh.jkind == kJobPass) {
        if (wid == 0) {
          float S = 0.f;
          for (int k2 = lane; k2 < K; k2 += 32) S += part_of(0, k2).x;
          S = warp_sum(S);
          if (lane == 0) sh.ctl.S = S;
        }
      } else if (wid == 0) {
        // ---- bonus: crossing slice, crossing tile, token ----
        const Job& job = sh.ctl.job;
        const bool leaf = (sh.jkind == kJobBonusLeaf);
        const int node = job.node;
        const int slice_len = sh.jslice;
        float Mg = TV_NEG_INF;
        if (leaf) {
          for (int k2 = lane; k2 < K; k2 += 32) Mg = fmaxf(Mg, part_of(0, k2).x);
          Mg = warp_max(Mg);
        }
        auto slice_scale = [&](float mx) -> float {
          return leaf ? ((mx == TV_NEG_INF) ? 0.f : L::exp_rel(mx, Mg, c_hi, c_lo)) : 1.f;
        };
        float W = 0.f;
        for (int k2 = lane; k2 < K; k2 += 32) {
          const float2 pk = part_of(0, k2);
          W += pk.y * slice_scale(pk.x);
        }
        W = warp_sum(W);
        const float target = args.uniforms[row0 + b + R] * W;
        // first slice whose running total exceeds the target (warp scan per 32 slices)
        int owner = -1, last_pos = -1;
        float before = 0.f, scale = 0.f, last_before = 0.f, last_scale = 0.f, base = 0.f;
        for (int k0 = 0; k0 < K && owner < 0; k0 += 32) {
          float wk = 0.f, sk = 0.f;
          if (k0 + lane < K) {
            const float2 pk = part_of(0, k0 + lane);
            sk = slice_scale(pk.x);
            wk = pk.y * sk;
          }
          float v = wk;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const float w2 = __shfl_up_sync(0xffffffffu, v, o);
            if (lane >= o) v += w2;
          }
          const unsigned pos = __ballot_sync(0xffffffffu, wk > 0.f);
          if (pos) {
            const int l = 31 - __clz(pos);
            last_pos = k0 + l;
            last_before = base + __shfl_sync(0xffffffffu, v - wk, l);
            last_scale = __shfl_sync(0xffffffffu, sk, l);
          }
          const unsigned hit = __ballot_sync(0xffffffffu, (k0 + lane < K) && (target < base + v));
          if (hit) {
            const int l = __ffs(hit) - 1;
            owner = k0 + l;
            before = base + __shfl_sync(0xffffffffu, v - wk, l);
            scale = __shfl_sync(0xffffffffu, sk, l);
          }
          base += __shfl_sync(0xffffffffu, v, 31);
        }
        if (owner < 0) {   // rounding put the target past the total: last slice with weight
          owner = (last_pos >= 0) ? last_pos : 0;
          before = (last_pos >= 0) ? last_before : 0.f;
          scale = (last_pos >= 0) ? last_scale : slice_scale(part_of(0, 0).x);
        }
        const float Mc = part_of(0, owner).x;
        const float lt = (scale > 0.f) ? (target - before) / scale : 0.f;
        // tiles of the crossing slice, in that slice's units
        const int sx0 = owner * slice_len, sx1 = min(V, sx0 + slice_len);
        const int t_lo = sx0 / kTileElems, t_hi = (sx1 + kTileElems - 1) / kTileElems;
        const float2* tl = f.tiles + (size_t)b * f.ntiles;
        auto tile_w = [&](float2 tv) -> float {
          return leaf ? ((tv.y == TV_NEG_INF) ? 0.f : tv.x * L::exp_rel(tv.y, Mc, c_hi, c_lo))
                      : tv.x;
        };
        int tile = -1, last_tile = -1;
        float tbase = 0.f, tb = 0.f, last_tbase = 0.f;
        for (int k0 = t_lo; k0 < t_hi && tile < 0; k0 += 32) {
          const float own = (k0 + lane < t_hi) ? tile_w(__ldcg(tl + k0 + lane)) : 0.f;
          float v = own;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const float w2 = __shfl_up_sync(0xffffffffu, v, o);
            if (lane >= o) v += w2;
          }
          const unsigned pos = __ballot_sync(0xffffffffu, own > 0.f);
          if (pos) {
            const int l = 31 - __clz(pos);
            last_tile = k0 + l;
            last_tbase = tb + __shfl_sync(0xffffffffu, v - own, l);
          }
          const unsigned hit = __ballot_sync(0xffffffffu, (k0 + lane < t_hi) && (lt < tb + v));
          if (hit) {
            const int l = __ffs(hit) - 1;
            tile = k0 + l;
            tbase = tb + __shfl_sync(0xffffffffu, v - own, l);
          }
          tb += __shfl_sync(0xffffffffu, v, 31);
        }
        if (tile < 0) {
          tile = (last_tile >= 0) ? last_tile : t_lo;
          tbase = (last_tile >= 0) ? last_tbase : 0.f;
        }
        const int xs = tile * kTileElems + lane * kChunk;
        const size_t rowoff = (row0 + node) * (size_t)V;
        float w[8];
        if (leaf) {
          float v[8];
          if (xs < sx1) load_logits<L, true>(logits + rowoff, xs, V, v);
          else {
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = TV_NEG_INF;
          }
#pragma unroll
          for (int e = 0; e < 8; ++e)
            w[e] = (v[e] == TV_NEG_INF) ? 0.f : L::exp_pass(v[e], Mc, c_hi, c_lo);
        } else {
          float v[8], q[8];
          if (xs < sx1) {
            load_logits<L, true>(logits + rowoff, xs, V, v);
            load_probs<true>(args.draft_probs + rowoff, xs, V, q);
          } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) { v[e] = TV_NEG_INF; q[e] = 0.f; }
          }
#pragma unroll
          for (int e = 0; e < 8; ++e)
            w[e] = (v[e] == TV_NEG_INF) ? 0.f
                   : fmaxf(fmaf(job.alpha1, L::exp_pass(v[e], job.rowmax, c_hi, c_lo),
                                -job.beta * q[e]), 0.f);
          for (int mq = 0; mq < job.nmask; ++mq) {
            const int off = s.mask_tok[mq] - xs;
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
        int yy;
        if (hit) {
          const int l = __ffs(hit) - 1;
          yy = tile * kTileElems + l * kChunk + __shfl_sync(0xffffffffu, found, l);
        } else {
          int last = -1;
#pragma unroll
          for (int e = 0; e < 8; ++e) if (w[e] > 0.f) last = xs + e;
          const unsigned any = __ballot_sync(0xffffffffu, last >= 0);
          yy = any ? __shfl_sync(0xffffffffu, last, 31 - __clz(any)) : sx1 - 1;
        }
        if (lane == 0) {
          args.out_bonus[b] = yy;
          sh.ctl.job.kind = kJobDone;
        }
      }
      __syncthreads();
      if (tid == 0 && sh.ctl.job.kind != kJobDone) {
        if (sh.ctl.bad & 64u) sh.ctl.job.kind = kJobDone;
        else control_step(s, sh.ctl, args.uniforms + row0 + b);
      }
    }
    // ---------------- post the own tree's next job, or finish the tree ----------------
    __syncthreads();
    if (sh.ctl.job.kind == kJobDone) {
      const bool ok = (sh.ctl.bad & (15u | 32u | 64u)) == 0u;
      const int N = args.N;
      for (int k2 = tid; k2 < N; k2 += kThreads) args.out_path[(size_t)b * N + k2] = -1;
      if (args.out_node_p)
        for (int i = tid; i < R; i += kThreads)
          args.out_node_p[row0 + i] = ok ? s.dbgp[i] : __int_as_float(0x7fc00000);
      __syncthreads();
      if (tid == 0) {
        const int acc_node = ok ? sh.ctl.accepted : -1;
        if (acc_node >= 0) {
          int depth = 0;
          for (int j = acc_node; j != 0; j = s.par[j]) ++depth;
          int k2 = depth - 1;
          for (int j = acc_node; j != 0; j = s.par[j]) args.out_path[(size_t)b * N + (k2--)] = j;
          args.out_accept_len[b] = depth;
        } else {
          args.out_accept_len[b] = -1;
          args.out_bonus[b] = -1;
        }
        if (args.out_stats) {
          int distinct = 0;
          for (int i = 0; i < R; ++i) distinct += (s.npass[i] > 0);
          int32_t* o = args.out_stats + (size_t)b * 4;
          o[0] = ok ? sh.ctl.n_tests : 0;
          o[1] = ok ? sh.ctl.n_passes : 0;
          o[2] = ok ? distinct : 0;
          o[3] = (acc_node >= 0 && s.first[acc_node] < 0) ? 1 : 0;
        }
        if (sh.ctl.bad) atomicOr(args.status, sh.ctl.bad);
        f.finished[b] = (unsigned)f.epoch;
        fence_gpu();
        sh.act = (atomicAdd(&f.ctr[kCtrDone], 1u) == (unsigned)B - 1u) ? 1 : 0;
        sh.my_tree = -1;
        sh.outstanding = 0;
      }
      __syncthreads();
      if (sh.act == 1 && wid == 0) {
        // last tree: the tickets now held (slots from the tail up to the head)
        // and the at most one more per CTA that may still be taken will see
        // an exit tag instead of an item
        unsigned lo = 0u, hi = 0u;
        if (lane == 0) {
          lo = atomicAdd(&f.ctr[kCtrTail], 0u);
          hi = atomicAdd(&f.ctr[kCtrHead], 0u) + gridDim.x;
        }
        lo = __shfl_sync(0xffffffffu, lo, 0);
        hi = min(__shfl_sync(0xffffffffu, hi, 0), (unsigned)f.cap);
        for (unsigned q = lo + lane; q < hi; q += 32)
          st_relaxed_u64(&f.items[q].tag, (f.epoch << 32) | q | kExitTag);
      }
    } else if (wid == 0) {
      post_job(s, sh, args, f, b, V, lane);
    }
  }

  // ---------------- exit ----------------
  __syncthreads();
  if (ld_relaxed_u32(&f.ctr[kCtrAbort])) {
    // after an abort, trees that did not finish report "invalid"
    for (int b = blockIdx.x * kThreads + tid; b < B; b += gridDim.x * kThreads) {
      if (ld_relaxed_u32(&f.finished[b]) != (unsigned)f.epoch) {
        args.out_accept_len[b] = -1;
        args.out_bonus[b] = -1;
      }
    }
  }
  if (tid == 0) {
    // the last CTA out leaves the counters at zero for the next call
    fence_gpu();
    if (atomicAdd(&f.ctr[kCtrExit], 1u) == gridDim.x - 1) {
      for (int k = 0; k < kNumCtr; ++k) atomicExch(&f.ctr[k], 0u);
    }
  }
}

}  // namespace flow
}  // namespace tvk

// --------------------------------------------------------------- launcher --

namespace {

struct FlowLayout {
  size_t kmax, cap, ntiles;
};

FlowLayout flow_layout(int B, int R, int V, int min_slice) {
  FlowLayout l;
  l.kmax = (size_t)((V + min_slice - 1) / min_slice);
  // per tree: at most R rows normalised and at most R - 1 passes plus the
  // bonus draw, each at most kmax slices
  l.cap = (size_t)B * (2 * (size_t)R + 1) * l.kmax + tvk::flow::kMaxGrid;
  l.ntiles = (size_t)((V + tvk::fused::kTileElems - 1) / tvk::fused::kTileElems);
  return l;
}

size_t up256(size_t n) { return (n + 255) & ~static_cast<size_t>(255); }

size_t flow_smem_bytes(int R, int ncw, int stages) {
  return (size_t)stages * tvk::fused::stage_bytes(ncw) +
         ((tvk::fused::tree_smem_bytes_nt(R, 0) + 15) & ~(size_t)15) + (size_t)R * 8 + 64;
}

}  // namespace

size_t tv_flow_workspace_bytes(int B, int R, int V, int min_slice) {
  const FlowLayout l = flow_layout(B, R, V, min_slice);
  return up256(256) + up256(l.cap * sizeof(FlowItem)) + 2 * up256((size_t)B * R * 4) +
         up256((size_t)B * R * l.kmax * 8) + up256((size_t)B * 4) +
         up256((size_t)B * l.ntiles * 8);
}

int tv_flow_bind(void* base, size_t bytes, int B, int R, int V, const FlowPlan& plan,
                 FlowArgs* f) {
  const FlowLayout l = flow_layout(B, R, V, plan.slice_pass < plan.slice_stats
                                                ? plan.slice_pass : plan.slice_stats);
  char* p = static_cast<char*>(base);
  auto take = [&](size_t n) {
    char* q = p;
    p += up256(n);
    return q;
  };
  f->ctr = reinterpret_cast<unsigned*>(take(256));
  f->items = reinterpret_cast<FlowItem*>(take(l.cap * sizeof(FlowItem)));
  f->job_mtok = reinterpret_cast<int*>(take((size_t)B * R * 4));
  f->job_mval = reinterpret_cast<float*>(take((size_t)B * R * 4));
  f->part = reinterpret_cast<unsigned long long*>(take((size_t)B * R * l.kmax * 8));
  f->finished = reinterpret_cast<unsigned*>(take((size_t)B * 4));
  f->tiles = reinterpret_cast<float2*>(take((size_t)B * l.ntiles * 8));
  f->cap = (int)l.cap;
  f->R = R;
  f->Kmax = (int)l.kmax;
  f->ntiles = (int)l.ntiles;
  f->slice_pass = plan.slice_pass;
  f->slice_stats = plan.slice_stats;
  return (size_t)(p - static_cast<char*>(base)) <= bytes ? 0 : -4;
}

FlowPlan tv_flow_plan(int R, int smem_per_sm, int smem_per_block, int force_ncw,
                      int force_stages, int force_slice_pass, int force_slice_stats) {
  FlowPlan p;
  if (force_ncw == 4 || force_ncw == 8) p.ncw = force_ncw;
  if (force_slice_pass >= 256 && force_slice_pass % 256 == 0) p.slice_pass = force_slice_pass;
  if (force_slice_stats >= 256 && force_slice_stats % 256 == 0) p.slice_stats = force_slice_stats;
  const int per_sm = 16 / p.ncw;   // CTAs per SM the kernel is built for
  if (force_stages >= 2 && force_stages <= tvk::fused::kMaxStages) {
    p.stages = force_stages;
  } else {
    p.stages = 2;
    for (int st = tvk::fused::kMaxStages; st >= 2; --st)
      if ((size_t)per_sm * (flow_smem_bytes(R, p.ncw, st) + 2048) <= (size_t)smem_per_sm) {
        p.stages = st;
        break;
      }
  }
  p.smem = flow_smem_bytes(R, p.ncw, p.stages);
  p.ok = p.smem + 2048 <= (size_t)smem_per_block;
  return p;
}

int tv_launch_flow(const TravArgs& a, FlowArgs f, int logit_is_bf16, const FlowPlan& plan,
                   int sm_count, cudaStream_t stream, cudaEvent_t* ev) {
  using namespace tvk::flow;
  const size_t smem = plan.smem;
  int stages = plan.stages;
  if (ev) {
    for (int k = 0; k < 3; ++k)
      if (cudaEventRecord(ev[k], stream) != cudaSuccess) return -5;
  }
  auto run = [&](auto kernel, int threads) -> int {
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return -5;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem) !=
            cudaSuccess ||
        per_sm < 1)
      return -5;
    const int grid = per_sm * sm_count;
    if (grid > kMaxGrid) return -5;
    void* params[] = {const_cast<TravArgs*>(&a), &f, &stages};
    if (cudaLaunchCooperativeKernel((const void*)kernel, dim3(grid), dim3(threads), params, smem,
                                    stream) != cudaSuccess) {
      cudaGetLastError();
      return -5;
    }
    return 0;
  };
  int rc;
  if (plan.ncw == 8)
    rc = logit_is_bf16 ? run(tv_flow_kernel<tvk::Bf16Logits, 8>, 288)
                       : run(tv_flow_kernel<tvk::F32Logits, 8>, 288);
  else
    rc = logit_is_bf16 ? run(tv_flow_kernel<tvk::Bf16Logits, 4>, 160)
                       : run(tv_flow_kernel<tvk::F32Logits, 4>, 160);
  if (rc) return rc;
  if (ev && cudaEventRecord(ev[3], stream) != cudaSuccess) return -5;
  return 0;
}
