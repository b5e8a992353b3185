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
// its tree.
//
// Each CTA is warp-specialised:
//   * an owner warp runs the serial control of the CTA's current tree (tree
//     set-up, combining partials, Eqs. (1)-(3), posting the next job);
//   * a fetcher warp takes tickets and copies the queued slices into the
//     CTA's slots, one slice ahead of the one being reduced (a second slice
//     held ahead made jobs wait longer behind other trees' slices: 3-5 %
//     slower at 128 to 1024 trees);
//   * a producer warp streams the fetched slices into a shared-memory ring
//     with 1-D bulk copies (TMA);
//   * NCW consumer warps reduce the ring stages and write each slice's
//     partial result.
// So the serial control of one tree overlaps the streaming of others, and
// consecutive slices of a CTA stream back to back.
//
// One cooperative launch keeps all CTAs resident, so CTAs may wait on work
// published by others; every wait is bounded, and a global abort flag ends
// the kernel cleanly if one ever gives up.  Consumer warps synchronise only
// through mbarriers (bounded waits), never through bar.sync, so a warp that
// gives up cannot leave the others blocked.
//
// Queue protocol: a poster reserves a range of slots with one atomicAdd on
// the tail, writes the slots' bodies, fences, then stores each slot's tag
// (call epoch, slot number).  A fetcher takes a ticket -- the next slot
// number, one atomicAdd on the head -- and processes that slot once its tag
// appears.  Slots are never reused within a call; when the last tree is done
// its owner writes an exit tag into every slot a ticket may still point to.
// A slice's partial is one 64-bit store that doubles as its completion flag.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <mutex>

#include "tv_control.cuh"
#include "tv_device.cuh"
#include "tv_launch.h"
#include "tv_ptx.cuh"

namespace tvk {
namespace flow {

using namespace tvk::fused;

constexpr int kMaxNCW = 8;
constexpr int kSlots = 2;           // queued slices a CTA holds: one streaming, one ahead
constexpr int kPBuf = 256;          // partials of a job kept in shared memory by the poll
constexpr unsigned long long kNoPart = ~0ull;   // a partial slot not written yet
constexpr unsigned kNoTicket = 0xffffffffu;
constexpr unsigned long long kExitTag = 0x80000000ull;   // tag bit: no more items, exit
constexpr int kMaxGrid = 4096;      // tickets taken past the last item: one per CTA at most
constexpr unsigned long long kIdleNs = 2000000000ull;   // 2 s without progress: abort

enum : int {
  kCtrTail = 0, kCtrHead = 1, kCtrDone = 2, kCtrNextTree = 3, kCtrAbort = 4, kCtrExit = 5,
  kNumCtr = 6
};
enum : int { kStageFirst = 1, kStageLast = 2, kStageExit = 4 };
constexpr int kSlotExit = -1;       // ItemSlot::kind of the fetcher's "no more slices"

// A queued slice as held by a CTA (the masks live in shared arrays of R).
struct ItemSlot {
  int b, node, row, slice;
  int kind, slice_len, nmask, pad0;
  float alpha1, beta, rowmax, pad1;
};

struct StageMeta {
  int slot, x, n, flags;
};

struct Shared {
  ItemSlot slots[kSlots];
  StageMeta meta[kMaxStages];
  float2 red[kMaxStages][kMaxNCW];   // per-warp partials of the slice ending in a stage
  Ctl ctl;                           // serial control state of the own tree (owner warp)
  Ahead ahead;                       // the next step, worked out while a pass runs
  Job fjob;                          // a job posted from `ahead`
  float2 pbuf[kPBuf];                // the own job's partials, as read by the poll
  int jkind, jrows, jK, jslice, outstanding;
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

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
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

// Ends the whole kernel cleanly: every role sees the flag at its next poll.
__device__ __forceinline__ void raise_abort(const TravArgs& a, const FlowArgs& f) {
  atomicOr(a.status, 32u);
  atomicExch(&f.ctr[kCtrAbort], 1u);
}

// An mbarrier wait whose outcome is the same for every lane of the warp (a
// lane that gave up makes the whole warp give up), so that no lane is left
// alone at a later warp-wide operation.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity) ? 1 : 0) != 0;
}

// Sleep of an idle poller: 32 ns, then 64 ns; false once the wait has
// lasted kIdleNs (the caller aborts).
struct Backoff {
  unsigned nap = 32u;
  unsigned long long since = 0ull;
  __device__ __forceinline__ void reset() {
    nap = 32u;
    since = 0ull;
  }
  __device__ __forceinline__ bool idle() {
    const unsigned long long now = global_ns();
    if (since == 0ull) since = now;
    else if (now - since > kIdleNs) return false;
    __nanosleep(nap);
    if (nap < 64u) nap <<= 1;
    return true;
  }
};

// ------------------------------------------------------------- shapes --

// Bytes of one ring stage: 4.5 KB per consumer warp, so that a stage holds 12
// tiles of bf16 target + fp32 draft values (three per warp with four warps).
// With the 228 KB of shared memory an SM has and four CTAs per SM this is two
// stages per CTA: against three stages of 3 KB per warp (the same bytes in
// flight), each warp waits on and releases a stage a third as often, 3.5-5.6 %
// faster from 128 to 1024 trees.
__host__ __device__ constexpr int flow_stage_bytes(int ncw) { return 4608 * ncw; }

template <typename L, int kNCW>
struct Shape {
  static constexpr int kConsumers = kNCW * 32;
  static constexpr int kThreads = kConsumers + 96;   // + producer, fetcher, owner warps
  static constexpr int kStageBytes = flow_stage_bytes(kNCW);
  static constexpr int kSweep = kConsumers * kChunk;
  static constexpr int kLB = L::kBytes;
  // tokens per stage: target and draft values together, or target only
  static constexpr int kPairElems = kStageBytes / (kLB + 4) / kTileElems * kTileElems;
  static constexpr int kRowElems = kStageBytes / kLB;
};

struct Smem {
  char* ring;
  TreeSmem s;
  int* mtok;     // [kSlots][R] removed tokens of the held slices
  float* mval;   // [kSlots][R] their stored masses
  float* u;      // [R + 1] the own tree's uniforms
  int* mtok2;    // [R] removed tokens of the pass worked out ahead
  uint64_t* full_bar;
  uint64_t* empty_bar;
  uint64_t* slot_free;
  uint64_t* slot_full;
  uint64_t* red_bar;
  Shared* sh;
};

// ------------------------------------------------------------- fetcher --

// Takes tickets and copies the published slices into the CTA's slots, at most
// kSlots - 1 ahead of the slice being reduced.
template <typename L, int kNCW>
__device__ void fetcher_role(const TravArgs& a, const FlowArgs& f, const Smem& m, int lane) {
  const int R = a.N + 1, B = a.B;
  int slot = 0, slot_phase = 0;
  unsigned polls = 0u;
  Backoff wait;
  bool have_slot = false;
  for (;;) {
    if (!have_slot) {
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&m.slot_free[slot], slot_phase ^ 1) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) raise_abort(a, f);
        return;   // the producer times out on its slot wait and stops the consumers
      }
      have_slot = true;
    }
    ItemSlot& it = m.sh->slots[slot];
    // ---- a ticket, then its slot's publication (lane 0) ----
    int cmd = 0;   // 1: a slice, 2: stop
    if (lane == 0) {
      unsigned ticket = kNoTicket;
      if (ld_relaxed_u32(&f.ctr[kCtrDone]) >= (unsigned)B) cmd = 2;   // nothing will come
      else ticket = atomicAdd(&f.ctr[kCtrHead], 1u);
      const unsigned long long want = (f.epoch << 32) | (unsigned long long)ticket;
      while (cmd == 0) {
        const unsigned long long tag =
            (ticket < (unsigned)f.cap) ? ld_acquire_u64(&f.items[ticket].tag) : 0ull;
        if (tag == want) {
          cmd = 1;
        } else if (tag == (want | kExitTag)) {
          cmd = 2;
        } else if ((++polls & 31u) == 0u && ld_relaxed_u32(&f.ctr[kCtrAbort])) {
          cmd = 2;
        } else if (!wait.idle()) {
          raise_abort(a, f);
          cmd = 2;
        }
      }
      wait.reset();
      int4 w[7];
      if (cmd == 1) {
        const int4* bp = reinterpret_cast<const int4*>(f.items + ticket);
#pragma unroll
        for (int k = 0; k < 7; ++k) w[k] = __ldcg(bp + k);   // one 112-byte read
      }
      if (cmd == 1) {
        it.b = w[0].x; it.node = w[0].y; it.row = w[0].z; it.slice = w[0].w;
        it.kind = w[1].x; it.slice_len = w[1].y; it.nmask = w[1].z;
        it.alpha1 = __int_as_float(w[2].x); it.beta = __int_as_float(w[2].y);
        it.rowmax = __int_as_float(w[2].z);
        int* mt = m.mtok + slot * R;
        float* mv = m.mval + slot * R;
        const int ni = min(w[1].z, kFlowInlineMask);
        const int tk[8] = {w[3].x, w[3].y, w[3].z, w[3].w, w[4].x, w[4].y, w[4].z, w[4].w};
        const int vk[8] = {w[5].x, w[5].y, w[5].z, w[5].w, w[6].x, w[6].y, w[6].z, w[6].w};
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (q < ni) { mt[q] = tk[q]; mv[q] = __int_as_float(vk[q]); }
      } else if (cmd == 2) {
        it.kind = kSlotExit;
      }
    }
    cmd = __shfl_sync(0xffffffffu, cmd, 0);
    __syncwarp();
    if (cmd == 1) {
      const int nmask = it.nmask;
      if (nmask > kFlowInlineMask) {   // rare: the rest of a long mask list
        const int b = it.b;
        fence_gpu();
        for (int q = kFlowInlineMask + lane; q < nmask; q += 32) {
          m.mtok[slot * R + q] = __ldcg(f.job_mtok + (size_t)b * R + q);
          m.mval[slot * R + q] = __ldcg(f.job_mval + (size_t)b * R + q);
        }
      }
      __syncwarp();
    }
    if (lane == 0) mbar_arrive(&m.slot_full[slot]);   // release: the slot's contents
    if (cmd == 2) return;
    have_slot = false;
    if (++slot == kSlots) { slot = 0; slot_phase ^= 1; }
  }
}

// ------------------------------------------------------------ producer --

// Streams the fetched slices through the ring, in slot order (one lane).
template <typename L, int kNCW>
__device__ void producer_loop(const TravArgs& a, const FlowArgs& f, const Smem& m,
                              int n_stages) {
  using S = Shape<L, kNCW>;
  using E = typename L::elem;
  const int R = a.N + 1, V = a.V;
  const E* logits = reinterpret_cast<const E*>(a.logits);
  int stage = 0, phase = 0, slot = 0, slot_phase = 0;
  for (;;) {
    if (!mbar_wait(&m.slot_full[slot], slot_phase)) {
      raise_abort(a, f);
      return;   // the consumers time out on their stage wait
    }
    const ItemSlot& it = m.sh->slots[slot];
    if (it.kind == kSlotExit) break;
    const bool pair = (it.kind == kJobPass || it.kind == kJobBonusRes);
    const int per = pair ? S::kPairElems : S::kRowElems;
    const int x0 = it.slice * it.slice_len;
    const int x1 = min(V, x0 + it.slice_len);
    const size_t row = ((size_t)it.b * R + it.node) * (size_t)V;
    for (int x = x0; x < x1; x += per) {
      const int n = min(per, x1 - x);
      if (!mbar_wait(&m.empty_bar[stage], phase ^ 1)) {
        raise_abort(a, f);
        return;
      }
      m.sh->meta[stage] = StageMeta{slot, x, n, (x == x0 ? kStageFirst : 0) |
                                                    (x + n >= x1 ? kStageLast : 0)};
      char* dst = m.ring + (size_t)stage * S::kStageBytes;
      const uint32_t lbytes = (uint32_t)n * S::kLB;
      const uint32_t qbytes = pair ? (uint32_t)n * 4u : 0u;
      mbar_arrive_expect_tx(&m.full_bar[stage], lbytes + qbytes);
      tma_load_1d(dst, logits + row + x, lbytes, &m.full_bar[stage]);
      if (pair)
        tma_load_1d(dst + (size_t)S::kPairElems * S::kLB, a.draft_probs + row + x, qbytes,
                    &m.full_bar[stage]);
      if (++stage == n_stages) { stage = 0; phase ^= 1; }
    }
    if (++slot == kSlots) { slot = 0; slot_phase ^= 1; }
  }
  // ---- tell the consumers to stop ----
  if (mbar_wait(&m.empty_bar[stage], phase ^ 1)) {
    m.sh->meta[stage] = StageMeta{0, 0, 0, kStageExit};
    mbar_arrive(&m.full_bar[stage]);
  } else {
    raise_abort(a, f);
  }
}

template <typename L, int kNCW>
__device__ void producer_role(const TravArgs& a, const FlowArgs& f, const Smem& m,
                              int n_stages, int lane) {
  if (lane == 0) producer_loop<L, kNCW>(a, f, m, n_stages);
  __syncwarp();
}

// ------------------------------------------------------------ consumers --

template <typename L, int kNCW>
__device__ void consumer_role(const TravArgs& a, const FlowArgs& f, const Smem& m,
                              int n_stages, int wid, int lane) {
  using S = Shape<L, kNCW>;
  using E = typename L::elem;
  const int R = a.N + 1, V = a.V;
  const float c_hi = a.c_hi, c_lo = a.c_lo;
  const float2 ch = make_float2(c_hi, c_hi), cl = make_float2(c_lo, c_lo);
  int stage = 0, phase = 0;
  unsigned red_phase = 0u;   // parity bit per stage of red_bar (warp 0 waits on it)
  // the slice in progress
  int kind = 0, b = 0, row_idx = 0, slice = 0, nmask = 0, slot = 0, x0 = 0, x1 = 0;
  float alpha1 = 0.f, beta = 0.f, rowmax = 0.f;
  float m_run = TV_NEG_INF;
  Comp acc;
  int mp = 0;
  for (;;) {
    if (!mbar_wait_warp(&m.full_bar[stage], phase)) {
      if (lane == 0) raise_abort(a, f);
      break;
    }
    const StageMeta meta = m.sh->meta[stage];
    if (meta.flags & kStageExit) break;
    if (meta.flags & kStageFirst) {
      const ItemSlot& it = m.sh->slots[meta.slot];
      kind = it.kind; b = it.b; row_idx = it.row; slice = it.slice; nmask = it.nmask;
      alpha1 = it.alpha1; beta = it.beta; rowmax = it.rowmax;
      slot = meta.slot;
      x0 = slice * it.slice_len;
      x1 = min(V, x0 + it.slice_len);
      m_run = TV_NEG_INF;
      acc = Comp();
      mp = 0;
    }
    const int* mtok = m.mtok + slot * R;
    const float* mval = m.mval + slot * R;
    const int x = meta.x, n = meta.n;
    const char* buf = m.ring + (size_t)stage * S::kStageBytes;
    const E* lb = reinterpret_cast<const E*>(buf);
    const float* qb = reinterpret_cast<const float*>(buf + (size_t)S::kPairElems * S::kLB);
    bool done_stage = false;
    if constexpr (S::kLB == 2) {
      if (kind == kJobStats) {
        // Row normaliser, bf16: this warp's maximum over its part of the stage
        // first (exact on bf16 pairs, after the same clamp as the sums), so
        // that the running sum is rescaled at most once per stage, then the
        // sum of e(x) relative to it.  exp2_corrected is used here as in the
        // passes: its small uniform bias then cancels in alpha1 e(x) = p a e(x)/s.
        const uint32_t lo_clamp = 0xC61CC61Cu;   // two bf16 -9984
        __nv_bfloat162 hm = *reinterpret_cast<const __nv_bfloat162*>(&lo_clamp);
        for (int t0 = wid * kTileElems; t0 < n; t0 += S::kSweep) {
          const int e0 = t0 + lane * kChunk;
          if (e0 < n) {
            const uint4 w = lds128(lb + e0);
            hm = __hmax2(hm, *reinterpret_cast<const __nv_bfloat162*>(&w.x));
            hm = __hmax2(hm, *reinterpret_cast<const __nv_bfloat162*>(&w.y));
            hm = __hmax2(hm, *reinterpret_cast<const __nv_bfloat162*>(&w.z));
            hm = __hmax2(hm, *reinterpret_cast<const __nv_bfloat162*>(&w.w));
          }
        }
        const uint32_t hb = *reinterpret_cast<uint32_t*>(&hm);
        const float stage_m =
            warp_max(fmaxf(__uint_as_float(hb << 16), __uint_as_float(hb & 0xffff0000u)));
        if (stage_m > m_run) {
          if (m_run != TV_NEG_INF) {
            const float sc = L::exp_rel(m_run, stage_m, c_hi, c_lo);
            acc.s *= sc;
            acc.c *= sc;
          }
          m_run = stage_m;
        }
        const float2 mm = make_float2(-m_run, -m_run);
        for (int t0 = wid * kTileElems; t0 < n; t0 += S::kSweep) {
          const int e0 = t0 + lane * kChunk;
          if (e0 < n) {
            float2 vp[4];
            bf16x8_pairs(lds128(lb + e0), vp);
            float2 e[4];
#pragma unroll
            for (int k2 = 0; k2 < 4; ++k2)
              e[k2] = exp2_corrected_x2(__fadd2_rn(vp[k2], mm), ch, cl);
            const float2 s2 = __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3]));
            acc.add(s2.x + s2.y);
          }
        }
        done_stage = true;
      }
    }
    for (int t0 = wid * kTileElems; !done_stage && t0 < n; t0 += S::kSweep) {
      const int e0 = t0 + lane * kChunk;
      const bool valid = e0 < n;
      const int xg = x + e0;
      float v[8];
      float2 vp[4];
      if constexpr (S::kLB == 2) {
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
          if constexpr (S::kLB == 2) {
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
          __stcg(f.tiles + (size_t)b * f.ntiles + (x + t0) / kTileElems, make_float2(ts, tm));
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
        if constexpr (S::kLB == 2) {
          const float2 mm = make_float2(-rowmax, -rowmax);
          const float2 al2 = make_float2(alpha1, alpha1);
          const float2 nb2 = make_float2(-beta, -beta);
#pragma unroll
          for (int k2 = 0; k2 < 4; ++k2) {
            const float2 e = exp2_corrected_x2(__fadd2_rn(vp[k2], mm), ch, cl);
            const float2 xx =
                __ffma2_rn(al2, e, __fmul2_rn(nb2, make_float2(q[2 * k2], q[2 * k2 + 1])));
            t[2 * k2] = fmaxf(xx.x, 0.f);
            t[2 * k2 + 1] = fmaxf(xx.y, 0.f);
          }
        } else {
#pragma unroll
          for (int k2 = 0; k2 < 8; ++k2)
            t[k2] = fmaxf(fmaf(alpha1, L::exp_pass(v[k2], rowmax, c_hi, c_lo), -beta * q[k2]),
                          0.f);
        }
        while (mp < nmask && mtok[mp] < xg) ++mp;
        for (int mq = mp; mq < nmask && mtok[mq] < xg + kChunk; ++mq) {
          const int off = mtok[mq] - xg;
          const float mv = (kind == kJobPass) ? 0.f : mval[mq];
#pragma unroll
          for (int k2 = 0; k2 < 8; ++k2) if (k2 == off) t[k2] = mv;
        }
        if (kind == kJobPass) {
          if (valid) acc.add(sum8(t));
        } else {
          const float ts = warp_sum(valid ? sum8(t) : 0.f);
          if (lane == 0)
            __stcg(f.tiles + (size_t)b * f.ntiles + (x + t0) / kTileElems, make_float2(ts, 0.f));
        }
      }
    }
    __syncwarp();
    const bool last = (meta.flags & kStageLast) != 0;
    if (!last) {
      if (lane == 0) mbar_arrive(&m.empty_bar[stage]);
    } else {
      // ---- the slice's partial: per-warp values, combined by warp 0 ----
      float2 mine;
      if (kind == kJobStats) {
        const float wm = warp_max(m_run);
        const float part =
            (m_run == TV_NEG_INF) ? 0.f : acc.value() * L::exp_rel(m_run, wm, c_hi, c_lo);
        mine = make_float2(wm, warp_sum(part));
      } else if (kind == kJobPass) {
        mine = make_float2(warp_sum(acc.value()), 0.f);
      } else {
        mine = make_float2(0.f, 0.f);
        fence_gpu();   // this warp's bonus tiles, before warp 0 reads them
      }
      if (lane == 0) {
        m.sh->red[stage][wid] = mine;
        mbar_arrive(&m.red_bar[stage]);      // release: red[] and the tiles
        mbar_arrive(&m.slot_free[slot]);     // done with the slot's masks
      }
      if (wid == 0) {
        const bool got = mbar_wait_warp(&m.red_bar[stage], (red_phase >> stage) & 1u);
        red_phase ^= 1u << stage;
        if (!got) {
          if (lane == 0) raise_abort(a, f);
          break;
        }
        float px = 0.f, py = 0.f;
        if (kind == kJobStats) {
          float M = TV_NEG_INF;
          for (int w = 0; w < kNCW; ++w) M = fmaxf(M, m.sh->red[stage][w].x);
          for (int w = 0; w < kNCW; ++w) {
            const float2 r = m.sh->red[stage][w];
            if (r.x != TV_NEG_INF) py += r.y * L::exp_rel(r.x, M, c_hi, c_lo);
          }
          px = M;
        } else if (kind == kJobPass) {
          for (int w = 0; w < kNCW; ++w) px += m.sh->red[stage][w].x;
        } else {
          // bonus: the slice's total (leaf: relative to the slice's own max)
          fence_gpu();
          const int t_lo = x0 / kTileElems, t_hi = (x1 + kTileElems - 1) / kTileElems;
          const float2* tl = f.tiles + (size_t)b * f.ntiles;
          if (kind == kJobBonusLeaf) {
            float lm = TV_NEG_INF;
            for (int k2 = t_lo + lane; k2 < t_hi; k2 += 32) lm = fmaxf(lm, __ldcg(tl + k2).y);
            px = warp_max(lm);
          }
          float W = 0.f;
          for (int k2 = t_lo + lane; k2 < t_hi; k2 += 32) {
            const float2 tv = __ldcg(tl + k2);
            W += (kind == kJobBonusLeaf)
                     ? ((tv.y == TV_NEG_INF) ? 0.f : tv.x * L::exp_rel(tv.y, px, c_hi, c_lo))
                     : tv.x;
          }
          py = warp_sum(W);
          fence_gpu();   // the tiles before the partial that announces them
        }
        if (lane == 0) {
          st_relaxed_u64(f.part + ((size_t)b * R + row_idx) * f.Kmax + slice, pack_part(px, py));
          mbar_arrive(&m.empty_bar[stage]);   // only now may the stage (and red[stage]) be reused
        }
      } else if (lane == 0) {
        mbar_arrive(&m.empty_bar[stage]);
      }
    }
    if (++stage == n_stages) { stage = 0; phase ^= 1; }
  }
}

// --------------------------------------------------------------- owner --

// Tokens per slice: enough slices per row to give every CTA one when each
// remaining tree has a job out, between the plan's largest and smallest
// slice.  Early on (many trees) this keeps slices large; towards the end,
// when a few trees' chains of jobs set the time, their jobs spread over more
// CTAs.  `done` is the number of finished trees as last read.
__device__ __forceinline__ int adaptive_slice(const FlowArgs& f, int V, int B, bool stats,
                                              int n_rows, unsigned done) {
  const int largest = stats ? f.slice_stats : f.slice_pass;
  const int active = max(1, B - (int)done);
  const int per_row = max(1, (int)gridDim.x / (active * n_rows));
  int want = (V + per_row - 1) / per_row;
  want = (want + kTileElems - 1) / kTileElems * kTileElems;
  return max(f.slice_min, min(largest, want));
}

// Publishes the own tree's current job (ctl.job) as slice items.  (Its queue
// slots are taken when the items are written: slots reserved earlier, to
// overlap that atomic with the combine, held the fetchers that drew them
// until the job was published, 1-1.5 % slower.)
__device__ void post_job(const TreeSmem& s, Shared& sh, const TravArgs& a, const FlowArgs& f,
                         int b, int V, int lane, unsigned done, const Job& j,
                         const int* mask_tok, const float* mask_val) {
  const bool stats = (j.kind == kJobStats);
  const int n_rows = stats ? j.n_rows : 1;
  const int slice = adaptive_slice(f, V, a.B, stats, n_rows, done);
  const int K = (V + slice - 1) / slice;
  const int nmask = (j.kind == kJobPass || j.kind == kJobBonusRes) ? j.nmask : 0;
  const int n = n_rows * K;
  const size_t R = (size_t)f.R;
  for (int q = kFlowInlineMask + lane; q < nmask; q += 32) {   // beyond the inline ones
    f.job_mtok[b * R + q] = mask_tok[q];
    f.job_mval[b * R + q] = (j.kind == kJobBonusRes) ? mask_val[q] : 0.f;
  }
  // the job's partial slots start as "not yet"
  for (int q = lane; q < n; q += 32) {
    const int r = q / K;
    __stcg(f.part + ((size_t)b * R + r) * f.Kmax + (q - r * K), kNoPart);
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
  const int4 w1 = make_int4(j.kind, slice, nmask, 0);
  const int4 w2 = make_int4(__float_as_int(j.alpha1), __float_as_int(j.beta),
                            __float_as_int(j.rowmax), 0);
  int tk[kFlowInlineMask];
  float vk[kFlowInlineMask];
#pragma unroll
  for (int q = 0; q < kFlowInlineMask; ++q) {
    tk[q] = (q < nmask) ? mask_tok[q] : 0x7fffffff;
    vk[q] = (q < nmask && j.kind == kJobBonusRes) ? mask_val[q] : 0.f;
  }
  const int4 w3 = make_int4(tk[0], tk[1], tk[2], tk[3]);
  const int4 w4 = make_int4(tk[4], tk[5], tk[6], tk[7]);
  const int4 w5 = make_int4(__float_as_int(vk[0]), __float_as_int(vk[1]),
                            __float_as_int(vk[2]), __float_as_int(vk[3]));
  const int4 w6 = make_int4(__float_as_int(vk[4]), __float_as_int(vk[5]),
                            __float_as_int(vk[6]), __float_as_int(vk[7]));
  for (int q = lane; q < n; q += 32) {
    const int r = q / K;
    int4* w = reinterpret_cast<int4*>(f.items + base + q);
    __stcg(w, make_int4(b, stats ? s.job_rows[r] : j.node, r, q - r * K));
    __stcg(w + 1, w1);
    __stcg(w + 2, w2);
    if (nmask > 0) {
      __stcg(w + 3, w3);
      __stcg(w + 4, w4);
      __stcg(w + 5, w5);
      __stcg(w + 6, w6);
    }
  }
  fence_gpu();   // bodies, masks and partial resets before tags
  __syncwarp();
  // (test hook: a withheld tree's job is never published, so the waits on it
  // run out and the kernel ends through its abort path)
  if (b != f.withhold_tree)
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

// Structure, validation and gathers of tree b; leaves ctl ready to run.
template <typename L, bool kGiven>
__device__ void owner_new_tree(const TravArgs& a, const TreeSmem& s, Shared& sh, float* u,
                               int b, int lane) {
  const int R = a.N + 1, V = a.V;
  const size_t row0 = (size_t)b * R;
  const typename L::elem* logits = reinterpret_cast<const typename L::elem*>(a.logits);
  if (lane == 0) {
    sh.outstanding = 0;
    sh.ahead.ok = 0;
    Ctl& c = sh.ctl;
    c.bad = 0u;
    c.accepted = -1;
    c.node = 0;
    c.pending = -1;
    c.masked_sum = 0.0;
    c.n_tests = c.n_passes = 0;
    c.job.kind = 0;
  }
  for (int i = lane; i <= R; i += 32) u[i] = a.uniforms[row0 + b + i];
  for (int i = lane; i < R; i += 32) {
    s.par[i] = a.parents[row0 + i];
    s.tok[i] = a.tokens[row0 + i];
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
  __syncwarp();
  uint32_t bad = 0u;
  for (int i = lane; i < R; i += 32) {
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
  bad = __reduce_or_sync(0xffffffffu, bad);
  __syncwarp();
  if (bad == 0u) {
    uint32_t bad2 = 0u;
    for (int i = lane; i < R; i += 32) {
      if (s.first[i] == 0x7fffffff) s.first[i] = -1;
      int nx = -1;
      if (i > 0) {
        const int p = s.par[i], t = s.tok[i];
        for (int j = i + 1; j < R; ++j) {
          if (s.par[j] != p) continue;
          if (nx < 0) nx = j;
          if (s.tok[j] == t) bad2 |= 4u;
        }
        const size_t prow = (row0 + p) * (size_t)V;
        s.gl[i] = L::at(logits + prow, t);
        s.gq[i] = __ldg(a.draft_probs + prow + t);
        if (!(s.gq[i] > 0.f)) bad2 |= 8u;
        s.invq[i] = 1.0 / (double)s.gq[i];
      }
      s.next[i] = nx;
    }
    bad = __reduce_or_sync(0xffffffffu, bad2);
  }
  __syncwarp();
  if (kGiven && bad == 0u) {
    // given normalisers (from the LM head's epilogue): every internal row is
    // normalised up front and no stats job is ever posted
    uint32_t bad3 = 0u;
    for (int i = lane; i < R; i += 32) {
      if (s.first[i] < 0) continue;
      const float2 st = a.row_stats[row0 + i];
      s.rowm[i] = st.x;
      s.rows[i] = st.y;
      s.invs[i] = 1.0 / (double)st.y;
      if (!(st.y > 0.f)) bad3 |= 64u;
    }
    __syncwarp();
    for (int i = lane + 1; i < R; i += 32) {
      const int p = s.par[i];
      s.mb0[i] = exp2(((double)s.gl[i] - (double)s.rowm[p]) * a.c) * s.invs[p];
    }
    bad = __reduce_or_sync(0xffffffffu, bad3);
    __syncwarp();
  }
  if (lane == 0) {
    sh.ctl.bad = bad;
    if (bad == 0u) {
      s.p[0] = 1.0;
      advance(s, sh.ctl, u, a.token_level != 0);
    } else {
      sh.ctl.job.kind = kJobDone;
    }
  }
  __syncwarp();
}

// Combines the finished job's partials (sh.pbuf or global) and advances.
template <typename L>
__device__ void owner_combine(const TravArgs& a, const FlowArgs& f, const TreeSmem& s,
                              Shared& sh, const float* u, int b, int lane) {
  const int R = a.N + 1, V = a.V;
  const size_t row0 = (size_t)b * R;
  const float c_hi = a.c_hi, c_lo = a.c_lo;
  const typename L::elem* logits = reinterpret_cast<const typename L::elem*>(a.logits);
  const int K = sh.jK;
  const bool in_smem = sh.outstanding <= kPBuf;
  auto part_of = [&](int r, int k) -> float2 {
    return in_smem ? sh.pbuf[r * K + k]
                   : unpack_part(__ldcg(f.part + (row0 + r) * f.Kmax + k));
  };
  if (sh.jkind == kJobStats) {
    // the rows' normalisers from their slices, one lane per row ...
    bool bad_row = false;
    for (int r = lane; r < sh.jrows; r += 32) {
      float M = TV_NEG_INF;
      for (int k2 = 0; k2 < K; ++k2) M = fmaxf(M, part_of(r, k2).x);
      float S = 0.f;
      for (int k2 = 0; k2 < K; ++k2) {
        const float2 pk = part_of(r, k2);
        if (pk.x != TV_NEG_INF) S += pk.y * L::exp_rel(pk.x, M, c_hi, c_lo);
      }
      const int node = s.job_rows[r];
      s.rowm[node] = M;
      s.rows[node] = S;
      s.invs[node] = 1.0 / (double)S;
      bad_row |= !(S > 0.f);
    }
    if (__any_sync(0xffffffffu, bad_row) && lane == 0) sh.ctl.bad |= 64u;
    __syncwarp();
    // ... then M_b^(0) of those rows' children, one lane per node (the same
    // value children_mb0 gives, see there)
    for (int i = lane + 1; i < R; i += 32) {
      const int p = s.par[i];
      bool mine = false;
      for (int r = 0; r < sh.jrows; ++r) mine |= (s.job_rows[r] == p);
      if (mine) s.mb0[i] = exp2(((double)s.gl[i] - (double)s.rowm[p]) * a.c) * s.invs[p];
    }
    __syncwarp();
  } else if (sh.jkind == kJobPass) {
    float S = 0.f;
    for (int k2 = lane; k2 < K; k2 += 32) S += part_of(0, k2).x;
    S = warp_sum(S);
    if (lane == 0) sh.ctl.S = S;
  } else {
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
    const float target = u[R] * W;
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
        load_probs<true>(a.draft_probs + rowoff, xs, V, q);
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
    if (a.out_margin) {
      // the draw's margin (kernel sums), in the crossing slice's units, then
      // relative to the total
      float clo = lbase, chi = lbase;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        if (e == found) chi = lbase + pre[e];
        if (e + 1 == found) clo = lbase + pre[e];
      }
      const float my_margin = fminf(lt - clo, chi - lt) * scale / W;
      const float bm = hit ? __shfl_sync(0xffffffffu, my_margin, __ffs(hit) - 1) : 0.f;
      if (lane == 0) sh.ctl.bmargin = bm;
    }
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
      a.out_bonus[b] = yy;
      sh.ctl.job.kind = kJobDone;
    }
  }
  __syncwarp();
  if (lane == 0 && sh.ctl.job.kind != kJobDone) {
    if (sh.ctl.bad & 64u) sh.ctl.job.kind = kJobDone;
    else advance(s, sh.ctl, u, a.token_level != 0);
  }
  __syncwarp();
}

// Writes tree b's outputs; true if it was the last tree of the call.
template <bool kGiven>
__device__ bool owner_finish(const TravArgs& a, const FlowArgs& f, const TreeSmem& s,
                             Shared& sh, const float* u, int b, int lane) {
  const int R = a.N + 1, N = a.N;
  const size_t row0 = (size_t)b * R;
  const bool ok = (sh.ctl.bad & (15u | 32u | 64u)) == 0u;
  for (int k2 = lane; k2 < N; k2 += 32) a.out_path[(size_t)b * N + k2] = -1;
  if (a.out_node_p)
    for (int i = lane; i < R; i += 32)
      a.out_node_p[row0 + i] = ok ? s.dbgp[i] : __int_as_float(0x7fc00000);
  __syncwarp();
  int last = 0;
  if (lane == 0) {
    const int acc_node = ok ? sh.ctl.accepted : -1;
    if (acc_node >= 0) {
      int depth = 0;
      for (int j = acc_node; j != 0; j = s.par[j]) ++depth;
      int k2 = depth - 1;
      for (int j = acc_node; j != 0; j = s.par[j]) a.out_path[(size_t)b * N + (k2--)] = j;
      a.out_accept_len[b] = depth;
    } else {
      a.out_accept_len[b] = -1;
      a.out_bonus[b] = -1;
    }
    if (a.out_stats) {
      int distinct = 0;
      for (int i = 0; i < R; ++i) distinct += (s.npass[i] > 0);
      int normalised = 0;
      for (int i = 0; i < R; ++i) normalised += (s.rows[i] > 0.f);
      int32_t* o = a.out_stats + (size_t)b * 5;
      o[0] = ok ? sh.ctl.n_tests : 0;
      o[1] = ok ? sh.ctl.n_passes : 0;
      o[2] = ok ? distinct : 0;
      o[3] = (acc_node >= 0 && s.first[acc_node] < 0) ? 1 : 0;
      o[4] = (ok && !kGiven) ? normalised : 0;   // rows this call streamed
    }
    if (a.out_margin) {
      const float nan = __int_as_float(0x7fc00000);
      a.out_margin[2 * (size_t)b] = acc_node >= 0 ? test_margin_serial(s.dbgp, u, R) : nan;
      a.out_margin[2 * (size_t)b + 1] = acc_node >= 0 ? sh.ctl.bmargin : nan;
    }
    if (sh.ctl.bad) atomicOr(a.status, sh.ctl.bad);
    f.finished[b] = (unsigned)f.epoch;
    fence_gpu();
    last = (atomicAdd(&f.ctr[kCtrDone], 1u) == (unsigned)a.B - 1u) ? 1 : 0;
    sh.outstanding = 0;
  }
  return __shfl_sync(0xffffffffu, last, 0) != 0;
}

template <typename L, bool kGiven>
__device__ void owner_role(const TravArgs& a, const FlowArgs& f, const Smem& m, int lane) {
  const int R = a.N + 1, V = a.V, B = a.B;
  Shared& sh = *m.sh;
  const TreeSmem& s = m.s;
  int my_tree = -1;
  unsigned polls = 0u;
  Backoff wait;
  unsigned done_est = 0u;      // trees finished, as read after the last post
  for (;;) {
    __syncwarp();   // lane 0's updates of sh (job shape, control state) seen by all lanes
    if (my_tree < 0) {
      unsigned t = 0u;
      if (lane == 0)
        t = (ld_relaxed_u32(&f.ctr[kCtrNextTree]) < (unsigned)B)
                ? atomicAdd(&f.ctr[kCtrNextTree], 1u) : (unsigned)B;
      t = __shfl_sync(0xffffffffu, t, 0);
      if (t >= (unsigned)B) break;   // no trees left for this CTA to own
      my_tree = (int)t;
      owner_new_tree<L, kGiven>(a, s, sh, m.u, my_tree, lane);
    } else {
      // poll the own job's partials (kept in pbuf for the combine)
      const int nout = sh.outstanding;
      const int K = sh.jK;
      bool all = true;
      for (int q = lane; q < nout; q += 32) {
        const int r = q / K;
        const unsigned long long v =
            ld_relaxed_u64(f.part + ((size_t)my_tree * R + r) * f.Kmax + (q - r * K));
        if (v == kNoPart) all = false;
        else if (q < kPBuf) sh.pbuf[q] = unpack_part(v);
      }
      const bool done = __all_sync(0xffffffffu, all);
      if (!done) {
        int stop = 0;
        if (lane == 0) {
          if ((++polls & 31u) == 0u && ld_relaxed_u32(&f.ctr[kCtrAbort])) stop = 1;
          else if (!wait.idle()) {
            raise_abort(a, f);
            stop = 1;
          }
        }
        if (__shfl_sync(0xffffffffu, stop, 0)) break;
        continue;
      }
      wait.reset();
      // the bonus draw reads tiles written before its partials
      if (sh.jkind == kJobBonusLeaf || sh.jkind == kJobBonusRes) fence_gpu();
      __syncwarp();
      if (sh.jkind == kJobPass && sh.ahead.ok && sh.outstanding <= kPBuf) {
        // ---- the next step was worked out ahead: decide, post, then update ----
        float S_pass = 0.f;
        for (int k2 = lane; k2 < sh.jK; k2 += 32) S_pass += sh.pbuf[k2].x;
        S_pass = warp_sum(S_pass);
        int fast = 0, post_first = 0, accept = 0;
        if (lane == 0) {
          const Ahead& ah = sh.ahead;
          const double S = (double)S_pass + s.p[ah.i] * sh.ctl.masked_sum;
          if (S > 1e-300) {
            fast = 1;
            const double D = S + ah.omp;
            Job& jf = sh.fjob;
            jf.n_rows = 1;
            if (ah.mode == 1) {
              accept = ((double)m.u[ah.c2] * D < ah.X) ? 1 : 0;
              post_first = 1;
              if (accept) {
                jf.kind = kJobBonusLeaf;
                jf.node = ah.c2;
                jf.nmask = 0;
              } else {
                const double invD = 1.0 / D;
                jf.kind = kJobPass;
                jf.node = ah.i;
                jf.nmask = ah.nmask;
                jf.alpha1 = (float)(ah.ainvs * invD);
                jf.beta = (float)(ah.beta * invD + ah.invZn);
                jf.rowmax = s.rowm[ah.i];
              }
            } else {
              accept = ((double)m.u[ah.i] * D < S) ? 1 : 0;
              if (!accept) {   // the pass at g that rejects i is known already
                post_first = 1;
                jf.kind = kJobPass;
                jf.node = ah.g;
                jf.nmask = ah.nmask;
                jf.alpha1 = ah.alpha1_g;
                jf.beta = ah.beta_g;
                jf.rowmax = ah.rowmax_g;
              }
            }
            sh.ctl.S = S_pass;
          }
        }
        fast = __shfl_sync(0xffffffffu, fast, 0);
        if (fast) {
          post_first = __shfl_sync(0xffffffffu, post_first, 0);
          accept = __shfl_sync(0xffffffffu, accept, 0);
          __syncwarp();
          if (post_first) {
            post_job(s, sh, a, f, my_tree, V, lane, __shfl_sync(0xffffffffu, done_est, 0),
                     sh.fjob, m.mtok2, s.mask_val);
            if (lane == 0) control_step_ahead(s, sh.ctl, sh.ahead, accept != 0);
          } else {
            if (lane == 0) control_step_ahead(s, sh.ctl, sh.ahead, accept != 0);
            __syncwarp();
            post_job(s, sh, a, f, my_tree, V, lane, __shfl_sync(0xffffffffu, done_est, 0),
                     sh.ctl.job, s.mask_tok, s.mask_val);
          }
          if (lane == 0) {
            done_est = ld_relaxed_u32(&f.ctr[kCtrDone]);
            if (a.token_level) sh.ahead.ok = 0;            // (Traversal Verification only)
            else prepare_ahead(s, sh.ctl, sh.ahead, m.mtok2);   // for the job just posted
          }
          continue;
        }
      }
      owner_combine<L>(a, f, s, sh, m.u, my_tree, lane);
    }
    if (sh.ctl.job.kind == kJobDone) {
      const bool last = owner_finish<kGiven>(a, f, s, sh, m.u, my_tree, lane);
      my_tree = -1;
      if (last) {
        // every tree is done: the tickets now held (slots from the tail up to
        // the head) and the at most one more per CTA that may still be taken
        // see an exit tag instead of an item
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
    } else {
      post_job(s, sh, a, f, my_tree, V, lane, __shfl_sync(0xffffffffu, done_est, 0),
               sh.ctl.job, s.mask_tok, s.mask_val);
      if (lane == 0) {
        done_est = ld_relaxed_u32(&f.ctr[kCtrDone]);   // used at the next job
        if (a.token_level) sh.ahead.ok = 0;             // (Traversal Verification only)
        else prepare_ahead(s, sh.ctl, sh.ahead, m.mtok2);    // while this job runs
      }
    }
  }
}

// ------------------------------------------------------------- the kernel --

// kGiven: the rows' normalisers come with the call (args.row_stats), so no
// stats job is ever posted; a separate instantiation keeps the owner code of
// the common case free of that branch
template <typename L, int kNCW, bool kGiven>
__global__ void __launch_bounds__(Shape<L, kNCW>::kThreads, 16 / kNCW)
    tv_flow_kernel(TravArgs args, FlowArgs f, int n_stages) {
  using S = Shape<L, kNCW>;
  extern __shared__ __align__(128) char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t red_bar[kMaxStages];
  __shared__ __align__(8) uint64_t slot_free[kSlots];
  __shared__ __align__(8) uint64_t slot_full[kSlots];
  __shared__ Shared sh;

  const int R = args.N + 1;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  Smem m;
  m.ring = smem_raw;
  char* tree_base = smem_raw + (size_t)n_stages * S::kStageBytes;
  m.s = carve_tree_nt(tree_base, R, 0);
  m.mtok = reinterpret_cast<int*>(tree_base + ((tree_smem_bytes_nt(R, 0) + 15) & ~(size_t)15));
  m.mval = reinterpret_cast<float*>(m.mtok + kSlots * R);
  m.u = m.mval + kSlots * R;
  m.mtok2 = reinterpret_cast<int*>(m.u + R + 1);
  m.full_bar = full_bar;
  m.empty_bar = empty_bar;
  m.slot_free = slot_free;
  m.slot_full = slot_full;
  m.red_bar = red_bar;
  m.sh = &sh;

  if (tid == 0) {
    for (int k = 0; k < n_stages; ++k) {
      mbar_init(&full_bar[k], 1);
      mbar_init(&empty_bar[k], kNCW);
      mbar_init(&red_bar[k], kNCW);
    }
    for (int k = 0; k < kSlots; ++k) {
      mbar_init(&slot_free[k], kNCW);
      mbar_init(&slot_full[k], 1);
    }
    fence_mbar_init();
    sh.outstanding = 0;
  }
  __syncthreads();

  if (wid < kNCW) consumer_role<L, kNCW>(args, f, m, n_stages, wid, lane);
  else if (wid == kNCW) producer_role<L, kNCW>(args, f, m, n_stages, lane);
  else if (wid == kNCW + 1) fetcher_role<L, kNCW>(args, f, m, lane);
  else owner_role<L, kGiven>(args, f, m, lane);

  // ---------------- exit ----------------
  __syncthreads();
  if (ld_relaxed_u32(&f.ctr[kCtrAbort])) {
    // after an abort, trees that did not finish report "invalid"
    for (int b = blockIdx.x * S::kThreads + tid; b < args.B; b += gridDim.x * S::kThreads) {
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
  // bonus draw, each at most kmax slices, with a factor of two to spare; then
  // room for the exit tags
  l.cap = (size_t)B * (4 * (size_t)R + 2) * l.kmax + tvk::flow::kMaxGrid;
  l.ntiles = (size_t)((V + tvk::fused::kTileElems - 1) / tvk::fused::kTileElems);
  return l;
}

size_t up256(size_t n) { return (n + 255) & ~static_cast<size_t>(255); }

size_t flow_smem_bytes(int R, int ncw, int stages) {
  return (size_t)stages * tvk::flow::flow_stage_bytes(ncw) +
         ((tvk::fused::tree_smem_bytes_nt(R, 0) + 15) & ~(size_t)15) +
         (size_t)tvk::flow::kSlots * R * 8 + (size_t)(R + 1) * 4 + (size_t)R * 4 + 64;
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
  const FlowLayout l = flow_layout(B, R, V, plan.slice_min);
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
  f->slice_min = plan.slice_min;
  f->withhold_tree = -1;
  return (size_t)(p - static_cast<char*>(base)) <= bytes ? 0 : -4;
}

FlowPlan tv_flow_plan(int R, int B, int V, int smem_per_sm, int smem_per_block, int force_ncw,
                      int force_stages, int force_slice_pass, int force_slice_stats,
                      int force_slice_min) {
  FlowPlan p;
  // the largest slices grow with the batch: while many trees stream at once
  // every CTA is busy anyway, and larger slices mean fewer queue items,
  // partials and combines per byte (at 1024 trees of 128256 tokens, 32768-
  // token slices stream 14 % faster than 8192; at 128 trees, where a job's
  // latency sets the time, 8192 is best).  From 1024 trees a pass takes a
  // quarter row per slice and a normaliser half a row when that is larger
  // (V = 151936: 4 % faster than 32768 for both; V = 128256: 64512-token
  // normaliser slices, 4 % faster), rounded up to whole ring stages of bf16
  // rows (3072 tokens of a pass, 9216 of a normaliser with four consumer
  // warps; V = 151936: 39936 and 82944 tokens, 0.8 % faster than 38144 and
  // 76032, whose last stages were partly empty)
  if (force_ncw == 4 || force_ncw == 8) p.ncw = force_ncw;
  const long long pass_unit = tvk::flow::flow_stage_bytes(p.ncw) / 6 / 256 * 256;
  const long long row_unit = tvk::flow::flow_stage_bytes(p.ncw) / 2;
  auto up_to = [](long long x, long long unit) { return (int)((x + unit - 1) / unit * unit); };
  p.slice_pass = B >= 1024 ? std::max(32768, up_to((V + 3LL) / 4, pass_unit))
                           : (B >= 256 ? 16384 : 8192);
  p.slice_stats = B >= 1024 ? std::max(32768, up_to((V + 1LL) / 2, row_unit))
                            : (B >= 256 ? 32768 : 16384);
  if (force_slice_pass >= 256 && force_slice_pass % 256 == 0) p.slice_pass = force_slice_pass;
  if (force_slice_stats >= 256 && force_slice_stats % 256 == 0) p.slice_stats = force_slice_stats;
  if (force_slice_min >= 256 && force_slice_min % 256 == 0) p.slice_min = force_slice_min;
  p.slice_min = std::min(p.slice_min, std::min(p.slice_pass, p.slice_stats));
  const int per_sm = 16 / p.ncw;   // CTAs per SM the kernel is built for
  if (force_stages >= 2 && force_stages <= tvk::fused::kMaxStages) {
    p.stages = force_stages;
  } else {
    p.stages = 2;
    for (int st = tvk::fused::kMaxStages; st >= 2; --st)
      if ((size_t)per_sm * (flow_smem_bytes(R, p.ncw, st) + 4096) <= (size_t)smem_per_sm) {
        p.stages = st;
        break;
      }
  }
  p.smem = flow_smem_bytes(R, p.ncw, p.stages);
  p.ok = p.smem + 4096 <= (size_t)smem_per_block;
  return p;
}

namespace {

// Per device and kernel variant: the dynamic shared memory limit already set
// and the CTAs per SM for the last size asked (attribute and occupancy
// queries cost far more host time than the launch itself).
struct LaunchCache {
  size_t smem_set = 0;
  size_t occ_smem = 0;
  int per_sm = 0;
};
constexpr int kCacheDevices = 64;
std::mutex g_launch_mutex;
LaunchCache g_launch_cache[kCacheDevices][8];

}  // namespace

int tv_launch_flow(const TravArgs& a, FlowArgs f, int logit_is_bf16, const FlowPlan& plan,
                   int sm_count, cudaStream_t stream, cudaEvent_t* ev) {
  using namespace tvk::flow;
  const size_t smem = plan.smem;
  int stages = plan.stages;
  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kCacheDevices) {
    cudaGetLastError();
    return -5;
  }
  if (ev) {
    for (int k = 0; k < 3; ++k)
      if (cudaEventRecord(ev[k], stream) != cudaSuccess) return -5;
  }
  auto run = [&](auto kernel, int threads, int variant) -> int {
    int per_sm = 0;
    {
      std::lock_guard<std::mutex> lock(g_launch_mutex);
      LaunchCache& c = g_launch_cache[device][variant];
      if (smem > c.smem_set) {
        if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess) {
          cudaGetLastError();
          return -5;
        }
        c.smem_set = smem;
      }
      if (c.occ_smem != smem || c.per_sm < 1) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&c.per_sm, kernel, threads, smem) !=
            cudaSuccess) {
          cudaGetLastError();
          c.per_sm = 0;
          return -5;
        }
        c.occ_smem = smem;
      }
      per_sm = c.per_sm;
    }
    if (per_sm < 1) return -5;
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
  using tvk::Bf16Logits;
  using tvk::F32Logits;
  const int given = a.row_stats != nullptr;
  int rc;
  if (plan.ncw == 8) {
    if (logit_is_bf16)
      rc = given ? run(tv_flow_kernel<Bf16Logits, 8, true>, Shape<Bf16Logits, 8>::kThreads, 4)
                 : run(tv_flow_kernel<Bf16Logits, 8, false>, Shape<Bf16Logits, 8>::kThreads, 0);
    else
      rc = given ? run(tv_flow_kernel<F32Logits, 8, true>, Shape<F32Logits, 8>::kThreads, 5)
                 : run(tv_flow_kernel<F32Logits, 8, false>, Shape<F32Logits, 8>::kThreads, 1);
  } else {
    if (logit_is_bf16)
      rc = given ? run(tv_flow_kernel<Bf16Logits, 4, true>, Shape<Bf16Logits, 4>::kThreads, 6)
                 : run(tv_flow_kernel<Bf16Logits, 4, false>, Shape<Bf16Logits, 4>::kThreads, 2);
    else
      rc = given ? run(tv_flow_kernel<F32Logits, 4, true>, Shape<F32Logits, 4>::kThreads, 7)
                 : run(tv_flow_kernel<F32Logits, 4, false>, Shape<F32Logits, 4>::kThreads, 3);
  }
  if (rc) return rc;
  if (ev && cudaEventRecord(ev[3], stream) != cudaSuccess) return -5;
  return 0;
}
