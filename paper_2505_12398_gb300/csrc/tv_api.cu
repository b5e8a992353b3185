// tv_api.cu -- host side of the C ABI declared in include/tv.h.
//
// Argument checks happen here, before anything is queued; the kernels and
// their launch sequence live in tv_kernels.cu.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/tv.h"
#include "tv_launch.h"

struct tv_handle {
  int device = 0;
  int vocab = 0;
  int max_nodes = 0;
  int max_batch = 0;
  tv_dtype dtype = TV_BF16;
  unsigned flags = 0;
  int sm_count = 0;
  int smem_per_sm = 0;
  int smem_per_block = 0;
  int force_ncw = 0, force_c = 0, force_stages = 0;   // tuning override (TV_FUSED_PLAN)
  int flow_force[5] = {0, 0, 0, 0, 0};                 // tuning override (TV_FLOW_PLAN)
  // device workspace
  int32_t* row_list = nullptr;   // [max_batch * (max_nodes + 1)]
  int32_t* n_rows = nullptr;     // [1]
  float2* stats = nullptr;       // [max_batch * (max_nodes + 1)]
  uint32_t* status = nullptr;    // [1]
  void* flow_ws = nullptr;       // persistent kernel's queue and partials
  size_t flow_ws_bytes = 0;
  unsigned long long epoch = 0;  // per-call tag of the persistent kernel's queue
  int withhold_tree = -1;        // test hook for the next persistent call (-1: none)
  // per-(row, tile) scratch of tv_lm_head (allocated on first use)
  float2* lmh_part = nullptr;
  size_t lmh_part_bytes = 0;
  // staging for tv_verify_batch_host (allocated on first use), and the bytes
  // its last call copied each way
  char* stage = nullptr;
  size_t stage_bytes = 0;
  uint64_t host_h2d_bytes = 0, host_d2h_bytes = 0;
  // optional per-kernel timing events
  bool timing = false;
  bool timed_call = false;
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  // tv_verify_batch_host: two copy streams (a 2-D host-to-device copy on one
  // stream reaches about 60 % of the link; split over two it saturates it)
  // and the events that order them against the caller's stream
  cudaStream_t copy_st[2] = {nullptr, nullptr};
  cudaEvent_t copy_ev[3] = {nullptr, nullptr, nullptr};
};

namespace {

constexpr int kMaxRows = 1024;   // N + 1
constexpr int kMaxVocab = 1 << 28;
constexpr unsigned kPathFlags = TV_FLAG_UNFUSED | TV_FLAG_CLUSTER | TV_FLAG_PERSISTENT;

enum Path { kPathThree = 0, kPathCluster = 1, kPathPersistent = 2 };

FlowPlan flow_plan(const tv_handle* h, int R, int B) {
  return tv_flow_plan(R, B, h->vocab, h->smem_per_sm, h->smem_per_block, h->flow_force[0],
                      h->flow_force[1],
                      h->flow_force[2], h->flow_force[3], h->flow_force[4]);
}

// Smallest slice the persistent kernel may use on this handle (sizes its queue).
int flow_min_slice(const tv_handle* h) {
  const FlowPlan p = flow_plan(h, h->max_nodes + 1, h->max_batch);
  return p.slice_min;
}

// Largest vocabulary and tree for which a handle that chose its path itself
// takes the cluster path rather than the persistent kernel.
constexpr int kClusterMaxVocab = 49152;
constexpr int kClusterMaxRows = 128;

Path choose_path(const tv_handle* h, int B, int R, FusedPlan* plan) {
  if ((h->vocab % 8) != 0 || (h->flags & TV_FLAG_UNFUSED)) return kPathThree;
  if (h->flags & TV_FLAG_CLUSTER) {
    *plan = tv_fused_plan(B, R, h->vocab, h->sm_count, h->smem_per_sm, h->smem_per_block,
                          h->force_ncw, h->force_c, h->force_stages);
    return plan->ok ? kPathCluster : kPathThree;
  }
  if (!h->flow_ws || !flow_plan(h, R, B).ok) return kPathThree;
  if (!(h->flags & TV_FLAG_PERSISTENT) && h->vocab <= kClusterMaxVocab && R <= kClusterMaxRows) {
    // short rows: a job of the persistent kernel costs more to publish and
    // combine through its global queue than to stream, and one cluster per
    // tree, exchanging partials through distributed shared memory, is faster
    // (V = 32000, EAGLE-shaped trees: 13-22 % less time at 16 to 2048 trees;
    // the persistent kernel is faster from V = 128256 and on deep trees)
    *plan = tv_fused_plan(B, R, h->vocab, h->sm_count, h->smem_per_sm, h->smem_per_block,
                          h->force_ncw, h->force_c, h->force_stages);
    if (plan->ok) return kPathCluster;
  }
  return kPathPersistent;
}

class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    ok_ = cudaGetDevice(&prev_) == cudaSuccess;
    if (ok_ && prev_ != dev) ok_ = cudaSetDevice(dev) == cudaSuccess;
    switched_ = ok_ && prev_ != dev;
  }
  ~DeviceGuard() {
    if (switched_) cudaSetDevice(prev_);
  }
  bool ok() const { return ok_; }

 private:
  int prev_ = 0;
  bool ok_ = false;
  bool switched_ = false;
};

// An NVTX range named after the entry point, for timeline tools (a few
// nanoseconds when no tool is attached).
class NvtxRange {
 public:
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Copies the rows (row bytes each) of nodes with children from host to
// device.  When every tree has the same parents, each run of consecutive rows
// with children is one 2-D copy over the batch; otherwise one copy per run per
// tree.  Adds the bytes copied to *bytes.
bool copy_internal_rows(void* dst_v, const void* src_v, size_t row, const int32_t* parents,
                        int B, size_t R, const cudaStream_t* sts, int n_st, size_t* bytes) {
  char* dst = static_cast<char*>(dst_v);
  const char* src = static_cast<const char*>(src_v);
  auto rows_with_children = [&](int b, std::vector<char>& kid) {
    std::fill(kid.begin(), kid.end(), 0);
    for (size_t i = 1; i < R; ++i) {
      const int p = parents[(size_t)b * R + i];
      if (p >= 0 && (size_t)p < i) kid[p] = 1;
    }
  };
  auto runs = [&](const std::vector<char>& kid, auto&& copy) {
    for (size_t r0 = 0; r0 < R;) {
      if (!kid[r0]) {
        ++r0;
        continue;
      }
      size_t r1 = r0;
      while (r1 < R && kid[r1]) ++r1;
      if (!copy(r0, r1)) return false;
      r0 = r1;
    }
    return true;
  };
  std::vector<char> kid(R);
  bool same = true;
  for (int b = 1; b < B && same; ++b)
    same = std::memcmp(parents, parents + (size_t)b * R, R * sizeof(int32_t)) == 0;
  if (same) {
    rows_with_children(0, kid);
    const bool ok = runs(kid, [&](size_t r0, size_t r1) {
      // the batch split between the streams, one 2-D copy each
      for (int k = 0; k < n_st; ++k) {
        const size_t b0 = (size_t)B * k / n_st, b1 = (size_t)B * (k + 1) / n_st;
        if (b1 == b0) continue;
        if (cudaMemcpy2DAsync(dst + (b0 * R + r0) * row, R * row, src + (b0 * R + r0) * row,
                              R * row, (r1 - r0) * row, b1 - b0, cudaMemcpyHostToDevice,
                              sts[k]) != cudaSuccess)
          return false;
      }
      *bytes += (r1 - r0) * row * (size_t)B;
      return true;
    });
    if (ok) return true;
    cudaGetLastError();   // (a pitch beyond the 2-D limit: copy tree by tree)
  }
  for (int b = 0; b < B; ++b) {
    rows_with_children(b, kid);
    const size_t base = (size_t)b * R;
    if (!runs(kid, [&](size_t r0, size_t r1) {
          if (cudaMemcpyAsync(dst + (base + r0) * row, src + (base + r0) * row, (r1 - r0) * row,
                              cudaMemcpyHostToDevice, sts[b % n_st]) != cudaSuccess)
            return false;
          *bytes += (r1 - r0) * row;
          return true;
        }))
      return false;
  }
  return true;
}

// True while `st` is capturing a CUDA graph.
bool capturing(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return cs == cudaStreamCaptureStatusActive;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t logit_bytes(const tv_handle* h) { return h->dtype == TV_BF16 ? 2 : 4; }

int check_call(const tv_handle* h, int B, int N, const void* parents, const void* tokens,
               const void* logits, const void* drafts, float temperature,
               const void* uniforms, const void* out_path, const void* out_len,
               const void* out_bonus, bool device_arrays = true) {
  if (!h) return TV_ERR_INVALID_ARG;
  if (B < 0 || N < 0) return TV_ERR_INVALID_ARG;
  if (B > h->max_batch || N > h->max_nodes) return TV_ERR_CAPACITY;
  if (!(std::isfinite(temperature) && temperature > 0.f)) return TV_ERR_TEMPERATURE;
  if (B == 0) return TV_OK;
  if (!parents || !tokens || !logits || !drafts || !uniforms || !out_len || !out_bonus)
    return TV_ERR_INVALID_ARG;
  if (N > 0 && !out_path) return TV_ERR_INVALID_ARG;
  if (device_arrays && (!aligned16(logits) || !aligned16(drafts))) return TV_ERR_INVALID_ARG;
  return TV_OK;
}

int verify_impl(tv_handle* h, int B, int N, const int32_t* parents, const int32_t* tokens,
                const void* logits, const float* drafts, float temperature,
                const float* uniforms, int32_t* out_path, int32_t* out_len, int32_t* out_bonus,
                float* out_node_p, int32_t* out_stats, void* stream,
                const float2* row_stats = nullptr, float* out_margin = nullptr) {
  int rc = check_call(h, B, N, parents, tokens, logits, drafts, temperature, uniforms,
                      out_path, out_len, out_bonus);
  if (rc != TV_OK || B == 0) return rc;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  TravArgs a;
  a.parents = parents;
  a.tokens = tokens;
  a.logits = logits;
  a.draft_probs = drafts;
  a.uniforms = uniforms;
  a.stats = h->stats;
  a.B = B;
  a.N = N;
  a.V = h->vocab;
  const double c = 1.4426950408889634 / static_cast<double>(temperature);
  a.c_hi = static_cast<float>(c);
  a.c_lo = static_cast<float>(c - static_cast<double>(a.c_hi));
  a.c = c;
  a.out_path = out_path;
  a.out_accept_len = out_len;
  a.out_bonus = out_bonus;
  a.out_node_p = out_node_p;
  a.out_stats = out_stats;
  a.out_margin = out_margin;
  a.status = h->status;
  a.token_level = (h->flags & TV_FLAG_TOKEN_LEVEL) ? 1 : 0;
  a.row_stats = row_stats;
  const int rows = B * (N + 1);
  int grid = h->sm_count * 4;
  if (grid > rows) grid = rows;
  if (grid < 1) grid = 1;
  FusedPlan plan;
  Path path = choose_path(h, B, N + 1, &plan);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (path == kPathPersistent && capturing(st)) {
    // a launch of the persistent kernel carries the call's queue epoch, so a
    // graph must not replay it: under capture, a handle that chose the path
    // itself uses the cluster path (else the three-kernel one)
    if ((h->flags & TV_FLAG_PERSISTENT) || row_stats) return TV_ERR_INVALID_ARG;
    plan = tv_fused_plan(B, N + 1, h->vocab, h->sm_count, h->smem_per_sm, h->smem_per_block,
                         h->force_ncw, h->force_c, h->force_stages);
    path = plan.ok ? kPathCluster : kPathThree;
  }
  // given row normalisers are read by the persistent kernel only: a handle
  // that chose the cluster path itself runs them there
  if (row_stats && path == kPathCluster && !(h->flags & TV_FLAG_CLUSTER) && h->flow_ws &&
      flow_plan(h, N + 1, B).ok)
    path = kPathPersistent;
  // the three-kernel path implements Traversal Verification only
  if (path == kPathThree && a.token_level) return TV_ERR_INVALID_ARG;
  // given row normalisers are read by the persistent kernel only
  if (row_stats && path != kPathPersistent) return TV_ERR_INVALID_ARG;
  const int bf16 = h->dtype == TV_BF16 ? 1 : 0;
  cudaEvent_t* ev = h->timing ? h->ev : nullptr;
  if (path == kPathCluster) {
    rc = tv_launch_fused(a, bf16, plan, st, ev);
  } else if (path == kPathPersistent) {
    FlowArgs f;
    const FlowPlan fp = flow_plan(h, N + 1, B);
    if (tv_flow_bind(h->flow_ws, h->flow_ws_bytes, B, N + 1, h->vocab, fp, &f) != 0)
      return TV_ERR_CAPACITY;
    f.epoch = ++h->epoch;
    f.withhold_tree = h->withhold_tree;
    h->withhold_tree = -1;
    rc = tv_launch_flow(a, f, bf16, fp, h->sm_count, st, ev);
  } else {
    rc = tv_launch_all(a, bf16, h->row_list, h->n_rows, grid, st, ev);
  }
  if (rc == TV_OK && h->timing) h->timed_call = true;
  return rc;
}

}  // namespace

extern "C" {

int tv_create(tv_handle** out, int device, int vocab, int max_nodes, int max_batch,
              tv_dtype logit_dtype, unsigned flags) {
  if (!out) return TV_ERR_INVALID_ARG;
  *out = nullptr;
  if (vocab < 1 || vocab > kMaxVocab) return TV_ERR_VOCAB;
  if (max_nodes < 0 || max_nodes + 1 > kMaxRows || max_batch < 1) return TV_ERR_INVALID_ARG;
  if (logit_dtype != TV_BF16 && logit_dtype != TV_FP32) return TV_ERR_INVALID_ARG;
  if ((flags & ~(kPathFlags | TV_FLAG_TOKEN_LEVEL)) ||
      __builtin_popcount(flags & kPathFlags) > 1)
    return TV_ERR_INVALID_ARG;
  // the token-level method runs on the single-kernel paths only
  if ((flags & TV_FLAG_TOKEN_LEVEL) && ((flags & TV_FLAG_UNFUSED) || (vocab % 8) != 0))
    return TV_ERR_INVALID_ARG;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, device) != cudaSuccess) return TV_ERR_CUDA;
  if (prop.major < 10) return TV_ERR_DEVICE;
  const size_t smem = tv_traverse_smem_bytes(max_nodes + 1, vocab);
  if (smem > static_cast<size_t>(prop.sharedMemPerBlockOptin)) return TV_ERR_VOCAB;

  tv_handle* h = new (std::nothrow) tv_handle;
  if (!h) return TV_ERR_CUDA;
  h->device = device;
  h->vocab = vocab;
  h->max_nodes = max_nodes;
  h->max_batch = max_batch;
  h->dtype = logit_dtype;
  h->flags = flags;
  h->sm_count = prop.multiProcessorCount;
  h->smem_per_sm = (int)prop.sharedMemPerMultiprocessor;
  h->smem_per_block = (int)prop.sharedMemPerBlockOptin;
  // TV_FUSED_PLAN="ncw,cluster,stages" overrides the fused kernel's launch
  // shape (tuning only; invalid values are ignored)
  if (const char* env = std::getenv("TV_FUSED_PLAN"))
    std::sscanf(env, "%d,%d,%d", &h->force_ncw, &h->force_c, &h->force_stages);
  // TV_FLOW_PLAN="ncw,stages,slice_pass,slice_stats,slice_min" does the same
  // for the persistent kernel
  if (const char* env = std::getenv("TV_FLOW_PLAN"))
    std::sscanf(env, "%d,%d,%d,%d,%d", &h->flow_force[0], &h->flow_force[1], &h->flow_force[2],
                &h->flow_force[3], &h->flow_force[4]);
  DeviceGuard guard(device);
  if (!guard.ok()) {
    delete h;
    return TV_ERR_CUDA;
  }
  const size_t rows = static_cast<size_t>(max_batch) * (max_nodes + 1);
  bool ok = cudaMalloc(&h->row_list, rows * sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&h->n_rows, sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&h->stats, rows * sizeof(float2)) == cudaSuccess &&
            cudaMalloc(&h->status, sizeof(uint32_t)) == cudaSuccess &&
            cudaMemset(h->status, 0, sizeof(uint32_t)) == cudaSuccess;
  if (ok && (vocab % 8) == 0 && !(flags & (TV_FLAG_UNFUSED | TV_FLAG_CLUSTER))) {
    // the queue's publication tags start at zero; calls use epochs 1, 2, ...
    // the queue is sized for the smallest slice; for very large handles the
    // smallest slice grows until the workspace stays within 1 GiB
    // (bounded by the pass slice of the smallest batches, so that every call's
    // slices stay at or above the size the queue was built for)
    const FlowPlan fp = flow_plan(h, max_nodes + 1, 1);
    int min_slice = fp.slice_min;
    while (tv_flow_workspace_bytes(max_batch, max_nodes + 1, vocab, min_slice) > (1ull << 30) &&
           min_slice < fp.slice_pass)
      min_slice *= 2;
    h->flow_force[4] = min_slice;
    h->flow_ws_bytes = tv_flow_workspace_bytes(max_batch, max_nodes + 1, vocab,
                                               flow_min_slice(h));
    ok = cudaMalloc(&h->flow_ws, h->flow_ws_bytes) == cudaSuccess &&
         cudaMemset(h->flow_ws, 0, h->flow_ws_bytes) == cudaSuccess;
  }
  if (!ok) {
    cudaGetLastError();
    tv_destroy(h);
    return TV_ERR_CUDA;
  }
  *out = h;
  return TV_OK;
}

int tv_verify_batch(tv_handle* h, int B, int N, const int32_t* parents,
                    const int32_t* draft_tokens, const void* target_logits,
                    const float* draft_probs, float temperature, const float* uniforms,
                    int32_t* out_accepted_path, int32_t* out_accept_len,
                    int32_t* out_bonus_token, void* cuda_stream) {
  NvtxRange range("tv_verify_batch");
  return verify_impl(h, B, N, parents, draft_tokens, target_logits, draft_probs, temperature,
                     uniforms, out_accepted_path, out_accept_len, out_bonus_token, nullptr,
                     nullptr, cuda_stream);
}

int tv_verify_batch_debug(tv_handle* h, int B, int N, const int32_t* parents,
                          const int32_t* draft_tokens, const void* target_logits,
                          const float* draft_probs, float temperature,
                          const float* uniforms, int32_t* out_accepted_path,
                          int32_t* out_accept_len, int32_t* out_bonus_token,
                          float* out_node_p, int32_t* out_stats, float* out_margin,
                          void* cuda_stream) {
  NvtxRange range("tv_verify_batch_debug");
  return verify_impl(h, B, N, parents, draft_tokens, target_logits, draft_probs, temperature,
                     uniforms, out_accepted_path, out_accept_len, out_bonus_token, out_node_p,
                     out_stats, cuda_stream, nullptr, out_margin);
}

int tv_verify_batch_host(tv_handle* h, int B, int N, const int32_t* parents,
                         const int32_t* draft_tokens, const void* target_logits,
                         const float* draft_probs, float temperature,
                         const float* uniforms, int32_t* out_accepted_path,
                         int32_t* out_accept_len, int32_t* out_bonus_token,
                         void* cuda_stream) {
  NvtxRange range("tv_verify_batch_host");
  int rc = check_call(h, B, N, parents, draft_tokens, target_logits, draft_probs, temperature,
                      uniforms, out_accepted_path, out_accept_len, out_bonus_token, false);
  if (rc != TV_OK || B == 0) return rc;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const size_t R = static_cast<size_t>(N) + 1;
  const size_t V = static_cast<size_t>(h->vocab);
  const size_t n_tree = static_cast<size_t>(B) * R * sizeof(int32_t);
  const size_t n_logit = static_cast<size_t>(B) * R * V * logit_bytes(h);
  const size_t n_draft = static_cast<size_t>(B) * R * V * sizeof(float);
  const size_t n_unif = static_cast<size_t>(B) * (R + 1) * sizeof(float);
  const size_t n_path = static_cast<size_t>(B) * N * sizeof(int32_t);
  const size_t n_out = static_cast<size_t>(B) * sizeof(int32_t);
  auto up = [](size_t x) { return (x + 255) & ~static_cast<size_t>(255); };
  const size_t need = up(n_logit) + up(n_draft) + 2 * up(n_tree) + up(n_unif) + up(n_path) +
                      2 * up(n_out);
  if (need > h->stage_bytes) {
    // sized for the handle's limits so that later calls never reallocate
    const size_t Rm = static_cast<size_t>(h->max_nodes) + 1;
    const size_t Bm = static_cast<size_t>(h->max_batch);
    const size_t cap = up(Bm * Rm * V * logit_bytes(h)) + up(Bm * Rm * V * 4) +
                       2 * up(Bm * Rm * 4) + up(Bm * (Rm + 1) * 4) + up(Bm * (Rm - 1) * 4) +
                       2 * up(Bm * 4);
    if (h->stage) cudaFree(h->stage);
    h->stage = nullptr;
    h->stage_bytes = 0;
    if (cudaMalloc(&h->stage, cap) != cudaSuccess) {
      cudaGetLastError();
      return TV_ERR_CUDA;
    }
    // every staged row starts defined: rows a call does not copy (leaves'
    // logit rows) then hold zeros or an earlier call's values, never garbage
    if (cudaMemset(h->stage, 0, cap) != cudaSuccess) {
      cudaGetLastError();
      cudaFree(h->stage);
      h->stage = nullptr;
      return TV_ERR_CUDA;
    }
    h->stage_bytes = cap;
  }
  char* p = h->stage;
  void* d_logit = p; p += up(n_logit);
  float* d_draft = reinterpret_cast<float*>(p); p += up(n_draft);
  int32_t* d_par = reinterpret_cast<int32_t*>(p); p += up(n_tree);
  int32_t* d_tok = reinterpret_cast<int32_t*>(p); p += up(n_tree);
  float* d_unif = reinterpret_cast<float*>(p); p += up(n_unif);
  int32_t* d_path = reinterpret_cast<int32_t*>(p); p += up(n_path);
  int32_t* d_len = reinterpret_cast<int32_t*>(p); p += up(n_out);
  int32_t* d_bonus = reinterpret_cast<int32_t*>(p);
  // Only rows the verification can need are copied: the logit and draft rows
  // of nodes with children.  Of the leaves' logit rows at most one per tree is
  // needed -- the accepted leaf's, for the bonus draw -- so the verification
  // runs first (its draw at a leaf then reads a stale row), and then only the
  // accepted leaves' rows are copied and their bonus tokens drawn again by
  // tv_launch_leaf_bonus.
  const bool two_phase = tv_leaf_bonus_smem_bytes(h->vocab) <= 48 * 1024;
  const size_t lrow = V * logit_bytes(h);
  size_t logit_copied = 0, draft_bytes = 0;
  bool ok = cudaMemcpyAsync(d_par, parents, n_tree, cudaMemcpyHostToDevice, st) == cudaSuccess &&
            cudaMemcpyAsync(d_tok, draft_tokens, n_tree, cudaMemcpyHostToDevice, st) == cudaSuccess &&
            cudaMemcpyAsync(d_unif, uniforms, n_unif, cudaMemcpyHostToDevice, st) == cudaSuccess;
  // the row copies run on the handle's two copy streams, after everything
  // queued on st so far and before the verification that follows on st
  if (!h->copy_st[0]) {
    for (int k = 0; k < 2; ++k)
      ok = ok && cudaStreamCreateWithFlags(&h->copy_st[k], cudaStreamNonBlocking) == cudaSuccess;
    for (int k = 0; k < 3; ++k)
      ok = ok && cudaEventCreateWithFlags(&h->copy_ev[k], cudaEventDisableTiming) == cudaSuccess;
  }
  ok = ok && cudaEventRecord(h->copy_ev[0], st) == cudaSuccess &&
       cudaStreamWaitEvent(h->copy_st[0], h->copy_ev[0], 0) == cudaSuccess &&
       cudaStreamWaitEvent(h->copy_st[1], h->copy_ev[0], 0) == cudaSuccess;
  if (two_phase) {
    ok = ok && copy_internal_rows(d_logit, target_logits, lrow, parents, B, R, h->copy_st, 2,
                                  &logit_copied);
  } else {
    ok = ok && cudaMemcpyAsync(d_logit, target_logits, n_logit, cudaMemcpyHostToDevice, st) ==
                   cudaSuccess;
    logit_copied = n_logit;
  }
  ok = ok && copy_internal_rows(d_draft, draft_probs, V * sizeof(float), parents, B, R,
                                h->copy_st, 2, &draft_bytes);
  ok = ok && cudaEventRecord(h->copy_ev[1], h->copy_st[0]) == cudaSuccess &&
       cudaEventRecord(h->copy_ev[2], h->copy_st[1]) == cudaSuccess &&
       cudaStreamWaitEvent(st, h->copy_ev[1], 0) == cudaSuccess &&
       cudaStreamWaitEvent(st, h->copy_ev[2], 0) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  rc = verify_impl(h, B, N, d_par, d_tok, d_logit, d_draft, temperature, d_unif, d_path, d_len,
                   d_bonus, nullptr, nullptr, cuda_stream);
  if (rc != TV_OK) return rc;
  ok = (N == 0 || cudaMemcpyAsync(out_accepted_path, d_path, n_path, cudaMemcpyDeviceToHost, st) ==
                      cudaSuccess) &&
       cudaMemcpyAsync(out_accept_len, d_len, n_out, cudaMemcpyDeviceToHost, st) == cudaSuccess &&
       cudaMemcpyAsync(out_bonus_token, d_bonus, n_out, cudaMemcpyDeviceToHost, st) == cudaSuccess &&
       cudaStreamSynchronize(st) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  size_t leaf_bytes = 0, pend_bytes = 0;
  if (two_phase) {
    // trees whose accepted node has no children: (tree, that node's row)
    std::vector<int2> pend;
    for (int b = 0; b < B; ++b) {
      const int tau = out_accept_len[b];
      if (tau < 0) continue;   // an invalid tree
      const int acc = tau > 0 ? out_accepted_path[(size_t)b * N + tau - 1] : 0;
      if (acc < 0 || (size_t)acc >= R) continue;
      bool leaf = true;
      for (size_t i = (size_t)acc + 1; i < R && leaf; ++i)
        leaf = parents[(size_t)b * R + i] != acc;
      if (leaf) pend.push_back(make_int2(b, acc));
    }
    if (!pend.empty()) {
      for (const int2& q : pend) {
        const size_t off = ((size_t)q.x * R + (size_t)q.y) * lrow;
        if (cudaMemcpyAsync(static_cast<char*>(d_logit) + off,
                            static_cast<const char*>(target_logits) + off, lrow,
                            cudaMemcpyHostToDevice, st) != cudaSuccess) {
          cudaGetLastError();
          return TV_ERR_CUDA;
        }
        leaf_bytes += lrow;
      }
      // the (tree, row) list is staged in the row-statistics buffer of the
      // three-kernel path ([max_batch (max_nodes + 1)] float2 >= B int2),
      // which no kernel reads once the verification above has finished
      int2* d_pend = reinterpret_cast<int2*>(h->stats);
      pend_bytes = pend.size() * sizeof(int2);
      const double c = 1.4426950408889634 / static_cast<double>(temperature);
      const float c_hi = static_cast<float>(c);
      const float c_lo = static_cast<float>(c - static_cast<double>(c_hi));
      ok = cudaMemcpyAsync(d_pend, pend.data(), pend_bytes, cudaMemcpyHostToDevice, st) ==
               cudaSuccess &&
           tv_launch_leaf_bonus(d_logit, h->dtype == TV_BF16 ? 1 : 0, d_unif, d_pend,
                                static_cast<int>(pend.size()), B, static_cast<int>(R),
                                h->vocab, c_hi, c_lo, d_bonus, st) == 0 &&
           cudaMemcpyAsync(out_bonus_token, d_bonus, n_out, cudaMemcpyDeviceToHost, st) ==
               cudaSuccess &&
           cudaStreamSynchronize(st) == cudaSuccess;
      if (!ok) {
        cudaGetLastError();
        return TV_ERR_CUDA;
      }
    }
  }
  h->host_h2d_bytes = 2 * n_tree + n_unif + logit_copied + draft_bytes + leaf_bytes + pend_bytes;
  h->host_d2h_bytes = (N > 0 ? n_path : 0) + 2 * n_out + (pend_bytes ? n_out : 0);
  return TV_OK;
}

int tv_last_host_copy_bytes(tv_handle* h, uint64_t* h2d, uint64_t* d2h) {
  if (!h) return TV_ERR_INVALID_ARG;
  if (h2d) *h2d = h->host_h2d_bytes;
  if (d2h) *d2h = h->host_d2h_bytes;
  return TV_OK;
}

int tv_verify_batch_stats(tv_handle* h, int B, int N, const int32_t* parents,
                          const int32_t* draft_tokens, const void* target_logits,
                          const float* draft_probs, float temperature, const float* uniforms,
                          const float* row_stats, int32_t* out_accepted_path,
                          int32_t* out_accept_len, int32_t* out_bonus_token, float* out_node_p,
                          int32_t* out_stats, void* cuda_stream) {
  NvtxRange range("tv_verify_batch_stats");
  if (!row_stats || (reinterpret_cast<uintptr_t>(row_stats) & 7u)) return TV_ERR_INVALID_ARG;
  return verify_impl(h, B, N, parents, draft_tokens, target_logits, draft_probs, temperature,
                     uniforms, out_accepted_path, out_accept_len, out_bonus_token, out_node_p,
                     out_stats, cuda_stream, reinterpret_cast<const float2*>(row_stats));
}

int tv_lm_head(tv_handle* h, int M, int K, const void* hidden, const void* weight,
               float temperature, void* out_logits, float* out_row_stats, void* cuda_stream) {
  NvtxRange range("tv_lm_head");
  if (!h || M < 0 || K < 64 || (K % 64) != 0) return TV_ERR_INVALID_ARG;
  if (h->dtype != TV_BF16 || (h->vocab % 8) != 0) return TV_ERR_INVALID_ARG;
  if ((size_t)M > (size_t)h->max_batch * (h->max_nodes + 1)) return TV_ERR_CAPACITY;
  if (!(std::isfinite(temperature) && temperature > 0.f)) return TV_ERR_TEMPERATURE;
  if (M == 0) return TV_OK;
  if (!hidden || !weight || !out_logits || !out_row_stats || !aligned16(hidden) ||
      !aligned16(weight) || !aligned16(out_logits) ||
      (reinterpret_cast<uintptr_t>(out_row_stats) & 7u))
    return TV_ERR_INVALID_ARG;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  const size_t need = (size_t)h->max_batch * (h->max_nodes + 1) *
                      (size_t)tv_lm_head_tiles(h->vocab) * sizeof(float2);
  if (h->lmh_part_bytes < need) {
    if (h->lmh_part) cudaFree(h->lmh_part);
    h->lmh_part = nullptr;
    h->lmh_part_bytes = 0;
    if (cudaMalloc(&h->lmh_part, need) != cudaSuccess) {
      cudaGetLastError();
      return TV_ERR_CUDA;
    }
    h->lmh_part_bytes = need;
  }
  const double c = 1.4426950408889634 / static_cast<double>(temperature);
  const float c_hi = static_cast<float>(c);
  const float c_lo = static_cast<float>(c - static_cast<double>(c_hi));
  const int rc = tv_launch_lm_head(hidden, weight, M, K, h->vocab, c_hi, c_lo, out_logits,
                                   h->lmh_part, reinterpret_cast<float2*>(out_row_stats),
                                   h->status, static_cast<cudaStream_t>(cuda_stream));
  return rc == 0 ? TV_OK : TV_ERR_CUDA;
}

int tv_draft_children(tv_handle* h, int B, int N, const int32_t* parents,
                      const float* draft_probs, const float* uniforms, int32_t* out_tokens,
                      void* cuda_stream) {
  NvtxRange range("tv_draft_children");
  if (!h || B < 0 || N < 0) return TV_ERR_INVALID_ARG;
  if (B > h->max_batch || N > h->max_nodes) return TV_ERR_CAPACITY;
  if (tv_draft_smem_bytes(N, h->vocab) > 48u * 1024u) return TV_ERR_VOCAB;
  if (B == 0) return TV_OK;
  if (!parents || !draft_probs || !uniforms || !out_tokens ||
      (reinterpret_cast<uintptr_t>(draft_probs) & 3u))
    return TV_ERR_INVALID_ARG;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  const int rc = tv_launch_draft(parents, draft_probs, uniforms, out_tokens, B, N, h->vocab,
                                 h->status, static_cast<cudaStream_t>(cuda_stream));
  return rc == 0 ? TV_OK : TV_ERR_CUDA;
}

int tv_debug_withhold_job(tv_handle* h, int tree) {
  if (!h || tree < 0 || tree >= h->max_batch) return TV_ERR_INVALID_ARG;
  h->withhold_tree = tree;
  return TV_OK;
}

int tv_get_status(tv_handle* h, uint32_t* status) {
  if (!h || !status) return TV_ERR_INVALID_ARG;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  uint32_t v = 0;
  if (cudaDeviceSynchronize() != cudaSuccess ||
      cudaMemcpy(&v, h->status, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemset(h->status, 0, sizeof(uint32_t)) != cudaSuccess) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  *status = v;
  return TV_OK;
}

int tv_set_phase_timing(tv_handle* h, int enable) {
  if (!h) return TV_ERR_INVALID_ARG;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  if (enable && !h->ev[0]) {
    for (int k = 0; k < 4; ++k) {
      if (cudaEventCreate(&h->ev[k]) != cudaSuccess) {
        cudaGetLastError();
        return TV_ERR_CUDA;
      }
    }
  }
  h->timing = enable != 0;
  h->timed_call = false;
  return TV_OK;
}

int tv_last_phase_ms(tv_handle* h, float* ms) {
  if (!h || !ms || !h->timing || !h->timed_call) return TV_ERR_INVALID_ARG;
  DeviceGuard guard(h->device);
  if (!guard.ok()) return TV_ERR_CUDA;
  if (cudaEventSynchronize(h->ev[3]) != cudaSuccess) return TV_ERR_CUDA;
  for (int k = 0; k < 3; ++k) {
    if (cudaEventElapsedTime(&ms[k], h->ev[k], h->ev[k + 1]) != cudaSuccess) {
      cudaGetLastError();
      return TV_ERR_CUDA;
    }
  }
  return TV_OK;
}

int tv_launch_shape(tv_handle* h, int B, int N, int* path, int* cluster, int* warps,
                    int* stages) {
  if (!h || B < 0 || N < 0) return TV_ERR_INVALID_ARG;
  if (B > h->max_batch || N > h->max_nodes) return TV_ERR_CAPACITY;
  FusedPlan plan;
  const Path p = choose_path(h, B, N + 1, &plan);
  if (path) *path = (int)p;
  if (cluster) *cluster = (p == kPathCluster) ? plan.C : 1;
  const FlowPlan fp = flow_plan(h, N + 1, B);
  if (warps) *warps = (p == kPathCluster) ? plan.ncw : (p == kPathPersistent ? fp.ncw : 16);
  if (stages)
    *stages = (p == kPathCluster) ? plan.stages : (p == kPathPersistent ? fp.stages : 0);
  return TV_OK;
}

int tv_destroy(tv_handle* h) {
  if (!h) return TV_ERR_INVALID_ARG;
  {
    DeviceGuard guard(h->device);
    if (guard.ok()) cudaDeviceSynchronize();
    for (int k = 0; k < 4; ++k)
      if (h->ev[k]) cudaEventDestroy(h->ev[k]);
    for (int k = 0; k < 2; ++k)
      if (h->copy_st[k]) cudaStreamDestroy(h->copy_st[k]);
    for (int k = 0; k < 3; ++k)
      if (h->copy_ev[k]) cudaEventDestroy(h->copy_ev[k]);
    cudaFree(h->row_list);
    cudaFree(h->n_rows);
    cudaFree(h->stats);
    cudaFree(h->status);
    if (h->flow_ws) cudaFree(h->flow_ws);
    if (h->stage) cudaFree(h->stage);
    if (h->lmh_part) cudaFree(h->lmh_part);
    cudaGetLastError();
  }
  delete h;
  return TV_OK;
}

const char* tv_strerror(int code) {
  switch (code) {
    case TV_OK: return "success";
    case TV_ERR_INVALID_ARG: return "invalid argument (null pointer, bad size or flag, misaligned array)";
    case TV_ERR_TEMPERATURE: return "temperature must be finite and > 0";
    case TV_ERR_VOCAB: return "vocabulary size out of range for this device";
    case TV_ERR_CAPACITY: return "batch or node count above the handle's limits";
    case TV_ERR_CUDA: return "CUDA runtime error";
    case TV_ERR_DEVICE: return "unsupported device (needs compute capability 10.x or newer)";
    default: return "unknown error code";
  }
}

int tv_version(void) { return 100; }

}  // extern "C"
