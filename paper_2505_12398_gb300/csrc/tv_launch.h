// tv_launch.h -- internal interface between the host API and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

struct TravArgs {
  const int32_t* parents;      // [B][N+1]
  const int32_t* tokens;       // [B][N+1]
  const void* logits;          // [B][N+1][V] bf16 or fp32
  const float* draft_probs;    // [B][N+1][V]
  const float* uniforms;       // [B][N+2]
  float2* stats;               // [B][N+1] row (max, sum of exp2) of internal rows
  int B, N, V;
  float c_hi, c_lo;            // log2(e) / temperature = c_hi + c_lo
  double c;                    // the same constant in float64
  int32_t* out_path;           // [B][N]
  int32_t* out_accept_len;     // [B]
  int32_t* out_bonus;          // [B]
  float* out_node_p;           // [B][N+1] or nullptr
  int32_t* out_stats;          // [B][5] or nullptr
  float* out_margin;           // [B][2] decision margins (test, bonus) or nullptr
  uint32_t* status;            // status word (OR of TV_STATUS_* bits)
  int token_level;             // 1: token-level (top-down) verification instead (fused paths)
  const float2* row_stats;     // [B][N+1] given row normalisers (max, sum), or nullptr
                               // (persistent path)
};

// The bonus draws at accepted original leaves, one CTA per entry of pending
// ((tree, leaf row) pairs, n_pending <= B): writes out_bonus[tree] (-1 for a
// row without a finite logit).  0, -1 (bad count), -3 (vocabulary too large for
// one CTA's tile sums) or -5 (launch failed).
int tv_launch_leaf_bonus(const void* logits, int logit_is_bf16, const float* uniforms,
                         const int2* pending, int n_pending, int B, int R, int V, float c_hi,
                         float c_lo, int32_t* out_bonus, cudaStream_t stream);
size_t tv_leaf_bonus_smem_bytes(int V);

// Launch plan of the fused kernel: cluster size, ring stages, shared memory.
struct FusedPlan {
  int ncw = 8;       // consumer warps per CTA (4 or 8)
  int C = 1;
  int stages = 0;
  size_t smem = 0;
  bool ok = false;
};

FusedPlan tv_fused_plan(int B, int R, int V, int sm_count, int smem_per_sm, int smem_per_block,
                        int force_ncw, int force_c, int force_stages);

// Queues the fused kernel (one cluster of plan.C CTAs per tree).  Requires
// V % 8 == 0 (16-byte aligned rows for the bulk copies).  With `events`,
// events[0..2] are recorded before and events[3] after it.
int tv_launch_fused(const TravArgs& a, int logit_is_bf16, const FusedPlan& plan,
                    cudaStream_t stream, cudaEvent_t* events);

// Dynamic shared memory the traversal kernel needs for R = N+1 rows.
size_t tv_traverse_smem_bytes(int R, int V);

// Queues the three kernels on `stream`; 0 on success, TV_ERR_CUDA otherwise.
// With `events` non-null, events[0..3] are recorded before the first kernel,
// between the kernels and after the last one.
int tv_launch_all(const TravArgs& a, int logit_is_bf16, int* row_list, int* n_rows,
                  int stats_grid, cudaStream_t stream, cudaEvent_t* events);

// ---- persistent load-balanced kernel (tv_flow.cu) ----

// One slot of the persistent kernel's work queue: a slice of one tree's
// current vocabulary job, self-contained (with up to kFlowInlineMask removed
// tokens) so that a claim is one 128-byte read.
constexpr int kFlowInlineMask = 8;
struct __align__(128) FlowItem {
  int tree, node, row, slice;   // tree, target row, row index within the job, slice
  int kind, slice_len, nmask, pad0;
  float alpha1, beta, rowmax, pad1;
  int mtok[kFlowInlineMask];    // first removed tokens of the row (ascending)
  float mval[kFlowInlineMask];  // their stored masses
  unsigned long long tag;       // epoch << 32 | slot, stored after the rest
  unsigned long long pad2;
};

// Device workspace of the persistent kernel (carved by tv_flow_bind).
struct FlowArgs {
  unsigned* ctr;                 // queue tail, head, trees done, next tree, abort, CTAs out
                                 // (zero between calls: the last CTA out resets them)
  FlowItem* items;               // [cap] queue slots
  int* job_mtok;                 // [B][R] removed tokens of a tree's current job row
  float* job_mval;               // [B][R] their stored masses (bonus residual)
  unsigned long long* part;      // [B][R][Kmax] partial (x, y) per (row, slice); all ones
                                 // until the slice is done
  unsigned* finished;            // [B] epoch of the call that finished the tree
  float2* tiles;                 // [B][ntiles] per-tile sums of the bonus draw
  unsigned long long epoch;      // differs between calls sharing the workspace
  int cap, R, Kmax, ntiles;
  int slice_pass, slice_stats;   // largest tokens per slice (multiples of 256)
  int slice_min;                 // smallest tokens per slice (multiple of 256)
  int withhold_tree;             // test hook: this tree's jobs are never published (-1: none)
};

// Launch shape of the persistent kernel.
struct FlowPlan {
  int ncw = 4;                   // consumer warps per CTA (4 or 8)
  int stages = 3;                // ring stages of 3 KB per consumer warp
  int slice_pass = 8192;         // largest slice of a pass / bonus draw (tokens; by batch)
  int slice_stats = 16384;       // largest slice of a row normaliser (tokens; by batch)
  int slice_min = 2048;          // slices shrink to this as fewer trees remain
  size_t smem = 0;
  bool ok = false;
};

// Default plan for R = N+1 rows and B trees (tuning overrides: force_* > 0).
FlowPlan tv_flow_plan(int R, int B, int V, int smem_per_sm, int smem_per_block, int force_ncw,
                      int force_stages, int force_slice_pass, int force_slice_stats,
                      int force_slice_min);
// Workspace for slices of at least `min_slice` tokens.
size_t tv_flow_workspace_bytes(int B, int R, int V, int min_slice);
// Carves the workspace; 0 on success, TV_ERR_CAPACITY if `bytes` is too small.
int tv_flow_bind(void* base, size_t bytes, int B, int R, int V, const FlowPlan& plan,
                 FlowArgs* f);
// Queues the cooperative persistent kernel.  The workspace must have been
// zeroed once before the first call.  Requires V % 8 == 0.  `events` as for
// tv_launch_fused.
int tv_launch_flow(const TravArgs& a, FlowArgs f, int logit_is_bf16, const FlowPlan& plan,
                   int sm_count, cudaStream_t stream, cudaEvent_t* events);

// ---- LM head fused with the row normalisers (tv_gemm.cu) ----

// Tiles of 256 logits per row (the per-row workspace of tv_launch_lm_head).
int tv_lm_head_tiles(int V);
// logits[M][V] (bf16) = hidden[M][K] x weight[V][K]^T (bf16) on the tensor
// cores, and row_stats[M] = (max, sum of 2^((l - max) (c_hi + c_lo))) of the
// stored logits.  part is [M][tv_lm_head_tiles(V)] scratch.  Requires K % 64
// == 0, V % 8 == 0 and 16-byte aligned arrays.  0 on success, -5 on a CUDA
// or tensor-map error.
int tv_launch_lm_head(const void* hidden, const void* weight, int M, int K, int V, float c_hi,
                      float c_lo, void* logits, float2* part, float2* row_stats,
                      uint32_t* status, cudaStream_t stream);

// Dynamic shared memory of one drafting CTA (tv_launch_draft) for N, V.
size_t tv_draft_smem_bytes(int N, int V);
// tokens[B][N+1]: every node's token drawn from its parent's draft row without
// the tokens of its earlier siblings (Definition 1), uniforms[b][c] for node c;
// one CTA per (tree, row).  0 or -5 (launch failed).
int tv_launch_draft(const int32_t* parents, const float* drafts, const float* uniforms,
                    int32_t* tokens, int B, int N, int V, uint32_t* status, cudaStream_t stream);

