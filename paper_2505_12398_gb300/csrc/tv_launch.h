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
  int32_t* out_stats;          // [B][4] or nullptr
  uint32_t* status;            // status word (OR of TV_STATUS_* bits)
};

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
