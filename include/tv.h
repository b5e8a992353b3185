/*
 * tv.h -- C ABI of the GB300 batched Traversal Verification library.
 *
 * Traversal Verification (arXiv 2505.12398, §3.1, Algorithm 3) verifies a
 * speculative-decoding draft token tree against the target model from the
 * leaves towards the root and accepts whole root-to-node sequences.  Given a
 * decoding tree T (Definition 1, §3.3), the draft distributions M_s(.|X^i) of
 * its non-leaf nodes and the target distributions M_b(.|X^i) of all its
 * nodes, it returns an accepted chain X^tau and one more token Y whose joint
 * law is the target model's (Definition 2, Theorem 1).  This library runs
 * that algorithm for a batch of independent trees on one GPU.
 *
 * Conventions shared by every call:
 *   - B trees, each with N draft nodes plus the root: N+1 rows per tree.
 *     Row 0 is the root (the prefix X_0); rows 1..N are draft nodes.
 *   - Every array pointer is a DEVICE pointer owned by the caller (except in
 *     tv_verify_batch_host).  The library never frees or retains it.
 *   - Layouts are dense, row-major, with no padding: [B][N+1] for tree
 *     arrays, [B][N+1][V] for the per-row distributions, [B][N+2] for the
 *     uniforms.  Distribution arrays must start on a 16-byte boundary.
 *   - All work is queued on the caller's CUDA stream (a cudaStream_t passed
 *     as void*; NULL = the legacy default stream).  Calls return as soon as
 *     the work is queued; nothing in the library synchronises the host
 *     except tv_get_status and tv_verify_batch_host.
 *   - Return values: 0 on success, a negative TV_ERR_* code otherwise.  Bad
 *     arguments are caught on the host before anything is launched.  Bad
 *     trees are found on the device: that tree's outputs are set to -1 and a
 *     TV_STATUS_* bit is raised in the handle's status word.
 *   - A handle owns its device workspace and may serve one stream at a time:
 *     calls on different streams that may overlap need different handles.
 */
#ifndef TV_H_
#define TV_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct tv_handle tv_handle;

/* Element type of the target logits. */
typedef enum { TV_BF16 = 0, TV_FP32 = 1 } tv_dtype;

/* Return codes. */
enum {
  TV_OK = 0,
  TV_ERR_INVALID_ARG = -1, /* null pointer, negative size, bad flag, misaligned array */
  TV_ERR_TEMPERATURE = -2, /* temperature not finite and > 0 (the method samples; §G) */
  TV_ERR_VOCAB = -3,       /* vocabulary size out of range */
  TV_ERR_CAPACITY = -4,    /* B or N above what the handle was created for */
  TV_ERR_CUDA = -5,        /* a CUDA runtime call failed (no device, launch error, ...) */
  TV_ERR_DEVICE = -6       /* the handle's device is not a supported GPU */
};

/* Device-side status bits, OR-ed into the handle's status word. */
enum {
  TV_STATUS_BAD_TREE = 1u,     /* parents[b][0] != -1 or parents[b][i] not in [0, i) */
  TV_STATUS_BAD_TOKEN = 2u,    /* a draft token outside [0, V) */
  TV_STATUS_DUP_SIBLING = 4u,  /* two siblings carry the same token (Definition 1
                                  draws children without replacement) */
  TV_STATUS_ZERO_DRAFT = 8u,   /* a drafted token has zero draft probability at its
                                  parent, so it cannot have come from M_s */
  TV_STATUS_DEGENERATE = 16u,  /* informational: S = 0 occurred in Eqs. (1)/(3); the
                                  0/0 was resolved as p' = 0 (p < 1) or p' = 1 (p = 1) */
  TV_STATUS_TIMEOUT = 32u,     /* a bounded device wait gave up (not expected; the tree's
                                  outputs are -1) */
  TV_STATUS_BAD_ROW = 64u,     /* a target row the traversal needed has no finite logit */
  TV_STATUS_DRAFT_EXHAUSTED = 128u  /* tv_draft_children: a node had more children than
                                       tokens of positive draft probability left (or a
                                       row without positive finite mass) */
};

/* Flags for tv_create.  At most one path flag may be given; with none the
   library picks the path: when V % 8 == 0, the cluster-per-tree kernel for
   V <= 49152 and N + 1 <= 128 (short rows, where one cluster per tree is
   faster than publishing every job through the persistent kernel's queue;
   calls with given row normalisers still run the persistent kernel), else the
   persistent kernel; the three-kernel path otherwise.  All paths compute the
   same results; the two single-kernel paths read rows with bulk copies and
   need V % 8 == 0, other vocabularies always take the three-kernel path. */
enum {
  TV_FLAG_NONE = 0u,
  /* Three kernels: row normalisers of every internal row, then one CTA per
     tree. */
  TV_FLAG_UNFUSED = 1u,
  /* One kernel, one thread-block cluster per tree (rows read lazily, the
     vocabulary split across the cluster's CTAs). */
  TV_FLAG_CLUSTER = 2u,
  /* One persistent cooperative kernel: each tree's serial control runs in an
     owner CTA, and the vocabulary work of every step is cut into slices that
     any CTA of the grid may process (load balancing across trees). */
  TV_FLAG_PERSISTENT = 4u,
  /* Method, combinable with TV_FLAG_CLUSTER or TV_FLAG_PERSISTENT (or none):
     token-level tree verification instead of Traversal Verification -- the
     top-down verifier the paper compares with (§2.2; "Tok.V" in §4).  At the
     current node (the root first) the children are tried in order by
     Recursive Rejection Sampling without replacement (Algorithm 2); an
     accepted child becomes the current node; the bonus token comes from an
     accepted leaf's row or from the residual once every child of the current
     node is rejected.  Same arguments, outputs and uniforms convention.
     Needs a single-kernel path: tv_create returns TV_ERR_INVALID_ARG with
     TV_FLAG_UNFUSED or when V % 8 != 0, and a call that could only run the
     three-kernel path returns TV_ERR_INVALID_ARG. */
  TV_FLAG_TOKEN_LEVEL = 8u
};

/*
 * tv_create -- allocate a handle and its device workspace.
 *   out        : receives the handle (set to NULL on failure).
 *   device     : CUDA device ordinal the handle works on.
 *   vocab      : V, the vocabulary size (1 <= V <= 2^28).
 *   max_nodes  : largest N (draft nodes per tree, root excluded) later calls
 *                may pass; 0 <= max_nodes <= 1023.
 *   max_batch  : largest B later calls may pass; >= 1.
 *   logit_dtype: element type of target_logits in later calls.
 *   flags      : TV_FLAG_NONE or one of TV_FLAG_UNFUSED, TV_FLAG_CLUSTER,
 *                TV_FLAG_PERSISTENT, optionally ORed with TV_FLAG_TOKEN_LEVEL.
 * Errors: TV_ERR_INVALID_ARG, TV_ERR_VOCAB, TV_ERR_CUDA, TV_ERR_DEVICE.
 */
int tv_create(tv_handle** out, int device, int vocab, int max_nodes, int max_batch,
              tv_dtype logit_dtype, unsigned flags);

/*
 * tv_verify_batch -- Traversal Verification of B trees (Algorithm 3, §3.1).
 *
 * Inputs (device pointers):
 *   parents          [B][N+1] int32.  parents[b][0] = -1; for i >= 1 the parent
 *                    row of node i, with 0 <= parents[b][i] < i.  Children of a
 *                    node are taken in increasing row order; the traversal
 *                    visits the tree in post-order (Appendix E).
 *   draft_tokens     [B][N+1] int32.  Token X_i of node i, 0 <= X_i < V;
 *                    entry 0 is ignored.  Siblings must carry distinct tokens.
 *   target_logits    [B][N+1][V], bf16 or fp32 (tv_create's logit_dtype).
 *                    Row i holds the target model's logits at node i;
 *                    M_b(.|X^i) = softmax(logits / temperature).  Rows of every
 *                    node are needed (a leaf's row when it is accepted).
 *   draft_probs      [B][N+1][V] fp32.  Row i holds M_s(.|X^i), used as given
 *                    (not renormalised, no temperature applied).  Rows of leaf
 *                    nodes are never read.
 *   temperature      > 0; scales the target logits only.
 *   uniforms         [B][N+2] fp32 in [0, 1).  uniforms[b][i] (1 <= i <= N) is the
 *                    eta of the test of node i (accepted iff eta < p, strict);
 *                    uniforms[b][N+1] draws the bonus token Y.  Entry 0 is unused.
 *                    Each node is tested at most once, so one uniform per node
 *                    has the law of Algorithm 3's fresh draw per test.
 * Outputs (device pointers, written for every tree b < B):
 *   out_accepted_path[B][N]  node ids of the accepted chain X^tau from depth 1
 *                    to depth tau (the root excluded), then -1 padding.
 *   out_accept_len   [B] tau, the number of accepted draft tokens (0..N);
 *                    -1 marks an invalid tree (see TV_STATUS_*).
 *   out_bonus_token  [B] Y, drawn by inverse CDF (smallest y with
 *                    u * W < sum_{x<=y} w(x)) from the accepted node's current
 *                    target distribution: its original M_b for an original
 *                    leaf, else the residual left by Eqs. (1)-(3); -1 if invalid.
 *   cuda_stream      cudaStream_t the work is queued on.
 * CUDA graphs: the call may be captured.  A launch of the persistent kernel
 * carries the call's queue epoch and must not be replayed, so while
 * cuda_stream is capturing, a handle that picks its path itself verifies with
 * the cluster path (else the three-kernel path), and a handle created with
 * TV_FLAG_PERSISTENT returns TV_ERR_INVALID_ARG.  Make one call outside the
 * capture first: first calls set kernel attributes and allocate scratch.
 * Errors (host-side, nothing launched): TV_ERR_INVALID_ARG, TV_ERR_TEMPERATURE,
 * TV_ERR_CAPACITY; TV_ERR_CUDA if a launch fails.  B = 0 is a no-op.
 */
int tv_verify_batch(tv_handle* h, int B, int N, const int32_t* parents,
                    const int32_t* draft_tokens, const void* target_logits,
                    const float* draft_probs, float temperature, const float* uniforms,
                    int32_t* out_accepted_path, int32_t* out_accept_len,
                    int32_t* out_bonus_token, void* cuda_stream);

/*
 * tv_verify_batch_debug -- tv_verify_batch plus per-node instrumentation.
 *   out_node_p  [B][N+1] fp32 (device): the acceptance rate p of node i at the
 *               moment it was tested (Algorithm 3's eta < p test); 0 for a node
 *               removed because its rate reached 0 (§3.2); NaN for nodes never
 *               tested; entry 0 (root) NaN.
 *   out_stats   [B][5] int32 (device): { number of tests, number of
 *               S-computations (Eqs. (1)/(3), one vocabulary pass each), number
 *               of distinct nodes with at least one S-computation, 1 if the
 *               bonus token came from an original leaf's row else 0, number of
 *               target rows whose normaliser (softmax denominator) the call
 *               computed }.  The first four follow from Algorithm 3; the last
 *               depends on the kernel path (the three-kernel path normalises
 *               every internal row, the single-kernel paths only the rows the
 *               traversal reaches).
 *   out_margin  [B][2] fp32 (device): the tree's decision margins, computed
 *               on the GPU, for counting near-ties on batches no oracle sees.
 *               [b][0] = min over the tree's tests of |eta - p| (Algorithm 3's
 *               strict eta < p test, p as recorded in out_node_p); +inf if
 *               the tree had no test.  [b][1] = the bonus draw's margin
 *               min(u W - CDF(Y - 1), CDF(Y) - u W) / W from the kernel's own
 *               float32 cumulative sums (0 when rounding put u W past the
 *               total).  A decision whose margin is below about 1e-6 may
 *               differ from an exact float64 evaluation.  NaN for an
 *               invalid tree.
 * Any of the three pointers may be NULL.  Other arguments and errors as
 * tv_verify_batch.
 */
int tv_verify_batch_debug(tv_handle* h, int B, int N, const int32_t* parents,
                          const int32_t* draft_tokens, const void* target_logits,
                          const float* draft_probs, float temperature,
                          const float* uniforms, int32_t* out_accepted_path,
                          int32_t* out_accept_len, int32_t* out_bonus_token,
                          float* out_node_p, int32_t* out_stats, float* out_margin,
                          void* cuda_stream);

/*
 * tv_verify_batch_host -- the same verification from HOST buffers: copies the
 * inputs to device staging owned by the handle (allocated and zeroed on first
 * use, sized by tv_create's limits), runs tv_verify_batch on cuda_stream,
 * copies the three outputs back and synchronises the stream before
 * returning.  All pointers are host pointers with the layouts above; pinned
 * (page-locked) memory gives the fastest copies.  Only rows the verification
 * can need are copied: the logit and draft rows of nodes with children (one
 * 2-D copy per run of such rows when all trees share their parents).  Of the
 * leaves' logit rows only the accepted leaf's is ever read, for the bonus
 * draw, so the call has two phases: the verification runs (its draw at a leaf
 * reads a stale staged row), then the accepted leaves' rows alone (at most one
 * per tree) are copied and their bonus tokens drawn again by a kernel of its
 * own (float64 prefix over float32 tile sums of the same e(x); a draw within
 * about 1e-6 W of a CDF step may differ from the device entry point's).
 * Errors as tv_verify_batch.
 */
int tv_verify_batch_host(tv_handle* h, int B, int N, const int32_t* parents,
                         const int32_t* draft_tokens, const void* target_logits,
                         const float* draft_probs, float temperature,
                         const float* uniforms, int32_t* out_accepted_path,
                         int32_t* out_accept_len, int32_t* out_bonus_token,
                         void* cuda_stream);

/*
 * tv_last_host_copy_bytes -- bytes the last successful tv_verify_batch_host
 * call on this handle copied host to device (*h2d) and device to host (*d2h).
 * Either pointer may be NULL.  Errors: TV_ERR_INVALID_ARG (no handle).
 */
int tv_last_host_copy_bytes(tv_handle* h, uint64_t* h2d, uint64_t* d2h);

/*
 * tv_lm_head -- the target model's last layer fused with the row normalisers
 * (the step before verification; not a step of the paper's method itself).
 * Computes the logits l = H W^T on the tensor cores and, in the same pass,
 * each stored row's normaliser (max_v l[v], sum_v 2^((l[v] - max) log2(e) / T)),
 * evaluated on the bf16 values stored.  Given those normalisers,
 * tv_verify_batch_stats does not stream any row to normalise it.
 *   M              rows (e.g. B * (N+1) for a batch of trees, rows in the
 *                  [B][N+1] order of target_logits); M <= max_batch * (max_nodes + 1).
 *   K              hidden size; K % 64 == 0.
 *   hidden         [M][K] bf16, 16-byte aligned.
 *   weight         [V][K] bf16 (output embedding, V = the handle's vocab), 16-byte aligned.
 *   temperature    > 0, the temperature the normalisers are for.
 *   out_logits     [M][V] bf16, 16-byte aligned.
 *   out_row_stats  [M][2] fp32 (max, sum), 8-byte aligned.
 * The handle must have been created for bf16 logits with V % 8 == 0.  The
 * first call allocates the handle's per-(row, 256-column tile) scratch for
 * max_batch * (max_nodes + 1) rows (a later call with a larger vocabulary
 * cannot happen: V is the handle's).
 * Errors: TV_ERR_INVALID_ARG, TV_ERR_CAPACITY, TV_ERR_TEMPERATURE, TV_ERR_CUDA.
 */
int tv_lm_head(tv_handle* h, int M, int K, const void* hidden, const void* weight,
               float temperature, void* out_logits, float* out_row_stats, void* cuda_stream);

/*
 * tv_draft_children -- the draft side of the tree (Definition 1): every node's
 * token drawn from its parent's draft distribution without replacement, the
 * children of a node in index order (the order the verification tests them).
 * Node c >= 1 with parent p takes uniforms[b][c] and gets the smallest token y
 * (ascending token order) with u W < CDF'(y), where CDF' is the cumulative
 * sum of draft_probs[b][p] with the tokens of p's earlier children removed and
 * W its total.  Deterministic given the inputs, so a caller drafting level by
 * level may call it on the tree drafted so far (rows of the new level's
 * parents filled in) and get the same tokens for the earlier levels.
 *   parents      [B][N+1] int32, as tv_verify_batch.
 *   draft_probs  [B][N+1][V] fp32 (V = the handle's vocab), rows of nodes
 *                without children are never read; 16-byte aligned rows read
 *                four tokens a load (V % 4 == 0), any alignment works.
 *   uniforms     [B][N+1] fp32 in [0, 1); column c draws node c, column 0 unused.
 *   out_tokens   [B][N+1] int32: entry 0 is 0 (the root's own token is not
 *                drawn here), entry c the token of node c, usable as
 *                tv_verify_batch's draft_tokens.
 * A tree with invalid parents gets -1 for every node (TV_STATUS_BAD_TREE).  A
 * node with more children than tokens of positive mass gets -1 for the
 * children that find none (TV_STATUS_DRAFT_EXHAUSTED).  The cumulative sums
 * are float64 over float32 tile sums: a draw within about 1e-6 W of a step
 * may fall on the neighbouring token.
 * Errors: TV_ERR_INVALID_ARG, TV_ERR_CAPACITY, TV_ERR_VOCAB (a draft row too
 * long for one CTA's shared memory, above about 600k tokens), TV_ERR_CUDA.
 */
int tv_draft_children(tv_handle* h, int B, int N, const int32_t* parents,
                      const float* draft_probs, const float* uniforms, int32_t* out_tokens,
                      void* cuda_stream);

/*
 * tv_verify_batch_stats -- tv_verify_batch with the target rows' normalisers
 * given (row_stats [B][N+1][2] fp32 (max, sum of 2^((l - max) log2(e) / T)) of
 * the bf16 or fp32 target_logits, as tv_lm_head writes them for the same
 * temperature), so no row is streamed to normalise it.  out_node_p and
 * out_stats are optional (NULL) and have the layouts of tv_verify_batch_debug
 * (out_stats[b][4], rows normalised by this call, is then 0).  Runs on the
 * persistent kernel only (a handle that picks its path itself uses it here
 * for every V): handles created for the other paths, and calls on a
 * capturing stream, return TV_ERR_INVALID_ARG.
 * Errors: those of tv_verify_batch.
 */
int tv_verify_batch_stats(tv_handle* h, int B, int N, const int32_t* parents,
                          const int32_t* draft_tokens, const void* target_logits,
                          const float* draft_probs, float temperature, const float* uniforms,
                          const float* row_stats, int32_t* out_accepted_path,
                          int32_t* out_accept_len, int32_t* out_bonus_token, float* out_node_p,
                          int32_t* out_stats, void* cuda_stream);

/*
 * tv_debug_withhold_job -- test hook for the failure path; no counterpart in
 * the paper.  The next call on this handle that runs the persistent kernel
 * writes tree `tree`'s first job into the work queue but never publishes it.
 * The CTAs holding its queue slots and the tree's owner wait on it until the
 * kernel's idle limit (2 s without progress).  The kernel then raises its abort
 * flag and every role exits.  That call returns normally, the status word gets
 * TV_STATUS_TIMEOUT, and every tree not finished by then reports -1
 * (accept_len, bonus, path).  Later calls on the handle are unaffected.  Calls
 * on the other paths ignore the request and leave it pending.
 *   tree : 0 <= tree < the handle's max_batch.
 * Errors: TV_ERR_INVALID_ARG.
 */
int tv_debug_withhold_job(tv_handle* h, int tree);

/*
 * tv_get_status -- synchronise the handle's device and return, in *status, the
 * OR of the TV_STATUS_* bits raised since the previous tv_get_status call
 * (then clear them).  Errors: TV_ERR_INVALID_ARG, TV_ERR_CUDA.
 */
int tv_get_status(tv_handle* h, uint32_t* status);

/*
 * tv_set_phase_timing -- when enable != 0, later verify calls on this handle
 * record CUDA events on their stream around each of the three kernels
 * (row preparation, row normalisers, traversal).  Costs three event records
 * per call; off by default.  Errors: TV_ERR_INVALID_ARG, TV_ERR_CUDA.
 */
int tv_set_phase_timing(tv_handle* h, int enable);

/*
 * tv_last_phase_ms -- waits for the events of the most recent timed call and
 * writes the device time of its three kernels, in milliseconds, to ms[0..2]
 * (preparation, row normalisers, traversal).  Errors: TV_ERR_INVALID_ARG
 * (timing off or no timed call yet), TV_ERR_CUDA.
 */
int tv_last_phase_ms(tv_handle* h, float* ms);

/*
 * tv_launch_shape -- how a call with these B and N would run on this handle:
 * *path = 0 for the three-kernel path, 1 for the cluster-per-tree kernel, 2
 * for the persistent kernel; *cluster = CTAs per tree (cluster path; 1
 * otherwise), *warps = consumer warps per CTA, *stages = ring stages (0 for
 * the three-kernel path).  Any output pointer may be NULL.
 * Errors: TV_ERR_INVALID_ARG, TV_ERR_CAPACITY.
 */
int tv_launch_shape(tv_handle* h, int B, int N, int* path, int* cluster, int* warps,
                    int* stages);

/*
 * tv_verify_batch_noalloc -- the same verification for callers that cannot
 * allocate device memory: a serving process whose allocator reserved the
 * device's memory up front and forbids new allocations once it has warmed
 * up, or an embedding in another runtime that owns every byte of the device.
 * tv_create allocates a handle's workspace, so such callers cannot use it.
 * The paper has no counterpart: this is a deployment entry point.
 *
 * Needs no handle and allocates nothing: its scratch (internal-row list, row
 * statistics, status word) is one fixed array of static device memory in the
 * library image (about 0.8 MB, held by every GPU that loads the library until
 * the process exits), used through the three-kernel path.  Limit:
 * B * (N + 1) <= 65536 rows; larger calls return TV_ERR_CAPACITY and launch
 * nothing.  The first call on a device makes that device current and looks up
 * the array's device address (cudaGetSymbolAddress) once; issue that first
 * call before any stream capture.  All calls share the array: each clears
 * what must start at zero, but calls whose work overlaps on the GPU race on it
 * and must not be issued.
 *
 * No TV_STATUS_* word is reported on this path: the status word lives in the
 * shared array and no call returns it.  An invalid tree (BAD_TREE, BAD_TOKEN,
 * DUP_SIBLING, ZERO_DRAFT, BAD_ROW) shows only as accept_len = -1, bonus = -1
 * and a path of -1 for that tree; the informational DEGENERATE bit is lost.
 *   device      : CUDA device ordinal (0..63) the pointers belong to.
 *   vocab, logit_dtype : as in tv_create.
 *   the rest    : as in tv_verify_batch (device pointers, caller-owned).
 * Errors: TV_ERR_INVALID_ARG, TV_ERR_TEMPERATURE, TV_ERR_VOCAB,
 * TV_ERR_CAPACITY, TV_ERR_DEVICE, TV_ERR_CUDA.
 */
int tv_verify_batch_noalloc(int device, int B, int N, int vocab, tv_dtype logit_dtype,
                            const int32_t* parents, const int32_t* draft_tokens,
                            const void* target_logits, const float* draft_probs,
                            float temperature, const float* uniforms,
                            int32_t* out_accepted_path, int32_t* out_accept_len,
                            int32_t* out_bonus_token, void* cuda_stream);

/* tv_destroy -- free the handle's workspace (synchronises its device). */
int tv_destroy(tv_handle* h);

/* tv_strerror -- static description of a return code. */
const char* tv_strerror(int code);

/* tv_version -- library version, major * 10000 + minor * 100 + patch. */
int tv_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TV_H_ */
