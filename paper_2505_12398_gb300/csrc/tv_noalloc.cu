// tv_noalloc.cu -- tv_verify_batch_noalloc: verification without any device
// allocation, for callers that cannot call cudaMalloc.
//
// Some callers cannot allocate device memory at all: a serving process whose
// memory pool reserved the device up front and forbids new allocations once
// it has warmed up, or an embedding whose allocator owns every byte of the
// device.  tv_create allocates a handle's workspace, so those callers cannot
// use it.  This entry point runs the three-kernel path (internal-row list,
// row normalisers, per-tree traversal) with its scratch -- the internal-row
// list, the row statistics and the status word -- in one fixed-size array of
// static device memory that is part of the library image: every GPU that
// loads the library holds those kScratchBytes (about 0.75 MiB) until the
// process exits.
//
// The caller still owns and passes every input and output.  All calls share
// the one array and it keeps whatever the last call left there; each call
// clears what must start at zero (the row counter, the status word) before
// its kernels run.  Calls whose work overlaps on the GPU (different streams,
// different host threads without ordering) race on the array and must not be
// issued.  The status word is written by the kernels but never returned:
// through this entry point an invalid tree shows only as -1 outputs.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "../../include/tv.h"
#include "tv_launch.h"

namespace {

constexpr int kMaxScratchRows = 1 << 16;   // B * (N + 1) rows at most
constexpr size_t kAlign = 256;
constexpr size_t kOffStatus = 0;
constexpr size_t kOffCount = kAlign;
constexpr size_t kOffRows = 2 * kAlign;
constexpr size_t kOffStats = kOffRows + (size_t)kMaxScratchRows * sizeof(int32_t);
constexpr size_t kScratchBytes = kOffStats + (size_t)kMaxScratchRows * sizeof(float2);
constexpr int kMaxDevices = 64;

// The scratch array.  In host code this name is only a host-side stand-in for
// the device object: kernels are given the address cudaGetSymbolAddress
// returns for the current device, never the name itself.
static __device__ __align__(256) unsigned char g_tv_scratch[kScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
int g_smem_optin[kMaxDevices] = {};

// Once per device, with that device current: the array's device address and
// the two device properties the launch needs.
int setup_device(int device) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_addr[device]) return TV_OK;
  void* ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_tv_scratch) != cudaSuccess || ptr == nullptr) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  int sms = 0, smem = 0, major = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, device) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, device) != cudaSuccess) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  if (major < 10) return TV_ERR_DEVICE;
  g_sm_count[device] = sms;
  g_smem_optin[device] = smem;
  g_scratch_addr[device] = ptr;
  return TV_OK;
}

}  // namespace

extern "C" int tv_verify_batch_noalloc(int device, int B, int N, int vocab, tv_dtype logit_dtype,
                                       const int32_t* parents, const int32_t* draft_tokens,
                                       const void* target_logits, const float* draft_probs,
                                       float temperature, const float* uniforms,
                                       int32_t* out_accepted_path, int32_t* out_accept_len,
                                       int32_t* out_bonus_token, void* cuda_stream) {
  if (B < 0 || N < 0 || N > 1023) return TV_ERR_INVALID_ARG;
  if (vocab < 1 || vocab > (1 << 28)) return TV_ERR_VOCAB;
  if (logit_dtype != TV_BF16 && logit_dtype != TV_FP32) return TV_ERR_INVALID_ARG;
  if (!(std::isfinite(temperature) && temperature > 0.f)) return TV_ERR_TEMPERATURE;
  if ((long long)B * (N + 1) > kMaxScratchRows) return TV_ERR_CAPACITY;
  if (device < 0 || device >= kMaxDevices) return TV_ERR_INVALID_ARG;
  if (B == 0) return TV_OK;
  if (!parents || !draft_tokens || !target_logits || !draft_probs || !uniforms ||
      !out_accept_len || !out_bonus_token || (N > 0 && !out_accepted_path))
    return TV_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(target_logits) & 15u) ||
      (reinterpret_cast<uintptr_t>(draft_probs) & 15u))
    return TV_ERR_INVALID_ARG;

  int prev = 0;
  if (cudaGetDevice(&prev) != cudaSuccess) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  if (prev != device && cudaSetDevice(device) != cudaSuccess) {
    cudaGetLastError();
    return TV_ERR_CUDA;
  }
  int rc = setup_device(device);
  if (rc == TV_OK && tv_traverse_smem_bytes(N + 1, vocab) > (size_t)g_smem_optin[device])
    rc = TV_ERR_VOCAB;
  if (rc == TV_OK) {
    unsigned char* base = static_cast<unsigned char*>(g_scratch_addr[device]);
    uint32_t* status = reinterpret_cast<uint32_t*>(base + kOffStatus);
    int32_t* n_rows = reinterpret_cast<int32_t*>(base + kOffCount);
    int32_t* row_list = reinterpret_cast<int32_t*>(base + kOffRows);
    float2* stats = reinterpret_cast<float2*>(base + kOffStats);
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    if (cudaMemsetAsync(status, 0, sizeof(uint32_t), st) != cudaSuccess) {
      cudaGetLastError();
      rc = TV_ERR_CUDA;
    } else {
      TravArgs a;
      a.parents = parents;
      a.tokens = draft_tokens;
      a.logits = target_logits;
      a.draft_probs = draft_probs;
      a.uniforms = uniforms;
      a.stats = stats;
      a.B = B;
      a.N = N;
      a.V = vocab;
      const double c = 1.4426950408889634 / static_cast<double>(temperature);
      a.c_hi = static_cast<float>(c);
      a.c_lo = static_cast<float>(c - static_cast<double>(a.c_hi));
      a.c = c;
      a.out_path = out_accepted_path;
      a.out_accept_len = out_accept_len;
      a.out_bonus = out_bonus_token;
      a.out_node_p = nullptr;
      a.out_stats = nullptr;
      a.out_margin = nullptr;
      a.status = status;
      a.token_level = 0;
      a.row_stats = nullptr;
      const int rows = B * (N + 1);
      int grid = g_sm_count[device] * 4;
      if (grid > rows) grid = rows;
      if (grid < 1) grid = 1;
      rc = tv_launch_all(a, logit_dtype == TV_BF16 ? 1 : 0, row_list, n_rows, grid, st, nullptr);
    }
  }
  if (prev != device) cudaSetDevice(prev);
  return rc;
}
