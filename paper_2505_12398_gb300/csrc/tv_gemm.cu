// tv_gemm.cu -- the target model's LM head fused with the row normalisers
// (sm_103a).
//
// The target distributions M_b(.|X^i) = softmax(l_i / T) that Traversal
// Verification reads (§3.1) come from the logits l = H W^T of the target
// model's last layer (hidden states H [M][K], output embedding W [V][K],
// bf16).  This kernel computes them on the 5th-generation tensor cores and, in
// the same pass, each stored row's normaliser: m = max_v l[v] and
// s = sum_v 2^((l[v] - m) c), c = log2(e) / T, evaluated on the bf16 values
// it stores.  Given those, verification never streams a row for its
// normaliser.
//
// A persistent kernel, one CTA per SM, walks 128 x 256 tiles of l in groups
// of row tiles holding 32 MiB of H, row tile fastest inside a group, so that
// the CTAs running at the same time share W tiles through L2 while the
// group's H stays resident: W is read from HBM once per group, H once.
//   * warp 0 (one lane) streams 128 x 64 tiles of H and 256 x 64 tiles of W
//     into a 4-stage shared-memory ring with 2-D TMA copies (128-byte
//     swizzle, the layout the tensor cores read), across tile boundaries;
//   * warp 1 allocates all 512 columns of tensor memory, two fp32
//     accumulators of 256 columns, and one lane issues tcgen05.mma (M=128,
//     N=256, K=16 per instruction) into them in turn, releasing each stage
//     with tcgen05.commit;
//   * warps 2-5 (one TMEM lane quarter each, one row per thread) read the
//     finished accumulator with tcgen05.ld, round to bf16, store the logits
//     and keep the row's running (max, sum) over the tile's columns, while
//     the tensor cores fill the other accumulator.
// A second kernel merges the per-tile (max, sum) of each row.
//
// Every mbarrier wait is bounded; a wait that gives up raises
// TV_STATUS_TIMEOUT in the status word and the CTA still frees its tensor
// memory before it exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <mutex>

#include "tv_device.cuh"
#include "tv_launch.h"
#include "tv_ptx.cuh"

namespace tvk {
namespace gemm {

constexpr int kBM = 128;          // rows of a tile (TMEM lanes)
constexpr int kBN = 256;          // columns of a tile (TMEM columns)
constexpr int kBK = 64;           // K per stage: 128 bytes of bf16, one swizzle row
constexpr int kUmmaK = 16;        // K per tcgen05.mma of kind::f16
constexpr int kStages = 4;
// Tile order: groups of row tiles holding about kGroupBytes of H, row tile
// fastest inside a group, so that the CTAs running at once share W tiles
// through L2 while the group's rows of H stay resident.  W is then read from
// HBM once per group and H once.
constexpr size_t kGroupBytes = 32u << 20;
constexpr int kThreads = 192;     // TMA warp, MMA warp, four epilogue warps
constexpr uint32_t kABytes = kBM * kBK * 2;   // 16 KB
constexpr uint32_t kBBytes = kBN * kBK * 2;   // 32 KB
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr int kAccBufs = 2;                   // accumulators in tensor memory
constexpr uint32_t kTmemCols = kAccBufs * kBN;   // fp32: one column per output column
constexpr size_t kSmemBytes = (size_t)kStages * kStageBytes + 1024;   // + alignment slack

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits
// 4-5 = 1), bf16 A and B (bits 7-9, 10-12 = 1), both K-major (bits 15, 16 =
// 0), N >> 3 in bits 17-22, M >> 4 in bits 24-28.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                            ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);

// Shared-memory matrix descriptor of a K-major operand tile written by TMA
// with the 128-byte swizzle: start address >> 4 (bits 0-13), leading byte
// offset (unused with this swizzle, set to 1; bits 16-29), stride byte offset
// 1024 B >> 4 between groups of 8 rows (bits 32-45), descriptor version 1
// (bit 46), swizzle mode 2 = 128 B (bits 61-63).  Tiles are 1024-byte aligned
// (base offset 0).  Stepping K by 16 bf16 inside the swizzled 128-byte row
// advances the start address by 32 bytes.
__device__ __forceinline__ uint64_t smem_desc(const void* p) {
  const uint64_t addr = smem_u32(p);
  return ((addr >> 4) & 0x3FFFull) | (1ull << 16) | ((uint64_t)(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}

// 2-D tiled TMA load of box {x .. x+box0, y .. y+box1} (x in elements, a
// multiple of 64 here, so 16-byte aligned) into shared memory.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Row and column tile of the t-th tile in the kernel's order.
__device__ __forceinline__ void tile_coords(int t, int m_tiles, int n_tiles, int group,
                                            int& mt, int& nt) {
  const int g = group > 0 && group < m_tiles ? group : m_tiles;
  const int full = (m_tiles / g) * g * n_tiles;       // tiles in whole groups
  if (t < full) {
    const int grp = t / (g * n_tiles), r = t - grp * g * n_tiles;
    mt = grp * g + r % g;
    nt = r / g;
  } else {
    const int gt = m_tiles - (m_tiles / g) * g, r = t - full;
    mt = (m_tiles / g) * g + r % gt;
    nt = r / gt;
  }
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

// Arrives on `bar` once every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::
                   "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* slot) {   // a whole warp
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(kTmemCols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr) {   // the allocating warp
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr),
               "r"(kTmemCols)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 accumulator columns of this warp's 32 TMEM lanes (lane
// i of the warp reads TMEM lane base + i): one row per thread.  The load and
// its wait are one statement, so no use of the registers precedes the wait.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
               "tcgen05.wait::ld.sync.aligned;"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Tiles t = blockIdx.x, blockIdx.x + gridDim.x, ... of l = H W^T (in the
// order of tile_coords), stored as bf16, and each row's
// (max, sum of 2^((l - max) c)) over a tile's columns in part[row][tile].
__global__ void __launch_bounds__(kThreads, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap map_h,
                   const __grid_constant__ CUtensorMap map_w, int M, int V, int K, float c_hi,
                   float c_lo, __nv_bfloat16* __restrict__ logits, float2* __restrict__ part,
                   int m_tiles, int n_tiles, int group, uint32_t* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t acc_full[kAccBufs];    // accumulator ready (tcgen05.commit)
  __shared__ __align__(8) uint64_t acc_empty[kAccBufs];   // accumulator read (4 epilogue warps)
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int failed;
  // the TMA tiles need 1024-byte alignment (128-byte swizzle atoms)
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nkb = K / kBK;
  const int n_total = m_tiles * n_tiles;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int k = 0; k < kAccBufs; ++k) {
      mbar_init(&acc_full[k], 1);
      mbar_init(&acc_empty[k], 4);
    }
    mbar_init(&drain_bar, 1);
    failed = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(&tmem_slot);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (warp == 0) {
    // ---- TMA producer: one ring across all of this CTA's tiles ----
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < n_total && ok; t += gridDim.x) {
        int mt, nt;
        tile_coords(t, m_tiles, n_tiles, group, mt, nt);
        const int m0 = mt * kBM, n0 = nt * kBN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % kStages;
          if (it >= kStages && !mbar_wait(&empty_bar[s], ((it / kStages) - 1) & 1)) {
            ok = false;
            break;
          }
          uint8_t* a = smem + (size_t)s * kStageBytes;
          mbar_arrive_expect_tx(&full_bar[s], kStageBytes);
          tma_load_2d(a, &map_h, kb * kBK, m0, &full_bar[s]);
          tma_load_2d(a + kABytes, &map_w, kb * kBK, n0, &full_bar[s]);
        }
      }
      if (!ok) failed = 1;
      // the copies issued last have landed before the CTA may exit
      for (uint32_t j = it > (uint32_t)kStages ? it - kStages : 0u; j < it; ++j)
        if (!mbar_wait(&full_bar[j % kStages], (j / kStages) & 1)) failed = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- tensor-core issue (one lane), the two accumulators in turn ----
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      int j = 0;
      for (int t = blockIdx.x; t < n_total && ok; t += gridDim.x, ++j) {
        const uint32_t acc = (uint32_t)j & 1u;
        if (j >= kAccBufs && !mbar_wait(&acc_empty[acc], ((j >> 1) - 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * (uint32_t)kBN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % kStages;
          if (!mbar_wait(&full_bar[s], (it / kStages) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint8_t* a = smem + (size_t)s * kStageBytes;
          const uint64_t da = smem_desc(a), db = smem_desc(a + kABytes);
#pragma unroll
          for (int k = 0; k < kBK / kUmmaK; ++k) {
            const uint64_t step = (uint64_t)((k * kUmmaK * 2) >> 4);   // 32 bytes of K
            umma_bf16(d, da + step, db + step, (kb > 0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&empty_bar[s]);   // the stage is free once these MMAs are done
        }
        if (ok) umma_commit(&acc_full[acc]);   // the accumulator is complete
      }
      if (!ok) failed = 1;
      // every MMA issued has finished before tensor memory is freed
      umma_commit(&drain_bar);
      if (!mbar_wait(&drain_bar, 0)) failed = 1;
    }
    __syncwarp();
  } else {
    // ---- epilogue: one row per thread ----
    const int q = warp & 3;                       // the TMEM lane quarter of this warp
    int j = 0;
    for (int t = blockIdx.x; t < n_total; t += gridDim.x, ++j) {
      const uint32_t acc = (uint32_t)j & 1u;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[acc], (j >> 1) & 1));
      if (!ok) {
        if (lane == 0) failed = 1;
        break;
      }
      tc_fence_after();
      int mt, n_tile;
      tile_coords(t, m_tiles, n_tiles, group, mt, n_tile);
      const int m0 = mt * kBM, n0 = n_tile * kBN;
      const int row = m0 + q * 32 + lane;
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + acc * (uint32_t)kBN;
      float m_run = TV_NEG_INF, s_run = 0.f;
      for (int c = 0; c < kBN; c += 32) {
        float v[32];
        tmem_ld32(tbase + (uint32_t)c, v);        // the whole warp, every row
        const int col0 = n0 + c;
        if (row >= M || col0 >= V) continue;
        uint32_t packed[16];
        float cm = TV_NEG_INF;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const __nv_bfloat16 b0 = __float2bfloat16_rn(v[2 * i]);
          const __nv_bfloat16 b1 = __float2bfloat16_rn(v[2 * i + 1]);
          v[2 * i] = __bfloat162float(b0);        // the stored values from here on
          v[2 * i + 1] = __bfloat162float(b1);
          if (col0 + 2 * i < V) cm = fmaxf(cm, v[2 * i]);
          if (col0 + 2 * i + 1 < V) cm = fmaxf(cm, v[2 * i + 1]);
          __nv_bfloat162 h2 = __halves2bfloat162(b0, b1);
          packed[i] = *reinterpret_cast<uint32_t*>(&h2);
        }
        __nv_bfloat16* dst = logits + (size_t)row * V + col0;
        if (col0 + 32 <= V) {                    // 64 aligned bytes (V % 8 == 0)
          uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            d4[i] = make_uint4(packed[4 * i], packed[4 * i + 1], packed[4 * i + 2],
                               packed[4 * i + 3]);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (col0 + i < V) dst[i] = __float2bfloat16_rn(v[i]);
        }
        if (cm > m_run) {
          if (m_run != TV_NEG_INF) s_run *= exp2_split(m_run - cm, 0.f, c_hi, c_lo);
          m_run = cm;
        }
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (col0 + i < V) s_run += exp2_corrected(v[i] - m_run, c_hi, c_lo);
      }
      // this accumulator may be overwritten once all four warps have read it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
      if (row < M) part[(size_t)row * n_tiles + n_tile] = make_float2(m_run, s_run);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem);
  }
  if (threadIdx.x == 0 && failed) atomicOr(status, 32u);
}

// Merges the per-tile (max, sum) of each row into the row's normaliser (one
// warp per row, tiles in order within each lane, then across lanes).
__global__ void lm_head_merge_kernel(const float2* __restrict__ part, int M, int n_tiles,
                                     float c_hi, float c_lo, float2* __restrict__ out) {
  const int row = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float2* p = part + (size_t)row * n_tiles;
  float mx = TV_NEG_INF;
  for (int t = lane; t < n_tiles; t += 32) mx = fmaxf(mx, p[t].x);
  mx = warp_max(mx);
  float s = 0.f;
  for (int t = lane; t < n_tiles; t += 32) {
    const float2 v = p[t];
    if (v.x != TV_NEG_INF) s += v.y * exp2_split(v.x - mx, 0.f, c_hi, c_lo);
  }
  s = warp_sum(s);
  if (lane == 0) out[row] = make_float2(mx, s);
}

}  // namespace gemm
}  // namespace tvk

// --------------------------------------------------------------- launcher --

namespace {

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                 const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                 const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, fetched once through the runtime (no link
// dependency on the driver library).
EncodeTiled encoder() {
  static std::once_flag once;
  static EncodeTiled fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiled>(p);
    else
      cudaGetLastError();
  });
  return fn;
}

// Row-major bf16 [rows][K] as a 2-D tensor with 64 x box_rows boxes and the
// 128-byte swizzle (rows past the end read as zeros).
bool make_map(CUtensorMap* map, const void* base, int rows, int K, int box_rows) {
  const EncodeTiled enc = encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)tvk::gemm::kBK, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
             box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

constexpr int kGemmDevices = 64;
std::mutex g_gemm_mutex;
bool g_gemm_smem_set[kGemmDevices] = {};
int g_gemm_sms[kGemmDevices] = {};

}  // namespace

int tv_lm_head_tiles(int V) { return (V + tvk::gemm::kBN - 1) / tvk::gemm::kBN; }

int tv_launch_lm_head(const void* hidden, const void* weight, int M, int K, int V, float c_hi,
                      float c_lo, void* logits, float2* part, float2* row_stats,
                      uint32_t* status, cudaStream_t stream) {
  using namespace tvk::gemm;
  if (M <= 0) return 0;
  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kGemmDevices) {
    cudaGetLastError();
    return -5;
  }
  CUtensorMap map_h, map_w;
  if (!make_map(&map_h, hidden, M, K, kBM) || !make_map(&map_w, weight, V, K, kBN)) return -5;
  {
    std::lock_guard<std::mutex> lock(g_gemm_mutex);
    if (!g_gemm_smem_set[device]) {
      if (cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)kSmemBytes) != cudaSuccess) {
        cudaGetLastError();
        return -5;
      }
      g_gemm_smem_set[device] = true;
    }
    if (g_gemm_sms[device] < 1 &&
        cudaDeviceGetAttribute(&g_gemm_sms[device], cudaDevAttrMultiProcessorCount, device) !=
            cudaSuccess) {
      cudaGetLastError();
      g_gemm_sms[device] = 0;
      return -5;
    }
  }
  const int n_tiles = tv_lm_head_tiles(V);
  const int m_tiles = (M + kBM - 1) / kBM;
  // one CTA per SM (its shared memory and all of tensor memory)
  const int grid = std::min(m_tiles * n_tiles, g_gemm_sms[device]);
  const int group = (int)std::max<size_t>(1, kGroupBytes / ((size_t)kBM * K * 2));
  lm_head_kernel<<<grid, kThreads, kSmemBytes, stream>>>(
      map_h, map_w, M, V, K, c_hi, c_lo, static_cast<__nv_bfloat16*>(logits), part, m_tiles,
      n_tiles, group, status);
  const int warps_per_block = 8;
  lm_head_merge_kernel<<<(M + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0,
                         stream>>>(part, M, n_tiles, c_hi, c_lo, row_stats);
  if (cudaGetLastError() != cudaSuccess) return -5;
  return 0;
}
