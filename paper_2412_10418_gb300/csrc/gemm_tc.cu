// gemm_tc.cu -- projection GEMMs on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Swap-AB: the weights are the M = 128 operand (one tile = 128 virtual output rows, loaded as
// two 64-row TMA boxes so that a tile may draw its halves from different segments: gate/up
// interleave, q/k/v boundaries) and the activation rows are the N operand (N = R rounded up
// to 16, 16..256). Both operands are K-major bf16 in 128-byte-swizzled shared-memory tiles;
// the accumulator lives in TMEM (fp32, N columns). The activations come as the hi and lo bf16
// planes of the split, so each 16-deep K step issues two MMAs into the same accumulator.
//
// Block = 4 warps: lane 0 of warp 0 issues TMA loads through a ring of mbarrier-guarded
// stages, lane 0 of warp 1 issues the MMAs and releases each stage with tcgen05.commit; then
// all four warps read their 32 TMEM lanes each. K is split across blocks when the tile count
// alone cannot fill the GPU; as in the weight-streaming kernel, partial tiles go to scratch
// and the last block of a tile sums them in split order and runs the fused epilogue.
// Every wait is bounded in time; on expiry the block latches CDSL_ETIMEOUT, waits (bounded)
// for its own copies in flight, frees its TMEM and returns.
#include <cudaTypedefs.h>

#include <algorithm>

#include "gemm.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace cdsl {
namespace {

constexpr int kMaxStages = 8;
constexpr int kStageBudget = 220 * 1024;            // ring memory a plan may use
constexpr int kMaxDynSmem = kStageBudget + 1024;    // + alignment slack (static smem is extra)
constexpr int kTileLd = 132;   // fp32 epilogue tile row pitch (128 + 4 against bank conflicts)
constexpr int kThreads = 128;

__device__ __forceinline__ uint32_t tmem_cols(int n_pad) {
  uint32_t c = 32;
  while (c < (uint32_t)n_pad) c <<= 1;
  return c;
}

// Source tensor map and first row of the 64-row half-tile starting at virtual row vstart.
__device__ __forceinline__ void half_source(const GemmArgs& a, int vstart, int* m, int* y) {
  if (a.mode == EPI_SWIGLU) {
    *m = (vstart >> 6) & 1;
    *y = (vstart >> 7) * 64;
    return;
  }
  int base = 0;
  for (int s = 0; s < a.n_seg; ++s) {
    if (vstart < base + a.seg_rows[s] || s == a.n_seg - 1) {
      *m = s;
      *y = vstart - base;
      return;
    }
    base += a.seg_rows[s];
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_tc(const __grid_constant__ TcMaps maps, const __grid_constant__ GemmArgs a, TcPlan p,
              float* part, int* tile_cnt) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int s_abort, s_last;

  uint8_t* smem = smem_raw + ((1024 - (tc::smem_u32(smem_raw) & 1023)) & 1023);
  const int tile = blockIdx.x, split = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int v0 = tile * 128;
  const int total_kb = a.K >> 6;
  const int kb0 = split * p.kb_per_split;
  const int nkb = min(p.kb_per_split, total_kb - kb0);
  const int S = p.stages, NP = p.n_pad;
  const uint32_t stage_bytes = 16384u + 256u * NP;
  const uint32_t ncols = tmem_cols(NP);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      tc::mbar_init(&full_bar[s], 1);
      tc::mbar_init(&empty_bar[s], 1);
    }
    tc::mbar_init(&done_bar, 1);
    s_abort = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(&tmem_base, ncols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    int m0, y0, m1, y1;
    half_source(a, v0, &m0, &y0);
    half_source(a, v0 + 64, &m1, &y1);
    const uint64_t pol = tc::policy_evict_first();
    int issued = 0;
    bool aborted = false;
    for (int i = 0; i < nkb; ++i) {
      const int s = i % S, use = i / S;
      if (use > 0 && !tc::mbar_wait(&empty_bar[s], (use - 1) & 1, a.status)) {
        aborted = true;
        break;
      }
      uint8_t* st = smem + (size_t)s * stage_bytes;
      tc::mbar_expect_tx(&full_bar[s], stage_bytes);
      const int x = (kb0 + i) * 64;
      tc::tma_load_2d_hint(st, &maps.w[m0], x, y0, &full_bar[s], pol);
      tc::tma_load_2d_hint(st + 8192, &maps.w[m1], x, y1, &full_bar[s], pol);
      for (int j = 0; j < NP / 16; ++j) {
        tc::tma_load_2d(st + 16384 + j * 2048, &maps.xh, x, j * 16, &full_bar[s]);
        tc::tma_load_2d(st + 16384 + NP * 128 + j * 2048, &maps.xl, x, j * 16, &full_bar[s]);
      }
      ++issued;
    }
    if (aborted) {
      s_abort = 1;
      // let the copies already in flight land before the block can exit
      for (int i = max(0, issued - S); i < issued; ++i)
        tc::mbar_wait(&full_bar[i % S], (i / S) & 1, a.status);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    const uint32_t idesc = tc::idesc_bf16_f32(128, NP);
    for (int i = 0; i < nkb; ++i) {
      const int s = i % S, use = i / S;
      if (!tc::mbar_wait(&full_bar[s], use & 1, a.status)) {
        s_abort = 1;
        break;
      }
      tc::tc_fence_after();
      const uint32_t sa = tc::smem_u32(smem + (size_t)s * stage_bytes);
      const uint64_t da = tc::desc_sw128(sa);
      const uint64_t dh = tc::desc_sw128(sa + 16384);
      const uint64_t dl = tc::desc_sw128(sa + 16384 + NP * 128);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {   // 4 x K=16 per 64-wide stage; +32 bytes = +2 in the desc
        tc::umma_bf16(tmem, da + 2 * kk, dh + 2 * kk, idesc, (i | kk) != 0);
        tc::umma_bf16(tmem, da + 2 * kk, dl + 2 * kk, idesc, 1);
      }
      tc::umma_commit(&empty_bar[s]);
    }
    tc::umma_commit(&done_bar);
  }
  __syncwarp();
  const bool ok = tc::mbar_wait(&done_bar, 0, a.status);
  tc::tc_fence_after();
  __syncthreads();

  float* tileS = reinterpret_cast<float*>(smem);   // [NP][kTileLd], reuses the drained stages
  const bool good = ok && !s_abort;
  if (good) {
    for (int c0 = 0; c0 < NP; c0 += 16) {
      float v[16];
      tc::tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) tileS[(c0 + i) * kTileLd + warp * 32 + lane] = v[i];
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) tc::tmem_dealloc(tmem, ncols);
  if (!good) return;

  const int R = min(a.R, NP);
  if (p.splits == 1) {
    tile_epilogue<__nv_bfloat16>(a, v0, 0, R, tileS, kTileLd);
    return;
  }
  const int tiles = gridDim.x;
  for (int i = threadIdx.x; i < R * 128; i += kThreads) {
    const int r = i >> 7, v = i & 127;
    part[((size_t)(split * NP + r) * tiles + tile) * 128 + v] = tileS[r * kTileLd + v];
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(tile_cnt + tile, 1) == p.splits - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int i = threadIdx.x; i < R * 128; i += kThreads) {
    const int r = i >> 7, v = i & 127;
    float s = 0.f;
    for (int sp = 0; sp < p.splits; ++sp)
      s += __ldcg(part + ((size_t)(sp * NP + r) * tiles + tile) * 128 + v);
    tileS[r * kTileLd + v] = s;
  }
  __syncthreads();
  tile_epilogue<__nv_bfloat16>(a, v0, 0, R, tileS, kTileLd);
  if (threadIdx.x == 0) tile_cnt[tile] = 0;
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

}  // namespace

bool tc_supported(const GemmArgs& a) {
  if (a.K % 64 || a.R < 1 || a.R > 256) return false;
  for (int s = 0; s + 1 < a.n_seg; ++s)
    if (a.mode != EPI_SWIGLU && a.seg_rows[s] % 64) return false;
  return true;
}

TcPlan plan_tc(int K, int n_virtual, int R, int n_sm) {
  TcPlan p{};
  p.n_pad = (R + 15) / 16 * 16;
  p.tiles = (n_virtual + 127) / 128;
  const int total_kb = K / 64;
  const size_t stage = 16384 + 256 * (size_t)p.n_pad;
  const int per_sm = (4 * stage + 2048 <= 113 * 1024) ? 2 : 1;
  p.stages = per_sm == 2 ? 4 : (int)std::max<size_t>(2, std::min<size_t>(kMaxStages, kStageBudget / stage));
  const int target = per_sm * n_sm;
  int splits = std::max(1, (target + p.tiles / 2) / p.tiles);
  splits = std::min(splits, total_kb);
  p.kb_per_split = (total_kb + splits - 1) / splits;
  p.splits = (total_kb + p.kb_per_split - 1) / p.kb_per_split;
  p.smem = std::max((size_t)p.stages * stage, (size_t)p.n_pad * kTileLd * 4) + 1024;
  return p;
}

int encode_bf16_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer) {
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return -1;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

int configure_gemm_tc() {
  return cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxDynSmem) ==
                 cudaSuccess
             ? 0
             : -1;
}

void launch_gemm_tc(const TcMaps& maps, const GemmArgs& a, const TcPlan& p, float* part,
                    int* tile_cnt, cudaStream_t s) {
  dim3 grid(p.tiles, p.splits);
  k_gemm_tc<<<grid, kThreads, p.smem, s>>>(maps, a, p, part, tile_cnt);
}

}  // namespace cdsl
