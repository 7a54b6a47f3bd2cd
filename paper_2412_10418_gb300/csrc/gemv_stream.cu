// gemv_stream.cu -- CUDA-core weight-streaming GEMM for few activation rows (R <= 8): the
// projections of bf16 models whose K the tensor-core kernel does not take (K % 64 != 0), and
// cdsl_gemv_noalloc. Every bf16 projection with K % 64 == 0 -- all of the synthetic workloads'
// -- runs on the tensor-core kernel (gemm_tc.cu) instead, which streams weights faster here.
//
// With R <= 8 rows a projection moves ~R*2 flops per weight byte: the kernel is bound by HBM
// bandwidth on the weights. Each block owns a tile of 128 virtual output rows and one K slice
// (split-K fills all SMs even for 2048-wide outputs). Weights are read exactly once with
// 128-bit non-allocating loads; the activation slice sits in shared memory as fp32 (hi + lo of
// the bf16 split). A warp streams 4 weight rows at a time, lanes striding K by 8 elements, and
// reduces its 4*R partial dot products across lanes with a transposing butterfly.
// Split-K partial tiles go to a scratch buffer; the last block of a tile to arrive (per-tile
// arrival counter) adds them in split order -- a deterministic sum -- and runs the fused
// epilogue. No block waits on another.
#include <algorithm>

#include "gemm.cuh"
#include "kernels.h"

namespace cdsl {
namespace {

constexpr int TV = 128;      // virtual output rows per tile
constexpr int KSTEP = 256;   // K elements covered by one warp-wide 128-bit load (32 lanes x 8)
constexpr int THREADS = 256;

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

__device__ __forceinline__ float dot8(const uint4& w, const float4& a, const float4& b) {
  float s = bf_lo(w.x) * a.x;
  s = fmaf(bf_hi(w.x), a.y, s);
  s = fmaf(bf_lo(w.y), a.z, s);
  s = fmaf(bf_hi(w.y), a.w, s);
  s = fmaf(bf_lo(w.z), b.x, s);
  s = fmaf(bf_hi(w.z), b.y, s);
  s = fmaf(bf_lo(w.w), b.z, s);
  s = fmaf(bf_hi(w.w), b.w, s);
  return s;
}

// Sum NV values held by every lane across the 32 lanes. Afterwards value index
// (lane >> shift) lives in v[0] of lane `lane`, shift = log2(32 / NV).
template <int NV>
__device__ __forceinline__ void transpose_reduce(float (&v)[NV]) {
  int n = NV;
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    if (n > 1) {
      const bool upper = (threadIdx.x & off) != 0;
#pragma unroll
      for (int i = 0; i < NV / 2; ++i) {
        if (i < n / 2) {
          const float send = upper ? v[i] : v[i + n / 2];
          const float keep = upper ? v[i + n / 2] : v[i];
          v[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
        }
      }
      n >>= 1;
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], off);
    }
  }
}

template <int RM>
__global__ void __launch_bounds__(THREADS) k_gemv(GemmArgs a, int k_split, int n_splits,
                                                 float* part, int* tile_cnt) {
  const LaunchStamp stamp(a.stamp);
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ float4 smem4[];
  float* xs = reinterpret_cast<float*>(smem4);   // [RM][k_split]
  float* tile = xs + RM * k_split;                // [RM][TV]
  __shared__ int s_last;
  const int tile_id = blockIdx.x, split = blockIdx.y, n_tiles = gridDim.x;
  const int v0 = tile_id * TV;
  const int k0 = split * k_split;
  const int ks = min(k_split, a.K - k0);
  const __nv_bfloat16* xb = reinterpret_cast<const __nv_bfloat16*>(a.x);

  for (int i = threadIdx.x; i < RM * ks; i += THREADS) {
    const int r = i / ks, kk = i - r * ks;
    xs[r * k_split + kk] =
        (r < a.R) ? load_act<__nv_bfloat16>(xb, a.x_plane, (size_t)r * a.ldx + k0 + kk) : 0.f;
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int NV = 4 * RM;
  constexpr int SHIFT = (NV == 32) ? 0 : (NV == 16 ? 1 : 2);
#pragma unroll 1
  for (int rg = 0; rg < 4; ++rg) {
    const int vb = warp * 16 + rg * 4;
    const uint4* wp[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat16* p = virtual_row<__nv_bfloat16>(a, v0 + vb + i);
      wp[i] = p ? reinterpret_cast<const uint4*>(p + k0) : nullptr;
    }
    float acc[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = 0.f;
#pragma unroll 2
    for (int kc = lane * 8; kc < ks; kc += KSTEP) {
      uint4 w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) w[i] = wp[i] ? ld_stream(wp[i] + (kc >> 3)) : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int r = 0; r < RM; ++r) {
        const float4 xa = *reinterpret_cast<const float4*>(xs + r * k_split + kc);
        const float4 xb4 = *reinterpret_cast<const float4*>(xs + r * k_split + kc + 4);
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i * RM + r] += dot8(w[i], xa, xb4);
      }
    }
    transpose_reduce<NV>(acc);
    if ((lane & ((1 << SHIFT) - 1)) == 0) {
      const int idx = lane >> SHIFT;      // = i * RM + r
      const int i = idx / RM, r = idx % RM;
      tile[r * TV + vb + i] = acc[0];
    }
  }
  __syncthreads();

  __shared__ float s_rs[RM];
  if (a.in_ss) {
    input_row_scales(a, 0, min(a.R, RM), s_rs, threadIdx.x, THREADS);
    __syncthreads();
  }
  if (n_splits == 1) {
    tile_epilogue<__nv_bfloat16>(a, v0, 0, min(a.R, RM), tile, TV, s_rs);
    return;
  }
  // split-K: publish this slice's partial tile, the last arriving block reduces and finishes
  float* mine = part + ((size_t)split * RM * n_tiles + tile_id) * TV;
  for (int i = threadIdx.x; i < RM * TV; i += THREADS) {
    const int r = i / TV, v = i % TV;
    mine[(size_t)r * n_tiles * TV + v] = tile[i];
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(tile_cnt + tile_id, 1) == n_splits - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int i = threadIdx.x; i < RM * TV; i += THREADS) {
    const int r = i / TV, v = i % TV;
    float s = 0.f;
    for (int sp = 0; sp < n_splits; ++sp)
      s += __ldcg(part + ((size_t)sp * RM * n_tiles + tile_id) * TV + (size_t)r * n_tiles * TV + v);
    tile[i] = s;
  }
  __syncthreads();
  tile_epilogue<__nv_bfloat16>(a, v0, 0, min(a.R, RM), tile, TV, s_rs);
  if (threadIdx.x == 0) tile_cnt[tile_id] = 0;  // ready for the next launch
}

}  // namespace

GemvPlan plan_gemv(int K, int n_virtual, int n_sm) {
  const int tiles = (n_virtual + TV - 1) / TV;
  const int target = 4 * n_sm;
  int splits = std::max(1, (target + tiles - 1) / tiles);
  int ks = (K + splits - 1) / splits;
  ks = (ks + KSTEP - 1) / KSTEP * KSTEP;
  ks = std::min(std::max(ks, KSTEP), 1024);
  GemvPlan p;
  p.k_split = ks;
  p.splits = (K + ks - 1) / ks;
  p.tiles = tiles;
  return p;
}

size_t gemv_smem_bytes(int rm, int k_split) { return sizeof(float) * ((size_t)rm * k_split + (size_t)rm * TV); }

void launch_gemv(const GemmArgs& a, const GemvPlan& p, float* part, int* tile_cnt, cudaStream_t s) {
  dim3 grid(p.tiles, p.splits);
  if (a.R <= 4) {
    k_gemv<4><<<grid, THREADS, gemv_smem_bytes(4, p.k_split), s>>>(a, p.k_split, p.splits, part, tile_cnt);
  } else {
    k_gemv<8><<<grid, THREADS, gemv_smem_bytes(8, p.k_split), s>>>(a, p.k_split, p.splits, part, tile_cnt);
  }
}

}  // namespace cdsl
