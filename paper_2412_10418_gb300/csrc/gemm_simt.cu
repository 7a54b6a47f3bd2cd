// gemm_simt.cu -- plain shared-memory tiled GEMM on the CUDA cores, y = x W^T + epilogue.
//
// The general fallback: any row count, float32 or bf16 operands, fp32 accumulation. It is
// the exact-fp32 path of the float32 workload (tensor cores would round to tf32) and the
// path for shapes the tensor-core and weight-streaming kernels do not cover.
// Tile: 128 virtual output rows x 32 activation rows per block, K in steps of 32.
#include "gemm.cuh"
#include "kernels.h"

namespace cdsl {
namespace {

constexpr int TV = 128, TR = 32, TK = 32;

template <typename T>
__global__ void __launch_bounds__(256) k_gemm_simt(GemmArgs a) {
  const LaunchStamp stamp(a.stamp);
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float Ws[TK][TV + 1];
  __shared__ float Xs[TK][TR + 1];
  __shared__ float Ys[TR * (TV + 4)];
  __shared__ float s_rs[TR];
  const int v0 = blockIdx.x * TV;
  const int tid = threadIdx.x;
  const int v = tid & (TV - 1);
  const int rb = (tid >> 7) * 16;
  const T* xw = reinterpret_cast<const T*>(a.x);
  // weight row pointers of this thread's loads: row (idx / TK) for idx = tid + i*256
  for (int r0 = 0; r0 < a.R; r0 += TR) {
    float acc[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = 0.f;
    for (int k0 = 0; k0 < a.K; k0 += TK) {
#pragma unroll 4
      for (int i = 0; i < (TV * TK) / 256; ++i) {
        const int idx = tid + i * 256;
        const int vv = idx / TK, kk = idx % TK;
        const T* wr = virtual_row<T>(a, v0 + vv);
        float w = 0.f;
        if (wr && k0 + kk < a.K) w = to_f32<T>(wr[k0 + kk]);
        Ws[kk][vv] = w;
      }
#pragma unroll
      for (int i = 0; i < (TR * TK) / 256; ++i) {
        const int idx = tid + i * 256;
        const int rr = idx / TK, kk = idx % TK;
        float xv = 0.f;
        if (r0 + rr < a.R && k0 + kk < a.K)
          xv = load_act<T>(xw, a.x_plane, (size_t)(r0 + rr) * a.ldx + k0 + kk);
        Xs[kk][rr] = xv;
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < TK; ++kk) {
        const float w = Ws[kk][v];
#pragma unroll
        for (int i = 0; i < 16; ++i) acc[i] += w * Xs[kk][rb + i];
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) Ys[(rb + i) * (TV + 4) + v] = acc[i];
    if (a.in_ss) input_row_scales(a, r0, min(TR, a.R - r0), s_rs, tid, 256);
    __syncthreads();
    tile_epilogue<T>(a, v0, r0, min(TR, a.R - r0), Ys, TV + 4, s_rs);
    __syncthreads();
  }
}

}  // namespace

void launch_gemm_simt(int dtype, const GemmArgs& a, cudaStream_t s) {
  const int tiles = (a.n_virtual + TV - 1) / TV;
  if (dtype == CDSL_DTYPE_BF16)
    k_gemm_simt<__nv_bfloat16><<<tiles, 256, 0, s>>>(a);
  else
    k_gemm_simt<float><<<tiles, 256, 0, s>>>(a);
}

}  // namespace cdsl
