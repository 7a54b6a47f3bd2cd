// noalloc.cu -- cdsl_gemv_noalloc: the weight-streaming GEMM for callers that cannot allocate.
//
// Some callers cannot hand this library a workspace: a host framework whose own caching
// allocator has already reserved the GPU's memory, a real-time loop that must not block on
// cudaMalloc / cudaFree, a runtime that forbids device allocation after start-up. For them this
// entry point runs the CUDA-core split-K GEMV (gemv_stream.cu) with every byte of its scratch --
// the hi/lo activation planes, the split-K partial tiles and the per-tile arrival counters --
// in one fixed device array below. The array is created with the library's module on every GPU
// that loads it and lives until the process exits; nothing is allocated per call.
//
// Host code must not pass the array's name to a kernel: on the host that name is only a
// stand-in symbol, not a device address. The device address is looked up once per CUDA
// context, with that context current, by cudaGetSymbolAddress, and passed to the kernels.
#include <cuda.h>

#include <mutex>
#include <utility>
#include <vector>

#include "gemm.cuh"
#include "kernels.h"

namespace cdsl {
namespace {

constexpr int kMaxR = 8;
constexpr int kMaxK = 8192;
constexpr int kMaxN = 32768;
constexpr int kMaxTiles = kMaxN / 128;
// Split-K partials: at most 8 splits x 8 rows x 256 tiles x 128 floats (the planner's worst
// case over the limits above; checked per call).
constexpr size_t kPartFloats = (size_t)8 * kMaxR * kMaxTiles * 128;
constexpr size_t kPartBytes = kPartFloats * sizeof(float);                 // 8 MiB
constexpr size_t kCntBytes = kMaxTiles * sizeof(int32_t);                  // 1 KiB
constexpr size_t kPlaneElems = (size_t)kMaxR * kMaxK;                      // per plane
constexpr size_t kPlaneBytes = 2 * kPlaneElems * sizeof(__nv_bfloat16);    // 256 KiB
constexpr size_t kScratchBytes = kPartBytes + kCntBytes + kPlaneBytes;

static __device__ __align__(256) unsigned char g_gemv_scratch[kScratchBytes];

std::mutex g_mu;
// (context, device address of the array in it), one entry per context set up so far
std::vector<std::pair<CUcontext, unsigned char*>> g_scratch_ctx;
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
CtxGetCurrentFn g_ctx_get_current = nullptr;

// x [n] fp32 -> hi plane [n], lo plane [n] (the GEMM-input format of bf16 models)
__global__ void k_split_planes(const float* x, int n, __nv_bfloat16* planes) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) store_act<__nv_bfloat16>(planes, (size_t)n, (size_t)i, x[i]);
}

// The current CUDA context (the runtime's primary context of the current device once a
// runtime call has made it current); nullptr where none is current yet.
CUcontext current_context() {
  if (!g_ctx_get_current) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return nullptr;
    g_ctx_get_current = reinterpret_cast<CtxGetCurrentFn>(fn);
  }
  CUcontext c = nullptr;
  return g_ctx_get_current(&c) == CUDA_SUCCESS ? c : nullptr;
}

// Device address of the scratch array in the current context (set-up on first use there).
int scratch_address(unsigned char** out, const char** why) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) {
    *why = "cdsl_gemv_noalloc: no usable current CUDA device";
    return CDSL_ECUDA;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  CUcontext ctx = current_context();
  for (const auto& e : g_scratch_ctx)
    if (ctx && e.first == ctx) {
      *out = e.second;
      return CDSL_OK;
    }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_gemv_scratch) != cudaSuccess || !p) {
    *why = "cdsl_gemv_noalloc: cudaGetSymbolAddress of the scratch array failed";
    return CDSL_ECUDA;
  }
  ctx = current_context();   // the lookup above made the device's primary context current
  if (!ctx) {
    *why = "cdsl_gemv_noalloc: no current CUDA context";
    return CDSL_ECUDA;
  }
  // the arrival counters must start at zero (each launch leaves them at zero again)
  if (cudaMemset(static_cast<unsigned char*>(p) + kPartBytes, 0, kCntBytes) != cudaSuccess) {
    *why = "cdsl_gemv_noalloc: clearing the arrival counters failed";
    return CDSL_ECUDA;
  }
  g_scratch_ctx.emplace_back(ctx, static_cast<unsigned char*>(p));
  *out = static_cast<unsigned char*>(p);
  return CDSL_OK;
}

}  // namespace
}  // namespace cdsl

using namespace cdsl;

extern "C" int32_t cdsl_gemv_noalloc(const void* d_w, int32_t N, int32_t K, const float* d_x,
                                     int32_t R, float* d_y, void* stream) {
  auto aligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  if (!d_w || !d_x || !d_y || !aligned(d_w) || !aligned(d_x) || !aligned(d_y)) {
    set_thread_error("cdsl_gemv_noalloc: pointers must be non-NULL and 16-byte aligned");
    return CDSL_EINVAL;
  }
  if (R < 1 || R > kMaxR || K < 8 || K > kMaxK || (K % 8) || N < 1 || N > kMaxN) {
    set_thread_error("cdsl_gemv_noalloc: sizes beyond the fixed scratch: need 1 <= R <= 8, "
                     "8 <= K <= 8192 with K % 8 == 0, 1 <= N <= 32768");
    return CDSL_EINVAL;
  }
  const GemvPlan plan = plan_gemv(K, N, kPlanSMs);
  if (plan.tiles > kMaxTiles || (size_t)plan.splits * kMaxR * plan.tiles * 128 > kPartFloats) {
    set_thread_error("cdsl_gemv_noalloc: split-K plan exceeds the fixed scratch");
    return CDSL_EINVAL;
  }
  unsigned char* base = nullptr;
  const char* why = nullptr;
  if (int e = scratch_address(&base, &why)) {
    set_thread_error(why);
    return e;
  }
  float* part = reinterpret_cast<float*>(base);
  int32_t* cnt = reinterpret_cast<int32_t*>(base + kPartBytes);
  __nv_bfloat16* planes = reinterpret_cast<__nv_bfloat16*>(base + kPartBytes + kCntBytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int n = R * K;
  k_split_planes<<<(n + 255) / 256, 256, 0, s>>>(d_x, n, planes);

  GemmArgs a{};
  a.w[0] = d_w;
  a.seg_rows[0] = N;
  a.n_seg = 1;
  a.mode = EPI_STORE;
  a.K = K;
  a.n_virtual = N;
  a.x = planes;
  a.ldx = K;
  a.x_plane = n;
  a.R = R;
  a.out_f32 = d_y;
  a.ld_out = N;
  launch_gemv(a, plan, part, cnt, s);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_thread_error(cudaGetErrorString(e));
    return CDSL_ECUDA;
  }
  return CDSL_OK;
}
