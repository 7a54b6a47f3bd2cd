// noalloc.cu -- cdsl_gemv_noalloc: the weight-streaming GEMM for callers that cannot allocate.
//
// Some callers cannot hand this library a workspace: code that runs while a stream is being
// captured in global capture mode (where cudaMalloc is an error), a host framework whose own
// allocator has already reserved the GPU's memory, or a latency-critical loop that must not
// block on cudaMalloc / cudaFree. For them this entry point runs the same split-K kernel the
// draft calls use, with every byte of its scratch -- the hi/lo activation planes, the split-K
// partial tiles and the per-tile arrival counters -- in one fixed device array below. The
// array is created with the library's module on every GPU that loads it and lives until the
// process exits; nothing is allocated per call.
//
// Host code must not pass the array's name to a kernel: on the host that name is only a
// stand-in symbol, not a device address. The device address is looked up once per device,
// with that device current, by cudaGetSymbolAddress, and passed to the kernels.
#include <mutex>

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

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char* g_scratch_dev[kMaxDevices] = {};

// x [n] fp32 -> hi plane [n], lo plane [n] (the GEMM-input format of bf16 models)
__global__ void k_split_planes(const float* x, int n, __nv_bfloat16* planes) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) store_act<__nv_bfloat16>(planes, (size_t)n, (size_t)i, x[i]);
}

// Device address of the scratch array on the current device (set-up on first use).
int scratch_address(unsigned char** out, const char** why) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *why = "cdsl_gemv_noalloc: no usable current CUDA device";
    return CDSL_ECUDA;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_gemv_scratch) != cudaSuccess || !p) {
      *why = "cdsl_gemv_noalloc: cudaGetSymbolAddress of the scratch array failed";
      return CDSL_ECUDA;
    }
    // the arrival counters must start at zero (each launch leaves them at zero again)
    if (cudaMemset(static_cast<unsigned char*>(p) + kPartBytes, 0, kCntBytes) != cudaSuccess) {
      *why = "cdsl_gemv_noalloc: clearing the arrival counters failed";
      return CDSL_ECUDA;
    }
    g_scratch_dev[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_dev[dev];
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
