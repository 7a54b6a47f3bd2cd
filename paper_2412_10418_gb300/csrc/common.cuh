// common.cuh -- shared device-side types of the CDSL step kernels.
//
// Row descriptors describe which token every row of a forward pass carries, where its K/V go
// and which keys it may attend to. One descriptor table serves prefill (causal prompt rows),
// the draft decode calls (one row per beam, plus the pending row of a fully accepted step) and
// the verify pass (k*(d+1) rows per prompt: the shared prefix plus the row's own beam up to
// itself). That is the whole of the "prefix sharing" of the k beams of Algorithm 2.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "../../include/cdsl.h"

namespace cdsl {

// --------------------------------------------------------------------------------------------
// Row descriptors
// --------------------------------------------------------------------------------------------
enum : int32_t { KV_PREFIX = -1, KV_NONE = -2 };

struct RowDesc {
  int32_t b;          // prompt index
  int32_t pos;        // absolute position (RoPE angle, prefix slot when kv_dst == KV_PREFIX)
  int32_t token;      // input token id
  int32_t n_prefix;   // prefix positions [0, n_prefix) visible
  int32_t tail_base;  // first visible tail slot (unused when n_tail == 0)
  int32_t n_tail;     // tail slots [tail_base, tail_base + n_tail) visible
  int32_t kv_dst;     // >= 0: tail slot; KV_PREFIX: prefix pages at pos; KV_NONE: not stored
  int32_t out_idx;    // index of the row's result (beam row / verify row / prompt), -1: none
};
static_assert(sizeof(RowDesc) == 32, "RowDesc is 32 bytes");

// --------------------------------------------------------------------------------------------
// Paged KV cache of one model (float32 elements for every model dtype)
//   pool: [n_layers][n_pages][2 (K,V)][kvh][page_size][hd]
//   tail: [n_layers][2 (K,V)][n_tail_slots][kvh][hd]          (per-beam rows of one step)
//   page_table: [B][max_pages] page ids, -1 = unallocated
// --------------------------------------------------------------------------------------------
struct KvStore {
  float* pool;
  float* tail;
  int32_t* page_table;
  int32_t n_pages;
  int32_t page_shift;  // log2(page_size)
  int32_t max_pages;   // page-table columns per prompt
  int32_t kvh;
  int32_t hd;
  int32_t n_tail_slots;
  int32_t n_layers;
  int32_t pad_;
};

__host__ __device__ inline size_t kv_prefix_offset(const KvStore& s, int layer, int page, int kv,
                                                   int head, int slot) {
  const size_t P = size_t(1) << s.page_shift;
  return ((((size_t)layer * s.n_pages + page) * 2 + kv) * s.kvh + head) * P * s.hd +
         (size_t)slot * s.hd;
}

__host__ __device__ inline size_t kv_tail_offset(const KvStore& s, int layer, int kv, int tslot,
                                                 int head) {
  return ((((size_t)layer * 2 + kv) * s.n_tail_slots + tslot) * s.kvh + head) * (size_t)s.hd;
}

// --------------------------------------------------------------------------------------------
// Element helpers (weights / KV / GEMM activations are float or bf16; math is fp32)
// --------------------------------------------------------------------------------------------
template <typename T> __device__ __forceinline__ float to_f32(T v);
template <> __device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}
template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// GEMM-input activations. float32 models: one fp32 plane. bf16 models: two bf16 planes,
// hi = bf16(x) and lo = bf16(x - hi), `plane` elements apart, so that tensor cores (whose two
// operands share one 16-bit type) see x to about 16 mantissa bits: y = W hi + W lo.
template <typename T> __device__ __forceinline__ void store_act(T* buf, size_t plane, size_t i, float v);
template <> __device__ __forceinline__ void store_act<float>(float* buf, size_t, size_t i, float v) {
  buf[i] = v;
}
template <> __device__ __forceinline__ void store_act<__nv_bfloat16>(__nv_bfloat16* buf, size_t plane,
                                                                    size_t i, float v) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  buf[i] = hi;
  buf[plane + i] = __float2bfloat16_rn(v - __bfloat162float(hi));
}
template <typename T> __device__ __forceinline__ float load_act(const T* buf, size_t plane, size_t i);
template <> __device__ __forceinline__ float load_act<float>(const float* buf, size_t, size_t i) {
  return buf[i];
}
template <> __device__ __forceinline__ float load_act<__nv_bfloat16>(const __nv_bfloat16* buf, size_t plane,
                                                                    size_t i) {
  return __bfloat162float(buf[i]) + __bfloat162float(buf[plane + i]);
}

// Device wall clock in nanoseconds (%globaltimer).
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// In-graph launch timing (cdsl_profile mode 2). A launch's record is three 64-bit words
// kStampStride apart: [0] the first block's entry, [1] the last block's exit (globaltimer ns,
// reset to ~0 and 0 before each step), [2] bytes the kernel counted itself (attention), or 0.
// Thread 0 of every block stamps its entry when constructed and its exit when destroyed.
constexpr int kStampStride = 16384;   // launches per stamped step, at most
struct LaunchStamp {
  unsigned long long* p;
  __device__ __forceinline__ explicit LaunchStamp(unsigned long long* rec)
      : p(threadIdx.x == 0 && threadIdx.y == 0 ? rec : nullptr) {
    if (p) atomicMin(p, (unsigned long long)globaltimer_ns());
  }
  __device__ __forceinline__ ~LaunchStamp() {
    if (p) atomicMax(p + kStampStride, (unsigned long long)globaltimer_ns());
  }
  __device__ __forceinline__ void add_bytes(unsigned long long b) const {
    if (p) atomicAdd(p + 2 * kStampStride, b);
  }
};

// Device status word: first error wins, later ones are dropped.
__device__ __forceinline__ void set_status(int32_t* status, int32_t code) {
  if (status) atomicCAS(status, 0, code);
}

// Orderable key for a (value, index) argmax with the lower index winning equal values:
// larger key <=> larger value, then smaller index.
__device__ __forceinline__ unsigned long long argmax_key(float v, int32_t idx) {
  uint32_t u = __float_as_uint(v);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (uint32_t)(~(uint32_t)idx);
}
__device__ __forceinline__ int32_t argmax_key_index(unsigned long long key) {
  return (int32_t)(~(uint32_t)(key & 0xffffffffull));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  return v;
}

// Programmatic dependent launch: wait for the producer grid's results / let the next grid in.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch with programmatic stream serialization allowed: the kernel may be scheduled while its
// predecessor is still running; it must execute pdl_wait() before touching anything the
// predecessor writes (every kernel of this library does).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Same, as thread-block clusters of cluster_x blocks along x (gridDim.x a multiple of it).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                      int cluster_x, cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)cluster_x;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace cdsl
