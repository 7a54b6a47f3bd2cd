// gemm.cuh -- the projection GEMMs of the decoder, y = x W^T, with fused epilogues.
//
// A GEMM runs over a "virtual" weight matrix made of up to three segments so that one launch
// covers the fused projections of a layer:
//   EPI_QKV    : [Wq; Wk; Wv] stacked            -> RoPE on q and k, q to a buffer, k/v to KV
//   EPI_SWIGLU : Wg and Wu interleaved in 64-row blocks (virtual rows 128t..128t+63 are gate
//                rows 64t.., the next 64 the matching up rows) -> silu(g) * u
//   EPI_RESID  : one matrix, h += y (residual stream, fp32)
//   EPI_STORE  : one matrix, fp32 store (logits)
// Output features are processed in tiles of 128 virtual rows; every pair the epilogue needs
// (RoPE's (i, i + hd/2), SwiGLU's (gate_j, up_j)) lies inside one tile.
#pragma once

#include "common.cuh"

namespace cdsl {

enum EpiMode : int32_t { EPI_STORE = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };

struct GemmArgs {
  const void* w[3];        // segment base pointers, [rows, K] row-major
  int32_t seg_rows[3];     // rows per segment (multiples of 64 except a final ragged one)
  int32_t n_seg;
  int32_t mode;            // EpiMode
  int32_t K;               // input features
  int32_t n_virtual;       // virtual output rows (padded to a multiple of 128 for SWIGLU)
  const void* x;           // activations [R, ldx] (store_act format of the weight dtype)
  int32_t ldx;
  int64_t x_plane;         // elements between the hi and lo planes of x (bf16 models)
  int32_t R;               // activation rows
  // epilogue outputs
  float* out_f32;          // STORE / RESID: [R, ld_out]
  int32_t ld_out;
  void* out_act;           // SWIGLU: [R, ld_act] (store_act format)
  int32_t ld_act;
  int64_t act_plane;       // SWIGLU: plane distance of out_act
  int32_t d_ffn;           // SWIGLU: valid features
  float* q_out;            // QKV: [R, n_heads * hd] fp32 (rotated)
  int32_t n_heads;
  KvStore kv;              // QKV: destination of k, v
  int32_t layer;
  const RowDesc* rows;     // QKV: per-row position and KV destination
  const float2* rope;      // QKV: [pos][hd/2] (cos, sin)
  int32_t* status;         // device status word (bounded waits report CDSL_ETIMEOUT here)
};

// Pointer to virtual row v of the segmented weight matrix, nullptr for padding rows.
template <typename T>
__device__ __forceinline__ const T* virtual_row(const GemmArgs& a, int v) {
  if (a.mode == EPI_SWIGLU) {
    const int blk = v >> 7, within = v & 127;
    const int row = blk * 64 + (within & 63);
    if (row >= a.d_ffn) return nullptr;
    return reinterpret_cast<const T*>(a.w[within >> 6]) + (size_t)row * a.K;
  }
  int base = 0;
  for (int s = 0; s < a.n_seg; ++s) {
    if (v < base + a.seg_rows[s]) return reinterpret_cast<const T*>(a.w[s]) + (size_t)(v - base) * a.K;
    base += a.seg_rows[s];
  }
  return nullptr;
}

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + expf(-g)); }

// Apply the epilogue to a finished fp32 tile: tile[r * ldt + v] holds y for activation row
// r0 + r and virtual row v0 + v (v in [0, 128)), for r in [0, rt). Run by `nthr` threads
// (tid = 0 .. nthr-1; all threads of the block by default); the caller synchronizes them
// before and after.
template <typename T>
__device__ void tile_epilogue(const GemmArgs& a, int v0, int r0, int rt, const float* tile,
                              int ldt, int tid = -1, int nthr = -1) {
  if (tid < 0) {
    tid = threadIdx.x;
    nthr = blockDim.x;
  }
  const int n_items = rt * 128;
  for (int idx = tid; idx < n_items; idx += nthr) {
    const int r = idx >> 7, v = idx & 127;
    const int row = r0 + r;
    if (row >= a.R) continue;
    const float y = tile[r * ldt + v];
    const int n = v0 + v;
    switch (a.mode) {
      case EPI_STORE:
        if (n < a.n_virtual) a.out_f32[(size_t)row * a.ld_out + n] = y;
        break;
      case EPI_RESID:
        if (n < a.n_virtual) a.out_f32[(size_t)row * a.ld_out + n] += y;
        break;
      case EPI_SWIGLU: {
        if (v >= 64) break;
        const int f = (v0 >> 7) * 64 + v;
        if (f >= a.d_ffn) break;
        const float u = tile[r * ldt + v + 64];
        store_act<T>(reinterpret_cast<T*>(a.out_act), a.act_plane, (size_t)row * a.ld_act + f,
                     silu_f(y) * u);
        break;
      }
      case EPI_QKV: {
        const int hd = a.kv.hd, half = hd >> 1;
        const int nq = a.n_heads * hd, nk = a.kv.kvh * hd;
        if (n >= nq + 2 * nk) break;
        const RowDesc rd = a.rows[row];
        float val = y;
        const int e = n % hd;  // segments start on head boundaries
        if (n < nq + nk) {     // q or k: rotate-half RoPE with the partner in this tile
          const float2 cs = a.rope[(size_t)rd.pos * half + (e % half)];
          const float other = (e < half) ? tile[r * ldt + v + half] : tile[r * ldt + v - half];
          val = (e < half) ? (y * cs.x - other * cs.y) : (y * cs.x + other * cs.y);
        }
        if (n < nq) {
          a.q_out[(size_t)row * nq + n] = val;
        } else {
          const int kvsel = (n < nq + nk) ? 0 : 1;
          const int head = (n - nq - kvsel * nk) / hd;
          float* dst = nullptr;
          if (rd.kv_dst >= 0) {
            dst = a.kv.tail + kv_tail_offset(a.kv, a.layer, kvsel, rd.kv_dst, head);
          } else if (rd.kv_dst == KV_PREFIX) {
            const int page = a.kv.page_table[rd.b * a.kv.max_pages + (rd.pos >> a.kv.page_shift)];
            if (page >= 0)
              dst = a.kv.pool + kv_prefix_offset(a.kv, a.layer, page, kvsel, head,
                                                 rd.pos & ((1 << a.kv.page_shift) - 1));
          }
          if (dst) dst[e] = val;
        }
        break;
      }
    }
  }
}

}  // namespace cdsl
