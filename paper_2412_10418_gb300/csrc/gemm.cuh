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
//
// RMSNorm is folded into the GEMMs: RMSNorm(h) g W^T = rsqrt(mean(h^2) + eps) * ((h . g) W^T),
// the row scale factoring out of the dot product. A RESID epilogue therefore also writes the
// next GEMM's input h . g_next (GEMM-input format) and per 32-feature chunk the partial sums
// of h^2 (and, for the reward head, of w . g . h); the consuming GEMM's epilogue multiplies by
// the row scale computed from those partials in a fixed order (deterministic).
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
  // input normalization: rows are h . g, scale by rsqrt(sum(in_ss[c][r]) / norm_D + eps)
  const float* in_ss;      // [norm_D / 32][ld_ss] partial sums of squares, or nullptr
  int32_t norm_D;
  int32_t ld_ss;           // row stride of the partial-sum arrays (>= R)
  float norm_eps;
  // RESID: next GEMM input and its partial sums
  void* next_x;            // [R, ld_out] GEMM-input format (plane distance act_plane), or nullptr
  const void* next_g;      // [ld_out] gain of the next RMSNorm (weight dtype)
  float* out_ss;           // [ld_out / 32][ld_ss]
  const float* head_w;     // reward head vector [ld_out] (last target layer only), or nullptr
  float* out_hw;           // [ld_out / 32][ld_ss] partial sums of head_w . g . h
};

// Row scale rsqrt(mean(h^2) + eps) from the 32-feature partial sums of row r. The partials
// are summed as four interleaved sequential sums S_q over chunks c = q (mod 4), combined as
// (S_0 + S_1) + (S_2 + S_3): input_row_scales below takes the same order across four lanes,
// so every consumer of a row derives the same bits.
__device__ __forceinline__ float row_scale(const float* ss, int chunks, int ld, int r, int D,
                                           float eps) {
  float q[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    q[j] = 0.f;
    for (int c = j; c < chunks; c += 4) q[j] += ss[(size_t)c * ld + r];
  }
  return rsqrtf(((q[0] + q[1]) + (q[2] + q[3])) / (float)D + eps);
}

// rs[i] = row scale of input row r0 + i for i < n (0 past a.R), computed by `nthr` threads
// (a multiple of 32, tid = 0 .. nthr-1): lane quads split each row's partials four ways so
// that all loads of a row are in flight together. The caller synchronizes afterwards.
__device__ __forceinline__ void input_row_scales(const GemmArgs& a, int r0, int n, float* rs,
                                                 int tid, int nthr);

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
// r0 + r and virtual row v0 + v (v in [0, 128)), for r in [0, rt). s_rs[r] is the input row
// scale of row r0 + r when a.in_ss is set (see input_row_scales). Run by `nthr` threads (a
// multiple of 32; tid = 0 .. nthr-1; all threads of the block by default), which the caller
// synchronizes before and after.
template <typename T>
__device__ void tile_epilogue(const GemmArgs& a, int v0, int r0, int rt, const float* tile,
                              int ldt, const float* s_rs, int tid = -1, int nthr = -1) {
  if (tid < 0) {
    tid = threadIdx.x;
    nthr = blockDim.x;
  }
  const int n_items = rt * 128;   // a multiple of 32: every warp sees 32 features of one row
  for (int idx = tid; idx < n_items; idx += nthr) {
    const int r = idx >> 7, v = idx & 127;
    const int row = r0 + r;
    const bool live = row < a.R;
    float y = tile[r * ldt + v];
    if (a.in_ss) y *= s_rs[r];
    const int n = v0 + v;
    switch (a.mode) {
      case EPI_STORE:
        if (live && n < a.n_virtual) a.out_f32[(size_t)row * a.ld_out + n] = y;
        break;
      case EPI_RESID: {
        float hn = 0.f;
        if (live && n < a.n_virtual) {
          float* hp = a.out_f32 + (size_t)row * a.ld_out + n;
          hn = *hp + y;
          *hp = hn;
          if (a.next_x)
            store_act<T>(reinterpret_cast<T*>(a.next_x), a.act_plane, (size_t)row * a.ld_out + n,
                         hn * to_f32<T>(reinterpret_cast<const T*>(a.next_g)[n]));
        }
        if (a.out_ss) {   // warp-uniform: 32 consecutive features of one row
          const float sq = warp_sum(hn * hn);
          float hw = 0.f;
          if (a.head_w) {
            const float gw = (live && n < a.n_virtual)
                                 ? a.head_w[n] * to_f32<T>(reinterpret_cast<const T*>(a.next_g)[n])
                                 : 0.f;
            hw = warp_sum(gw * hn);
          }
          if ((v & 31) == 0 && live && n < a.n_virtual) {
            a.out_ss[(size_t)(n >> 5) * a.ld_ss + row] = sq;
            if (a.head_w) a.out_hw[(size_t)(n >> 5) * a.ld_ss + row] = hw;
          }
        }
        break;
      }
      case EPI_SWIGLU: {
        if (!live || v >= 64) break;
        const int f = (v0 >> 7) * 64 + v;
        if (f >= a.d_ffn) break;
        float u = tile[r * ldt + v + 64];
        if (a.in_ss) u *= s_rs[r];
        store_act<T>(reinterpret_cast<T*>(a.out_act), a.act_plane, (size_t)row * a.ld_act + f,
                     silu_f(y) * u);
        break;
      }
      case EPI_QKV: {
        if (!live) break;
        const int hd = a.kv.hd, half = hd >> 1;
        const int nq = a.n_heads * hd, nk = a.kv.kvh * hd;
        if (n >= nq + 2 * nk) break;
        const RowDesc rd = a.rows[row];
        float val = y;
        const int e = n % hd;  // segments start on head boundaries
        if (n < nq + nk) {     // q or k: rotate-half RoPE with the partner in this tile
          const float2 cs = a.rope[(size_t)rd.pos * half + (e % half)];
          float other = (e < half) ? tile[r * ldt + v + half] : tile[r * ldt + v - half];
          if (a.in_ss) other *= s_rs[r];
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

__device__ __forceinline__ void input_row_scales(const GemmArgs& a, int r0, int n, float* rs,
                                                 int tid, int nthr) {
  const int chunks = a.norm_D >> 5, items = n * 4;
  for (int base = tid & ~31; base < items; base += nthr) {   // warp-uniform trip count
    const int idx = base + (tid & 31), r = idx >> 2, q = idx & 3, row = r0 + r;
    const bool live = idx < items && row < a.R;
    float acc = 0.f;
    if (live) {
#pragma unroll 8
      for (int c = q; c < chunks; c += 4) acc += a.in_ss[(size_t)c * a.ld_ss + row];
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);   // (S_0 + S_1), (S_2 + S_3)
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);   // (S_0 + S_1) + (S_2 + S_3)
    if (idx < items && q == 0) rs[r] = live ? rsqrtf(acc / (float)a.norm_D + a.norm_eps) : 0.f;
  }
}

}  // namespace cdsl
