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
  uint64_t wait_ns;        // limit of the tensor-core kernel's pipeline waits (nanoseconds)
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
  unsigned long long* stamp;  // in-graph launch timing record (LaunchStamp), or nullptr
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

// Items of a tile each epilogue thread works on per pass in the batched epilogues (their loads
// in flight together).
constexpr int kEpiBatch = 8;

// What the QKV epilogue needs of one activation row: the RoPE position and where the row's k
// and v go (element offset of k, head 0 in the prefix pool or the beam tails). A kernel that
// finishes many tiles over the same rows gathers these once (qkv_rows) instead of every tile
// reading the row descriptor and the page table again.
struct QkvRow {
  int32_t pos;
  int32_t where;   // 0: not stored, 1: prefix pool, 2: beam tail
  int64_t base;
};

// rows[i] for activation rows i < n (by `nthr` threads, tid = 0 .. nthr-1; the caller
// synchronizes afterwards).
__device__ __forceinline__ void qkv_rows(const GemmArgs& a, int n, QkvRow* rows, int tid,
                                         int nthr) {
  const KvStore& kv = a.kv;
  for (int r = tid; r < n; r += nthr) {
    const RowDesc rd = a.rows[r];
    QkvRow m{rd.pos, 0, 0};
    if (rd.kv_dst >= 0) {
      m.where = 2;
      m.base = (int64_t)kv_tail_offset(kv, a.layer, 0, rd.kv_dst, 0);
    } else if (rd.kv_dst == KV_PREFIX) {
      const int page = kv.page_table[rd.b * kv.max_pages + (rd.pos >> kv.page_shift)];
      if (page >= 0) {
        m.where = 1;
        m.base = (int64_t)kv_prefix_offset(kv, a.layer, page, 0, 0,
                                           rd.pos & ((1 << kv.page_shift) - 1));
      }
    }
    rows[r] = m;
  }
}

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + expf(-g)); }

// Apply the epilogue to a finished fp32 tile: tile[r * ldt + v] holds y for activation row
// r0 + r and virtual row v0 + v (v in [0, 128)), for r in [0, rt). s_rs[r] is the input row
// scale of row r0 + r when a.in_ss is set (see input_row_scales). kBatch: the residual and
// QKV epilogues issue kEpiBatch items' loads per thread before their stores (for tiles of many
// rows); the QKV one then takes the rows' QkvRow from qrows (indexed by row, not r). Run by
// `nthr` threads (a multiple of 32; tid = 0 .. nthr-1; all threads of the block by default),
// which the caller synchronizes before and after.
template <typename T, bool kBatch = false>
__device__ void tile_epilogue(const GemmArgs& a, int v0, int r0, int rt, const float* tile,
                              int ldt, const float* s_rs, int tid = -1, int nthr = -1,
                              const QkvRow* qrows = nullptr) {
  if (tid < 0) {
    tid = threadIdx.x;
    nthr = blockDim.x;
  }
  // Every field is read once, into registers, before the stores: `a` is reached through a
  // reference (to the kernel parameter), which the compiler must otherwise assume the stores
  // below may alias, re-reading it on every item.
  const int mode = a.mode, R = a.R, nv = a.n_virtual;
  const bool scaled = a.in_ss != nullptr;
  const float* __restrict__ tl = tile;   // shared memory: never aliases the outputs
  if (mode == EPI_STORE) {
    float* __restrict__ const out = a.out_f32;
    const size_t ld = (size_t)a.ld_out;
    for (int idx = tid; idx < rt * 128; idx += nthr) {
      const int r = idx >> 7, v = idx & 127, row = r0 + r, n = v0 + v;
      float y = tl[r * ldt + v];
      if (scaled) y *= s_rs[r];
      if (row < R && n < nv) out[(size_t)row * ld + n] = y;
    }
  } else if (mode == EPI_RESID && !kBatch) {
    float* __restrict__ const out = a.out_f32;
    const size_t ld = (size_t)a.ld_out, plane = (size_t)a.act_plane, ld_ss = (size_t)a.ld_ss;
    T* const next_x = reinterpret_cast<T*>(a.next_x);
    const T* const next_g = reinterpret_cast<const T*>(a.next_g);
    float* const out_ss = a.out_ss;
    const float* const head_w = a.head_w;
    float* const out_hw = a.out_hw;
    // a multiple of 32 items per thread pass: every warp sees 32 features of one row
    for (int idx = tid; idx < rt * 128; idx += nthr) {
      const int r = idx >> 7, v = idx & 127, row = r0 + r, n = v0 + v;
      const bool ok = row < R && n < nv;
      float y = tl[r * ldt + v];
      if (scaled) y *= s_rs[r];
      float hn = 0.f;
      if (ok) {
        float* hp = out + (size_t)row * ld + n;
        hn = *hp + y;
        *hp = hn;
        if (next_x)
          store_act<T>(next_x, plane, (size_t)row * ld + n, hn * to_f32<T>(next_g[n]));
      }
      if (out_ss) {   // warp-uniform
        const float sq = warp_sum(hn * hn);
        float hw = 0.f;
        if (head_w) {
          const float gw = ok ? head_w[n] * to_f32<T>(next_g[n]) : 0.f;
          hw = warp_sum(gw * hn);
        }
        if ((v & 31) == 0 && ok) {
          out_ss[(size_t)(n >> 5) * ld_ss + row] = sq;
          if (head_w) out_hw[(size_t)(n >> 5) * ld_ss + row] = hw;
        }
      }
    }
  } else if (mode == EPI_RESID) {
    float* __restrict__ const out = a.out_f32;
    const size_t ld = (size_t)a.ld_out, plane = (size_t)a.act_plane, ld_ss = (size_t)a.ld_ss;
    T* const next_x = reinterpret_cast<T*>(a.next_x);
    const T* const next_g = reinterpret_cast<const T*>(a.next_g);
    float* const out_ss = a.out_ss;
    const float* const head_w = a.head_w;
    float* const out_hw = a.out_hw;
    // kEpiBatch items per thread per pass: every residual load of a pass is issued
    // before its first store, so a tile of many rows costs rt / kEpiBatch round trips to
    // memory instead of rt. Every warp sees 32 features of one row (warp_sum below).
    const int items = rt * 128;
    for (int base = tid; base < items; base += nthr * kEpiBatch) {
      float hres[kEpiBatch];
#pragma unroll
      for (int u = 0; u < kEpiBatch; ++u) {
        const int idx = base + u * nthr, r = idx >> 7, v = idx & 127, row = r0 + r, n = v0 + v;
        hres[u] = (idx < items && row < R && n < nv) ? out[(size_t)row * ld + n] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kEpiBatch; ++u) {
        const int idx = base + u * nthr;
        if (idx >= items) break;   // warp-uniform (items and nthr are multiples of 32)
        const int r = idx >> 7, v = idx & 127, row = r0 + r, n = v0 + v;
        const bool ok = row < R && n < nv;
        float y = tl[r * ldt + v];
        if (scaled) y *= s_rs[r];
        float hn = 0.f;
        if (ok) {
          hn = hres[u] + y;
          out[(size_t)row * ld + n] = hn;
          if (next_x)
            store_act<T>(next_x, plane, (size_t)row * ld + n, hn * to_f32<T>(next_g[n]));
        }
        if (out_ss) {   // warp-uniform
          const float sq = warp_sum(hn * hn);
          float hw = 0.f;
          if (head_w) {
            const float gw = ok ? head_w[n] * to_f32<T>(next_g[n]) : 0.f;
            hw = warp_sum(gw * hn);
          }
          if ((v & 31) == 0 && ok) {
            out_ss[(size_t)(n >> 5) * ld_ss + row] = sq;
            if (head_w) out_hw[(size_t)(n >> 5) * ld_ss + row] = hw;
          }
        }
      }
    }
  } else if (mode == EPI_SWIGLU) {
    T* const out_act = reinterpret_cast<T*>(a.out_act);
    const size_t ld_act = (size_t)a.ld_act, plane = (size_t)a.act_plane;
    const int d_ffn = a.d_ffn, f0 = (v0 >> 7) * 64;
    for (int idx = tid; idx < rt * 64; idx += nthr) {   // gate v, up v + 64
      const int r = idx >> 6, v = idx & 63, row = r0 + r, f = f0 + v;
      if (row >= R || f >= d_ffn) continue;
      float g = tl[r * ldt + v], u = tl[r * ldt + v + 64];
      if (scaled) {
        g *= s_rs[r];
        u *= s_rs[r];
      }
      store_act<T>(out_act, plane, (size_t)row * ld_act + f, silu_f(g) * u);
    }
  } else {   // EPI_QKV
    const KvStore kv = a.kv;
    float* const q_out = a.q_out;
    const RowDesc* const rows = a.rows;
    const float2* const rope = a.rope;
    const int layer = a.layer;
    const int hd = kv.hd, half = hd >> 1;
    const int nq = a.n_heads * hd, nk = kv.kvh * hd;
    if constexpr (kBatch) if (qrows) {
      const int items = rt * 128;
      // kEpiBatch items per thread per pass: their RoPE factors in flight together
      const size_t kv_pool = (size_t)kv.kvh * hd << kv.page_shift, h_pool = (size_t)hd
                                                                             << kv.page_shift;
      const size_t kv_tail = (size_t)kv.n_tail_slots * kv.kvh * hd, h_tail = (size_t)hd;
      for (int base = tid; base < items; base += nthr * kEpiBatch) {
        float2 cs[kEpiBatch];
#pragma unroll
        for (int u = 0; u < kEpiBatch; ++u) {
          const int idx = base + u * nthr, row = r0 + (idx >> 7), n = v0 + (idx & 127);
          cs[u] = (idx < items && row < R && n < nq + nk)
                      ? rope[(size_t)qrows[row].pos * half + ((n % hd) % half)]
                      : make_float2(1.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kEpiBatch; ++u) {
          const int idx = base + u * nthr, r = idx >> 7, v = idx & 127, row = r0 + r,
                    n = v0 + v;
          if (idx >= items || row >= R || n >= nq + 2 * nk) continue;
          float y = tl[r * ldt + v];
          if (scaled) y *= s_rs[r];
          float val = y;
          const int e = n % hd;
          if (n < nq + nk) {
            float other = (e < half) ? tl[r * ldt + v + half] : tl[r * ldt + v - half];
            if (scaled) other *= s_rs[r];
            val = (e < half) ? (y * cs[u].x - other * cs[u].y) : (y * cs[u].x + other * cs[u].y);
          }
          if (n < nq) {
            q_out[(size_t)row * nq + n] = val;
          } else {
            const QkvRow m = qrows[row];
            const int kvsel = (n < nq + nk) ? 0 : 1;
            const int head = (n - nq - kvsel * nk) / hd;
            if (m.where == 1)
              kv.pool[(size_t)m.base + kvsel * kv_pool + head * h_pool + e] = val;
            else if (m.where == 2)
              kv.tail[(size_t)m.base + kvsel * kv_tail + head * h_tail + e] = val;
          }
        }
      }
      return;
    }
    for (int idx = tid; idx < rt * 128; idx += nthr) {
      const int r = idx >> 7, v = idx & 127, row = r0 + r, n = v0 + v;
      if (row >= R || n >= nq + 2 * nk) continue;
      float y = tl[r * ldt + v];
      if (scaled) y *= s_rs[r];
      const RowDesc rd = rows[row];
      float val = y;
      const int e = n % hd;  // segments start on head boundaries
      if (n < nq + nk) {     // q or k: rotate-half RoPE with the partner in this tile
        const float2 cs = rope[(size_t)rd.pos * half + (e % half)];
        float other = (e < half) ? tl[r * ldt + v + half] : tl[r * ldt + v - half];
        if (scaled) other *= s_rs[r];
        val = (e < half) ? (y * cs.x - other * cs.y) : (y * cs.x + other * cs.y);
      }
      if (n < nq) {
        q_out[(size_t)row * nq + n] = val;
      } else {
        const int kvsel = (n < nq + nk) ? 0 : 1;
        const int head = (n - nq - kvsel * nk) / hd;
        float* dst = nullptr;
        if (rd.kv_dst >= 0) {
          dst = kv.tail + kv_tail_offset(kv, layer, kvsel, rd.kv_dst, head);
        } else if (rd.kv_dst == KV_PREFIX) {
          const int page = kv.page_table[rd.b * kv.max_pages + (rd.pos >> kv.page_shift)];
          if (page >= 0)
            dst = kv.pool + kv_prefix_offset(kv, layer, page, kvsel, head,
                                             rd.pos & ((1 << kv.page_shift) - 1));
        }
        if (dst) dst[e] = val;
      }
    }
  }
}

__device__ __forceinline__ void input_row_scales(const GemmArgs& a, int r0, int n, float* rs,
                                                 int tid, int nthr) {
  const int D = a.norm_D, chunks = D >> 5, items = n * 4, R = a.R;
  const float* const ss = a.in_ss;
  const size_t ld = (size_t)a.ld_ss;
  const float eps = a.norm_eps;
  for (int base = tid & ~31; base < items; base += nthr) {   // warp-uniform trip count
    const int idx = base + (tid & 31), r = idx >> 2, q = idx & 3, row = r0 + r;
    const bool live = idx < items && row < R;
    float acc = 0.f;
    if (live) {
#pragma unroll 8
      for (int c = q; c < chunks; c += 4) acc += ss[(size_t)c * ld + row];
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);   // (S_0 + S_1), (S_2 + S_3)
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);   // (S_0 + S_1) + (S_2 + S_3)
    if (idx < items && q == 0) rs[r] = live ? rsqrtf(acc / (float)D + eps) : 0.f;
  }
}

}  // namespace cdsl
