// attention.cu -- attention of every row of a pass over its prompt's shared prefix pages and
// its own beam tail (decode rows of the draft, the tree-masked verify rows, causal prefill).
//
// Prefix sharing: all rows of one prompt read the same prefix K/V. A block owns one prompt,
// one KV head, one chunk of 64 prefix positions and 32 query vectors (query vector =
// (row, query head of the GQA group)); it loads the chunk's K and V once into shared memory
// and scores all its query vectors against them (split-KV, flash-decoding style). One more
// chunk per query block holds each row's own tail keys (its beam's rows of this pass, causal
// within the beam). Each query vector's partial result (max score m, sum of exponentials l,
// unnormalized output o) goes to scratch; the last block of a (prompt, head, query block) to
// arrive merges the chunks in order (lanes over chunks, all loads in flight) and writes the
// normalized output in the GEMM-input format. fp32 throughout.
//
// Score loop: a warp owns 4 query vectors (broadcast reads), its lanes own keys lane and
// lane + 32 (rows of 132 floats: conflict-free 128-bit reads). Output loop: lanes own 4 (or 2)
// consecutive dims of the 4 query vectors, reading P by broadcast and V row-contiguously.
#include <algorithm>

#include "kernels.h"

namespace cdsl {
namespace {

constexpr int ACH = 64;   // prefix positions per block
constexpr int AQB = 32;   // query vectors per block
constexpr int ATHREADS = 256;

template <int HD>
struct AttnSmem {
  static constexpr int QP = HD + 4;        // padded row pitch of Q and K
  static constexpr size_t floats = (size_t)AQB * QP + (size_t)ACH * QP + (size_t)ACH * HD + (size_t)ACH * AQB;
  static constexpr size_t bytes = floats * sizeof(float);
};

template <typename T, int HD>
__global__ void __launch_bounds__(ATHREADS) k_attn(AttnArgs a) {
  using L = AttnSmem<HD>;
  extern __shared__ float4 sm4[];
  float* qS = reinterpret_cast<float*>(sm4);   // [AQB][QP]  pre-scaled queries
  float* kS = qS + AQB * L::QP;                 // [ACH][QP]
  float* vS = kS + ACH * L::QP;                 // [ACH][HD]
  float* pS = vS + ACH * HD;                    // [ACH][AQB] probabilities
  __shared__ int s_row[AQB], s_gg[AQB], s_np[AQB];
  __shared__ int s_wcnt[ATHREADS / 32];
  __shared__ int s_nrows, s_last;
  __shared__ float s_m[AQB], s_l[AQB];
  __shared__ int s_page[ACH];

  const int chunk = blockIdx.x, g = blockIdx.y;
  const int n_pchunks = gridDim.x - 1;          // prefix chunks; x == n_pchunks: tail keys
  const bool tail_chunk = chunk == n_pchunks;
  int b, qb;
  if (a.zmap) {
    b = a.zmap[2 * blockIdx.z];
    qb = a.zmap[2 * blockIdx.z + 1];
  } else {
    b = blockIdx.z / a.qb_count;
    qb = blockIdx.z % a.qb_count;
  }
  const int G = a.G, H = a.n_heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = chunk * ACH;

  // ---- this block's query vectors: rows of prompt b in order, G heads each
  if (threadIdx.x < AQB) s_row[threadIdx.x] = -1;
  if (threadIdx.x == 0) s_nrows = 0;
  __syncthreads();
  for (int base = 0; base < a.R; base += ATHREADS) {
    const int r = base + threadIdx.x;
    const bool mine = r < a.R && a.rows[r].b == b;
    const unsigned bal = __ballot_sync(0xffffffffu, mine);
    if (lane == 0) s_wcnt[warp] = __popc(bal);
    __syncthreads();
    int off = s_nrows;
    for (int w = 0; w < warp; ++w) off += s_wcnt[w];
    const int local = off + __popc(bal & ((1u << lane) - 1));
    if (mine) {
      for (int gg = 0; gg < G; ++gg) {
        const int qi = local * G + gg - qb * AQB;
        if (qi >= 0 && qi < AQB) {
          s_row[qi] = r;
          s_gg[qi] = gg;
          s_np[qi] = a.rows[r].n_prefix;
        }
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < ATHREADS / 32; ++w) tot += s_wcnt[w];
      s_nrows += tot;
    }
    __syncthreads();
  }
  const int nq = min(AQB, s_nrows * G - qb * AQB);
  int maxnp = 0;
  for (int i = 0; i < nq; ++i) maxnp = max(maxnp, s_np[i]);
  // Page ids of this chunk: the rows (plan kernel) and the committed page-table entries come
  // from kernels the launch chain has already completed, so they are read before the wait.
  if (!tail_chunk && nq > 0 && threadIdx.x < ACH) {
    const int t = t0 + threadIdx.x;
    s_page[threadIdx.x] =
        (t < maxnp) ? a.kv.page_table[b * a.kv.max_pages + (t >> a.kv.page_shift)] : -1;
  }
  pdl_wait();                 // q, K/V and the scratch of the previous kernels are ready
  pdl_launch_dependents();
  if (nq <= 0) return;   // no query vector in this block (no block of this group has any)
  const size_t grp = ((size_t)blockIdx.z * gridDim.y + g);
  float* po = a.part_o + (grp * gridDim.x + chunk) * AQB * HD;
  float* pml = a.part_ml + (grp * gridDim.x + chunk) * AQB * 2;

  constexpr int DPL = HD / 32;
  if (tail_chunk) {
    // ---- each row's own tail keys (at most 17): lanes over keys for the scores, over dims
    //      for the output
    for (int qi = warp; qi < nq; qi += ATHREADS / 32) {
      const RowDesc rd = a.rows[s_row[qi]];
      const int nt = min(rd.n_tail, 17);
      const float* qrow = a.q + (size_t)s_row[qi] * H * HD + (size_t)(g * G + s_gg[qi]) * HD;
      float sc = -INFINITY;
      if (lane < nt) {
        const float* kt = a.kv.tail + kv_tail_offset(a.kv, a.layer, 0, rd.tail_base + lane, g);
        float d = 0.f;
#pragma unroll 8
        for (int e = 0; e < HD; e += 4) {
          const float4 qv = *reinterpret_cast<const float4*>(qrow + e);
          const float4 kv = *reinterpret_cast<const float4*>(kt + e);
          d += qv.x * kv.x + qv.y * kv.y + qv.z * kv.z + qv.w * kv.w;
        }
        sc = d * a.scale;
      }
      const float m = warp_max(sc);
      const float pj = (lane < nt) ? expf(sc - m) : 0.f;
      const float l = warp_sum(pj);
      float o[DPL];
#pragma unroll
      for (int c = 0; c < DPL; ++c) o[c] = 0.f;
      for (int j = 0; j < nt; ++j) {
        const float w = __shfl_sync(0xffffffffu, pj, j);
        const float* vt = a.kv.tail + kv_tail_offset(a.kv, a.layer, 1, rd.tail_base + j, g);
#pragma unroll
        for (int c = 0; c < DPL; ++c) o[c] = fmaf(w, vt[DPL * lane + c], o[c]);
      }
#pragma unroll
      for (int c = 0; c < DPL; ++c) po[qi * HD + DPL * lane + c] = o[c];
      if (lane == 0) {
        pml[2 * qi] = (nt > 0) ? m : -INFINITY;
        pml[2 * qi + 1] = l;
      }
    }
  } else if (t0 < maxnp) {
    // ---- stage Q (scaled), K and V of positions t0 .. t0 + ACH - 1
    for (int idx = threadIdx.x; idx < AQB * (HD / 4); idx += ATHREADS) {
      const int qi = idx / (HD / 4), e4 = idx % (HD / 4);
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (qi < nq) {
        v = *reinterpret_cast<const float4*>(a.q + (size_t)s_row[qi] * H * HD +
                                             (size_t)(g * G + s_gg[qi]) * HD + 4 * e4);
        v.x *= a.scale; v.y *= a.scale; v.z *= a.scale; v.w *= a.scale;
      }
      *reinterpret_cast<float4*>(qS + qi * L::QP + 4 * e4) = v;
    }
    const int pmask = (1 << a.kv.page_shift) - 1;
    __syncthreads();   // s_page complete
    // every thread first issues all of its K and V loads, then stores them
    constexpr int PER = ACH * (HD / 4) / ATHREADS;   // float4 per thread per matrix
    float4 kr[PER], vr[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int idx = threadIdx.x + i * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      const int page = s_page[j];
      kr[i] = vr[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (page >= 0) {
        const size_t ko = kv_prefix_offset(a.kv, a.layer, page, 0, g, (t0 + j) & pmask) + 4 * e4;
        kr[i] = __ldg(reinterpret_cast<const float4*>(a.kv.pool + ko));
        vr[i] = __ldg(reinterpret_cast<const float4*>(a.kv.pool + ko + ((size_t)a.kv.kvh << a.kv.page_shift) * HD));
      }
    }
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int idx = threadIdx.x + i * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      *reinterpret_cast<float4*>(kS + j * L::QP + 4 * e4) = kr[i];
      *reinterpret_cast<float4*>(vS + j * HD + 4 * e4) = vr[i];
    }
    __syncthreads();

    // ---- scores: warp -> 4 query vectors, lane -> keys lane, lane + 32
    const int q0 = warp * 4;
    float s[4][2];
#pragma unroll
    for (int i = 0; i < 4; ++i) s[i][0] = s[i][1] = 0.f;
#pragma unroll 4
    for (int e = 0; e < HD; e += 4) {
      const float4 k0 = *reinterpret_cast<const float4*>(kS + lane * L::QP + e);
      const float4 k1 = *reinterpret_cast<const float4*>(kS + (lane + 32) * L::QP + e);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float4 qv = *reinterpret_cast<const float4*>(qS + (q0 + i) * L::QP + e);
        s[i][0] += qv.x * k0.x + qv.y * k0.y + qv.z * k0.z + qv.w * k0.w;
        s[i][1] += qv.x * k1.x + qv.y * k1.y + qv.z * k1.z + qv.w * k1.w;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int qi = q0 + i;
      const int np = (qi < nq) ? s_np[qi] : 0;
      const bool ok0 = t0 + lane < np, ok1 = t0 + lane + 32 < np;
      const float a0 = ok0 ? s[i][0] : -INFINITY, a1 = ok1 ? s[i][1] : -INFINITY;
      const float m = warp_max(fmaxf(a0, a1));
      const float p0 = ok0 ? expf(a0 - m) : 0.f, p1 = ok1 ? expf(a1 - m) : 0.f;
      const float l = warp_sum(p0 + p1);
      pS[lane * AQB + qi] = p0;
      pS[(lane + 32) * AQB + qi] = p1;
      if (lane == 0) {
        s_m[qi] = m;
        s_l[qi] = l;
      }
    }
    __syncwarp();

    // ---- partial output: lane -> dims [DPL*lane, DPL*lane + DPL)
    float o[4][DPL];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int c = 0; c < DPL; ++c) o[i][c] = 0.f;
#pragma unroll 4
    for (int t = 0; t < ACH; ++t) {
      const float4 p4 = *reinterpret_cast<const float4*>(pS + t * AQB + q0);
      float v[DPL];
      if constexpr (DPL == 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(vS + t * HD + 4 * lane);
        v[0] = v4.x; v[1] = v4.y; v[2] = v4.z; v[3] = v4.w;
      } else {
        const float2 v2 = *reinterpret_cast<const float2*>(vS + t * HD + 2 * lane);
        v[0] = v2.x; v[1] = v2.y;
      }
      const float pp[4] = {p4.x, p4.y, p4.z, p4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int c = 0; c < DPL; ++c) o[i][c] = fmaf(pp[i], v[c], o[i][c]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int qi = q0 + i;
#pragma unroll
      for (int c = 0; c < DPL; ++c) po[qi * HD + DPL * lane + c] = o[i][c];
      if (lane == 0) {
        pml[2 * qi] = s_m[qi];
        pml[2 * qi + 1] = s_l[qi];
      }
    }
  }

  // ---- last block of this (prompt, head, query block): merge chunks + tail, normalize
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(a.cnt + grp, 1) == (int)gridDim.x - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // (1) per query vector: max over its chunks and the softmax weight of every chunk
  constexpr int MAXP = 64;   // prefix chunks + the tail chunk (n_chunks <= 63, checked on the host)
  float* wS = pS;            // [AQB][MAXP] reuses the probability tile (ACH * AQB floats)
  static_assert(AQB * MAXP <= ACH * AQB, "merge weights fit in the probability tile");
  for (int i = threadIdx.x; i < nq * MAXP; i += ATHREADS) {
    const int qi = i / MAXP, j = i % MAXP;
    const int ncv = (s_np[qi] + ACH - 1) / ACH;
    float mc = -INFINITY;
    if (j <= ncv) {
      const int cj = j < ncv ? j : n_pchunks;
      mc = __ldcg(a.part_ml + ((grp * gridDim.x + cj) * AQB + qi) * 2);
    }
    wS[i] = mc;
  }
  __syncthreads();
  if (threadIdx.x < nq) {
    const int qi = threadIdx.x;
    const int ncv = (s_np[qi] + ACH - 1) / ACH;
    float m = -INFINITY;
    for (int j = 0; j <= ncv; ++j) m = fmaxf(m, wS[qi * MAXP + j]);
    float l = 0.f;
    for (int j = 0; j <= ncv; ++j) {
      const float mc = wS[qi * MAXP + j];
      const int cj = j < ncv ? j : n_pchunks;
      const float w = (mc > -INFINITY) ? expf(mc - m) : 0.f;
      l += w * __ldcg(a.part_ml + ((grp * gridDim.x + cj) * AQB + qi) * 2 + 1);
      wS[qi * MAXP + j] = w;
    }
    s_l[qi] = 1.0f / l;
  }
  __syncthreads();
  // (2) outputs: items (query vector, 4 dims), every item's chunk loads in flight together
  {
    T* out = reinterpret_cast<T*>(a.out);
    for (int i = threadIdx.x; i < nq * (HD / 4); i += ATHREADS) {
      const int qi = i / (HD / 4), e4 = i % (HD / 4);
      const int ncv = (s_np[qi] + ACH - 1) / ACH;
      float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
      for (int j = 0; j <= ncv; ++j) {
        const int cj = j < ncv ? j : n_pchunks;
        const float w = wS[qi * MAXP + j];
        const float4 v = __ldcg(reinterpret_cast<const float4*>(
            a.part_o + ((grp * gridDim.x + cj) * AQB + qi) * HD + 4 * e4));
        o.x = fmaf(w, v.x, o.x); o.y = fmaf(w, v.y, o.y);
        o.z = fmaf(w, v.z, o.z); o.w = fmaf(w, v.w, o.w);
      }
      const float inv = s_l[qi];
      const size_t dst = (size_t)s_row[qi] * H * HD + (size_t)(g * G + s_gg[qi]) * HD + 4 * e4;
      store_act<T>(out, a.plane, dst + 0, o.x * inv);
      store_act<T>(out, a.plane, dst + 1, o.y * inv);
      store_act<T>(out, a.plane, dst + 2, o.z * inv);
      store_act<T>(out, a.plane, dst + 3, o.w * inv);
    }
  }
  if (threadIdx.x == 0) a.cnt[grp] = 0;
}

template <typename T, int HD>
void launch_t(const AttnArgs& a, int n_z, cudaStream_t s) {
  dim3 grid(a.n_chunks + 1, a.kv.kvh, n_z);   // + the tail-key chunk
  launch_pdl(k_attn<T, HD>, grid, dim3(ATHREADS), AttnSmem<HD>::bytes, s, a);
}

}  // namespace

int attn_chunk() { return ACH; }
int attn_max_chunks() { return 63; }
int attn_qblock() { return AQB; }

int configure_attention() {
  int e = 0;
  e |= cudaFuncSetAttribute(k_attn<float, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<64>::bytes);
  e |= cudaFuncSetAttribute(k_attn<float, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<128>::bytes);
  e |= cudaFuncSetAttribute(k_attn<__nv_bfloat16, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<64>::bytes);
  e |= cudaFuncSetAttribute(k_attn<__nv_bfloat16, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<128>::bytes);
  return e ? -1 : 0;
}

void launch_attn(int dtype, const AttnArgs& a, int n_z, cudaStream_t s) {
  if (dtype == CDSL_DTYPE_BF16) {
    if (a.kv.hd == 128) launch_t<__nv_bfloat16, 128>(a, n_z, s);
    else launch_t<__nv_bfloat16, 64>(a, n_z, s);
  } else {
    if (a.kv.hd == 128) launch_t<float, 128>(a, n_z, s);
    else launch_t<float, 64>(a, n_z, s);
  }
}

}  // namespace cdsl
