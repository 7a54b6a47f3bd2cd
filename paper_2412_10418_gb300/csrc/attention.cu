// attention.cu -- attention of every row of a pass over its prompt's shared prefix pages and
// its own beam tail (decode rows of the draft, the tree-masked verify rows, causal prefill).
//
// Prefix sharing: all rows of one prompt read the same prefix K/V. The keys of a pass are cut
// into chunks of 64 slots: prefix chunks of 64 consecutive prefix positions, then tail chunks
// holding the distinct beam tails of a query block's rows (each row masked to its own beam and
// causal within it). A thread-block cluster of up to 16 blocks owns one prompt, one KV head
// and one query block of 16 or 32 query vectors (query vector = (row, query head of the GQA
// group)); block r of the cluster takes chunks r, r + C, ... (one chunk each while the pass
// has at most 16). For each chunk it loads K and V once into shared memory and scores all its
// query vectors against them, keeping a running (max m, sum of exponentials l, unnormalized
// output o) per query vector (split-KV with an online softmax, fp32). The cluster then merges
// its blocks' partials through distributed shared memory, each block finishing a share of the
// query vectors, and writes the normalized output in the GEMM-input format. No global scratch,
// no atomics.
//
// Per chunk: S = Q K^T and o += P V run on the tensor cores in 3xTF32 (mma.sync m16n8k8, each
// fp32 operand split into a tf32 high part and a tf32 remainder: fp32-level accuracy), their
// 16x8 tiles spread evenly over the 8 warps; the online softmax between them runs on the CUDA
// cores, a warp owning QPW (2 or 4) query vectors and its lanes keys lane and lane + 32. A
// query block is 8 * QPW query vectors.
#include <algorithm>

#include <cooperative_groups.h>

#include "kernels.h"

namespace cdsl {
namespace {

namespace cg = cooperative_groups;

constexpr int ACH = 64;              // key slots per chunk
constexpr int AQB = 32;              // query vectors per cluster (at most)
constexpr int MAXP = 64;             // chunks (prefix + tail) of a pass
constexpr int ACL = 16;              // blocks per cluster (at most)
constexpr int MAXCB = MAXP / 8;      // chunks per block (at most; clusters have >= 8 blocks
                                     // whenever a pass has more than 8 chunks)
constexpr int ATHREADS = 256;
constexpr int AWARPS = ATHREADS / 32;

int g_max_cluster = 8;               // 16 where non-portable clusters of this kernel fit

template <int HD>
struct AttnSmem {
  static constexpr int QP = HD + 4;        // row pitch of Q and K (conflict-free fragments)
  static constexpr int VP = HD + 8;        // row pitch of V
  static constexpr int SP = ACH + 4;       // row pitch of the scores / probabilities
  static constexpr size_t floats = (size_t)AQB * QP + (size_t)ACH * QP + (size_t)ACH * VP + (size_t)AQB * SP;
  static constexpr size_t bytes = floats * sizeof(float);
};

// ---- 3xTF32 tensor-core products (mma.sync m16n8k8): x = hi + lo with hi = tf32(x),
//      lo = tf32(x - hi); a.b ~ a_hi.b_hi + a_hi.b_lo + a_lo.b_hi (the a_lo.b_lo term and the
//      rounding of the lo parts are below 2^-21 relative: fp32-level accuracy)
__device__ __forceinline__ void split_tf32(float x, uint32_t& hi, uint32_t& lo) {
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(hi) : "f"(x));
  const float rest = x - __uint_as_float(hi);
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(lo) : "f"(rest));
}
__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
// Fragments of one 16x8x8 step, split into tf32 high and low parts: A from a row-major [m][k]
// tile (element (m, k) at A[m * lda + k]); B from a [n][k] tile (B[n * ldb + k]) or, with kn,
// a [k][n] tile (B[k * ldb + n]).
struct FragA { uint32_t h[4], l[4]; };
struct FragB { uint32_t h[2], l[2]; };
__device__ __forceinline__ FragA load_a(const float* A, int lda, int lane) {
  const int g = lane >> 2, t = lane & 3;
  FragA f;
  split_tf32(A[g * lda + t], f.h[0], f.l[0]);
  split_tf32(A[(g + 8) * lda + t], f.h[1], f.l[1]);
  split_tf32(A[g * lda + t + 4], f.h[2], f.l[2]);
  split_tf32(A[(g + 8) * lda + t + 4], f.h[3], f.l[3]);
  return f;
}
template <bool kn>
__device__ __forceinline__ FragB load_b(const float* B, int ldb, int lane) {
  const int g = lane >> 2, t = lane & 3;
  FragB f;
  if (kn) {
    split_tf32(B[t * ldb + g], f.h[0], f.l[0]);
    split_tf32(B[(t + 4) * ldb + g], f.h[1], f.l[1]);
  } else {
    split_tf32(B[g * ldb + t], f.h[0], f.l[0]);
    split_tf32(B[g * ldb + t + 4], f.h[1], f.l[1]);
  }
  return f;
}
__device__ __forceinline__ void mma3(float (&d)[4], const FragA& a, const FragB& b) {
  mma_tf32(d, a.l, b.h);   // small terms first
  mma_tf32(d, a.h, b.l);
  mma_tf32(d, a.h, b.h);
}

template <typename T, int HD, int QPW>
__global__ void __launch_bounds__(ATHREADS, 2) k_attn(AttnArgs a) {
  using L = AttnSmem<HD>;
  constexpr int QB = AWARPS * QPW;              // query vectors of the cluster
  extern __shared__ float4 sm4[];
  float* qS = reinterpret_cast<float*>(sm4);   // [QB][QP]  pre-scaled queries
  float* kS = qS + AQB * L::QP;                 // [ACH][QP]; after the chunks: partial o [QB][HD]
  float* vS = kS + ACH * L::QP;                 // [ACH][VP]
  float* pS = vS + ACH * L::VP;                 // [QB][SP] scores, then probabilities
  __shared__ int s_row[QB], s_gg[QB], s_np[QB], s_tb[QB], s_nt[QB];
  __shared__ int s_toff[32], s_tlen[32];        // per query vector: its tail's slot range
  __shared__ int s_wcnt[AWARPS];
  __shared__ int s_nrows, s_maxnp;
  __shared__ float s_pm[QB], s_pl[QB];          // running (m, l) per query vector
  __shared__ float s_alpha[QB];                 // this chunk's rescale of o per query vector
  __shared__ const float* s_kp[MAXCB * ACH];    // K row of every key slot of the block's chunks
  __shared__ int s_ktb[MAXCB * ACH];            // tail slots: tail base of the beam,
  __shared__ uint8_t s_kj[MAXCB * ACH];         //   index in it

  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)gridDim.x;                 // = cluster size
  const int cx = (int)blockIdx.x;               // = rank in the cluster
  const int g = blockIdx.y;
  const int n_p = a.n_chunks, NC = a.n_chunks + a.n_tchunks;
  const int nb_chunks = (NC - cx + C - 1) / C;  // this block's chunks cx, cx + C, ...
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

  // ---- this cluster's query vectors: rows of prompt b in order, G heads each. The rows (plan
  //      kernel), the committed page table and the tail layout come from kernels the launch
  //      chain has already completed, so everything up to the key slots precedes the wait.
  if (threadIdx.x < QB) s_row[threadIdx.x] = -1;
  for (int i = threadIdx.x; i < MAXCB * ACH; i += ATHREADS) s_kp[i] = nullptr;
  if (threadIdx.x == 0) s_nrows = 0;
  __syncthreads();
  for (int base = 0; base < a.R; base += ATHREADS) {
    const int r = base + threadIdx.x;
    RowDesc rd;
    const bool mine = r < a.R && (rd = a.rows[r]).b == b;
    const unsigned bal = __ballot_sync(0xffffffffu, mine);
    if (lane == 0) s_wcnt[warp] = __popc(bal);
    __syncthreads();
    int off = s_nrows;
    for (int w = 0; w < warp; ++w) off += s_wcnt[w];
    const int local = off + __popc(bal & ((1u << lane) - 1));
    if (mine) {
      for (int gg = 0; gg < G; ++gg) {
        const int qi = local * G + gg - qb * QB;
        if (qi >= 0 && qi < QB) {
          s_row[qi] = r;
          s_gg[qi] = gg;
          s_np[qi] = rd.n_prefix;
          s_tb[qi] = rd.tail_base;
          s_nt[qi] = rd.n_tail;
        }
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < AWARPS; ++w) tot += s_wcnt[w];
      s_nrows += tot;
    }
    __syncthreads();
  }
  const int nq = max(0, min(QB, s_nrows * G - qb * QB));
  if (warp == 0) {
    // longest prefix, and the distinct tails (lane = query vector) in order of first
    // appearance, each as long as its longest row: slot offsets in their concatenation
    int np = (lane < nq) ? s_np[lane] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) np = max(np, __shfl_xor_sync(0xffffffffu, np, o));
    const int tb = (lane < nq) ? s_tb[lane] : -1;
    const int nt = (lane < nq) ? s_nt[lane] : 0;
    int len = 0;
    bool first = nt > 0;
    for (int j = 0; j < 32; ++j) {
      const int tbj = __shfl_sync(0xffffffffu, tb, j), ntj = __shfl_sync(0xffffffffu, nt, j);
      if (tbj == tb && ntj > 0) {
        len = max(len, ntj);
        if (j < lane) first = false;
      }
    }
    if (!first) len = 0;
    int off = len;   // inclusive scan of the lengths over the lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, off, o);
      if (lane >= o) off += v;
    }
    const int total = __shfl_sync(0xffffffffu, off, 31);
    s_toff[lane] = off - len;
    s_tlen[lane] = len;
    if (lane == 0) {
      s_maxnp = np;
      if (cx == 0 && total > a.n_tchunks * ACH) set_status(a.status, CDSL_ERANGE);
    }
  }
  __syncthreads();
  const int maxnp = s_maxnp;
  // key slots of this block's chunks
  for (int i = 0; i < nb_chunks; ++i) {
    const int c = cx + i * C;
    if (c < n_p) {   // prefix positions c*64 .. c*64 + 63 below the longest prefix
      const int t = c * ACH + (threadIdx.x & (ACH - 1));
      if (threadIdx.x < ACH && t < maxnp) {
        const int page = a.kv.page_table[b * a.kv.max_pages + (t >> a.kv.page_shift)];
        if (page >= 0)
          s_kp[i * ACH + threadIdx.x] = a.kv.pool + kv_prefix_offset(a.kv, a.layer, page, 0, g,
                                                                     t & ((1 << a.kv.page_shift) - 1));
      }
    } else if (warp == 0 && lane < nq) {   // tail slots [lo, lo + 64) of the concatenation
      const int lo = (c - n_p) * ACH, off = s_toff[lane], len = s_tlen[lane], tb = s_tb[lane];
      for (int e = max(0, lo - off); e < len && off + e < lo + ACH; ++e) {
        const int sl = i * ACH + off + e - lo;
        s_kp[sl] = a.kv.tail + kv_tail_offset(a.kv, a.layer, 0, tb + e, g);
        s_ktb[sl] = tb;
        s_kj[sl] = (uint8_t)e;
      }
    }
  }
  __syncthreads();
  pdl_wait();                 // q and K/V of the previous kernels are ready
  pdl_launch_dependents();

  constexpr int DPL = HD / 32;
  const int q0 = warp * QPW;      // softmax rows of this warp
  // tensor-core tiles: scores QB x 64 and outputs QB x HD in 16x8 tiles, spread evenly over
  // the 8 warps (a warp's tiles share their 16 query rows)
  constexpr int MT = QB / 16;
  constexpr int ST = MT * (ACH / 8) / AWARPS;   // score tiles per warp
  constexpr int OT = MT * (HD / 8) / AWARPS;    // output tiles per warp
  const int s_m = (warp * ST) / (ACH / 8), s_n0 = (warp * ST) % (ACH / 8);
  const int o_m = (warp * OT) / (HD / 8), o_n0 = (warp * OT) % (HD / 8);
  const int fg = lane >> 2, ft = lane & 3;      // fragment row group, column pair
  float oacc[OT][4];                            // rows o_m*16 + fg (+8), cols n*8 + 2*ft (+1)
#pragma unroll
  for (int i = 0; i < OT; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  if (threadIdx.x < QB) {
    s_pm[threadIdx.x] = -INFINITY;
    s_pl[threadIdx.x] = 0.f;
  }
  bool q_staged = false;
  for (int i = 0; i < nb_chunks && nq > 0; ++i) {
    const int c = cx + i * C;
    const bool tail = c >= n_p;
    const int t0 = c * ACH;
    if (!tail && t0 >= maxnp) continue;   // beyond every query vector's prefix
    // ---- stage K and V of the chunk's 64 slots (and Q the first time), loads in flight
    //      together
    constexpr int QPER = QB * (HD / 4) / ATHREADS;
    constexpr int PER = ACH * (HD / 4) / ATHREADS;   // float4 per thread per matrix
    const size_t v_delta = tail ? (size_t)a.kv.n_tail_slots * a.kv.kvh * HD
                                : ((size_t)a.kv.kvh << a.kv.page_shift) * HD;
    float4 qr[QPER], kr[PER], vr[PER];
    if (!q_staged) {
#pragma unroll
      for (int u = 0; u < QPER; ++u) {
        const int idx = threadIdx.x + u * ATHREADS;
        const int qi = idx / (HD / 4), e4 = idx % (HD / 4);
        qr[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (qi < nq)
          qr[u] = *reinterpret_cast<const float4*>(a.q + (size_t)s_row[qi] * H * HD +
                                                   (size_t)(g * G + s_gg[qi]) * HD + 4 * e4);
      }
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int idx = threadIdx.x + u * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      const float* kp = s_kp[i * ACH + j];
      kr[u] = vr[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (kp) {
        kr[u] = __ldg(reinterpret_cast<const float4*>(kp + 4 * e4));
        vr[u] = __ldg(reinterpret_cast<const float4*>(kp + v_delta + 4 * e4));
      }
    }
    __syncthreads();   // the previous chunk's readers of kS / vS are done
    if (!q_staged) {
#pragma unroll
      for (int u = 0; u < QPER; ++u) {
        const int idx = threadIdx.x + u * ATHREADS;
        const int qi = idx / (HD / 4), e4 = idx % (HD / 4);
        float4 v = qr[u];
        v.x *= a.scale; v.y *= a.scale; v.z *= a.scale; v.w *= a.scale;
        *reinterpret_cast<float4*>(qS + qi * L::QP + 4 * e4) = v;
      }
      q_staged = true;
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int idx = threadIdx.x + u * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      *reinterpret_cast<float4*>(kS + j * L::QP + 4 * e4) = kr[u];
      *reinterpret_cast<float4*>(vS + j * L::VP + 4 * e4) = vr[u];
    }
    __syncthreads();

    // ---- scores S = Q K^T on the tensor cores (3xTF32): Q rows s_m*16.., keys n*8..
    {
      float sacc[ST][4];
#pragma unroll
      for (int i = 0; i < ST; ++i) sacc[i][0] = sacc[i][1] = sacc[i][2] = sacc[i][3] = 0.f;
#pragma unroll 4
      for (int k0 = 0; k0 < HD; k0 += 8) {
        const FragA fa = load_a(qS + (s_m * 16) * L::QP + k0, L::QP, lane);
#pragma unroll
        for (int i = 0; i < ST; ++i)
          mma3(sacc[i], fa, load_b<false>(kS + ((s_n0 + i) * 8) * L::QP + k0, L::QP, lane));
      }
#pragma unroll
      for (int i = 0; i < ST; ++i) {
        float* dst = pS + (s_m * 16 + fg) * L::SP + (s_n0 + i) * 8 + 2 * ft;
        dst[0] = sacc[i][0];
        dst[1] = sacc[i][1];
        dst[8 * L::SP] = sacc[i][2];
        dst[8 * L::SP + 1] = sacc[i][3];
      }
    }
    __syncthreads();

    // ---- online softmax over the chunk: warp -> QPW query vectors, lane -> keys lane, lane+32
#pragma unroll
    for (int q = 0; q < QPW; ++q) {
      const int qi = q0 + q;
      float* srow = pS + qi * L::SP;
      bool ok0, ok1;
      if (qi >= nq) {
        ok0 = ok1 = false;
      } else if (!tail) {         // prefix: positions before the row's prefix length
        ok0 = t0 + lane < s_np[qi];
        ok1 = t0 + lane + 32 < s_np[qi];
      } else {                    // tail: the row's own beam, causal within it
        const int tb = s_tb[qi], nt = s_nt[qi];
        const int k0 = i * ACH + lane, k1 = k0 + 32;
        ok0 = s_kp[k0] && s_ktb[k0] == tb && s_kj[k0] < nt;
        ok1 = s_kp[k1] && s_ktb[k1] == tb && s_kj[k1] < nt;
      }
      const float a0 = ok0 ? srow[lane] : -INFINITY, a1 = ok1 ? srow[lane + 32] : -INFINITY;
      const float m_old = s_pm[qi];
      const float m_new = fmaxf(m_old, warp_max(fmaxf(a0, a1)));
      float alpha = 1.f, p0 = 0.f, p1 = 0.f;
      if (m_new > -INFINITY) {
        alpha = (m_old > -INFINITY) ? expf(m_old - m_new) : 0.f;
        p0 = ok0 ? expf(a0 - m_new) : 0.f;
        p1 = ok1 ? expf(a1 - m_new) : 0.f;
      }
      const float psum = warp_sum(p0 + p1);
      srow[lane] = p0;
      srow[lane + 32] = p1;
      if (lane == 0) {
        s_pl[qi] = alpha * s_pl[qi] + psum;
        s_pm[qi] = m_new;
        s_alpha[qi] = alpha;
      }
    }
    __syncthreads();

    // ---- o = alpha o + P V on the tensor cores (3xTF32): rows o_m*16.., dims n*8..
    {
      const float al0 = s_alpha[o_m * 16 + fg], al1 = s_alpha[o_m * 16 + fg + 8];
#pragma unroll
      for (int n = 0; n < OT; ++n) {
        oacc[n][0] *= al0; oacc[n][1] *= al0;
        oacc[n][2] *= al1; oacc[n][3] *= al1;
      }
#pragma unroll 2
      for (int k0 = 0; k0 < ACH; k0 += 8) {
        const FragA fa = load_a(pS + (o_m * 16) * L::SP + k0, L::SP, lane);
#pragma unroll
        for (int n = 0; n < OT; ++n)
          mma3(oacc[n], fa, load_b<true>(vS + k0 * L::VP + (o_n0 + n) * 8, L::VP, lane));
      }
    }
  }

  // ---- the block's partial o per query vector into shared memory (over kS); (m, l) are in
  //      s_pm / s_pl
  __syncthreads();
  float* s_po = kS;
#pragma unroll
  for (int n = 0; n < OT; ++n) {
    float* dst = s_po + (o_m * 16 + fg) * HD + (o_n0 + n) * 8 + 2 * ft;
    dst[0] = oacc[n][0];
    dst[1] = oacc[n][1];
    dst[8 * HD] = oacc[n][2];
    dst[8 * HD + 1] = oacc[n][3];
  }
  cluster.sync();   // every block's partials are visible to the cluster

  // ---- merge: block cx finishes query vectors cx, cx + C, ... (a warp per query vector),
  //      reading the C partials through distributed shared memory, 8 blocks at a time
  for (int qi = cx + warp * C; qi < nq; qi += C * AWARPS) {
    float mr = -INFINITY, lr = 0.f;
    if (lane < C) {
      mr = cluster.map_shared_rank(s_pm, lane)[qi];
      lr = cluster.map_shared_rank(s_pl, lane)[qi];
    }
    const float M = warp_max(mr);
    const float w = (lane < C && mr > -INFINITY) ? expf(mr - M) : 0.f;
    const float Lsum = warp_sum(w * lr);
    float acc[DPL];
#pragma unroll
    for (int c2 = 0; c2 < DPL; ++c2) acc[c2] = 0.f;
    for (int r0 = 0; r0 < C; r0 += 8) {
      float vv[8][DPL];
#pragma unroll
      for (int r = 0; r < 8; ++r) {
#pragma unroll
        for (int c2 = 0; c2 < DPL; ++c2) vv[r][c2] = 0.f;
        if (r0 + r < C) {
          const float* src = cluster.map_shared_rank(s_po, r0 + r) + qi * HD + DPL * lane;
          if constexpr (DPL == 4) {
            const float4 t4 = *reinterpret_cast<const float4*>(src);
            vv[r][0] = t4.x; vv[r][1] = t4.y; vv[r][2] = t4.z; vv[r][3] = t4.w;
          } else {
            const float2 t2 = *reinterpret_cast<const float2*>(src);
            vv[r][0] = t2.x; vv[r][1] = t2.y;
          }
        }
      }
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const float wr = __shfl_sync(0xffffffffu, w, (r0 + r) & 31);
#pragma unroll
        for (int c2 = 0; c2 < DPL; ++c2) acc[c2] = fmaf(wr, vv[r][c2], acc[c2]);
      }
    }
    const float inv = Lsum > 0.f ? 1.0f / Lsum : 0.f;
    T* out = reinterpret_cast<T*>(a.out);
    const size_t dst = (size_t)s_row[qi] * H * HD + (size_t)(g * G + s_gg[qi]) * HD + DPL * lane;
#pragma unroll
    for (int c2 = 0; c2 < DPL; ++c2) store_act<T>(out, a.plane, dst + c2, acc[c2] * inv);
  }
  cluster.sync();   // no block leaves while the others may still read its shared memory
}

template <typename T, int HD, int QPW>
void launch_t(const AttnArgs& a, int n_z, cudaStream_t s) {
  const int cl = std::min(g_max_cluster, a.n_chunks + a.n_tchunks);
  launch_pdl_cluster(k_attn<T, HD, QPW>, dim3(cl, a.kv.kvh, n_z), dim3(ATHREADS),
                     AttnSmem<HD>::bytes, cl, s, a);
}

template <typename T, int HD, int QPW>
int configure_t() {
  auto k = k_attn<T, HD, QPW>;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<HD>::bytes) !=
      cudaSuccess)
    return -1;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
    return 1;   // portable clusters only
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ACL, 1, 1);
  cfg.blockDim = dim3(ATHREADS);
  cfg.dynamicSmemBytes = AttnSmem<HD>::bytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = ACL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess || n < 1) {
    cudaGetLastError();
    return 1;
  }
  return 0;
}

}  // namespace

int attn_chunk() { return ACH; }
int attn_max_chunks() { return MAXP; }
int attn_qblock() { return AQB; }
int attn_qblock_for(int rows_per_prompt, int G) {
  return rows_per_prompt * G <= AWARPS * 2 ? AWARPS * 2 : AQB;
}

int attn_tail_chunks(int rows_per_prompt, int G, int rows_per_tail, int max_tail) {
  if (max_tail <= 0 || rows_per_prompt <= 0) return 0;
  // rows met by one query block (it may straddle a row at either end), and the distinct
  // tails among them when consecutive runs of rows_per_tail rows share one
  const int rows = std::min(rows_per_prompt, (AQB + G - 1) / G + 1);
  const int tails = std::min(rows, (rows - 1) / std::max(1, rows_per_tail) + 2);
  return (tails * max_tail + ACH - 1) / ACH;
}

int configure_attention() {
  int worst = 0;
  for (int r : {configure_t<float, 64, 2>(), configure_t<float, 64, 4>(),
                configure_t<float, 128, 2>(), configure_t<float, 128, 4>(),
                configure_t<__nv_bfloat16, 64, 2>(), configure_t<__nv_bfloat16, 64, 4>(),
                configure_t<__nv_bfloat16, 128, 2>(), configure_t<__nv_bfloat16, 128, 4>()}) {
    if (r < 0) return -1;
    worst = std::max(worst, r);
  }
  g_max_cluster = worst ? 8 : ACL;
  return 0;
}

void launch_attn(int dtype, const AttnArgs& a, int n_z, cudaStream_t s) {
  const bool q2 = a.qblock <= AWARPS * 2;
  if (dtype == CDSL_DTYPE_BF16) {
    if (a.kv.hd == 128) q2 ? launch_t<__nv_bfloat16, 128, 2>(a, n_z, s) : launch_t<__nv_bfloat16, 128, 4>(a, n_z, s);
    else q2 ? launch_t<__nv_bfloat16, 64, 2>(a, n_z, s) : launch_t<__nv_bfloat16, 64, 4>(a, n_z, s);
  } else {
    if (a.kv.hd == 128) q2 ? launch_t<float, 128, 2>(a, n_z, s) : launch_t<float, 128, 4>(a, n_z, s);
    else q2 ? launch_t<float, 64, 2>(a, n_z, s) : launch_t<float, 64, 4>(a, n_z, s);
  }
}

}  // namespace cdsl
