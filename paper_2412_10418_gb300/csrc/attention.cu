// attention.cu -- attention of every row of a pass over its prompt's shared prefix pages and
// its own beam tail (decode rows of the draft, the tree-masked verify rows, causal prefill).
//
// Prefix sharing: all rows of one prompt read the same prefix K/V. The keys of a pass are cut
// into chunks of 64 slots: prefix chunks of 64 consecutive prefix positions, then tail chunks
// holding the distinct beam tails of a query block's rows (each row masked to its own beam and
// causal within it). A thread-block cluster of up to 16 blocks owns one prompt, one KV head
// and one query block of 16, 32 or 40 query vectors (query vector = (row, query head of the
// GQA group)); the chunks that hold keys are dealt to the cluster's blocks in turn (one chunk
// each while the pass has no more chunks than blocks; attn_layout.cuh). For each chunk it loads K and V once into shared memory and scores all its
// query vectors against them, keeping a running (max m, sum of exponentials l, unnormalized
// output o) per query vector (split-KV with an online softmax, fp32). The cluster then merges
// its blocks' partials through distributed shared memory, each block finishing a share of the
// query vectors, and writes the normalized output in the GEMM-input format. No global scratch,
// no atomics.
//
// Score loop: a warp owns QPW (2, 4 or 5) query vectors (broadcast reads), its lanes own keys lane
// and lane + 32 (rows of 132 floats: conflict-free 128-bit reads). Output loop: lanes own 4
// (or 2) consecutive dims of the warp's query vectors, reading P by broadcast and V
// row-contiguously. All 8 warps have query vectors: a query block is 8 * QPW of them.
#include <algorithm>

#include <cooperative_groups.h>

#include "attn_layout.cuh"
#include "kernels.h"

namespace cdsl {
namespace {

namespace cg = cooperative_groups;

using attn::ACH;
using attn::MAXP;
using attn::MAXCB;
constexpr int AQB = 40;              // query vectors per cluster (at most)
constexpr int ACL = 16;              // blocks per cluster (at most)
constexpr int ATHREADS = 256;
constexpr int AWARPS = ATHREADS / 32;

int g_max_cluster = 8;               // 16 where non-portable clusters of this kernel fit

template <int HD>
struct AttnSmem {
  static constexpr int QP = HD + 4;        // padded row pitch of Q and K
  static constexpr int PP = AQB + 4;       // row pitch of P (4-way store conflicts at most)
  static constexpr size_t floats = (size_t)AQB * QP + (size_t)ACH * QP + (size_t)ACH * HD + (size_t)ACH * PP;
  static constexpr size_t bytes = floats * sizeof(float);
};

template <typename T, int HD, int QPW>
__global__ void __launch_bounds__(ATHREADS, 2) k_attn(AttnArgs a) {
  const LaunchStamp stamp(a.stamp);
  using SL = AttnSmem<HD>;
  constexpr int QB = AWARPS * QPW;              // query vectors of the cluster
  extern __shared__ float4 sm4[];
  float* qS = reinterpret_cast<float*>(sm4);   // [QB][QP]  pre-scaled queries
  float* kS = qS + AQB * SL::QP;                 // [ACH][QP]; after the chunks: partial o [QB][HD]
  float* vS = kS + ACH * SL::QP;                 // [ACH][HD]
  float* pS = vS + ACH * HD;                    // [ACH][PP] probabilities
  __shared__ attn::Layout<QB> L;
  __shared__ int s_nkeys;
  __shared__ float s_pm[QB], s_pl[QB];          // the block's partial (m, l) per query vector

  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)gridDim.x;                 // = cluster size
  const int cx = (int)blockIdx.x;               // = rank in the cluster
  const int g = blockIdx.y;
  const int n_p = a.n_chunks;
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

  // ---- this cluster's query vectors and this block's key slots. The rows (plan kernel), the
  //      committed page table and the tail layout come from kernels the launch chain has
  //      already completed, so all of it precedes the wait.
  const int nq = attn::build_layout<QB, ATHREADS>(L, a, b, qb, cx, C);
  const int nb_chunks = L.nb;                     // chunk_of(L, n_p, cx, C, 0 .. nb_chunks - 1)
  const int maxnp = L.maxnp;
  if (a.stamp) attn::count_bytes<QB, ATHREADS, HD>(L, stamp, qb, cx, nb_chunks, nq, &s_nkeys);
  pdl_wait();                 // q and K/V of the previous kernels are ready
  pdl_launch_dependents();

  constexpr int DPL = HD / 32;
  const int q0 = warp * QPW;
  const bool active = q0 < nq;   // warps without query vectors only help to stage
  float o[QPW][DPL], m_run[QPW], l_run[QPW];
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    m_run[i] = -INFINITY;
    l_run[i] = 0.f;
#pragma unroll
    for (int c = 0; c < DPL; ++c) o[i][c] = 0.f;
  }
  bool q_staged = false;
  for (int i = 0; i < nb_chunks && nq > 0; ++i) {
    const int c = attn::chunk_of(L, n_p, cx, C, i);
    const bool tail = c >= n_p;
    const int t0 = c * ACH;
    if (!tail && t0 >= maxnp) continue;   // beyond every query vector's prefix
    // ---- stage K and V of the chunk's 64 slots (and Q the first time), loads in flight
    //      together
    constexpr int QPER = (QB * (HD / 4) + ATHREADS - 1) / ATHREADS;   // (last pass partial)
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
        if (qi < nq && qi < QB)
          qr[u] = *reinterpret_cast<const float4*>(a.q + (size_t)L.row[qi] * H * HD +
                                                   (size_t)(g * G + L.gg[qi]) * HD + 4 * e4);
      }
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int idx = threadIdx.x + u * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      const int ks = L.kslot[i * ACH + j];
      kr[u] = vr[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ks >= 0) {
        const float* kp = tail ? a.kv.tail + kv_tail_offset(a.kv, a.layer, 0, ks, g)
                               : a.kv.pool + kv_prefix_offset(a.kv, a.layer, ks, 0, g,
                                                              (t0 + j) & ((1 << a.kv.page_shift) - 1));
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
        if (qi < QB) *reinterpret_cast<float4*>(qS + qi * SL::QP + 4 * e4) = v;
      }
      q_staged = true;
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int idx = threadIdx.x + u * ATHREADS;
      const int j = idx / (HD / 4), e4 = idx % (HD / 4);
      *reinterpret_cast<float4*>(kS + j * SL::QP + 4 * e4) = kr[u];
      *reinterpret_cast<float4*>(vS + j * HD + 4 * e4) = vr[u];
    }
    __syncthreads();
    if (!active) continue;

    // ---- scores: warp -> QPW query vectors, lane -> keys lane, lane + 32
    float s[QPW][2];
#pragma unroll
    for (int q = 0; q < QPW; ++q) s[q][0] = s[q][1] = 0.f;
#pragma unroll 4
    for (int e = 0; e < HD; e += 4) {
      const float4 k0 = *reinterpret_cast<const float4*>(kS + lane * SL::QP + e);
      const float4 k1 = *reinterpret_cast<const float4*>(kS + (lane + 32) * SL::QP + e);
#pragma unroll
      for (int q = 0; q < QPW; ++q) {
        const float4 qv = *reinterpret_cast<const float4*>(qS + (q0 + q) * SL::QP + e);
        s[q][0] += qv.x * k0.x + qv.y * k0.y + qv.z * k0.z + qv.w * k0.w;
        s[q][1] += qv.x * k1.x + qv.y * k1.y + qv.z * k1.z + qv.w * k1.w;
      }
    }
    // ---- online softmax: running max, rescale of l and o, probabilities of this chunk;
    //      every stage runs over all QPW query vectors, so their shuffles are in flight
    //      together (the same butterflies as warp_max / warp_sum)
    float p0[QPW], p1[QPW], mx[QPW], alpha[QPW];
#pragma unroll
    for (int q = 0; q < QPW; ++q) {
      const int qi = q0 + q;
      bool ok0, ok1;
      if (qi >= nq) {
        ok0 = ok1 = false;
      } else if (!tail) {         // prefix: positions before the row's prefix length
        ok0 = t0 + lane < L.np[qi];
        ok1 = t0 + lane + 32 < L.np[qi];
      } else {                    // tail: the row's own beam, causal within it
        const int tb = L.tb[qi], nt = L.nt[qi];
        const int k0 = i * ACH + lane, k1 = k0 + 32;
        ok0 = L.kslot[k0] >= 0 && L.ktb[k0] == tb && L.kj[k0] < nt;
        ok1 = L.kslot[k1] >= 0 && L.ktb[k1] == tb && L.kj[k1] < nt;
      }
      s[q][0] = ok0 ? s[q][0] : -INFINITY;   // masked keys: exp(-inf - m) = 0 below
      s[q][1] = ok1 ? s[q][1] : -INFINITY;
      mx[q] = fmaxf(s[q][0], s[q][1]);
    }
#pragma unroll
    for (int o2 = 16; o2 > 0; o2 >>= 1)
#pragma unroll
      for (int q = 0; q < QPW; ++q) mx[q] = fmaxf(mx[q], __shfl_xor_sync(0xffffffffu, mx[q], o2));
#pragma unroll
    for (int q = 0; q < QPW; ++q) {
      const float m_new = fmaxf(m_run[q], mx[q]);
      alpha[q] = 1.f;
      p0[q] = p1[q] = 0.f;
      if (m_new > -INFINITY) {
        alpha[q] = (m_run[q] > -INFINITY) ? expf(m_run[q] - m_new) : 0.f;
        p0[q] = expf(s[q][0] - m_new);
        p1[q] = expf(s[q][1] - m_new);
      }
      m_run[q] = m_new;
      mx[q] = p0[q] + p1[q];   // from here: this lane's share of the sum
    }
#pragma unroll
    for (int o2 = 16; o2 > 0; o2 >>= 1)
#pragma unroll
      for (int q = 0; q < QPW; ++q) mx[q] += __shfl_xor_sync(0xffffffffu, mx[q], o2);
#pragma unroll
    for (int q = 0; q < QPW; ++q) {
      l_run[q] = alpha[q] * l_run[q] + mx[q];
#pragma unroll
      for (int c2 = 0; c2 < DPL; ++c2) o[q][c2] *= alpha[q];
    }
    if constexpr (QPW == 4) {
      *reinterpret_cast<float4*>(pS + lane * SL::PP + q0) = make_float4(p0[0], p0[1], p0[2], p0[3]);
      *reinterpret_cast<float4*>(pS + (lane + 32) * SL::PP + q0) =
          make_float4(p1[0], p1[1], p1[2], p1[3]);
    } else if constexpr (QPW == 2) {
      *reinterpret_cast<float2*>(pS + lane * SL::PP + q0) = make_float2(p0[0], p0[1]);
      *reinterpret_cast<float2*>(pS + (lane + 32) * SL::PP + q0) = make_float2(p1[0], p1[1]);
    } else {
#pragma unroll
      for (int q = 0; q < QPW; ++q) {
        pS[lane * SL::PP + q0 + q] = p0[q];
        pS[(lane + 32) * SL::PP + q0 + q] = p1[q];
      }
    }
    __syncwarp();

    // ---- o += P V: lane -> dims [DPL*lane, DPL*lane + DPL)
#pragma unroll 4
    for (int t = 0; t < ACH; ++t) {
      float pp[QPW];
      if constexpr (QPW == 4) {
        const float4 p4 = *reinterpret_cast<const float4*>(pS + t * SL::PP + q0);
        pp[0] = p4.x; pp[1] = p4.y; pp[2] = p4.z; pp[3] = p4.w;
      } else if constexpr (QPW == 2) {
        const float2 p2 = *reinterpret_cast<const float2*>(pS + t * SL::PP + q0);
        pp[0] = p2.x; pp[1] = p2.y;
      } else {
#pragma unroll
        for (int q = 0; q < QPW; ++q) pp[q] = pS[t * SL::PP + q0 + q];
      }
      float v[DPL];
      if constexpr (DPL == 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(vS + t * HD + 4 * lane);
        v[0] = v4.x; v[1] = v4.y; v[2] = v4.z; v[3] = v4.w;
      } else {
        const float2 v2 = *reinterpret_cast<const float2*>(vS + t * HD + 2 * lane);
        v[0] = v2.x; v[1] = v2.y;
      }
#pragma unroll
      for (int q = 0; q < QPW; ++q)
#pragma unroll
        for (int c2 = 0; c2 < DPL; ++c2) o[q][c2] = fmaf(pp[q], v[c2], o[q][c2]);
    }
    __syncwarp();   // pS columns of this warp are rewritten by its next chunk
  }

  // ---- the block's partial (m, l, o) per query vector into shared memory (o over kS)
  __syncthreads();
  float* s_po = kS;
  if (active) {
#pragma unroll
    for (int q = 0; q < QPW; ++q) {
      const int qi = q0 + q;
      if (qi >= nq) continue;
#pragma unroll
      for (int c2 = 0; c2 < DPL; ++c2) s_po[qi * HD + DPL * lane + c2] = o[q][c2];
      if (lane == 0) {
        s_pm[qi] = m_run[q];
        s_pl[qi] = l_run[q];
      }
    }
  }
  cluster.sync();   // every block's partials are visible to the cluster

  // ---- merge: block cx finishes query vectors cx, cx + C, ... (a warp per query vector),
  //      reading the C partials through distributed shared memory, 8 blocks at a time
  for (int qi = cx + warp * C; qi < nq; qi += C * AWARPS) {
    // the first 8 blocks' partial o go out with (m, l): one round trip for C <= 8
    float vv[8][DPL];
    auto load_o = [&](int r0) {
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
    };
    load_o(0);
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
      if (r0 > 0) load_o(r0);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const float wr = __shfl_sync(0xffffffffu, w, (r0 + r) & 31);
#pragma unroll
        for (int c2 = 0; c2 < DPL; ++c2) acc[c2] = fmaf(wr, vv[r][c2], acc[c2]);
      }
    }
    const float inv = Lsum > 0.f ? 1.0f / Lsum : 0.f;
    T* out = reinterpret_cast<T*>(a.out);
    const size_t dst = (size_t)L.row[qi] * H * HD + (size_t)(g * G + L.gg[qi]) * HD + DPL * lane;
#pragma unroll
    for (int c2 = 0; c2 < DPL; ++c2) store_act<T>(out, a.plane, dst + c2, acc[c2] * inv);
  }
  cluster.sync();   // no block leaves while the others may still read its shared memory
}

template <typename T, int HD, int QPW>
ClusterFit g_fit;   // cluster residency of k_attn<T, HD, QPW> (configure_t)

template <typename T, int HD, int QPW>
void launch_t(const AttnArgs& a, int n_z, cudaStream_t s) {
  const int cl = attn_cluster_size(g_fit<T, HD, QPW>, g_max_cluster, a.n_chunks + a.n_tchunks,
                                   a.kv.kvh * n_z);
  launch_pdl_cluster(k_attn<T, HD, QPW>, dim3(cl, a.kv.kvh, n_z), dim3(ATHREADS),
                     AttnSmem<HD>::bytes, cl, s, a);
}

template <typename T, int HD, int QPW>
int configure_t() {
  auto k = k_attn<T, HD, QPW>;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnSmem<HD>::bytes) !=
      cudaSuccess)
    return -1;
  const bool nonportable =
      cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  cudaGetLastError();
  fill_cluster_fit(&g_fit<T, HD, QPW>, k, ATHREADS, AttnSmem<HD>::bytes, nonportable ? ACL : 8);
  return nonportable && g_fit<T, HD, QPW>.active[ACL] >= 1 ? 0 : 1;   // 1: portable only
}

}  // namespace

int attn_chunk() { return ACH; }
int attn_max_chunks() { return MAXP; }
int attn_qblock() { return AWARPS * 4; }
int attn_qblock_for(int rows_per_prompt, int G) {
  // 8 warps x 2, 4 or 5 query vectors: the fewest query blocks (each of them loads the K/V
  // chunks once), the smallest block that still takes them. Blocks of 40 need G >= 2 (at most
  // 32 rows per block: the tail layout runs one lane per row).
  const int nq = rows_per_prompt * G;
  if (nq <= AWARPS * 2) return AWARPS * 2;
  if (nq <= AWARPS * 4 || G < 2) return AWARPS * 4;
  const int n_qb = (nq + AQB - 1) / AQB;
  return (nq + n_qb - 1) / n_qb <= AWARPS * 4 ? AWARPS * 4 : AQB;
}

int attn_tail_chunks(int rows_per_prompt, int G, int rows_per_tail, int max_tail) {
  if (max_tail <= 0 || rows_per_prompt <= 0) return 0;
  // rows met by one query block (at most 32 in either attention kernel), and the distinct
  // tails among them when consecutive runs of rows_per_tail rows share one
  (void)G;
  const int rows = std::min(rows_per_prompt, 32);
  const int tails = std::min(rows, (rows - 1) / std::max(1, rows_per_tail) + 2);
  return (tails * max_tail + ACH - 1) / ACH;
}

int configure_attention() {
  int worst = 0;
  for (int r : {configure_t<float, 64, 2>(), configure_t<float, 64, 4>(),
                configure_t<float, 64, 5>(), configure_t<float, 128, 2>(),
                configure_t<float, 128, 4>(), configure_t<float, 128, 5>(),
                configure_t<__nv_bfloat16, 64, 2>(), configure_t<__nv_bfloat16, 64, 4>(),
                configure_t<__nv_bfloat16, 64, 5>(), configure_t<__nv_bfloat16, 128, 2>(),
                configure_t<__nv_bfloat16, 128, 4>(), configure_t<__nv_bfloat16, 128, 5>()}) {
    if (r < 0) return -1;
    worst = std::max(worst, r);
  }
  g_max_cluster = worst ? 8 : ACL;
  return 0;
}

template <typename T, int HD>
void launch_hd(const AttnArgs& a, int n_z, cudaStream_t s) {
  if (a.qblock <= AWARPS * 2) launch_t<T, HD, 2>(a, n_z, s);
  else if (a.qblock <= AWARPS * 4) launch_t<T, HD, 4>(a, n_z, s);
  else launch_t<T, HD, 5>(a, n_z, s);
}

void launch_attn(int dtype, const AttnArgs& a, int n_z, cudaStream_t s) {
  if (dtype == CDSL_DTYPE_BF16) {
    if (a.kv.hd == 128) launch_hd<__nv_bfloat16, 128>(a, n_z, s);
    else launch_hd<__nv_bfloat16, 64>(a, n_z, s);
  } else {
    if (a.kv.hd == 128) launch_hd<float, 128>(a, n_z, s);
    else launch_hd<float, 64>(a, n_z, s);
  }
}

}  // namespace cdsl
