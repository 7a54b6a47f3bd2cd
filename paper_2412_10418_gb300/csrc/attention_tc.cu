// attention_tc.cu -- attention of the decode and verify passes of bf16 models on the
// 5th-generation tensor cores (tcgen05 MMA into TMEM).
//
// The pass is split as in attention.cu (attn_layout.cuh): a thread-block cluster of up to 16
// blocks owns one (prompt, KV head, query block), and the chunks of 64 key slots that hold
// keys (prefix positions, then the query block's beam tails) are dealt to its blocks in turn.
// A query block holds up to 128 query vectors -- the MMA's M -- so the 7B verify pass (80
// query vectors per KV head) is one block per chunk and KV head.
//
// Per chunk, with every operand a K-major bf16 tile in 128-byte-swizzled shared memory:
//   S = Q K^T      M = 128 query vectors, N = 64 keys, K = head_dim  -> TMEM columns [0, 64)
//   O += P V       M = 128 query vectors, N = head_dim, K = 64 keys   -> TMEM columns [64, ..)
// fp32 accuracy from bf16 operands: every fp32 input x is split into hi = bf16(x) and
// lo = bf16(x - hi), and each product is hi.hi + hi.lo + lo.hi (lo.lo, about 2^-18 of the
// product, is dropped), accumulated in fp32. The K/V cache stays fp32 in HBM; the block
// converts each chunk while staging it (K row-major as the score product's B operand, V
// transposed as the P V product's B operand). Staging is software-pipelined: the next
// chunk's rows are loaded into registers while this chunk's softmax runs and stored once
// its P V has completed. Q is split once per block, pre-scaled by log2(e) / sqrt(head_dim)
// (scores in base 2).
//
// Softmax: warps w and w + 4 read TMEM lanes 32(w % 4) .. +31, so each thread owns one query
// vector's row of scores over half the chunk's keys (the two halves exchange their row
// maxima through shared memory; each keeps its own share of the row sum). The running
// reference m is raised only when a chunk's maximum exceeds it by more than kLazy (then O in
// TMEM and l are rescaled); otherwise p = 2^(s - m) <= e^8, and the final o / l does not
// depend on the reference. The block's partial (m, l, o) are merged across the cluster
// through distributed shared memory as in attention.cu, and the normalized output is written
// as the O projection's hi/lo input.
//
// One thread issues every MMA; tcgen05.commit arrives on an mbarrier that the consumers wait
// on (bounded by the launch's wait limit: on expiry CDSL_ETIMEOUT is latched and the block
// skips its remaining chunks, waits for its own MMAs in flight and still meets every cluster
// barrier).
#include <algorithm>

#include <cooperative_groups.h>

#include "attn_layout.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace cdsl {
namespace {

namespace cg = cooperative_groups;
using attn::ACH;
using attn::MAXCB;

constexpr int TQB = 128;             // query vectors per block (at most): the MMA's M
constexpr int TTHREADS = 256;
constexpr int TWARPS = TTHREADS / 32;
constexpr int TACL = 16;             // blocks per cluster (at most)
constexpr int kIssuer = 128;         // thread that issues the MMAs (warp 4, lane 0)
constexpr float kLazy = 11.5415602f; // raise the softmax reference only past this margin
                                     // (base-2 scores: 8 / ln 2, so p <= e^8)
constexpr float kLog2e = 1.44269504088896341f;

int g_tc_max_cluster = 8;

template <int HD>
struct TcSmem {
  static constexpr int KB = HD / 64;                        // 64-wide K blocks of Q and K
  static constexpr uint32_t Q_KB = TQB * 128;               // bytes of one K block of Q
  static constexpr uint32_t K_KB = ACH * 128;               // bytes of one K block of K
  static constexpr uint32_t Q_PLANE = KB * Q_KB;            // Q [128][HD] bf16, one plane
  static constexpr uint32_t K_PLANE = KB * K_KB;            // K [64][HD]
  static constexpr uint32_t V_PLANE = HD * 128;             // V^T [HD][64 keys]
  static constexpr uint32_t P_PLANE = TQB * 128;            // P [128][64 keys]
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t K_OFF = Q_OFF + 2 * Q_PLANE;
  static constexpr uint32_t V_OFF = K_OFF + 2 * K_PLANE;
  static constexpr uint32_t P_OFF = V_OFF + 2 * V_PLANE;
  static constexpr uint32_t TOTAL = P_OFF + 2 * P_PLANE;
  static constexpr int OP = HD + 4;                         // row pitch of the partial o (floats)
  static constexpr uint32_t O_OFF = K_OFF;                  // partial o [128][OP] fp32, after the
  static_assert(TQB * OP * 4 <= TOTAL - K_OFF, "partial o fits over K, V and P");   // chunks
  static constexpr uint32_t TMEM_COLS = (64 + HD) <= 128 ? 128 : 256;
  static constexpr size_t bytes = TOTAL + 1024;             // + 1024-byte alignment of the base
};

// 8 fp32 values -> 8 bf16 hi values and 8 bf16 lo values (x = hi + lo to about 2^-17).
__device__ __forceinline__ void split8(const float (&x)[8], uint4& hi, uint4& lo) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(x[2 * i]), h1 = __float2bfloat16_rn(x[2 * i + 1]);
    const __nv_bfloat16 l0 = __float2bfloat16_rn(x[2 * i] - __bfloat162float(h0));
    const __nv_bfloat16 l1 = __float2bfloat16_rn(x[2 * i + 1] - __bfloat162float(h1));
    h[i] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    l[i] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
  }
  hi = make_uint4(h[0], h[1], h[2], h[3]);
  lo = make_uint4(l[0], l[1], l[2], l[3]);
}

__device__ __forceinline__ void st_shared16(uint8_t* base, uint32_t off, const uint4& v) {
  *reinterpret_cast<uint4*>(base + off) = v;
}

template <int HD>
__global__ void __launch_bounds__(TTHREADS, 1) k_attn_tc(AttnArgs a) {
  const LaunchStamp stamp(a.stamp);
  using SM = TcSmem<HD>;
  constexpr int KB = SM::KB;
  constexpr int DCH = HD / 8;                    // 16-byte bf16 chunks per row of Q and K
  constexpr int K_IT = ACH * DCH / TTHREADS;     // staging items per thread: K (key, chunk)
  constexpr int V_IT = HD * (ACH / 8) / TTHREADS;  //   and V^T (dim, 8 keys)
  constexpr int Q_IT = TQB * DCH / TTHREADS;     //   and Q (query vector, chunk)
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = smem_raw + ((1024 - (tc::smem_u32(smem_raw) & 1023)) & 1023);
  __shared__ attn::Layout<TQB> L;
  __shared__ __align__(8) uint64_t bar_s, bar_o;   // score / P V products complete
  __shared__ __align__(8) uint64_t bar_d;          // every MMA of the block has completed
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_nkeys;
  __shared__ const float* s_kptr[2][ACH];         // K of each key slot of a chunk (V follows);
                                                  // chunk i uses buffer i & 1
  __shared__ float s_pm[TQB], s_pl[TQB];          // the block's partial (m, l) per query vector
  __shared__ float s_mx[2][TQB];                  // per half: a chunk's row maxima, then l

  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)gridDim.x;                   // = cluster size
  const int cx = (int)blockIdx.x;                 // = rank in the cluster
  const int g = blockIdx.y;
  const int n_p = a.n_chunks;
  const int b = blockIdx.z / a.qb_count, qb = blockIdx.z % a.qb_count;
  const int G = a.G, H = a.n_heads;
  const int warp = threadIdx.x >> 5;

  // ---- query vectors and key slots (before the wait: inputs of completed kernels only)
  const int nq = attn::build_layout<TQB, TTHREADS>(L, a, b, qb, cx, C);
  const int nb_chunks = L.nb;                     // chunk_of(L, n_p, cx, C, 0 .. nb_chunks - 1)
  if (a.stamp) attn::count_bytes<TQB, TTHREADS, HD>(L, stamp, qb, cx, nb_chunks, nq, &s_nkeys);
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar_s, 1);
    tc::mbar_init(&bar_o, 1);
    tc::mbar_init(&bar_d, 1);
    s_abort = 0;
    tc::fence_mbar_init();
  }
  pdl_wait();                 // q and K/V of the previous kernels are ready
  pdl_launch_dependents();
  if (warp == 0) tc::tmem_alloc(&s_tmem, SM::TMEM_COLS);

  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t t_s = tmem, t_o = tmem + 64;      // columns: S [0, 64), O [64, 64 + HD)
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  const uint32_t sbase = tc::smem_u32(sm);
  const uint32_t idesc_s = tc::idesc_bf16_f32(128, ACH), idesc_o = tc::idesc_bf16_f32(128, HD);
  const size_t v_delta_tail = (size_t)a.kv.n_tail_slots * a.kv.kvh * HD;
  const size_t v_delta_pfx = ((size_t)a.kv.kvh << a.kv.page_shift) * HD;
  const int qi = threadIdx.x & (TQB - 1);          // softmax: TMEM lane (query vector) and
  const int half = threadIdx.x / TQB;              //   half of the chunk's keys
  float m_ref = -INFINITY, l_run = 0.f;
  int nproc = 0;                                    // chunks whose P V has been issued

  // Staging is software-pipelined: chunk i + 1's K and V rows are loaded from the fp32 cache
  // into registers right after chunk i's score MMAs are issued (in flight during its
  // softmax), and converted and stored once chunk i's P V has completed.
  auto kptrs = [&](int i) {   // threads 0 .. ACH-1: key slot pointers of chunk i
    if (threadIdx.x < ACH) {
      const int c = attn::chunk_of(L, n_p, cx, C, i);
      const int ks = L.kslot[i * ACH + threadIdx.x];
      const float* kp = nullptr;
      if (ks >= 0) {
        const int slot = (c * ACH + threadIdx.x) & ((1 << a.kv.page_shift) - 1);
        kp = c >= n_p ? a.kv.tail + kv_tail_offset(a.kv, a.layer, 0, ks, g)
                      : a.kv.pool + kv_prefix_offset(a.kv, a.layer, ks, 0, g, slot);
      }
      s_kptr[i & 1][threadIdx.x] = kp;
    }
  };
  float4 kr[K_IT][2];   // raw K and V of the next chunk to stage
  float vr[V_IT][8];
  auto load_kv = [&](int i) {   // all loads of chunk i in flight together (pointers ready)
    const size_t v_delta = attn::chunk_of(L, n_p, cx, C, i) >= n_p ? v_delta_tail : v_delta_pfx;
    const float* const* kps = s_kptr[i & 1];
#pragma unroll
    for (int u = 0; u < K_IT; ++u) {
      const int idx = threadIdx.x + u * TTHREADS, j = idx / DCH, dc = idx % DCH;
      const float* kp = kps[j];
      kr[u][0] = kr[u][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (kp) {
        kr[u][0] = __ldg(reinterpret_cast<const float4*>(kp + dc * 8));
        kr[u][1] = __ldg(reinterpret_cast<const float4*>(kp + dc * 8 + 4));
      }
    }
#pragma unroll
    for (int u = 0; u < V_IT; ++u) {
      const int idx = threadIdx.x + u * TTHREADS, d = idx % HD, jc = idx / HD;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float* kp = kps[jc * 8 + q];
        vr[u][q] = kp ? __ldg(kp + v_delta + d) : 0.f;
      }
    }
  };
  if (nb_chunks > 0 && nq > 0) {
    // ---- Q once per block: query vector qi is row qi of the A operand (zero rows from nq
    //      on), pre-scaled by log2(e) / sqrt(head_dim) (base-2 scores); and chunk 0's loads
    kptrs(0);
    float4 qr[Q_IT][2];
#pragma unroll
    for (int u = 0; u < Q_IT; ++u) {
      const int it = threadIdx.x + u * TTHREADS, qv = it / DCH, dc = it % DCH;
      qr[u][0] = qr[u][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (qv < nq) {
        const float* src =
            a.q + (size_t)L.row[qv] * H * HD + (size_t)(g * G + L.gg[qv]) * HD + dc * 8;
        qr[u][0] = *reinterpret_cast<const float4*>(src);
        qr[u][1] = *reinterpret_cast<const float4*>(src + 4);
      }
    }
    __syncthreads();   // chunk 0's pointers
    load_kv(0);
#pragma unroll
    for (int u = 0; u < Q_IT; ++u) {
      const int it = threadIdx.x + u * TTHREADS, qv = it / DCH, dc = it % DCH;
      const float sc = a.scale * kLog2e;
      const float x[8] = {qr[u][0].x * sc, qr[u][0].y * sc, qr[u][0].z * sc, qr[u][0].w * sc,
                          qr[u][1].x * sc, qr[u][1].y * sc, qr[u][1].z * sc, qr[u][1].w * sc};
      uint4 hi, lo;
      split8(x, hi, lo);
      const uint32_t off = SM::Q_OFF + (dc >> 3) * SM::Q_KB + tc::sw128_offset(qv, dc & 7);
      st_shared16(sm, off, hi);
      st_shared16(sm, off + SM::Q_PLANE, lo);
    }
  }

  for (int i = 0; i < nb_chunks && nq > 0; ++i) {
    const int c = attn::chunk_of(L, n_p, cx, C, i);
    const bool tail = c >= n_p;
    const int t0 = c * ACH;
    // the previous chunk's P V has completed: K, V and P may be overwritten
    if (nproc > 0 && !tc::mbar_wait(&bar_o, (nproc - 1) & 1, a.status, a.wait_ns)) s_abort = 1;
    if (i + 1 < nb_chunks) kptrs(i + 1);
    // ---- stage the chunk: split the loaded K and V into hi/lo and store
#pragma unroll
    for (int u = 0; u < K_IT; ++u) {
      const int idx = threadIdx.x + u * TTHREADS, j = idx / DCH, dc = idx % DCH;
      const float x[8] = {kr[u][0].x, kr[u][0].y, kr[u][0].z, kr[u][0].w,
                          kr[u][1].x, kr[u][1].y, kr[u][1].z, kr[u][1].w};
      uint4 hi, lo;
      split8(x, hi, lo);
      const uint32_t off = SM::K_OFF + (dc >> 3) * SM::K_KB + tc::sw128_offset(j, dc & 7);
      st_shared16(sm, off, hi);
      st_shared16(sm, off + SM::K_PLANE, lo);
    }
#pragma unroll
    for (int u = 0; u < V_IT; ++u) {
      const int idx = threadIdx.x + u * TTHREADS, d = idx % HD, jc = idx / HD;
      uint4 hi, lo;
      split8(vr[u], hi, lo);
      const uint32_t off = SM::V_OFF + tc::sw128_offset(d, jc);
      st_shared16(sm, off, hi);
      st_shared16(sm, off + SM::V_PLANE, lo);
    }
    tc::fence_proxy_async();
    __syncthreads();
    if (s_abort) break;
    // ---- S = Q K^T (hi.hi + hi.lo + lo.hi over the head dimension)
    if (threadIdx.x == kIssuer) {
      tc::tc_fence_after();
#pragma unroll
      for (int kb = 0; kb < KB; ++kb) {
        const uint64_t qh = tc::desc_sw128(sbase + SM::Q_OFF + kb * SM::Q_KB);
        const uint64_t ql = tc::desc_sw128(sbase + SM::Q_OFF + SM::Q_PLANE + kb * SM::Q_KB);
        const uint64_t kh = tc::desc_sw128(sbase + SM::K_OFF + kb * SM::K_KB);
        const uint64_t kl = tc::desc_sw128(sbase + SM::K_OFF + SM::K_PLANE + kb * SM::K_KB);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {   // K = 16 per MMA: +32 bytes = +2 in the descriptor
          tc::umma_bf16(t_s, qh + 2 * kk, kh + 2 * kk, idesc_s, (kb | kk) ? 1u : 0u);
          tc::umma_bf16(t_s, qh + 2 * kk, kl + 2 * kk, idesc_s, 1u);
          tc::umma_bf16(t_s, ql + 2 * kk, kh + 2 * kk, idesc_s, 1u);
        }
      }
      tc::umma_commit(&bar_s);
    }
    if (i + 1 < nb_chunks) load_kv(i + 1);   // in flight during this chunk's softmax
    // ---- softmax over the chunk: thread t owns TMEM lane qi = t % 128 (a query vector) and
    //      the chunk's keys 32h .. 32h + 31, h = t / 128 (warps w and w + 4 read the same
    //      lanes; tcgen05.ld is warp-collective, so a warp takes every branch as a whole)
    const bool sok = __all_sync(0xffffffffu, tc::mbar_wait(&bar_s, nproc & 1, a.status, a.wait_ns));
    float s[2][16];
    float mx = -INFINITY;
    if (!sok) {
      s_abort = 1;
    } else {
      tc::tc_fence_after();
      uint32_t r[2][16];
#pragma unroll
      for (int q = 0; q < 2; ++q)
        tc::tmem_ld16_nowait(t_s + lane_base + 32 * half + 16 * q, r[q]);
      tc::tmem_wait_ld();
      // prefix chunk: key j is visible below the row's prefix length (one limit per row)
      const int lim = (!tail && qi < nq) ? L.np[qi] - t0 - 32 * half : 0;
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int j = 32 * half + 16 * q + e;
          const bool vis = tail ? (qi < nq && attn::key_visible(L, qi, i, c, n_p, j))
                                : 16 * q + e < lim;
          s[q][e] = vis ? __uint_as_float(r[q][e]) : -INFINITY;   // masked: 2^(-inf - m) = 0
          mx = fmaxf(mx, s[q][e]);
        }
      s_mx[half][qi] = mx;
    }
    __syncthreads();
    if (s_abort) break;
    mx = fmaxf(s_mx[0][qi], s_mx[1][qi]);   // the row's maximum, the same in both halves
    {
      // raise the reference where a row's maximum passed it by more than kLazy: its earlier
      // sum and output are rescaled by alpha = exp(m_old - m_new) (both halves decide alike)
      float alpha = 1.f;
      bool rescale_o = false;
      if (mx > -INFINITY && (m_ref == -INFINITY || mx > m_ref + kLazy)) {
        alpha = m_ref == -INFINITY ? 0.f : exp2f(m_ref - mx);
        rescale_o = nproc > 0 && m_ref > -INFINITY;
        l_run *= alpha;
        m_ref = mx;
      }
      // each half rescales its half of the output row's columns, each lane by its own factor
      // (1 where its reference stayed)
      if (__any_sync(0xffffffffu, rescale_o)) {
        const float f = rescale_o ? alpha : 1.f;
#pragma unroll 1
        for (int q = 0; q < HD / 32; ++q) {
          float o[16];
          const uint32_t col = t_o + lane_base + half * (HD / 2) + 16 * q;
          tc::tmem_ld16(col, o);
#pragma unroll
          for (int e = 0; e < 16; ++e) o[e] *= f;
          tc::tmem_st16(col, o);
        }
      }
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          s[q][e] = m_ref == -INFINITY ? 0.f : exp2f(s[q][e] - m_ref);
          sum += s[q][e];
        }
      l_run += sum;   // this half's share of the row's sum; the halves are added at the end
      // P row qi: keys 8ch..8ch+7 are 16-byte chunk ch (hi and lo planes); this half writes
      // chunks 4h .. 4h + 3
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        float x[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) x[e] = s[cc >> 1][(cc & 1) * 8 + e];
        uint4 hi, lo;
        split8(x, hi, lo);
        const uint32_t off = SM::P_OFF + tc::sw128_offset(qi, 4 * half + cc);
        st_shared16(sm, off, hi);
        st_shared16(sm, off + SM::P_PLANE, lo);
      }
      tc::fence_proxy_async();
      tc::tc_fence_before();
    }
    __syncthreads();
    // ---- O += P V (hi.hi + hi.lo + lo.hi over the chunk's 64 keys)
    if (threadIdx.x == kIssuer) {
      tc::tc_fence_after();
      const uint64_t ph = tc::desc_sw128(sbase + SM::P_OFF);
      const uint64_t pl = tc::desc_sw128(sbase + SM::P_OFF + SM::P_PLANE);
      const uint64_t vh = tc::desc_sw128(sbase + SM::V_OFF);
      const uint64_t vl = tc::desc_sw128(sbase + SM::V_OFF + SM::V_PLANE);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        tc::umma_bf16(t_o, ph + 2 * kk, vh + 2 * kk, idesc_o, (nproc | kk) ? 1u : 0u);
        tc::umma_bf16(t_o, ph + 2 * kk, vl + 2 * kk, idesc_o, 1u);
        tc::umma_bf16(t_o, pl + 2 * kk, vh + 2 * kk, idesc_o, 1u);
      }
      tc::umma_commit(&bar_o);
    }
    ++nproc;
  }

  // ---- every MMA issued here completes before its operands are overwritten and TMEM is
  //      released (fixed limit, also after a give-up)
  if (threadIdx.x == kIssuer) {
    tc::umma_commit(&bar_d);
    tc::mbar_wait(&bar_d, 0, a.status);
  }
  // ---- the block's partial (m, l, o) per query vector into shared memory (o over K, V, P):
  //      each half writes its half of the row's columns; l is the sum of the halves' shares
  if (nproc > 0 && !tc::mbar_wait(&bar_o, (nproc - 1) & 1, a.status, a.wait_ns)) s_abort = 1;
  if (half == 1) s_mx[1][qi] = l_run;
  __syncthreads();
  float* s_po = reinterpret_cast<float*>(sm + SM::O_OFF);   // [TQB][OP]
  const bool have_o = nproc > 0 && !s_abort;
  if (have_o) tc::tc_fence_after();
#pragma unroll 1
  for (int q0 = 0; q0 < HD / 32; q0 += 4) {   // 64 columns per wait
    uint32_t o[4][16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (have_o && q0 + q < HD / 32) {
        tc::tmem_ld16_nowait(t_o + lane_base + half * (HD / 2) + 16 * (q0 + q), o[q]);
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) o[q][e] = 0u;
      }
    }
    if (have_o) tc::tmem_wait_ld();
    if (qi < nq) {
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (q0 + q < HD / 32)
#pragma unroll
          for (int e = 0; e < 16; e += 4) {
            float* dst = s_po + qi * SM::OP + half * (HD / 2) + 16 * (q0 + q) + e;
            *reinterpret_cast<float4*>(dst) =
                make_float4(__uint_as_float(o[q][e]), __uint_as_float(o[q][e + 1]),
                            __uint_as_float(o[q][e + 2]), __uint_as_float(o[q][e + 3]));
          }
    }
  }
  if (half == 0 && qi < nq) {
    s_pm[qi] = have_o ? m_ref : -INFINITY;
    s_pl[qi] = have_o ? l_run + s_mx[1][qi] : 0.f;
  }
  tc::tc_fence_before();
  cluster.sync();   // every block's partials are visible to the cluster

  // ---- merge: block cx finishes query vectors cx, cx + C, ... (a warp per query vector),
  //      reading the C partials through distributed shared memory, 8 blocks at a time
  constexpr int DPL = HD / 32;
  const int lane = threadIdx.x & 31;
  for (int qv = cx + warp * C; qv < nq; qv += C * TWARPS) {
    float vv[8][DPL];
    auto load_o = [&](int r0) {
#pragma unroll
      for (int r = 0; r < 8; ++r) {
#pragma unroll
        for (int c2 = 0; c2 < DPL; ++c2) vv[r][c2] = 0.f;
        if (r0 + r < C) {
          const float* src = cluster.map_shared_rank(s_po, r0 + r) + qv * SM::OP + DPL * lane;
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
      mr = cluster.map_shared_rank(s_pm, lane)[qv];
      lr = cluster.map_shared_rank(s_pl, lane)[qv];
    }
    const float M = warp_max(mr);
    const float w = (lane < C && mr > -INFINITY) ? exp2f(mr - M) : 0.f;
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
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
    const size_t dst = (size_t)L.row[qv] * H * HD + (size_t)(g * G + L.gg[qv]) * HD + DPL * lane;
#pragma unroll
    for (int c2 = 0; c2 < DPL; ++c2) store_act<__nv_bfloat16>(out, a.plane, dst + c2, acc[c2] * inv);
  }
  cluster.sync();   // no block leaves while the others may still read its shared memory
  if (warp == 0) tc::tmem_dealloc(tmem, SM::TMEM_COLS);
}

template <int HD>
ClusterFit g_tc_fit;   // cluster residency of k_attn_tc<HD> (configure_tc)

template <int HD>
int configure_tc() {
  auto k = k_attn_tc<HD>;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TcSmem<HD>::bytes) !=
      cudaSuccess)
    return -1;
  const bool nonportable =
      cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  cudaGetLastError();
  fill_cluster_fit(&g_tc_fit<HD>, k, TTHREADS, TcSmem<HD>::bytes, nonportable ? TACL : 8);
  return nonportable && g_tc_fit<HD>.active[TACL] >= 1 ? 0 : 1;   // 1: portable only
}

}  // namespace

int attn_tc_qblock(int rows_per_prompt, int G) {
  // up to 128 query vectors, and at most 32 rows meeting in one block (the tail layout runs
  // one lane per row): 32 G vectors (whole rows) when that is smaller; no larger than a
  // prompt's vectors rounded up to whole rows of 16
  const int cap = std::min(128, 32 * G);
  const int nq = rows_per_prompt * G;
  return std::max(16, std::min(cap, (nq + 15) / 16 * 16));
}

int configure_attention_tc() {
  const int r128 = configure_tc<128>(), r64 = configure_tc<64>();
  if (r128 < 0 || r64 < 0) return -1;
  g_tc_max_cluster = (r128 || r64) ? 8 : TACL;
  return 0;
}

void launch_attn_tc(const AttnArgs& a, int n_z, cudaStream_t s) {
  const int cl = attn_cluster_size(a.kv.hd == 128 ? g_tc_fit<128> : g_tc_fit<64>,
                                   g_tc_max_cluster, a.n_chunks + a.n_tchunks, a.kv.kvh * n_z);
  if (a.kv.hd == 128)
    launch_pdl_cluster(k_attn_tc<128>, dim3(cl, a.kv.kvh, n_z), dim3(TTHREADS),
                       TcSmem<128>::bytes, cl, s, a);
  else
    launch_pdl_cluster(k_attn_tc<64>, dim3(cl, a.kv.kvh, n_z), dim3(TTHREADS),
                       TcSmem<64>::bytes, cl, s, a);
}

}  // namespace cdsl
