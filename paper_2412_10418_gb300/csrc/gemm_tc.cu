// gemm_tc.cu -- projection GEMMs on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Swap-AB: the weights are the M = 128 operand (one tile = 128 virtual output rows, loaded as
// two 64-row TMA boxes so that a tile may draw its halves from different segments: gate/up
// interleave, q/k/v boundaries) and the activation rows are the N operand (N = R rounded up
// to 16, 16..256). Both operands are K-major bf16 in 128-byte-swizzled shared-memory tiles;
// the accumulator lives in TMEM (fp32). The activations come as the hi and lo bf16 planes of
// the split, so each 16-deep K step issues two MMAs into the same accumulator.
//
// Persistent stream-K schedule: a fixed grid of blocks (two per SM when the ring fits in half
// the shared memory) divides the tiles x 64-wide K blocks evenly, so there is no partial last
// wave. With as many tiles as block slots or fewer the same code runs one block per whole tile
// (data-parallel: every segment is a whole tile, no fixup). A block walks its contiguous range
// of (tile, k-block) units; a run of units within one tile is a segment. Warp 0 (one lane)
// streams weights and activations with TMA through a ring of mbarrier-guarded stages; warp 1
// (one lane) issues the MMAs into one of two TMEM accumulators and commits; warps 2-5 drain a
// finished accumulator (TMEM -> registers -> shared memory) while the next segment
// accumulates into the other one. A segment covering a whole tile runs the fused epilogue
// directly; otherwise its partial tile goes to scratch and the tile is finished from the
// partials summed in block order (a deterministic sum): by the last contributing block
// (k_gemm_tc<false>), or above 64 activation rows (k_gemm_tc<true>) by every contributor for
// its share of the rows, after its own last segment, once all partials are in.
//
// Cluster split-K (GEMMs with few tiles): a thread-block cluster of S blocks owns one tile and
// block r of it the r-th of S even K ranges. Each block drains its partial tile into shared
// memory; after a cluster barrier every block sums a share of the tile's activation rows over
// the S partials (in block order, through distributed shared memory) and runs the epilogue on
// them. No global partials, no atomics.
//
// Programmatic dependent launch: weights do not depend on the previous kernel, so the TMA
// lane issues the first ring's weight loads before griddepcontrol.wait and the activation
// loads after it; every other dependent access comes after the wait. Every wait on an mbarrier
// is bounded in time; on expiry the block latches CDSL_ETIMEOUT and winds down.
#include <cudaTypedefs.h>

#include <algorithm>

#include "gemm.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace cdsl {
namespace {

constexpr int kMaxStages = 8;
constexpr int kTileLd = 132;     // fp32 epilogue tile row pitch (128 + 4 against bank conflicts)
constexpr int kEpRowsMax = 64;   // activation rows drained per epilogue chunk (at most)
constexpr int kThreads = 192;    // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kEpThreads = 128;

__host__ __device__ __forceinline__ uint32_t tmem_cols_for(int n_pad) {
  uint32_t c = 32;
  while (c < (uint32_t)n_pad) c <<= 1;
  return c;
}

// Source tensor map and first row of the 64-row half-tile starting at virtual row vstart.
__device__ __forceinline__ void half_source(const GemmArgs& a, int vstart, int* m, int* y) {
  if (a.mode == EPI_SWIGLU) {
    *m = (vstart >> 6) & 1;
    *y = (vstart >> 7) * 64;
    return;
  }
  int base = 0;
  for (int s = 0; s < a.n_seg; ++s) {
    if (vstart < base + a.seg_rows[s] || s == a.n_seg - 1) {
      *m = s;
      *y = vstart - base;
      return;
    }
    base += a.seg_rows[s];
  }
}

// Stream-K partition: block c owns units [start(c), start(c + 1)) (U * C < 2^31, checked on
// the host).
__device__ __forceinline__ int unit_start(int c, int U, int C) { return c * U / C; }
__device__ __forceinline__ int unit_owner(int u, int U, int C) { return ((u + 1) * C - 1) / U; }

constexpr int kMaxContrib = 256;   // contributors to one tile (bounded on the host)
constexpr int kMaxSplit = 8;       // target blocks per tile when tiles are few
constexpr int kRedBatch = 4;       // float4 groups per thread per pass of the large-row fixup
constexpr int kBigRows = 64;       // padded activation rows above which k_gemm_tc<true> runs

// kBig: the variant for more than 64 activation rows: its epilogue, stream-K fixup and
// cluster reduction keep several loads per thread in flight (a tile's epilogue then costs a
// few round trips to memory instead of one per row), and its QKV epilogue reads each row's
// position and K/V destination gathered once per block. The plain loops of the other
// variant keep its register count low, so that neighbouring launches overlap.
template <bool kBig>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_tc(const __grid_constant__ TcMaps maps, const __grid_constant__ GemmArgs a, TcPlan p,
              float* part, int* tile_cnt) {
  extern __shared__ uint8_t smem_raw[];
  const LaunchStamp stamp(a.stamp);
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t accf_bar[2];
  __shared__ __align__(8) uint64_t acce_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;   // every MMA this block issued has completed
  __shared__ uint32_t tmem_base;
  __shared__ int s_abort, s_last;
  __shared__ int s_slot_off[kMaxContrib];   // reducer: scratch offset (floats) per contributor
  __shared__ float s_rs[256];                // input row scales (RMSNorm folded into the GEMM)
  __shared__ QkvRow s_qkv[kBig ? 256 : 1];   // QKV: RoPE position and K/V destination per row
  __shared__ int s_pend[2], s_npend;         // kBig stream-K: tiles this block helps finish

  uint8_t* smem = smem_raw + ((1024 - (tc::smem_u32(smem_raw) & 1023)) & 1023);
  const int NP = p.n_pad, S = p.stages, KBT = p.kb_total;
  const uint32_t stage_bytes = 16384u + 256u * NP;
  const int kEpRows = p.ep_rows;
  float* tileS = reinterpret_cast<float*>(smem + (size_t)S * stage_bytes);  // [ep_rows][kTileLd]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x, C = gridDim.x;
  const int U = p.tiles * KBT;
  const int SK = p.cluster;   // > 0: cluster split-K, block (tile c / SK, K range c % SK)
  int u0, u1;
  if (SK > 0) {
    const int t = c / SK, r = c % SK;
    u0 = t * KBT + r * KBT / SK;
    u1 = t * KBT + (r + 1) * KBT / SK;
  } else {
    u0 = unit_start(c, U, C);
    u1 = unit_start(c + 1, U, C);
  }
  // hi and lo rows are contiguous in each stage: one MMA with N = 2*NP covers both (the
  // accumulator then holds W.hi in columns [0, NP) and W.lo in [NP, 2NP)); above N = 256 they
  // are two MMAs into one accumulator.
  const bool fused = 2 * NP <= 256;
  const uint32_t acc_cols = tmem_cols_for(fused ? 2 * NP : NP);

  // TMA producer state (thread 0): unit u0 + i is (t_cur, kb_cur) for the next i to issue
  const int n_units = u1 - u0;
  const int pre = min(S, n_units);
  int t_cur = u0 / KBT, kb_cur = u0 % KBT;
  int n_issued = 0;   // (thread 0) units whose copies were issued
  uint64_t pol = 0;
  auto load_w = [&](int i, int t, int kb) {
    int m0, y0, m1, y1;
    half_source(a, t * 128, &m0, &y0);
    half_source(a, t * 128 + 64, &m1, &y1);
    uint8_t* st = smem + (size_t)(i % S) * stage_bytes;
    tc::tma_load_2d_hint(st, &maps.w[m0], kb * 64, y0, &full_bar[i % S], pol);
    tc::tma_load_2d_hint(st + 8192, &maps.w[m1], kb * 64, y1, &full_bar[i % S], pol);
  };
  auto load_x = [&](int i, int kb) {   // one box of NP rows per plane (the maps' box)
    uint8_t* st = smem + (size_t)(i % S) * stage_bytes;
    tc::tma_load_2d(st + 16384, &maps.xh, kb * 64, 0, &full_bar[i % S]);
    tc::tma_load_2d(st + 16384 + NP * 128, &maps.xl, kb * 64, 0, &full_bar[i % S]);
  };
  if (threadIdx.x == 0) {
    for (int m = 0; m < 3; ++m) tc::tma_prefetch_map(&maps.w[m]);
    tc::tma_prefetch_map(&maps.xh);
    tc::tma_prefetch_map(&maps.xl);
    for (int s = 0; s < S; ++s) {
      tc::mbar_init(&full_bar[s], 1);
      tc::mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&accf_bar[i], 1);
      tc::mbar_init(&acce_bar[i], kEpThreads);
    }
    tc::mbar_init(&drain_bar, 1);
    s_abort = 0;
    s_npend = 0;
    tc::fence_mbar_init();
    tc::fence_proxy_async();
    // the first ring's weights do not depend on the previous kernel: issue them while warp 1
    // allocates TMEM
    pol = tc::policy_evict_first();
    for (int i = 0; i < pre; ++i) {
      tc::mbar_expect_tx(&full_bar[i], stage_bytes);
      load_w(i, t_cur, kb_cur);
      if (++kb_cur == KBT) { kb_cur = 0; ++t_cur; }
    }
  }
  if (warp == 1) tc::tmem_alloc(&tmem_base, 2 * acc_cols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  pdl_launch_dependents();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      bool aborted = false;
      int issued = 0;
      pdl_wait();
      {
        int kb = u0 % KBT;
        for (int i = 0; i < pre; ++i) {
          load_x(i, kb);
          if (++kb == KBT) kb = 0;
        }
      }
      issued = pre;
      for (int i = pre; i < n_units; ++i) {
        const int s = i % S, use = i / S;
        if (!tc::mbar_wait(&empty_bar[s], (use - 1) & 1, a.status, a.wait_ns)) {
          aborted = true;
          break;
        }
        tc::mbar_expect_tx(&full_bar[s], stage_bytes);
        load_w(i, t_cur, kb_cur);
        load_x(i, kb_cur);
        if (++kb_cur == KBT) { kb_cur = 0; ++t_cur; }
        ++issued;
      }
      if (aborted) s_abort = 1;
      n_issued = issued;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc = tc::idesc_bf16_f32(128, fused ? 2 * NP : NP);
      int seg = 0;
      int u = u0;
      bool ok = true;
      while (u < u1 && ok) {
        const int seg_end = min(u1, (u / KBT + 1) * KBT);
        const int acc = seg & 1;
        if (seg >= 2 &&
            !tc::mbar_wait(&acce_bar[acc], ((seg >> 1) - 1) & 1, a.status, a.wait_ns)) {
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t d = tmem + (uint32_t)acc * acc_cols;
        const int seg_begin = u;
        for (; u < seg_end; ++u) {
          const int i = (int)(u - u0), s = i % S, use = i / S;
          if (!tc::mbar_wait(&full_bar[s], use & 1, a.status, a.wait_ns)) {
            ok = false;
            break;
          }
          tc::tc_fence_after();
          const uint32_t sa = tc::smem_u32(smem + (size_t)s * stage_bytes);
          const uint64_t da = tc::desc_sw128(sa);
          const uint64_t dh = tc::desc_sw128(sa + 16384);
          const uint64_t dl = tc::desc_sw128(sa + 16384 + NP * 128);
          const bool first = (u == seg_begin);
          if (fused) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)   // 4 x K=16 per stage; +32 bytes = +2 in the desc
              tc::umma_bf16(d, da + 2 * kk, dh + 2 * kk, idesc, (first && kk == 0) ? 0u : 1u);
          } else {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              tc::umma_bf16(d, da + 2 * kk, dh + 2 * kk, idesc, (first && kk == 0) ? 0u : 1u);
              tc::umma_bf16(d, da + 2 * kk, dl + 2 * kk, idesc, 1u);
            }
          }
          tc::umma_commit(&empty_bar[s]);
        }
        if (!ok) break;   // an unfinished accumulator is never handed to the epilogue
        tc::umma_commit(&accf_bar[acc]);
        ++seg;
      }
      if (!ok) s_abort = 1;
      // every MMA issued here completes before TMEM is released (fixed limit)
      tc::umma_commit(&drain_bar);
      tc::mbar_wait(&drain_bar, 0, a.status);
    }
  } else {
    // ---------------- epilogue warps 2..5: TMEM lanes 32*(warp % 4) .. +31
    const int etid = threadIdx.x - 64;
    const int quarter = warp & 3;
    pdl_wait();
    int seg = 0;
    int u = u0;
    const int R = min(a.R, NP);
    if (a.in_ss || (kBig && a.mode == EPI_QKV)) {   // once per block, while the first
      if (a.in_ss) input_row_scales(a, 0, R, s_rs, etid, kEpThreads);   // accumulator fills
      if (kBig && a.mode == EPI_QKV) qkv_rows(a, R, s_qkv, etid, kEpThreads);
      tc::named_barrier(1, kEpThreads);
    }
    while (u < u1) {
      const int t = u / KBT;
      const int seg_end = min(u1, (t + 1) * KBT);
      const bool whole = (u % KBT) == 0 && seg_end == (t + 1) * KBT;
      const int acc = seg & 1;
      const bool ready = tc::mbar_wait(&accf_bar[acc], (seg >> 1) & 1, a.status, a.wait_ns);
      // the epilogue warps give up together or not at all: named barriers and warp-collective
      // TMEM loads follow
      if (tc::named_barrier_or(1, kEpThreads, !ready)) {
        s_abort = 1;
        break;
      }
      tc::tc_fence_after();
      const uint32_t d = tmem + (uint32_t)acc * acc_cols + ((uint32_t)(quarter * 32) << 16);
      const int slot = (t == u0 / KBT) ? 0 : 1;
      float* my_part = part + ((size_t)(c * 2 + slot) * NP) * 128;
      for (int r0 = 0; r0 < NP; r0 += kEpRows) {
        const int rows = min(kEpRows, NP - r0);
        for (int c0 = 0; c0 < rows; c0 += 16) {
          float v[16];
          tc::tmem_ld16(d + (uint32_t)(r0 + c0), v);
          if (fused) {
            float w[16];
            tc::tmem_ld16(d + (uint32_t)(NP + r0 + c0), w);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += w[i];
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) tileS[(c0 + i) * kTileLd + quarter * 32 + lane] = v[i];
        }
        tc::named_barrier(1, kEpThreads);
        const int rt = max(0, min(rows, R - r0));
        if (SK > 0) {
          // cluster split-K: the partial stays in tileS (ep_rows == NP: one chunk) until the
          // cluster reduction at the end
        } else if (whole) {
          tile_epilogue<__nv_bfloat16, kBig>(a, t * 128, r0, rt, tileS, kTileLd, s_rs + r0,
                                             etid, kEpThreads, kBig ? s_qkv : nullptr);
        } else if (kBig) {
          for (int i = etid; i < rt * 32; i += kEpThreads) {   // float4 groups
            const int r = i >> 5, v = (i & 31) * 4;
            *reinterpret_cast<float4*>(my_part + (size_t)(r0 + r) * 128 + v) =
                *reinterpret_cast<const float4*>(tileS + r * kTileLd + v);
          }
        } else {
          for (int i = etid; i < rt * 128; i += kEpThreads) {
            const int r = i >> 7, v = i & 127;
            my_part[(size_t)(r0 + r) * 128 + v] = tileS[r * kTileLd + v];
          }
        }
        tc::named_barrier(1, kEpThreads);
      }
      tc::tc_fence_before();
      tc::mbar_arrive(&acce_bar[acc]);   // accumulator drained: the MMA lane may reuse it
      if (!whole && SK == 0) {
        const int cf = unit_owner(t * KBT, U, C);
        const int cl = unit_owner((t + 1) * KBT - 1, U, C);
        // publish this block's partial and count it (one acquire-release atomic after the
        // barrier)
        tc::named_barrier(1, kEpThreads);
        if constexpr (kBig) {
          // the tile is finished after this block's last segment, by all its contributors
          if (etid == 0) {
            tc::atom_add_acq_rel_gpu(tile_cnt + t, 1);
            s_pend[s_npend++] = t;
          }
        } else {
          // the last block to arrive sees every contributor's partial and finishes the tile
          if (etid == 0) s_last = (tc::atom_add_acq_rel_gpu(tile_cnt + t, 1) == cl - cf);
          tc::named_barrier(1, kEpThreads);
          if (s_last) {
            // scratch slot of every contributor: its first segment -> 0, its last -> 1
            for (int j = etid; j <= cl - cf; j += kEpThreads) {
              const int cc = cf + j;
              const int sl = (t == unit_start(cc, U, C) / KBT) ? 0 : 1;
              s_slot_off[j] = (cc * 2 + sl) * NP * 128;
            }
            tc::named_barrier(1, kEpThreads);
            const int ncontrib = cl - cf + 1;
            for (int r0 = 0; r0 < R; r0 += kEpRows) {
              const int rt = min(kEpRows, R - r0);
              // float4 groups: 32 per activation row; all contributors' loads in flight together
              for (int i = etid; i < rt * 32; i += kEpThreads) {
                const int off = (r0 + (i >> 5)) * 128 + (i & 31) * 4;
                float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                int j = 0;
                for (; j + 4 <= ncontrib; j += 4) {
                  float4 v[4];
#pragma unroll
                  for (int q = 0; q < 4; ++q)
                    v[q] = __ldcg(reinterpret_cast<const float4*>(part + s_slot_off[j + q] + off));
#pragma unroll
                  for (int q = 0; q < 4; ++q) {
                    sum.x += v[q].x; sum.y += v[q].y; sum.z += v[q].z; sum.w += v[q].w;
                  }
                }
                for (; j < ncontrib; ++j) {
                  const float4 v = __ldcg(reinterpret_cast<const float4*>(part + s_slot_off[j] + off));
                  sum.x += v.x; sum.y += v.y; sum.z += v.z; sum.w += v.w;
                }
                *reinterpret_cast<float4*>(tileS + (i >> 5) * kTileLd + (i & 31) * 4) = sum;
              }
              tc::named_barrier(1, kEpThreads);
              tile_epilogue<__nv_bfloat16, false>(a, t * 128, r0, rt, tileS, kTileLd, s_rs + r0,
                                                  etid, kEpThreads);
              tc::named_barrier(1, kEpThreads);
            }
            if (etid == 0) tile_cnt[t] = 0;
          }
        }
      }
      u = seg_end;
      ++seg;
    }
    if constexpr (kBig) {
      // Distributed stream-K fixup: every contributor of a partially owned tile sums its share
      // of the tile's activation rows over all contributors' partials (block order, as the
      // single-finisher form would) and runs the epilogue on them, once every partial of the
      // tile is published. Each block publishes all its partials before it waits, and every
      // block of the grid is resident at once (one block per SM, no more blocks than SMs), so
      // every wait ends; it is still bounded. tile_cnt[tiles + t] counts the finished shares;
      // the last one resets both counters for the next launch.
      const bool gave_up = tc::named_barrier_or(1, kEpThreads, s_abort != 0);
      const int npend = gave_up ? 0 : s_npend;
      for (int q = 0; q < npend; ++q) {
        const int t = s_pend[q];
        const int cf = unit_owner(t * KBT, U, C);
        const int cl = unit_owner((t + 1) * KBT - 1, U, C);
        const int ncontrib = cl - cf + 1, jme = c - cf;
        bool ok = true;
        if (etid == 0) ok = tc::wait_count_gpu(tile_cnt + t, ncontrib, a.status, a.wait_ns);
        if (tc::named_barrier_or(1, kEpThreads, !ok)) {
          s_abort = 1;
          break;
        }
        // scratch slot of every contributor: its first segment -> 0, its last -> 1
        for (int j = etid; j < ncontrib; j += kEpThreads) {
          const int cc = cf + j;
          const int sl = (t == unit_start(cc, U, C) / KBT) ? 0 : 1;
          s_slot_off[j] = (cc * 2 + sl) * NP * 128;
        }
        tc::named_barrier(1, kEpThreads);
        const int ra = jme * R / ncontrib, rb = (jme + 1) * R / ncontrib;
        for (int rs = ra; rs < rb; rs += kEpRows) {
          const int rt = min(kEpRows, rb - rs), r0 = rs;
          // float4 groups, 32 per activation row, kRedBatch groups per thread per pass: the
          // loads of kRedBatch groups x up to four contributors are in flight together. The
          // contributors are summed in block order (deterministic).
          for (int i0 = etid; i0 < rt * 32; i0 += kEpThreads * kRedBatch) {
            float4 sum[kRedBatch];
            int off[kRedBatch];
#pragma unroll
            for (int g = 0; g < kRedBatch; ++g) {
              const int i = min(i0 + g * kEpThreads, rt * 32 - 1);   // clamped: in bounds
              off[g] = (r0 + (i >> 5)) * 128 + (i & 31) * 4;
              sum[g] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
            for (int j = 0; j < ncontrib; j += 4) {
              const int nj = min(4, ncontrib - j);
              float4 v[4][kRedBatch];
#pragma unroll
              for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int g = 0; g < kRedBatch; ++g)
                  if (q < nj)
                    v[q][g] = __ldcg(
                        reinterpret_cast<const float4*>(part + s_slot_off[j + q] + off[g]));
#pragma unroll
              for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int g = 0; g < kRedBatch; ++g)
                  if (q < nj) {
                    sum[g].x += v[q][g].x; sum[g].y += v[q][g].y;
                    sum[g].z += v[q][g].z; sum[g].w += v[q][g].w;
                  }
            }
#pragma unroll
            for (int g = 0; g < kRedBatch; ++g) {
              const int i = i0 + g * kEpThreads;
              if (i < rt * 32)
                *reinterpret_cast<float4*>(tileS + (i >> 5) * kTileLd + (i & 31) * 4) = sum[g];
            }
          }
          tc::named_barrier(1, kEpThreads);
          tile_epilogue<__nv_bfloat16, true>(a, t * 128, r0, rt, tileS, kTileLd, s_rs + r0, etid,
                                             kEpThreads, s_qkv);
          tc::named_barrier(1, kEpThreads);
        }
        if (etid == 0 && tc::atom_add_acq_rel_gpu(tile_cnt + p.tiles + t, 1) == ncontrib - 1) {
          tile_cnt[t] = 0;
          tile_cnt[p.tiles + t] = 0;
        }
      }
    }
  }
  if (SK > 0) {
    // ---- cluster split-K reduction: rank r sums rows [r*R/SK, (r+1)*R/SK) of the SK partial
    //      tiles in rank order (distributed shared memory) into a free pipeline stage and runs
    //      the epilogue on them
    // the epilogue warps agree on whether the block gave up (the two named barriers below
    // must be reached by all of them or by none)
    const bool gave_up = warp >= 2 ? tc::named_barrier_or(1, kEpThreads, s_abort != 0) : true;
    tc::cluster_arrive();               // this block's partial tile is complete (release)
    tc::cluster_wait();                 // every block's is (acquire)
    const bool reduce = warp >= 2 && !gave_up;
    const int R = min(a.R, NP), r = c % SK, t = c / SK;
    const int ra = r * R / SK, rb = (r + 1) * R / SK;
    float* red = reinterpret_cast<float*>(smem);   // stage 0 (idle): [rb - ra][kTileLd]
    if (reduce) {
      const int etid = threadIdx.x - 64;
      const uint32_t tile_s = tc::smem_u32(tileS);
      for (int i = etid; i < (rb - ra) * 32; i += kEpThreads) {
        const uint32_t off = ((ra + (i >> 5)) * kTileLd + (i & 31) * 4) * 4;
        float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
        if constexpr (kBig) {
          // eight blocks' loads in flight together, summed in rank order
          for (int q0 = 0; q0 < SK; q0 += 8) {
            float4 v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q)
              if (q0 + q < SK)
                v[q] = tc::ld_cluster_f32x4(tc::map_cluster_rank(tile_s + off, q0 + q));
#pragma unroll
            for (int q = 0; q < 8; ++q)
              if (q0 + q < SK) {
                sum.x += v[q].x; sum.y += v[q].y; sum.z += v[q].z; sum.w += v[q].w;
              }
          }
        } else {
          for (int q = 0; q < SK; ++q) {
            const float4 v = tc::ld_cluster_f32x4(tc::map_cluster_rank(tile_s + off, q));
            sum.x += v.x; sum.y += v.y; sum.z += v.z; sum.w += v.w;
          }
        }
        *reinterpret_cast<float4*>(red + (i >> 5) * kTileLd + (i & 31) * 4) = sum;
      }
    }
    // this block has read the others' tiles (the sums above consumed every load): the
    // barrier's second phase runs while the epilogue writes
    tc::cluster_arrive();
    if (reduce) {
      const int etid = threadIdx.x - 64;
      tc::named_barrier(1, kEpThreads);
      if (rb > ra)
        tile_epilogue<__nv_bfloat16, kBig>(a, t * 128, ra, rb - ra, red, kTileLd, s_rs + ra,
                                           etid, kEpThreads, kBig ? s_qkv : nullptr);
    }
    tc::cluster_wait();                 // no block leaves while its tile may still be read
  }
  tc::tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && s_abort) {
    // a block that gave up waits for the copies it issued last to land before it leaves (the
    // earlier ones were consumed, so they have landed); fixed limit
    for (int i = max(0, n_issued - S); i < n_issued; ++i)
      tc::mbar_wait(&full_bar[i % S], (i / S) & 1, a.status);
  }
  if (warp == 1) tc::tmem_dealloc(tmem, 2 * acc_cols);
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
size_t g_static_smem[2] = {4096, 8192};   // static shared memory of k_gemm_tc<false / true>
                                          // (queried at configuration)
int g_max_cluster = 8;         // 16 where non-portable clusters of k_gemm_tc are allowed
// Clusters of k_gemm_tc<big> resident at once with one or two blocks' shared memory budget per
// SM ([big][blocks per SM - 1]; configure_gemm_tc fills [1][0], the one in use; until then no
// plan is limited).
ClusterFit g_cfit[2][2];
bool g_cfit_ready = false;

}  // namespace

bool tc_supported(const GemmArgs& a) {
  if (a.K % 64 || a.R < 1 || a.R > 256) return false;
  // 32-bit stream-K unit arithmetic and at most kMaxContrib blocks per tile
  const long long units = (long long)((a.n_virtual + 127) / 128) * (a.K / 64);
  if (a.K / 64 >= kMaxContrib || units * 4 * kPlanSMs >= (1LL << 31)) return false;
  for (int s = 0; s + 1 < a.n_seg; ++s)
    if (a.mode != EPI_SWIGLU && a.seg_rows[s] % 64) return false;
  return true;
}

TcPlan plan_tc(int K, int n_virtual, int R, int n_sm, int force_per_sm, int max_split,
               int cluster) {
  TcPlan p{};
  p.n_pad = (R + 15) / 16 * 16;
  p.tiles = (n_virtual + 127) / 128;
  p.kb_total = K / 64;
  const size_t stage = 16384 + 256 * (size_t)p.n_pad;
  p.big = p.n_pad > kBigRows;
  // two blocks per SM when three stages fit in half the shared memory (228 KB per SM, less
  // each block's static part and the 1 KB the runtime reserves per block), else one; the
  // epilogue drains 16 activation rows at a time when that frees room for another stage
  const size_t half = 114 * 1024 - g_static_smem[p.big] - 1024;
  auto fit = [&](size_t budget, int ep) {
    return (int)std::min<size_t>(kMaxStages, (budget - (size_t)ep * kTileLd * 4 - 1024) / stage);
  };
  int per_sm = 1;
  size_t budget = std::min<size_t>(220 * 1024, 227 * 1024 - g_static_smem[p.big]);
  const int ep_big = std::min(p.n_pad, kEpRowsMax);
  if (force_per_sm >= 3 && !p.big) {   // more, shallower blocks (measurement aid; the
                                         // large-row variant's fixup needs one block per SM)
    per_sm = force_per_sm;
    budget = (227 * 1024) / force_per_sm - 1024;
  } else if ((force_per_sm == 2 || force_per_sm == 0) && fit(half, 16) >= 3) {
    per_sm = 2;
    budget = half;
  }
  p.ep_rows = fit(budget, 16) > fit(budget, ep_big) ? 16 : ep_big;
  p.stages = fit(budget, p.ep_rows);
  // at most kMaxSplit blocks share a tile: the fixup then stays cheap next to the streaming
  const long long units = (long long)p.tiles * p.kb_total;
  p.ctas = (int)std::min<long long>(std::min<long long>(units, (long long)per_sm * n_sm),
                                    (long long)p.tiles * (max_split > 0 ? max_split : kMaxSplit));
  // few tiles: a cluster of S <= 12 blocks per tile, all tiles resident at once. Clusters are
  // placed whole within a GPC; on 152 SMs at two blocks each, grids of clusters past ~87 % of
  // the block slots no longer fit in one wave (measured), hence the cap.
  const int cap = per_sm * n_sm * 87 / 100;
  // (the whole partial tile, n_pad rows, stays in shared memory: two stages must still fit)
  const bool tile_fits = fit(budget, p.n_pad) >= 2;
  // Up to 12 blocks per tile while the grid stays within 64 % of the block slots (measured
  // at two blocks per SM, 7B draft down projection 2048 x 5504, 16 tiles: 8.43 us at 12
  // blocks against 9.02 us at 8; larger non-portable clusters or grids lose, e.g. 16 x 16
  // blocks: 14.3 us).
  const int wide = per_sm * n_sm * 64 / 100;
  int S = cluster;
  if (S < 0)
    S = (tile_fits && 2 * p.tiles <= cap)
            ? std::max(std::min(8, cap / p.tiles), std::min(12, wide / p.tiles))
            : 0;
  S = std::min(std::min(S, p.kb_total), g_max_cluster);
  // large-row plans (one block per SM): every cluster must be resident at once. A cluster is
  // placed whole within a GPC, so fewer clusters fit than the SMs suggest (g_cfit: e.g. the
  // small model's 18-tile QKV at 160 rows, 7-block clusters: 42.9 -> 28.2 us with 6). The
  // reported residency at two blocks per SM is below what the 7B plans measurably get
  // (limiting them by it: 7B step 5.95 -> 7.10 ms), so those keep the measured caps above.
  if (g_cfit_ready && p.big && per_sm == 1)
    while (S >= 2 && g_cfit[1][0].active[S] < p.tiles) --S;
  if (S >= 2 && tile_fits) {
    p.cluster = S;
    p.ctas = p.tiles * S;
    p.ep_rows = p.n_pad;   // the whole partial tile stays in shared memory
    p.stages = fit(budget, p.ep_rows);
  } else if (cluster < 0 && max_split == 0 && p.tiles <= per_sm * n_sm &&
             10 * p.tiles >= 9 * n_sm) {
    // about one tile per SM or more, but too many for clusters: one block per whole tile (no
    // split, no fixup). Measured against stream-K over all 304 slots: 38.4 vs 41.2 us (7B
    // gate/up), 46.2 vs 55.2 us (7B LM head), 22.8 vs 25.2 us (draft LM head). With fewer
    // tiles than that (e.g. the 40-tile projections of the 13B verify pass at 224 rows, whose
    // partial tiles are too large for clusters) whole tiles would leave most SMs idle:
    // stream-K over every block slot instead.
    p.ctas = p.tiles;
  }
  p.smem = (size_t)p.stages * stage + (size_t)p.ep_rows * kTileLd * 4 + 1024;
  return p;
}

size_t tc_scratch_floats(const TcPlan& p) {
  return p.cluster ? 0 : (size_t)p.ctas * 2 * p.n_pad * 128;
}

int encode_bf16_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer) {
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return -1;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

int configure_gemm_tc() {
  int rc = 0;
  bool nonportable = true;
  auto setup = [&](auto kernel, int big) {
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, kernel) != cudaSuccess) {
      rc = -1;
      return;
    }
    g_static_smem[big] = fa.sharedSizeBytes;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
        cudaSuccess)
      nonportable = false;
    cudaGetLastError();
    // plans use at most 220 KB + 1 KB of alignment slack; a block has at most 227 KB in all
    const int dyn = (int)std::min<size_t>(220 * 1024 + 1024, 227 * 1024 - fa.sharedSizeBytes);
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn) !=
        cudaSuccess)
      rc = -1;
  };
  setup(k_gemm_tc<false>, 0);
  setup(k_gemm_tc<true>, 1);
  g_max_cluster = nonportable ? 16 : 8;
  if (rc == 0) {
    const size_t one = std::min<size_t>(220 * 1024 + 1024, 227 * 1024 - g_static_smem[1]);
    fill_cluster_fit(&g_cfit[1][0], k_gemm_tc<true>, kThreads, one, g_max_cluster);
    g_cfit_ready = true;
  }
  return rc;
}

void launch_gemm_tc(const TcMaps& maps, const GemmArgs& a, const TcPlan& p, float* part,
                    int* tile_cnt, cudaStream_t s) {
  auto kernel = p.big ? k_gemm_tc<true> : k_gemm_tc<false>;
  if (p.cluster)
    launch_pdl_cluster(kernel, dim3(p.ctas), dim3(kThreads), p.smem, p.cluster, s, maps, a, p,
                       part, tile_cnt);
  else
    launch_pdl(kernel, dim3(p.ctas), dim3(kThreads), p.smem, s, maps, a, p, part, tile_cnt);
}

}  // namespace cdsl
