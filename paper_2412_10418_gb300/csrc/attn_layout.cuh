// attn_layout.cuh -- which query vectors and which key slots one attention block works on.
//
// Both attention kernels (attention.cu: CUDA cores, any model dtype; attention_tc.cu: tensor
// cores, bf16 models) split a pass the same way. The keys a prompt's rows may see are cut into
// chunks of ACH slots: prefix chunks (ACH consecutive positions of the prompt's shared prefix
// pages) and then tail chunks (the distinct beam tails of a query block's rows, concatenated,
// each as long as its longest row). A cluster of blocks owns one (prompt b, KV head, query
// block qb). The launch sizes for the most chunks a pass can have (n_chunks prefix chunks,
// n_tchunks tail chunks); the chunks that hold keys -- prefix chunks below the block's longest
// prefix, tail chunks up to the tails' total length -- are numbered in order, and block cx of
// the C blocks takes numbers cx, cx + C, ..., so the cluster's work is spread evenly over
// the chunks that exist at run time. A query vector is a (row,
// query head of the KV head's GQA group) pair; the rows of prompt b are taken in row order,
// G vectors each, and query block qb holds vectors [qb * QB, qb * QB + QB).
#pragma once

#include <algorithm>

#include "kernels.h"

namespace cdsl {
namespace attn {

constexpr int ACH = 64;              // key slots per chunk
constexpr int MAXP = 128;            // chunks (prefix + tail) of a pass
constexpr int MAXCB = MAXP / 8;      // chunks per block (at most; clusters have >= 8 blocks
                                     // whenever a pass has more than 8 chunks)

// Per-block layout in shared memory. QB: capacity in query vectors (the launch's query block,
// a.qblock, is at most QB).
template <int QB>
struct Layout {
  int row[QB], gg[QB], np[QB], tb[QB], nt[QB];   // per query vector: row, head in the group,
                                                 // prefix length, tail base, tail length
  int toff[32], tlen[32], ttb[32];   // per row of the block (first row of a tail only): the
                                     // tail's offset in the concatenation, length, base slot
  int wcnt[32];                      // scratch: rows of prompt b per warp
  int nrows, maxnp;                  // rows of prompt b seen so far; longest prefix
  int nr_p, nr_t, nb;                // prefix and tail chunks holding keys; this block's chunks
  int kslot[MAXCB * ACH];            // every key slot of the block's chunks: the page (prefix
                                     // chunk) or tail row (tail chunk), -1 empty
  int ktb[MAXCB * ACH];              // tail slots: tail base of the beam,
  uint8_t kj[MAXCB * ACH];           //   index in it
};

// Pass chunk (prefix chunks first, n_p of them) of this block's i-th chunk: number cx + i * C
// among the chunks that hold keys (L.nr_p prefix, then L.nr_t tail chunks).
template <int QB>
__device__ __forceinline__ int chunk_of(const Layout<QB>& L, int n_p, int cx, int C, int i) {
  const int k = cx + i * C;
  return k < L.nr_p ? k : n_p + (k - L.nr_p);
}

// Fill L for query block qb of prompt b and this block's chunks (L.nb of them, chunk_of);
// called by all NTHREADS threads of the block (a multiple of 32, at most 1024), which it
// leaves synchronized. Reads only what the launch chain has already completed (row
// descriptors, committed page table), so it may run before griddepcontrol.wait. Returns the
// number of the block's query vectors (0..a.qblock). At most 32 rows may meet in one query block
// (the tail layout runs one lane per row). More tail keys than the tail chunks hold latch
// CDSL_ERANGE.
template <int QB, int NTHREADS>
__device__ int build_layout(Layout<QB>& L, const AttnArgs& a, int b, int qb, int cx, int C) {
  constexpr int NWARPS = NTHREADS / 32;
  const int G = a.G, QBr = a.qblock;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < QB; i += NTHREADS) L.row[i] = -1;
  for (int i = threadIdx.x; i < MAXCB * ACH; i += NTHREADS) L.kslot[i] = -1;
  if (threadIdx.x == 0) L.nrows = 0;
  __syncthreads();
  // this block's query vectors: rows of prompt b in order, G heads each
  for (int base = 0; base < a.R; base += NTHREADS) {
    const int r = base + threadIdx.x;
    RowDesc rd;
    const bool mine = r < a.R && (rd = a.rows[r]).b == b;
    const unsigned bal = __ballot_sync(0xffffffffu, mine);
    if (lane == 0) L.wcnt[warp] = __popc(bal);
    __syncthreads();
    int off = L.nrows;
    for (int w = 0; w < warp; ++w) off += L.wcnt[w];
    const int local = off + __popc(bal & ((1u << lane) - 1));
    if (mine) {
      for (int gg = 0; gg < G; ++gg) {
        const int qi = local * G + gg - qb * QBr;
        if (qi >= 0 && qi < QBr) {
          L.row[qi] = r;
          L.gg[qi] = gg;
          L.np[qi] = rd.n_prefix;
          L.tb[qi] = rd.tail_base;
          L.nt[qi] = rd.n_tail;
        }
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < NWARPS; ++w) tot += L.wcnt[w];
      L.nrows += tot;
    }
    __syncthreads();
  }
  const int nq = max(0, min(QBr, L.nrows * G - qb * QBr));
  if (warp == 0) {
    // longest prefix, and the distinct tails (lane = row of the block) in order of first
    // appearance, each as long as its longest row: slot offsets in their concatenation
    const int first_local = (qb * QBr) / G;
    const int qi_l = max(0, (first_local + lane) * G - qb * QBr);   // the row's first vector
    const bool row_ok = nq > 0 && qi_l < nq && lane <= (qb * QBr + nq - 1) / G - first_local;
    int np = row_ok ? L.np[qi_l] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) np = max(np, __shfl_xor_sync(0xffffffffu, np, o));
    const int tb = row_ok ? L.tb[qi_l] : -1;
    const int nt = row_ok ? L.nt[qi_l] : 0;
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
    L.toff[lane] = off - len;
    L.tlen[lane] = len;
    L.ttb[lane] = tb;
    if (lane == 0) {
      L.maxnp = np;
      if (cx == 0 && total > a.n_tchunks * ACH) set_status(a.status, CDSL_ERANGE);
      L.nr_p = min(a.n_chunks, (np + ACH - 1) / ACH);
      L.nr_t = min(a.n_tchunks, (total + ACH - 1) / ACH);
      L.nb = max(0, (L.nr_p + L.nr_t - cx + C - 1) / C);   // <= MAXCB: C >= chunks / MAXCB
    }
  }
  __syncthreads();
  const int maxnp = L.maxnp, n_p = a.n_chunks, nb_chunks = L.nb;
  // key slots of this block's chunks
  for (int i = 0; i < nb_chunks; ++i) {
    const int c = chunk_of(L, n_p, cx, C, i);
    if (c < n_p) {   // prefix positions c*ACH .. c*ACH + ACH-1 below the longest prefix
      for (int j = threadIdx.x; j < ACH; j += NTHREADS) {
        const int t = c * ACH + j;
        if (t < maxnp)
          L.kslot[i * ACH + j] = a.kv.page_table[b * a.kv.max_pages + (t >> a.kv.page_shift)];
      }
    } else if (warp == 0) {   // tail slots [lo, lo + ACH) of the concatenation
      const int lo = (c - n_p) * ACH, off = L.toff[lane], len = L.tlen[lane], tb = L.ttb[lane];
      for (int e = max(0, lo - off); e < len && off + e < lo + ACH; ++e) {
        const int sl = i * ACH + off + e - lo;
        L.kslot[sl] = tb + e;
        L.ktb[sl] = tb;
        L.kj[sl] = (uint8_t)e;
      }
    }
  }
  __syncthreads();
  return nq;
}

// Whether query vector qi (of a block with layout L) may see key j of the block's chunk i,
// chunk c of the pass (prefix chunks first): a prefix position before the row's prefix length,
// or a slot of the row's own beam tail up to itself.
template <int QB>
__device__ __forceinline__ bool key_visible(const Layout<QB>& L, int qi, int i, int c, int n_p,
                                            int j) {
  if (c < n_p) return c * ACH + j < L.np[qi];
  const int k = i * ACH + j;
  return L.kslot[k] >= 0 && L.ktb[k] == L.tb[qi] && L.kj[k] < L.nt[qi];
}

// Algorithmic bytes of the block for in-graph timing: K and V (fp32) of every key slot of its
// chunks once per (prompt, KV head) -- counted by the first query block's clusters -- plus,
// from block 0 of the cluster, every query vector read and its output written once.
template <int QB, int NTHREADS, int HD>
__device__ void count_bytes(const Layout<QB>& L, const LaunchStamp& stamp, int qb, int cx,
                            int nb_chunks, int nq, int* s_cnt) {
  if (threadIdx.x == 0) *s_cnt = 0;
  __syncthreads();
  int mine = 0;
  if (qb == 0)
    for (int i = threadIdx.x; i < nb_chunks * ACH; i += NTHREADS) mine += L.kslot[i] >= 0;
  if (mine) atomicAdd(s_cnt, mine);
  __syncthreads();
  if (threadIdx.x == 0)
    stamp.add_bytes((unsigned long long)*s_cnt * HD * 8 +
                    (cx == 0 ? (unsigned long long)nq * HD * 8 : 0));
}

}  // namespace attn

// Blocks per cluster of an attention launch with `groups` clusters (prompt x KV head x query
// block) over `chunks` key chunks: the size C with the least estimated time, waves(C) x
// (2 ceil(chunks / C) + 1) in half chunk-times -- a block's chunks one after another, then
// about half a chunk's time of merging -- where a wave is f.active[C] clusters. One chunk per
// block while the groups leave room (the latency-bound decode and verify passes); fewer blocks
// with more chunks each when one chunk per block would need more than a wave (a cluster too
// large to be placed as often as the groups need it, e.g. 16 blocks, or too many groups). A
// block takes at most attn::MAXCB chunks (its key-slot table), so C >= ceil(chunks / MAXCB);
// ties go to the smaller cluster.
inline int attn_cluster_size(const ClusterFit& f, int max_cluster, int chunks, int groups) {
  const int least = std::max(1, (chunks + attn::MAXCB - 1) / attn::MAXCB);
  const int most = std::max(least, std::min(std::min(max_cluster, 16), chunks));
  int best = least;
  long long best_cost = -1;
  for (int c = least; c <= most; ++c) {
    if (f.active[c] < 1) continue;
    const long long waves = (groups + f.active[c] - 1) / f.active[c];
    const long long cost = waves * (2LL * ((chunks + c - 1) / c) + 1);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = c;
    }
  }
  return best;
}

}  // namespace cdsl
