// kernels.cu -- embedding, RMSNorm (+ reward head), logits row statistics, row plans, and the
// CDSL acceptance decision / commit.
#include <cuda_bf16.h>
#include <math.h>

#include "gemm.cuh"
#include "kernels.h"

namespace cdsl {

namespace {

constexpr int kMaxWarps = 32;

__device__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  float t = (threadIdx.x < nw) ? red[threadIdx.x] : 0.f;
  if (wid == 0) t = warp_sum(t);
  if (threadIdx.x == 0) red[0] = t;
  __syncthreads();
  return red[0];
}

__device__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_max_u64(v);
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  unsigned long long t = (threadIdx.x < nw) ? red[threadIdx.x] : 0ull;
  if (wid == 0) t = warp_max_u64(t);
  if (threadIdx.x == 0) red[0] = t;
  __syncthreads();
  return red[0];
}

// ------------------------------------------------------------------------------ embedding
// h = E[token]; also the first GEMM input x = h . g (GEMM-input format) and the 32-feature
// partial sums of h^2 from which the consuming GEMM takes the RMSNorm row scale.
template <typename T>
__global__ void k_embed(const RowDesc* rows, const T* E, int D, float* h, T* x, size_t plane,
                        const T* g, float* ss, int ld_ss) {
  pdl_wait();
  pdl_launch_dependents();
  const int r = blockIdx.x;
  const T* e = E + (size_t)rows[r].token * D;
  for (int c0 = 0; c0 < D; c0 += blockDim.x) {   // blockDim is a multiple of 32, D of 64
    const int c = c0 + threadIdx.x;
    const float v = c < D ? to_f32<T>(e[c]) : 0.f;
    if (c < D) {
      h[(size_t)r * D + c] = v;
      store_act<T>(x, plane, (size_t)r * D + c, v * to_f32<T>(g[c]));
    }
    const float sq = warp_sum(v * v);
    if ((threadIdx.x & 31) == 0 && c < D) ss[(size_t)(c >> 5) * ld_ss + r] = sq;
  }
}

// ------------------------------------------------------------------------------ RMSNorm
// out[r] = h[src] / sqrt(mean(h[src]^2) + eps) * g, src = gather ? gather[r] : r.
// With head_w: head_out[r] = sigmoid(head_w . normalized row) (fp32, before rounding).
template <typename T>
__global__ void __launch_bounds__(256) k_rmsnorm(const float* h, int D, const T* g, float eps,
                                                T* out, size_t plane, const int32_t* gather,
                                                const float* head_w, float* head_out) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float red[kMaxWarps];
  constexpr int MAXV = 8;   // float4 per thread: D <= 8 * 4 * 256 = 8192
  const int r = blockIdx.x;
  const int src = gather ? gather[r] : r;
  const float4* x = reinterpret_cast<const float4*>(h + (size_t)src * D);
  const int n4 = D >> 2;
  float4 v[MAXV];
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < MAXV; ++i) {
    const int c = threadIdx.x + i * 256;
    v[i] = c < n4 ? x[c] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
#pragma unroll
  for (int i = 0; i < MAXV; ++i) ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
  ss = block_sum(ss, red);
  const float inv = rsqrtf(ss / (float)D + eps);
  float hw = 0.f;
#pragma unroll
  for (int i = 0; i < MAXV; ++i) {
    const int c = threadIdx.x + i * 256;
    if (c >= n4) continue;
    const float e[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float y = e[q] * inv * to_f32<T>(g[4 * c + q]);
      store_act<T>(out, plane, (size_t)r * D + 4 * c + q, y);
      if (head_w) hw += head_w[4 * c + q] * y;
    }
  }
  if (head_w) {
    hw = block_sum(hw, red);
    if (threadIdx.x == 0) head_out[r] = 1.0f / (1.0f + expf(-hw));
  }
}

// ------------------------------------------------------------------------------ row stats
// One block per logits row; each thread holds its slice of the row in registers (one load
// pass), then max / argmax, log-sum-exp and the top-k passes run on the registers.
constexpr int RS_THREADS = 512;
constexpr int RS_MAXV = 16;   // float4 per thread: V <= 16 * 4 * 512 = 32768

__global__ void __launch_bounds__(RS_THREADS) k_row_stats(RowStatsArgs a) {
  const LaunchStamp stamp(a.stamp);
  pdl_wait();
  pdl_launch_dependents();
  __shared__ unsigned long long redk[kMaxWarps];
  __shared__ float red[kMaxWarps];
  __shared__ int bad_s;
  const int r = blockIdx.x;
  const float* row = a.logits + (size_t)r * a.V;
  const float4* v4 = reinterpret_cast<const float4*>(row);
  const int n4 = a.V >> 2;
  if (threadIdx.x == 0) bad_s = 0;
  float4 x[RS_MAXV];
#pragma unroll
  for (int i = 0; i < RS_MAXV; ++i) {
    const int c = threadIdx.x + i * RS_THREADS;
    x[i] = c < n4 ? v4[c] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  }
  __syncthreads();
  unsigned long long best = 0;
  int bad = 0;
#pragma unroll
  for (int i = 0; i < RS_MAXV; ++i) {
    const int c = threadIdx.x + i * RS_THREADS;
    if (c >= n4) continue;
    const float e[4] = {x[i].x, x[i].y, x[i].z, x[i].w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (!isfinite(e[q])) bad = 1;
      const unsigned long long key = argmax_key(e[q], 4 * c + q);
      best = key > best ? key : best;
    }
  }
  if (bad) atomicOr(&bad_s, 1);
  best = block_max_u64(best, redk);
  const int amax = argmax_key_index(best);
  const float m = row[amax];
  float z = 0.f;
#pragma unroll
  for (int i = 0; i < RS_MAXV; ++i) {
    const int c = threadIdx.x + i * RS_THREADS;
    if (c >= n4) continue;
    z += expf(x[i].x - m) + expf(x[i].y - m) + expf(x[i].z - m) + expf(x[i].w - m);
  }
  z = block_sum(z, red);
  const float lse = m + logf(z);
  if (threadIdx.x == 0 && bad_s) set_status(a.status, CDSL_ENONFINITE);

  if (a.x_out) {  // draft rollout: greedy token and its log-probability
    if (threadIdx.x == 0) {
      a.x_out[r * a.out_stride + a.out_off] = amax;
      a.logq_out[r * a.out_stride + a.out_off] = m - lse;
    }
    return;
  }
  if (a.amax && threadIdx.x == 0) a.amax[r] = amax;
  if (a.head_out && threadIdx.x < 32) {   // sigmoid(w . g . h * row scale) from the partials
    float hw = 0.f;
    for (int c = threadIdx.x; c < (a.norm_D >> 5); c += 32) hw += a.hw[(size_t)c * a.ld_ss + r];
    hw = warp_sum(hw);
    if (threadIdx.x == 0) {
      const float rs = row_scale(a.ss, a.norm_D >> 5, a.ld_ss, r, a.norm_D, a.norm_eps);
      a.head_out[r] = 1.0f / (1.0f + expf(-hw * rs));
    }
  }
  if (a.dp1 > 0 && threadIdx.x == 0) {
    const int j = r % a.dp1, bi = r / a.dp1, d = a.dp1 - 1;
    if (j < d && a.logp) {
      const int tok = a.next_x[bi * d + j];
      a.logp[bi * d + j] = row[tok] - lse;
    }
  }
  if (a.topk) {
    int dst = r;
    if (a.dst) dst = a.dst[r];
    if (dst < 0) return;
    unsigned long long prev = best;
    if (threadIdx.x == 0) a.topk[dst * a.k] = amax;
    for (int p = 1; p < a.k; ++p) {
      unsigned long long cur = 0;
#pragma unroll
      for (int i = 0; i < RS_MAXV; ++i) {
        const int c = threadIdx.x + i * RS_THREADS;
        if (c >= n4) continue;
        const float e[4] = {x[i].x, x[i].y, x[i].z, x[i].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const unsigned long long key = argmax_key(e[q], 4 * c + q);
          if (key < prev && key > cur) cur = key;
        }
      }
      cur = block_max_u64(cur, redk);
      if (threadIdx.x == 0) a.topk[dst * a.k + p] = argmax_key_index(cur);
      prev = cur;
    }
  }
}

// ------------------------------------------------------------------------------ plans
// Draft call j (1..d): beam rows (b, i) carry c_bi (j = 1) or x_bi,j-1 at position L + j - 1,
// see the prefix and their own tail slots 0..j-1. Call 1 adds one row per prompt: the pending
// token L-1 of a fully accepted step, written straight into the draft prefix pages.
__global__ void k_plan_draft(StepState st, int j, int spb, RowDesc* rows) {
  pdl_wait();
  pdl_launch_dependents();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  const int nbk = st.B * st.k;
  if (r < nbk) {
    const int b = r / st.k;
    const int L = st.len[b];
    RowDesc rd;
    rd.b = b;
    rd.pos = L + j - 1;
    rd.token = (j == 1) ? st.roots[r] : st.x[r * st.d + j - 2];
    rd.n_prefix = L;
    rd.tail_base = r * spb;
    rd.n_tail = j;
    rd.kv_dst = r * spb + j - 1;
    rd.out_idx = r;
    rows[r] = rd;
  } else if (j == 1 && r < nbk + st.B) {
    const int b = r - nbk;
    const int L = st.len[b];
    RowDesc rd;
    rd.b = b;
    rd.tail_base = 0;
    rd.n_tail = 0;
    rd.out_idx = -1;
    if (st.pend[b]) {
      rd.pos = L - 1;
      rd.token = st.tokens[b * st.lcap + L - 1];
      rd.n_prefix = L;
      rd.kv_dst = KV_PREFIX;
    } else {  // idle row: reads position 0, stores nothing
      rd.pos = 0;
      rd.token = 0;
      rd.n_prefix = 1;
      rd.kv_dst = KV_NONE;
    }
    rows[r] = rd;
  }
}

// Verify rows (b, i, j), j = 0..d: token c_bi (j = 0) or x_bi,j at position L + j; they see
// the prefix and their beam's tail slots 0..j (causal within the beam, nothing across beams).
__global__ void k_plan_verify(StepState st, RowDesc* rows) {
  pdl_wait();
  pdl_launch_dependents();
  const int dp1 = st.d + 1;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= st.B * st.k * dp1) return;
  const int bi = r / dp1, j = r % dp1, b = bi / st.k;
  const int L = st.len[b];
  RowDesc rd;
  rd.b = b;
  rd.pos = L + j;
  rd.token = (j == 0) ? st.roots[bi] : st.x[bi * st.d + j - 1];
  rd.n_prefix = L;
  rd.tail_base = bi * dp1;
  rd.n_tail = j + 1;
  rd.kv_dst = r;
  rd.out_idx = r;
  rows[r] = rd;
}

// Step-1 round 2, draft call j (1..d), in the round's own tail region of d+1 slots per prompt
// (slot 0 c_1, slot 1 x', slot j lh_j-1): rows [0, B) carry x' at L + 1 (j = 1, which also
// records x' = argmax M_p(pfx + c_1), verify row (b, 1, 0)) or lh_j-1 at L + j; rows [B, 2B)
// of call 1 carry c_1 at L.
__global__ void k_plan_s1_draft(StepState st, int j, RowDesc* rows) {
  pdl_wait();
  pdl_launch_dependents();
  const int B = st.B, dp1 = st.d + 1;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= (j == 1 ? 2 * B : B)) return;
  const int b = r % B;
  const int L = st.len[b], base = st.s1_dbase + b * dp1;
  RowDesc rd;
  rd.b = b;
  rd.n_prefix = L;
  rd.tail_base = base;
  if (r >= B) {
    rd.pos = L;
    rd.token = st.roots[b * st.k];
    rd.n_tail = 1;
    rd.kv_dst = base;
    rd.out_idx = -1;
  } else if (j == 1) {
    const int xp = st.v_amax[b * st.k * dp1];
    st.s1_tok[b * dp1] = xp;
    rd.pos = L + 1;
    rd.token = xp;
    rd.n_tail = 2;
    rd.kv_dst = base + 1;
    rd.out_idx = b;
  } else {
    rd.pos = L + j;
    rd.token = st.s1_tok[b * dp1 + j - 1];
    rd.n_tail = j + 1;
    rd.kv_dst = base + j;
    rd.out_idx = b;
  }
  rows[r] = rd;
}

// Step-1 round 2, the target pass, in its tail region of d+2 slots per prompt (c_1, x',
// lh_1..lh_d): rows [0, B) x' at L + 1 (the LM rows: M_p(pfx + c_1 + x')), [B, 2B) c_1 at L,
// then lh_j at L + 1 + j, prompt-major (the reward head reads lh_d's row).
__global__ void k_plan_s1_verify(StepState st, RowDesc* rows) {
  pdl_wait();
  pdl_launch_dependents();
  const int B = st.B, d = st.d, dp1 = d + 1;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= B * (d + 2)) return;
  int b, slot;
  if (r < B) {
    b = r; slot = 1;
  } else if (r < 2 * B) {
    b = r - B; slot = 0;
  } else {
    b = (r - 2 * B) / d; slot = 2 + (r - 2 * B) % d;
  }
  const int L = st.len[b], base = st.s1_tbase + b * (d + 2);
  RowDesc rd;
  rd.b = b;
  rd.pos = L + slot;
  rd.token = slot == 0 ? st.roots[b * st.k] : st.s1_tok[b * dp1 + slot - 1];
  rd.n_prefix = L;
  rd.tail_base = base;
  rd.n_tail = slot + 1;
  rd.kv_dst = base + slot;
  rd.out_idx = r < B ? b : -1;
  rows[r] = rd;
}

// ------------------------------------------------------------------------------ decision
__device__ void alloc_pages(const KvStore& kv, int b, int from, int to, int32_t* next_page,
                            int32_t* status) {
  if (to <= from) return;
  for (int p = from >> kv.page_shift; p <= (to - 1) >> kv.page_shift; ++p) {
    int32_t* e = kv.page_table + b * kv.max_pages + p;
    if (p >= kv.max_pages) { set_status(status, CDSL_ERANGE); return; }
    if (*e < 0) {
      const int id = atomicAdd(next_page, 1);
      if (id >= kv.n_pages) { set_status(status, CDSL_ERANGE); return; }
      *e = id;
    }
  }
}

// One warp per prompt, one lane per beam: n_b, rewards, b*, state, emission, page allocation.
// Draw number c of the SplitMix64 generator seeded with `seed` (Steele, Lea, Flood, 2014:
// state_c = seed + (c + 1) * golden gamma, output = the variant-13 mix of the state), reduced
// to its top 24 bits as a float in [0, 1) (exact in float32).
__device__ __forceinline__ float uniform24(uint32_t seed, unsigned long long c) {
  unsigned long long z = (unsigned long long)seed + (c + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z ^= z >> 31;
  return (float)(z >> 40) * (1.0f / 16777216.0f);
}

__global__ void k_select(StepState st, KvStore tkv, KvStore dkv, int commit) {
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.x, lane = threadIdx.x;
  const int k = st.k, d = st.d, dp1 = d + 1;
  if (st.gen[b] >= st.max_new) {
    if (lane < k) {
      st.reward[(b * k + lane) * 2] = 0.f;
      st.reward[(b * k + lane) * 2 + 1] = 0.f;
      st.n_acc[b * k + lane] = 0;
    }
    if (lane < dp1) st.emitted[b * dp1 + lane] = -1;
    if (lane == 0) {
      st.beam[b] = -1; st.state[b] = 0; st.n_emit[b] = 0;
      st.s1_need[b] = 0; st.s1_used[b] = 0;
    }
    return;
  }
  float rf = -INFINITY, ra = -INFINITY;
  int n = 0;
  if (lane < k) {
    const int bi = b * k + lane;
    if (st.acceptance == 0) {   // hard rejection: M_p's argmax must equal the drafted token
      for (int j = 0; j < d; ++j) {
        if (st.v_amax[bi * dp1 + j] != st.x[bi * d + j]) break;
        ++n;
      }
    } else {                    // speculative sampling: u_j <= min(1, p_j(x_j) / q_j(x_j))
      const unsigned long long step = (unsigned long long)st.counters[0];
      const unsigned long long c0 = ((step * st.B + b) * k + lane) * d;
      for (int j = 0; j < d; ++j) {
        const float u = uniform24(st.seed, c0 + j);
        if (!(logf(u) <= st.v_logp[bi * d + j] - st.logq[bi * d + j])) break;
        ++n;
      }
    }
    const int root = st.roots[bi];
    uint32_t cf = st.cov[b], ca = st.cov[b];
    for (int q = 0; q < st.nk; ++q) {
      const int kwq = st.kw[b * st.nk + q];
      bool in_full = (root == kwq), in_acc = (root == kwq);
      for (int j = 0; j < d; ++j) {
        const bool hit = st.x[bi * d + j] == kwq;
        in_full |= hit;
        in_acc |= hit && (j < n);
      }
      if (in_full) cf |= 1u << q;
      if (in_acc) ca |= 1u << q;
    }
    const float covf = (float)__popc(cf) / (float)st.nk;
    const float cova = (float)__popc(ca) / (float)st.nk;
    if (st.reward_head) {
      rf = 0.5f * covf + 0.5f * st.v_head[bi * dp1 + d];
      ra = 0.5f * cova + 0.5f * st.v_head[bi * dp1 + n];
    } else {
      rf = covf;
      ra = cova;
    }
    st.n_acc[bi] = n;
    st.reward[bi * 2] = rf;
    st.reward[bi * 2 + 1] = ra;
  }
  const unsigned long long key = (lane < k) ? argmax_key(rf, lane) : 0ull;
  const int bs = argmax_key_index(warp_max_u64(key));   // first beam with the largest r^full
  const int nb = __shfl_sync(0xffffffffu, n, bs);
  const float rab = __shfl_sync(0xffffffffu, ra, bs);
  const bool s1 = (nb >= st.n_min) && (rab >= st.r_t);
  // Step-1 (b = 1) of S2/S3: M_p's greedy token c_1 when its lookahead's reward reaches r_t
  const float rf1 = __shfl_sync(0xffffffffu, rf, 0);
  const bool step1 = !s1 && nb < st.n_min && st.step1 >= 1 && rf1 >= st.r_t;
  const int win = step1 ? 0 : bs;   // the beam whose tokens are emitted
  int cnt = s1 ? 1 + nb : 1;
  cnt = min(cnt, st.max_new - st.gen[b]);
  const int bbi = b * k + win;
  if (lane < dp1) {
    int tok = -1;
    if (lane < cnt) tok = (lane == 0) ? st.roots[bbi] : st.x[bbi * d + lane - 1];
    st.emitted[b * dp1 + lane] = tok;
  }
  if (lane == 0) {
    st.beam[b] = win;
    st.state[b] = s1 ? 1 : (step1 ? 3 : (nb < st.n_min ? 2 : 4));
    st.n_emit[b] = cnt;
    // budget 2: round 1 failed in S2/S3, round 2 may still replace this Step-2 emission
    st.s1_need[b] = (!s1 && nb < st.n_min && st.step1 >= 2 && !(rf1 >= st.r_t)) ? 1 : 0;
    st.s1_used[b] = 0;
    if (!commit) return;
    const int L = st.len[b];
    alloc_pages(tkv, b, L, L + cnt, st.next_page + 0, st.status);
    alloc_pages(dkv, b, L, L + cnt, st.next_page + 1, st.status);
  }
}

// Step-1 round 2 (Alg. 1 S2/S3, Sec. 3.2.3, budget b = 2): X = [c_1, x'] with the lookahead
// lh of x'; R(T + X + lh) from the keyword bits and M_p's hidden state at lh_d (the same
// arithmetic as the verify rows' head). One warp per prompt.
__global__ void k_select_s1(StepState st, KvStore tkv, KvStore dkv, const float* ss,
                            const float* hw, int norm_D, int ld_ss, float eps) {
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.x, lane = threadIdx.x;
  const int d = st.d, dp1 = d + 1;
  if (!st.s1_need[b]) return;
  const int c1 = st.roots[b * st.k];
  uint32_t bits = 0;
  if (lane < st.nk) {
    const int kwq = st.kw[b * st.nk + lane];
    bool hit = c1 == kwq;
    for (int j = 0; j < dp1; ++j) hit |= st.s1_tok[b * dp1 + j] == kwq;
    if (hit) bits = 1u << lane;
  }
  for (int o = 16; o > 0; o >>= 1) bits |= __shfl_xor_sync(0xffffffffu, bits, o);
  const float cov = (float)__popc(st.cov[b] | bits) / (float)st.nk;
  float r = cov;
  if (st.reward_head) {
    const int row = 2 * st.B + b * d + d - 1;   // lh_d
    float h = 0.f;
    for (int c = lane; c < (norm_D >> 5); c += 32) h += hw[(size_t)c * ld_ss + row];
    h = warp_sum(h);
    const float rs = row_scale(ss, norm_D >> 5, ld_ss, row, norm_D, eps);
    r = 0.5f * cov + 0.5f * (1.0f / (1.0f + expf(-h * rs)));
  }
  if (lane == 0) st.s1_reward[b] = r;
  if (!(r >= st.r_t)) return;   // Step-2 (the c_b* emission of k_select) stands
  const int cnt = min(2, st.max_new - st.gen[b]);
  if (lane < dp1)
    st.emitted[b * dp1 + lane] = lane == 0 ? c1 : ((lane == 1 && cnt == 2) ? st.s1_tok[b * dp1] : -1);
  if (lane == 0) {
    st.beam[b] = 0;
    st.state[b] = 3;
    st.n_emit[b] = cnt;
    st.s1_used[b] = cnt == 2 ? 1 : 0;   // one token left: c_1 from beam 1's tails
    const int L = st.len[b];
    alloc_pages(tkv, b, L, L + cnt, st.next_page + 0, st.status);
    alloc_pages(dkv, b, L, L + cnt, st.next_page + 1, st.status);
  }
}

// Copy the winner's tail K/V rows 0..cnt-1 to prefix positions L..L+cnt-1 (after a Step-1
// round-2 emission: rows 0, 1 of the round's tail region).
__global__ void k_commit_kv(StepState st, KvStore kv, int spb, int is_draft) {
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.x, layer = blockIdx.y, kvsel = blockIdx.z;
  int cnt = st.n_emit[b];
  const bool s1 = st.s1_used[b] != 0;
  if (is_draft && !s1) cnt = min(cnt, st.d);
  if (cnt <= 0) return;
  const int bs = st.beam[b], L = st.len[b];
  const int src0 = !s1 ? (b * st.k + bs) * spb
                       : (is_draft ? st.s1_dbase + b * (st.d + 1) : st.s1_tbase + b * (st.d + 2));
  const int per_row = kv.kvh * kv.hd;
  for (int e = threadIdx.x; e < cnt * per_row; e += blockDim.x) {
    const int j = e / per_row, rest = e % per_row, head = rest / kv.hd, c = rest % kv.hd;
    const int pos = L + j;
    const int page = kv.page_table[b * kv.max_pages + (pos >> kv.page_shift)];
    if (page < 0) continue;
    const float* src = kv.tail + kv_tail_offset(kv, layer, kvsel, src0 + j, head);
    float* dst = kv.pool + kv_prefix_offset(kv, layer, page, kvsel, head, pos & ((1 << kv.page_shift) - 1));
    dst[c] = src[c];
  }
}

// pfx <- pfx + O, T <- T + O; the next beams are the top-k of the winner's row cnt-1.
__global__ void k_advance(StepState st) {
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.x, lane = threadIdx.x;
  const int k = st.k, d = st.d, dp1 = d + 1;
  if (b == 0 && lane == 0) {
    const int rounds = st.step1 >= 2 ? 2 : 1;   // the Step-1 round runs every step
    st.counters[0] += 1;                        // steps
    st.counters[1] += d * rounds;               // draft forward passes
    st.counters[2] += rounds;                   // target forward passes
  }
  const int cnt = st.n_emit[b];
  if (cnt <= 0) return;
  const int L = st.len[b], bs = st.beam[b];
  if (lane < cnt) st.tokens[b * st.lcap + L + lane] = st.emitted[b * dp1 + lane];
  uint32_t bits = 0;
  if (lane < st.nk) {
    const int kwq = st.kw[b * st.nk + lane];
    for (int t = 0; t < cnt; ++t)
      if (st.emitted[b * dp1 + t] == kwq) bits = 1u << lane;
  }
  for (int o = 16; o > 0; o >>= 1) bits |= __shfl_xor_sync(0xffffffffu, bits, o);
  const bool s1 = st.s1_used[b] != 0;   // next roots: top-k of M_p(pfx + c_1 + x')
  const int root_row = (b * k + bs) * dp1 + cnt - 1;
  if (lane < k)
    st.roots[b * k + lane] = s1 ? st.s1_topk[b * k + lane] : st.v_topk[root_row * k + lane];
  if (lane == 0) {
    st.cov[b] |= bits;
    st.len[b] = L + cnt;
    st.gen[b] += cnt;
    st.pend[b] = (!s1 && cnt == dp1) ? 1 : 0;
    atomicAdd((unsigned long long*)&st.counters[3], (unsigned long long)cnt);
    if (st.state[b] == 1) atomicAdd((unsigned long long*)&st.counters[4], 1ull);
    atomicAdd((unsigned long long*)&st.counters[5], 1ull);
  }
}

__global__ void k_rope_table(float2* table, int n_pos, int hd, double theta) {
  const int half = hd / 2;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_pos * half) return;
  const int pos = i / half, m = i % half;
  const double ang = (double)pos * pow(theta, -2.0 * m / hd);
  double s, c;
  sincos(ang, &s, &c);
  table[i] = make_float2((float)c, (float)s);
}

}  // namespace

// ------------------------------------------------------------------------------ launchers
#define DISPATCH(dtype, ...)                                   \
  do {                                                         \
    if ((dtype) == CDSL_DTYPE_BF16) {                          \
      using T = __nv_bfloat16;                                 \
      __VA_ARGS__;                                             \
    } else {                                                   \
      using T = float;                                         \
      __VA_ARGS__;                                             \
    }                                                          \
  } while (0)

void launch_embed(int dtype, const RowDesc* rows, int R, const void* embed, int D, float* h,
                  void* x, size_t plane, const void* g, float* ss, int ld_ss, cudaStream_t s) {
  DISPATCH(dtype, launch_pdl(k_embed<T>, dim3(R), dim3(256), 0, s, rows, (const T*)embed, D, h,
                             (T*)x, plane, (const T*)g, ss, ld_ss));
}

void launch_rmsnorm(int dtype, const float* h, int R, int D, const void* gain, float eps,
                    void* out, size_t plane, const int32_t* gather, const float* head_w,
                    float* head_out, cudaStream_t s) {
  DISPATCH(dtype, launch_pdl(k_rmsnorm<T>, dim3(R), dim3(256), 0, s, h, D, (const T*)gain, eps,
                             (T*)out, plane, gather, head_w, head_out));
}

void launch_row_stats(const RowStatsArgs& a, cudaStream_t s) {
  launch_pdl(k_row_stats, dim3(a.R), dim3(RS_THREADS), 0, s, a);
}

void launch_plan_draft(const StepState& st, int j, int spb, RowDesc* rows, cudaStream_t s) {
  const int n = st.B * st.k + (j == 1 ? st.B : 0);
  launch_pdl(k_plan_draft, dim3((n + 127) / 128), dim3(128), 0, s, st, j, spb, rows);
}

void launch_plan_verify(const StepState& st, RowDesc* rows, cudaStream_t s) {
  const int n = st.B * st.k * (st.d + 1);
  launch_pdl(k_plan_verify, dim3((n + 127) / 128), dim3(128), 0, s, st, rows);
}

void launch_plan_s1_draft(const StepState& st, int j, RowDesc* rows, cudaStream_t s) {
  const int n = j == 1 ? 2 * st.B : st.B;
  launch_pdl(k_plan_s1_draft, dim3((n + 127) / 128), dim3(128), 0, s, st, j, rows);
}

void launch_plan_s1_verify(const StepState& st, RowDesc* rows, cudaStream_t s) {
  const int n = st.B * (st.d + 2);
  launch_pdl(k_plan_s1_verify, dim3((n + 127) / 128), dim3(128), 0, s, st, rows);
}

void launch_select_s1(const StepState& st, KvStore tkv, KvStore dkv, const float* ss,
                      const float* hw, int norm_D, int ld_ss, float norm_eps, cudaStream_t s) {
  launch_pdl(k_select_s1, dim3(st.B), dim3(32), 0, s, st, tkv, dkv, ss, hw, norm_D, ld_ss,
             norm_eps);
}

void launch_select(const StepState& st, KvStore tkv, KvStore dkv, int commit, cudaStream_t s) {
  launch_pdl(k_select, dim3(st.B), dim3(32), 0, s, st, tkv, dkv, commit);
}

void launch_commit_kv(const StepState& st, KvStore kv, int spb, int is_draft, cudaStream_t s) {
  dim3 grid(st.B, kv.n_layers, 2);
  launch_pdl(k_commit_kv, grid, dim3(256), 0, s, st, kv, spb, is_draft);
}

void launch_advance(const StepState& st, cudaStream_t s) {
  launch_pdl(k_advance, dim3(st.B), dim3(32), 0, s, st);
}

void launch_rope_table(float2* table, int n_pos, int hd, float theta, cudaStream_t s) {
  const int n = n_pos * (hd / 2);
  k_rope_table<<<(n + 255) / 256, 256, 0, s>>>(table, n_pos, hd, (double)theta);
}

}  // namespace cdsl
