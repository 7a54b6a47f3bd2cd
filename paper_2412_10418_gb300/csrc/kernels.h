// kernels.h -- host launchers of the CDSL step kernels (declarations).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "gemm.cuh"

namespace cdsl {

// Per-prompt decoding state on the device (all pointers into the workspace).
struct StepState {
  int32_t B, k, d, nk, max_new, lcap, n_min, reward_head;
  float r_t;
  int32_t acceptance;  // 0 hard rejection, 1 speculative sampling
  uint32_t seed;       // SplitMix64 seed of the speculative-sampling draws
  int32_t step1;       // Step-1 budget b (0, 1 or 2)
  int32_t s1_dbase;    // Step-1 round 2: first draft tail slot of its region (d+1 per prompt)
  int32_t s1_tbase;    //   and first target tail slot (d+2 per prompt)
  int32_t* len;        // [B] committed prefix length L (target; draft up to the pending row)
  int32_t* pend;       // [B] 1: the draft still lacks the KV of token L-1
  int32_t* gen;        // [B] tokens generated (len(T))
  int32_t* tokens;     // [B, lcap]
  int32_t* roots;      // [B, k]
  int32_t* kw;         // [B, nk]
  uint32_t* cov;       // [B] keyword bits already covered by T
  int32_t* x;          // [B, k, d] drafted tokens
  float* logq;         // [B, k, d]
  int32_t* v_amax;     // [B*k*(d+1)] verify row argmax
  float* v_logp;       // [B, k, d] log p_j(x_j)
  int32_t* v_topk;     // [B*k*(d+1), k]
  float* v_head;       // [B*k*(d+1)] sigmoid(w . h)
  int32_t* n_acc;      // [B, k]
  float* reward;       // [B, k, 2]
  int32_t* beam;       // [B]
  int32_t* state;      // [B]
  int32_t* emitted;    // [B, d+1]
  int32_t* n_emit;     // [B]
  int32_t* next_page;  // [2] bump allocators (target, draft)
  int32_t* status;     // device status word
  long long* counters; // [8]
  // Step-1 round 2 (budget b = 2): x' = argmax M_p(pfx + c_1), its d-token M_q lookahead
  int32_t* s1_need;    // [B] 1: round 1 failed in S2/S3 and round 2 decides the step
  int32_t* s1_tok;     // [B, d+1] x', lh_1..lh_d
  float* s1_logq;      // [B, d+1] log q of lh_1..lh_d (index 1..d)
  float* s1_reward;    // [B] R(T + c_1 + x' + lh)
  int32_t* s1_topk;    // [B, k] top-k of M_p(pfx + c_1 + x')
  int32_t* s1_used;    // [B] 1: c_1, x' were emitted (K/V from the round's tails)
};

// elementwise / row kernels (T = float or __nv_bfloat16, the model dtype)
// h = E[token]; x = h . g in the GEMM-input format; ss = 32-feature partial sums of h^2
void launch_embed(int dtype, const RowDesc* rows, int R, const void* embed, int D, float* h,
                  void* x, size_t plane, const void* g, float* ss, int ld_ss, cudaStream_t s);
// out: GEMM-input activations (store_act format, hi/lo planes `plane` elements apart)
void launch_rmsnorm(int dtype, const float* h, int R, int D, const void* gain, float eps,
                    void* out, size_t plane, const int32_t* gather, const float* head_w,
                    float* head_out, cudaStream_t s);
// Attention of a pass (attention.cu). Chunks 0 .. n_chunks-1 hold attn_chunk() prefix
// positions each, the n_tchunks after them the query blocks' beam tails (n_chunks + n_tchunks
// <= attn_max_chunks()). Grid: (cluster of up to 16 blocks over the chunks, kv head, z) with
// z -> (prompt, query block of `qblock` query vectors: attn_qblock_for(), or attn_qblock()
// with a zmap) either dense (b = z / qb_count) or from zmap[2z], zmap[2z+1]. More tail keys
// than the tail chunks hold latch CDSL_ERANGE in *status.
struct AttnArgs {
  const float* q; int32_t n_heads, G;
  KvStore kv; int32_t layer;
  const RowDesc* rows; int32_t R;
  void* out; size_t plane; float scale;
  int32_t n_chunks, n_tchunks, qb_count, qblock;
  const int32_t* zmap;
  int32_t* status;
  unsigned long long* stamp;   // in-graph launch timing record (LaunchStamp), or nullptr
  uint64_t wait_ns;            // limit of the tensor-core kernel's MMA waits (nanoseconds)
};
int attn_chunk();
int attn_max_chunks();
int attn_qblock();
// Query vectors per block of a dense pass with rows_per_prompt rows per prompt, GQA group G.
int attn_qblock_for(int rows_per_prompt, int G);
// Tail chunks a pass needs: rows_per_prompt rows per prompt, GQA group G, consecutive runs of
// rows_per_tail rows sharing one beam tail, tails of at most max_tail keys.
int attn_tail_chunks(int rows_per_prompt, int G, int rows_per_tail, int max_tail);
int configure_attention();
void launch_attn(int dtype, const AttnArgs& a, int n_z, cudaStream_t s);
// Tensor-core attention (attention_tc.cu) for dense passes of bf16 models (no zmap): query
// blocks of attn_tc_qblock() vectors (at most 128), head_dim 64 or 128.
int attn_tc_qblock(int rows_per_prompt, int G);
int configure_attention_tc();
void launch_attn_tc(const AttnArgs& a, int n_z, cudaStream_t s);
// Row statistics of logits rows: argmax (lower id on ties), log-sum-exp, top-k, log p.
//   draft mode  (dp1 == 0): x[r*out_stride + out_off] = argmax, logq[...] = log q(argmax)
//   verify mode (dp1 == d+1): amax[r], topk[r, k], logp of the next drafted token
//   roots mode  (topk only): topk of row r written to row dst[r] of topk
struct RowStatsArgs {
  const float* logits; int32_t R, V, k;
  int32_t dp1;                 // d+1 in verify mode, else 0
  const int32_t* next_x;       // verify: drafted tokens [B,k,d]
  int32_t* amax; float* logp;  // verify: [R], [B,k,d]
  int32_t* topk;               // verify / roots: [R or B, k]
  const int32_t* dst;          // roots: destination row per logits row
  int32_t* x_out; float* logq_out; int32_t out_stride, out_off;  // draft
  int32_t* status;
  // verify: reward head sigmoid(w . RMSNorm(h)) from the last layer's partial sums
  const float* ss; const float* hw; int32_t norm_D, ld_ss; float norm_eps; float* head_out;
  unsigned long long* stamp;   // in-graph launch timing record (LaunchStamp), or nullptr
};
void launch_row_stats(const RowStatsArgs& a, cudaStream_t s);

void launch_gemm_simt(int dtype, const GemmArgs& a, cudaStream_t s);

// Weight-streaming GEMM for R <= 8 activation rows (bf16 weights), split-K over `splits`
// slices of k_split elements. Scratch: part [splits][8][tiles][128] floats and one arrival
// counter per tile (zero between launches).
// Clusters of each size (1..16 blocks) that one kernel can keep resident at once
// (cudaOccupancyMaxActiveClusters, queried at configuration; 0 where a size does not fit).
struct ClusterFit {
  int active[17] = {};
};

template <typename Kernel>
void fill_cluster_fit(ClusterFit* f, Kernel kernel, int threads, size_t smem, int max_cluster) {
  for (int c = 1; c <= max_cluster && c <= 16; ++c) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(c, 1, 1);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = c;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    f->active[c] = n;
  }
}

struct GemvPlan { int splits, k_split, tiles; };
constexpr int kPlanSMs = 152;  // GB300: split-K is planned for this many SMs
GemvPlan plan_gemv(int K, int n_virtual, int n_sm);
void launch_gemv(const GemmArgs& a, const GemvPlan& p, float* part, int* tile_cnt, cudaStream_t s);

// Tensor-core GEMM (tcgen05, TMEM, TMA) for bf16 weights and 1..256 activation rows, on a
// persistent stream-K grid of `ctas` blocks. maps: TMA descriptors of the weight segments
// (128-byte swizzle, 64x64 boxes) and of the hi / lo activation planes (64x16 boxes).
// Scratch: part [ctas][2][n_pad][128] floats (tc_scratch_floats), one arrival counter per
// tile (zero between launches). Launched with programmatic dependent launch allowed.
struct TcMaps { CUtensorMap w[3]; CUtensorMap xh, xl; };
// cluster > 0: cluster split-K with that many blocks per tile (ctas = tiles * cluster); 0:
// persistent stream-K over ctas blocks.
// big: the variant for more than 64 activation rows (k_gemm_tc<true>)
struct TcPlan { int tiles, kb_total, ctas, n_pad, stages, ep_rows, cluster, big; size_t smem; };
bool tc_supported(const GemmArgs& a);
// cluster: -1 chooses (split-K clusters when every tile fits at once with >= 2 blocks), 0
// stream-K, > 0 that cluster size.
TcPlan plan_tc(int K, int n_virtual, int R, int n_sm, int force_per_sm = 0, int max_split = 0,
               int cluster = -1);
size_t tc_scratch_floats(const TcPlan& p);
int encode_bf16_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer);
int configure_gemm_tc();
void launch_gemm_tc(const TcMaps& maps, const GemmArgs& a, const TcPlan& p, float* part,
                    int* tile_cnt, cudaStream_t s);

// Message returned by cdsl_last_error(NULL) on this thread.
void set_thread_error(const char* msg);

// plans and the decision
void launch_plan_draft(const StepState& st, int j, int tail_slots_per_beam, RowDesc* rows,
                       cudaStream_t s);
void launch_plan_verify(const StepState& st, RowDesc* rows, cudaStream_t s);
// Step-1 round 2: draft call j (1..d) over [x' (+ c_1 when j = 1)] or lh_j-1, and the target
// pass over [x', c_1, lh_1..lh_d] of every prompt
void launch_plan_s1_draft(const StepState& st, int j, RowDesc* rows, cudaStream_t s);
void launch_plan_s1_verify(const StepState& st, RowDesc* rows, cudaStream_t s);
// commit = 0: decide only (n_b, rewards, b*, state, emission); 1: also allocate KV pages
void launch_select(const StepState& st, KvStore tkv, KvStore dkv, int commit, cudaStream_t s);
// Step-1 round 2's decision: R(T + c_1 + x' + lh) >= r_t emits c_1, x' (state 3). ss / hw:
// the target pass's final-norm and reward-head partial sums (ld_ss rows apart).
void launch_select_s1(const StepState& st, KvStore tkv, KvStore dkv, const float* ss,
                      const float* hw, int norm_D, int ld_ss, float norm_eps, cudaStream_t s);
void launch_commit_kv(const StepState& st, KvStore kv, int slots_per_beam, int is_draft,
                      cudaStream_t s);
void launch_advance(const StepState& st, cudaStream_t s);
void launch_rope_table(float2* table, int n_pos, int hd, float theta, cudaStream_t s);

}  // namespace cdsl
