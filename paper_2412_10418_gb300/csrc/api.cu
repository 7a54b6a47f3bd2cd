// api.cu -- the C ABI of include/cdsl.h: context, workspace layout, forward passes of the
// draft and target models, and the CDSL-k step (lookahead, verify, select) on one stream.
#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <map>
#include <tuple>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "kernels.h"

using namespace cdsl;

namespace {

thread_local std::string g_init_error;

enum Phase { PH_NEW = 0, PH_READY = 1, PH_LOOKED = 2, PH_VERIFIED = 3 };

struct ModelW {
  cdsl_model_cfg cfg{};
  const void* embed = nullptr;
  const void* final_norm = nullptr;
  const void* lm_head = nullptr;
  std::vector<std::array<const void*, 9>> layers;
  KvStore kv{};
  float2* rope = nullptr;
  int32_t spb = 0;  // tail slots per beam
};

enum { W_ATTN_NORM = 0, W_Q, W_K, W_V, W_O, W_FFN_NORM, W_GATE, W_UP, W_DOWN };

// Bump allocator over the caller's workspace; with base == nullptr it only measures.
struct Carver {
  char* base;
  size_t off = 0;
  explicit Carver(void* b) : base(static_cast<char*>(b)) {}
  template <typename T>
  T* take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

}  // namespace

struct cdsl_ctx {
  cdsl_model_cfg tcfg{}, dcfg{};
  cdsl_run_cfg run{};
  ModelW tgt, dft;
  cudaStream_t stream = nullptr;
  const float* head_w = nullptr;
  int dtype = 0;
  int B = 0, k = 0, d = 0, nk = 0, lcap = 0, lrope = 0, max_pages = 0, page_shift = 0;
  int R_v = 0, R_d = 0, R_p = 0, R_s1 = 0, R_max = 0, R_pad = 0, V = 0;
  int d_max = 0, act_cols = 0, q_cols = 0;
  size_t act_plane = 0;  // elements between hi and lo planes of X1 / X2 (bf16 models)
  // buffers
  float* h = nullptr;
  void* X1 = nullptr;
  void* X2 = nullptr;
  void* Xa = nullptr;           // attention output (input of the O projection)
  float* ss_a = nullptr;        // partial sums of h^2 (RMSNorm row scales), two ping-pong sets
  float* ss_b = nullptr;
  float* ss_hw = nullptr;       // reward-head partial sums
  float* qbuf = nullptr;
  float* logits = nullptr;
  RowDesc* rows_d = nullptr;
  RowDesc* rows_v = nullptr;
  RowDesc* rows_p = nullptr;
  int32_t* lm_gather = nullptr;
  int32_t* lm_dst = nullptr;
  float* gemv_part = nullptr;   // split-K partial tiles of the weight-streaming GEMM
  int32_t* gemv_cnt = nullptr;  // per-tile arrival counters, then per-tile finished shares
  int plan_sms = kPlanSMs;      // SMs the tensor-core GEMM plans for: min(kPlanSMs, device's)
  int32_t* attn_zmap = nullptr; // prefill: z -> (prompt, query block)
  int attn_zmax = 0, attn_chunks = 0;
  StepState st{};
  size_t ws_total = 0;
  int phase = PH_NEW;
  cudaGraphExec_t graph = nullptr;
  long long graph_nodes = 0;
  uint64_t wait_ns = 2000000000ull;   // limit of the tensor-core kernels' pipeline waits
  // kernel timing (cdsl_profile): mode 1 events around direct launches, mode 2 in-graph stamps
  struct ProfRec { int impl; double bytes, flops; size_t ev; };
  int prof_mode = 0;
  bool profiling = false;       // mode 1
  // mode 2: launch records of the stamped graph (LaunchStamp; kStampStride apart)
  unsigned long long* stamps = nullptr;   // [3][kStampStride]
  bool stamping = false;        // capturing the stamped graph
  unsigned long long* cur_stamp = nullptr;   // record of the launch being issued
  cudaGraphExec_t graph_st = nullptr;
  struct StampRec { int impl; double bytes, flops; };
  std::vector<StampRec> st_recs;          // per launch of the stamped step, in stream order
  std::vector<double> st_ms;              // attributed in-graph milliseconds per launch, summed
  std::vector<double> st_kbytes;          // kernel-counted bytes per launch, summed
  int st_steps = 0;
  double st_span_ms = 0;                  // first stamped entry to last stamped exit, summed
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  std::vector<ProfRec> prof;
  // TMA descriptors, built on first use: (base, inner, outer, box_outer) -> map
  std::map<std::tuple<uintptr_t, int, int, int>, CUtensorMap> maps;
  int map_error = 0;
  std::string err;
};

namespace {

int fail(cdsl_ctx* c, int code, const std::string& msg) {
  if (c) c->err = msg; else g_init_error = msg;
  return code;
}

int cuda_check(cdsl_ctx* c, const char* where) {
  if (c && c->map_error) {
    const int m = c->map_error;
    c->map_error = 0;
    return fail(c, CDSL_ECUDA, std::string(where) + ": cuTensorMapEncodeTiled failed (" +
                                   std::to_string(m) + ")");
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess)
    return fail(c, CDSL_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
  return CDSL_OK;
}

int check_model(const cdsl_model_cfg* m, const char* name, std::string* why) {
  char buf[256];
  auto bad = [&](const char* what) {
    snprintf(buf, sizeof buf, "%s config: %s", name, what);
    *why = buf;
    return CDSL_EINVAL;
  };
  if (!m) return bad("NULL");
  if (m->n_layers < 1 || m->n_layers > 512) return bad("n_layers out of range");
  if (m->d_model < 64 || m->d_model % 64) return bad("d_model must be a positive multiple of 64");
  if (m->head_dim != 64 && m->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (m->n_heads < 1 || m->n_kv_heads < 1 || m->n_heads % m->n_kv_heads)
    return bad("n_heads must be a positive multiple of n_kv_heads");
  if (m->n_heads / m->n_kv_heads > 16) return bad("more than 16 query heads per kv head");
  if (m->d_ffn < 8 || m->d_ffn % 8) return bad("d_ffn must be a positive multiple of 8");
  if (m->vocab < 2 || m->vocab % 8 || m->vocab > 32768)
    return bad("vocab must be a multiple of 8, at most 32768");
  if (m->d_model > 8192) return bad("d_model must be at most 8192");
  if (m->dtype != CDSL_DTYPE_F32 && m->dtype != CDSL_DTYPE_BF16) return bad("unknown dtype");
  if (!(m->rope_theta > 0.f) || !(m->norm_eps > 0.f)) return bad("rope_theta and norm_eps must be > 0");
  return CDSL_OK;
}

int check_run(const cdsl_run_cfg* r, int vocab, std::string* why) {
  auto bad = [&](const char* what) { *why = std::string("run config: ") + what; return CDSL_EINVAL; };
  if (!r) return bad("NULL");
  if (r->batch < 1 || r->batch > 4096) return bad("batch out of range");
  if (r->k < 1 || r->k > 16 || r->k > vocab) return bad("k must be in 1..16");
  if (r->d < 1 || r->d > 16) return bad("d must be in 1..16");
  if (r->max_prompt < 1 || r->max_new < 1) return bad("max_prompt and max_new must be >= 1");
  if ((long long)r->max_prompt + r->max_new > (long long)(attn_max_chunks() - 1) * attn_chunk())
    return bad("max_prompt + max_new exceeds the attention limit (8128 positions)");
  if (r->n_keywords < 1 || r->n_keywords > 32) return bad("n_keywords must be in 1..32");
  const int ps = r->page_size ? r->page_size : 64;
  if (ps < 16 || ps > 256 || (ps & (ps - 1))) return bad("page_size must be a power of two in 16..256");
  if (r->max_chunk < 0) return bad("max_chunk must be >= 0");
  if (r->acceptance != 0 && r->acceptance != 1)
    return bad("acceptance must be 0 (hard rejection) or 1 (speculative sampling)");
  if (r->step1_budget < 0 || r->step1_budget > 2) return bad("step1_budget must be 0, 1 or 2");
  return CDSL_OK;
}

int group_size(const cdsl_model_cfg& m) { return m.n_heads / m.n_kv_heads; }
int prefix_chunks(const cdsl_run_cfg& r) {
  return (r.max_prompt + r.max_new + attn_chunk() - 1) / attn_chunk();
}
// Tail-key chunks of the Step-1 round's passes (budget 2): the target's d+2 rows per prompt
// and the draft's (at most 2 rows, d+1 tail slots).
int s1_tail_chunks_t(const cdsl_model_cfg& t, const cdsl_run_cfg& r) {
  return attn_tail_chunks(r.d + 2, group_size(t), r.d + 2, r.d + 2);
}
int s1_tail_chunks_d(const cdsl_model_cfg& dr, const cdsl_run_cfg& r, int j) {
  const int rows = j == 1 ? 2 : 1;
  return attn_tail_chunks(rows, group_size(dr), rows, j + 1);
}
// Most tail-key chunks of any pass: the verify rows of the target, the draft rollout rows
// (and the Step-1 round's passes).
int tail_chunks_max(const cdsl_model_cfg& t, const cdsl_model_cfg& dr, const cdsl_run_cfg& r) {
  int m = std::max(attn_tail_chunks(r.k * (r.d + 1), group_size(t), r.d + 1, r.d + 1),
                   attn_tail_chunks(r.k + 1, group_size(dr), 1, r.d));
  if (r.step1_budget >= 2) {
    m = std::max(m, s1_tail_chunks_t(t, r));
    for (int j = 1; j <= r.d; ++j) m = std::max(m, s1_tail_chunks_d(dr, r, j));
  }
  return m;
}

// Sizes derived from the configurations (shared by cdsl_workspace_size and cdsl_init).
void derive_dims(cdsl_ctx* c) {
  const cdsl_run_cfg& r = c->run;
  c->dtype = c->tcfg.dtype;
  c->B = r.batch; c->k = r.k; c->d = r.d; c->nk = r.n_keywords;
  c->V = c->tcfg.vocab;
  c->lcap = r.max_prompt + r.max_new + 1;
  c->lrope = r.max_prompt + r.max_new + r.d + 2;
  const int ps = r.page_size ? r.page_size : 64;
  c->page_shift = 0;
  while ((1 << c->page_shift) < ps) ++c->page_shift;
  c->max_pages = (c->lcap + ps - 1) / ps;
  c->R_v = c->B * c->k * (c->d + 1);
  c->R_d = c->B * c->k + c->B;
  // Step-1 round 2: the target pass holds d+2 rows per prompt (draft calls fit in R_d)
  c->R_s1 = r.step1_budget >= 2 ? c->B * (c->d + 2) : 0;
  // default 256 prefill rows (the most the tensor-core GEMM takes): the large-row GEMM then
  // streams each weight once per 256 prompt tokens (measured, 512-token 7B prefill: 43 ms at
  // 64 rows, 35 at 128, 33 at 256; 13B, 4 x 1024 tokens: 564, 464, 428 ms)
  const int chunk = r.max_chunk ? r.max_chunk : 256;
  c->R_p = std::min(chunk, c->B * r.max_prompt);
  c->R_max = std::max(std::max(c->R_v, c->R_s1), std::max(c->R_d, c->R_p));
  c->R_pad = (c->R_max + 31) / 32 * 32;
  c->d_max = std::max(c->tcfg.d_model, c->dcfg.d_model);
  c->q_cols = std::max(c->tcfg.n_heads * c->tcfg.head_dim, c->dcfg.n_heads * c->dcfg.head_dim);
  c->act_cols = std::max(std::max(c->d_max, c->q_cols), std::max(c->tcfg.d_ffn, c->dcfg.d_ffn));
}

KvStore make_kv(const cdsl_model_cfg& m, cdsl_ctx* c, int slots) {
  KvStore s{};
  s.n_pages = c->B * c->max_pages;
  s.page_shift = c->page_shift;
  s.max_pages = c->max_pages;
  s.kvh = m.n_kv_heads;
  s.hd = m.head_dim;
  s.n_tail_slots = slots;
  s.n_layers = m.n_layers;
  return s;
}

// Carve every buffer; returns total bytes. With base == nullptr only the size is computed.
size_t carve(cdsl_ctx* c, void* base) {
  Carver cv(base);
  const int B = c->B, k = c->k, d = c->d;
  auto model_kv = [&](ModelW& m, const cdsl_model_cfg& cfg, int spb, int extra) {
    const int slots = B * k * spb + extra;
    m.kv = make_kv(cfg, c, slots);
    const size_t per_page = (size_t)2 * cfg.n_kv_heads * ((size_t)1 << c->page_shift) * cfg.head_dim;
    m.kv.pool = cv.take<float>((size_t)cfg.n_layers * m.kv.n_pages * per_page);
    m.kv.tail = cv.take<float>((size_t)cfg.n_layers * 2 * slots * cfg.n_kv_heads * cfg.head_dim);
    m.kv.page_table = cv.take<int32_t>((size_t)B * c->max_pages);
    m.rope = cv.take<float2>((size_t)c->lrope * (cfg.head_dim / 2));
    m.spb = spb;
  };
  // per beam: target d+1 verify rows, draft d rollout rows; the Step-1 round (budget 2) adds
  // d+2 target and d+1 draft slots per prompt after them
  const bool s1 = c->run.step1_budget >= 2;
  model_kv(c->tgt, c->tcfg, d + 1, s1 ? B * (d + 2) : 0);
  model_kv(c->dft, c->dcfg, d, s1 ? B * (d + 1) : 0);
  c->h = cv.take<float>((size_t)c->R_pad * c->d_max);
  // GEMM inputs: one fp32 plane, or hi/lo bf16 planes (4 bytes per element either way)
  c->act_plane = (size_t)c->R_pad * c->act_cols;
  c->X1 = cv.take<float>(c->act_plane);
  c->X2 = cv.take<float>(c->act_plane);
  c->Xa = cv.take<float>(c->act_plane);
  const size_t ss_n = (size_t)(c->d_max / 32) * c->R_pad;
  c->ss_a = cv.take<float>(ss_n);
  c->ss_b = cv.take<float>(ss_n);
  c->ss_hw = cv.take<float>(ss_n);
  c->qbuf = cv.take<float>((size_t)c->R_pad * c->q_cols);
  const int lm_rows = std::max(c->R_v, std::max(B * k, B));
  c->logits = cv.take<float>((size_t)lm_rows * c->V);
  c->rows_d = cv.take<RowDesc>(c->R_d);
  c->rows_v = cv.take<RowDesc>(std::max(c->R_v, c->R_s1));
  c->rows_p = cv.take<RowDesc>(c->R_p);
  c->lm_gather = cv.take<int32_t>(c->R_p);
  c->lm_dst = cv.take<int32_t>(c->R_p);
  {  // split-K scratch for the weight-streaming GEMM: the largest projection of either model
    size_t part = 0, tiles = 0;
    for (const cdsl_model_cfg* m : {&c->tcfg, &c->dcfg}) {
      const int D = m->d_model, QH = m->n_heads * m->head_dim, KVH = m->n_kv_heads * m->head_dim;
      const int shapes[5][2] = {{D, QH + 2 * KVH}, {QH, D}, {D, (m->d_ffn + 63) / 64 * 128},
                                {m->d_ffn, D}, {D, m->vocab}};
      for (const auto& sh : shapes) {
        const GemvPlan p = plan_gemv(sh[0], sh[1], kPlanSMs);
        part = std::max(part, (size_t)p.splits * 8 * p.tiles * 128);
        tiles = std::max(tiles, (size_t)p.tiles);
        if (c->dtype == CDSL_DTYPE_BF16 && sh[0] % 64 == 0) {
          for (int R = 9; R <= std::min(c->R_max, 256); R += 16) {  // every n_pad in use
            // the plan, and stream-K, which a plan falls back to where clusters do not fit
            const TcPlan t = plan_tc(sh[0], sh[1], R, kPlanSMs);
            const TcPlan sk = plan_tc(sh[0], sh[1], R, kPlanSMs, 0, 0, 0);
            part = std::max(part, std::max(tc_scratch_floats(t), tc_scratch_floats(sk)));
            tiles = std::max(tiles, (size_t)t.tiles);
          }
        }
      }
    }
    c->gemv_part = cv.take<float>(part);
    c->gemv_cnt = cv.take<int32_t>(2 * tiles);
  }
  {  // attention: the prefill's (prompt, query block) map
    const int QB = attn_qblock();
    const int G = std::max(group_size(c->tcfg), group_size(c->dcfg));
    auto qbs = [&](int rows) { return (rows * G + QB - 1) / QB; };
    c->attn_zmax = qbs(c->R_p) + B;   // dense passes need no map
    c->attn_chunks = prefix_chunks(c->run);
    c->attn_zmap = cv.take<int32_t>((size_t)2 * c->attn_zmax);
  }
  StepState& s = c->st;
  s.B = B; s.k = k; s.d = d; s.nk = c->nk; s.max_new = c->run.max_new; s.lcap = c->lcap;
  s.reward_head = c->run.reward_head;
  s.r_t = c->run.r_t;
  s.acceptance = c->run.acceptance;
  s.seed = c->run.seed;
  s.step1 = c->run.step1_budget;
  s.s1_tbase = B * k * (d + 1);
  s.s1_dbase = B * k * d;
  s.n_min = d + 1;
  for (int n = 0; n <= d; ++n)
    if ((float)n / (float)d >= c->run.a_t) { s.n_min = n; break; }
  s.len = cv.take<int32_t>(B);
  s.pend = cv.take<int32_t>(B);
  s.gen = cv.take<int32_t>(B);
  s.tokens = cv.take<int32_t>((size_t)B * c->lcap);
  s.roots = cv.take<int32_t>((size_t)B * k);
  s.kw = cv.take<int32_t>((size_t)B * c->nk);
  s.cov = cv.take<uint32_t>(B);
  s.x = cv.take<int32_t>((size_t)B * k * d);
  s.logq = cv.take<float>((size_t)B * k * d);
  s.v_amax = cv.take<int32_t>(c->R_v);
  s.v_logp = cv.take<float>((size_t)B * k * d);
  s.v_topk = cv.take<int32_t>((size_t)c->R_v * k);
  s.v_head = cv.take<float>(c->R_v);
  s.n_acc = cv.take<int32_t>((size_t)B * k);
  s.reward = cv.take<float>((size_t)B * k * 2);
  s.beam = cv.take<int32_t>(B);
  s.state = cv.take<int32_t>(B);
  s.emitted = cv.take<int32_t>((size_t)B * (d + 1));
  s.n_emit = cv.take<int32_t>(B);
  s.next_page = cv.take<int32_t>(2);
  s.status = cv.take<int32_t>(1);
  s.counters = cv.take<long long>(8);
  s.s1_need = cv.take<int32_t>(B);
  s.s1_tok = cv.take<int32_t>((size_t)B * (d + 1));
  s.s1_logq = cv.take<float>((size_t)B * (d + 1));
  s.s1_reward = cv.take<float>(B);
  s.s1_topk = cv.take<int32_t>((size_t)B * k);
  s.s1_used = cv.take<int32_t>(B);
  c->stamps = cv.take<unsigned long long>((size_t)3 * kStampStride);
  return (cv.off + 255) & ~size_t(255);
}

const CUtensorMap& tensor_map(cdsl_ctx* c, const void* base, int inner, int outer, int box_outer);

// Algorithmic bytes of one projection GEMM: every weight once, the activations read once
// (4 bytes per element: fp32, or bf16 hi + lo), the outputs written once (read-modify-write
// for the residual add).
double gemm_bytes(const cdsl_ctx* c, const GemmArgs& a, double* flops) {
  const double wsz = c->dtype == CDSL_DTYPE_BF16 ? 2.0 : 4.0;
  double rows = 0;
  for (int s = 0; s < a.n_seg; ++s) rows += a.seg_rows[s];
  *flops = 2.0 * a.R * rows * a.K;
  double out = 0;
  switch (a.mode) {
    case EPI_STORE: out = 4.0 * a.R * rows; break;
    case EPI_RESID: out = (a.next_x ? 12.0 : 8.0) * a.R * rows; break;   // h r/w (+ next input)
    case EPI_SWIGLU: out = 4.0 * a.R * a.d_ffn; break;
    case EPI_QKV: out = 4.0 * a.R * rows; break;
  }
  return rows * a.K * wsz + 4.0 * a.R * a.K + out;
}

// Kernel timing (cdsl_profile): bracket one launch of class `cls` with CUDA events.
enum { K_GEMM_SIMT = 0, K_GEMV = 1, K_GEMM_TC = 2, K_ATTN = 3, K_NORM = 4, K_ROWSTATS = 5,
       K_EMBED = 6, K_STEPLOGIC = 7, K_CLASSES = 8 };

template <typename F>
void timed(cdsl_ctx* c, int cls, double bytes, double flops, F&& launch) {
  if (c->stamping) {   // capturing the stamped graph: give the launch its record
    const size_t i = c->st_recs.size();
    c->cur_stamp = i < (size_t)kStampStride ? c->stamps + i : nullptr;
    c->st_recs.push_back({cls, bytes, flops});
    launch();
    c->cur_stamp = nullptr;
    return;
  }
  if (!c->profiling) {
    launch();
    return;
  }
  while (c->ev_pool.size() < c->ev_used + 2) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    c->ev_pool.push_back(e);
  }
  const size_t ev = c->ev_used;
  c->ev_used += 2;
  cudaEventRecord(c->ev_pool[ev], c->stream);
  launch();
  cudaEventRecord(c->ev_pool[ev + 1], c->stream);
  c->prof.push_back({cls, bytes, flops, ev});
}

void gemm(cdsl_ctx* c, const GemmArgs& a) {
  // bf16: the tensor-core kernel for every shape it supports (it streams weights faster than
  // the CUDA-core GEMV even at 4-8 rows); the weight-streaming GEMV otherwise at <= 8 rows;
  // float32 (and anything else): the CUDA-core tiled GEMM.
  const bool bf16 = c->dtype == CDSL_DTYPE_BF16;
  const int impl = (bf16 && tc_supported(a)) ? K_GEMM_TC : (bf16 && a.R <= 8) ? K_GEMV : K_GEMM_SIMT;
  double fl = 0;
  const double by = (c->profiling || c->stamping) ? gemm_bytes(c, a, &fl) : 0.0;
  GemmArgs as = a;   // as launched: with the launch's timing record, if any
  if (impl == K_GEMV) {
    timed(c, impl, by, fl, [&] {
      as.stamp = c->cur_stamp;
      launch_gemv(as, plan_gemv(a.K, a.n_virtual, kPlanSMs), c->gemv_part, c->gemv_cnt, c->stream);
    });
  } else if (impl == K_GEMM_TC) {
    TcMaps maps;
    for (int s = 0; s < 3; ++s) {
      const int seg = s < a.n_seg ? s : 0;
      maps.w[s] = tensor_map(c, a.w[seg], a.K, a.seg_rows[seg], 64);
    }
    const __nv_bfloat16* xb = reinterpret_cast<const __nv_bfloat16*>(a.x);
    const TcPlan p = plan_tc(a.K, a.n_virtual, a.R, c->plan_sms);
    // activation boxes: 64 features x n_pad rows (<= 256 <= R_pad), one per plane and stage
    maps.xh = tensor_map(c, xb, a.ldx, c->R_pad, p.n_pad);
    maps.xl = tensor_map(c, xb + a.x_plane, a.ldx, c->R_pad, p.n_pad);
    timed(c, impl, by, fl, [&] {
      as.stamp = c->cur_stamp;
      launch_gemm_tc(maps, as, p, c->gemv_part, c->gemv_cnt, c->stream);
    });
  } else {
    timed(c, impl, by, fl, [&] {
      as.stamp = c->cur_stamp;
      launch_gemm_simt(c->dtype, as, c->stream);
    });
  }
}

GemmArgs gemm_base(const cdsl_ctx* c, const ModelW& m, int mode, int K, const void* x, int ldx,
                   int R) {
  GemmArgs a{};
  a.mode = mode;
  a.K = K;
  a.x = x;
  a.ldx = ldx;
  a.x_plane = (int64_t)c->act_plane;
  a.act_plane = (int64_t)c->act_plane;
  a.R = R;
  a.n_heads = m.cfg.n_heads;
  a.kv = m.kv;
  a.status = c->st.status;
  a.wait_ns = c->wait_ns;
  return a;
}

const CUtensorMap& tensor_map(cdsl_ctx* c, const void* base, int inner, int outer, int box_outer) {
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(base), inner, outer, box_outer);
  auto it = c->maps.find(key);
  if (it != c->maps.end()) return it->second;
  CUtensorMap m;
  std::memset(&m, 0, sizeof m);
  const int e = encode_bf16_map(&m, base, (uint64_t)inner, (uint64_t)outer, 64, (uint32_t)box_outer);
  if (e && !c->map_error) c->map_error = e;
  return c->maps.emplace(key, m).first->second;
}

// Query vectors per prompt and KV head from which a dense pass of a bf16 model runs on the
// tensor-core attention (attention_tc.cu) rather than the CUDA-core one (attention.cu). The
// 7B verify pass (80) measured 16.3 us per launch on the former against 20.1 us on the
// latter; decode passes (16-36) stay on the CUDA cores, where a block's 64-key chunk is too
// small for the MMA's 128 rows to pay.
constexpr int kAttnTcMinVectors = 64;

// One forward pass of a model over R rows described by `rows`; for lm_rows > 0 the final
// norm + LM head run over rows gather[i] (or the first lm_rows rows) into logits.
// Attention layout of a pass: rows per prompt (dense z mapping) or a host-built z map.
struct AttnPass {
  int rows_per_prompt = 0;            // dense: z = b * qb_count + qb
  const std::vector<int32_t>* zmap = nullptr;  // prefill: (b, qb) pairs for this model
  int n_chunks = 0;
  int n_tchunks = 0;                  // tail-key chunks (attn_tail_chunks)
};

// One forward pass of a model over R rows described by `rows`; for lm_rows > 0 the final
// norm + LM head run over rows gather[i] (or the first lm_rows rows) into logits. RMSNorm is
// folded into the GEMMs (the residual epilogues write h . g_next and the partial sums of h^2,
// the consumers scale by the row factor); only a gathered LM input is normalized by a kernel.
// With want_head, the last layer also leaves the reward-head partials in c->ss_hw.
void forward(cdsl_ctx* c, ModelW& m, const RowDesc* rows, int R, int lm_rows,
             const int32_t* gather, float* logits, bool want_head, const AttnPass& ap) {
  const cdsl_model_cfg& cfg = m.cfg;
  const int D = cfg.d_model, hd = cfg.head_dim, H = cfg.n_heads, KVH = cfg.n_kv_heads;
  const int F = cfg.d_ffn, L = cfg.n_layers;
  cudaStream_t s = c->stream;
  AttnArgs at{};
  at.q = c->qbuf; at.n_heads = H; at.G = H / KVH; at.kv = m.kv; at.rows = rows; at.R = R;
  at.out = c->Xa; at.plane = c->act_plane; at.scale = 1.0f / sqrtf((float)hd);
  at.n_chunks = ap.n_chunks ? ap.n_chunks : c->attn_chunks;
  at.n_tchunks = ap.n_tchunks;
  at.status = c->st.status;
  at.wait_ns = c->wait_ns;
  int n_z;
  // dense passes of bf16 models with many query vectors per KV head on the tensor-core
  // attention (kAttnTcMinVectors)
  const bool attn_tc = c->dtype == CDSL_DTYPE_BF16 && !ap.zmap &&
                       ap.rows_per_prompt * (H / KVH) >= kAttnTcMinVectors;
  if (attn_tc) {
    at.qblock = attn_tc_qblock(ap.rows_per_prompt, at.G);
    at.qb_count = (ap.rows_per_prompt * at.G + at.qblock - 1) / at.qblock;
    n_z = c->B * at.qb_count;
  } else if (ap.zmap) {
    n_z = (int)ap.zmap->size() / 2;
    at.zmap = c->attn_zmap;
    at.qblock = attn_qblock();
    cudaMemcpyAsync(c->attn_zmap, ap.zmap->data(), ap.zmap->size() * 4, cudaMemcpyHostToDevice, s);
  } else {
    at.qblock = attn_qblock_for(ap.rows_per_prompt, at.G);
    at.qb_count = (ap.rows_per_prompt * at.G + at.qblock - 1) / at.qblock;
    n_z = c->B * at.qb_count;
  }
  const int ld_ss = c->R_pad;
  auto normed_input = [&](GemmArgs& a, const float* ss) {
    a.in_ss = ss; a.norm_D = D; a.ld_ss = ld_ss; a.norm_eps = cfg.norm_eps;
  };
  auto residual_out = [&](GemmArgs& a, const void* g_next, float* ss_out, bool head) {
    a.out_f32 = c->h; a.ld_out = D;
    a.next_x = c->X1; a.next_g = g_next; a.out_ss = ss_out; a.ld_ss = ld_ss;
    if (head) { a.head_w = c->head_w; a.out_hw = c->ss_hw; }
  };
  timed(c, K_EMBED, 0, 0, [&] {
    launch_embed(c->dtype, rows, R, m.embed, D, c->h, c->X1, c->act_plane,
                 m.layers[0][W_ATTN_NORM], c->ss_a, ld_ss, s);
  });
  for (int l = 0; l < L; ++l) {
    const auto& W = m.layers[l];
    GemmArgs q = gemm_base(c, m, EPI_QKV, D, c->X1, D, R);
    q.w[0] = W[W_Q]; q.w[1] = W[W_K]; q.w[2] = W[W_V];
    q.seg_rows[0] = H * hd; q.seg_rows[1] = KVH * hd; q.seg_rows[2] = KVH * hd;
    q.n_seg = 3;
    q.n_virtual = (H + 2 * KVH) * hd;
    q.q_out = c->qbuf;
    q.layer = l;
    q.rows = rows;
    q.rope = m.rope;
    normed_input(q, c->ss_a);
    gemm(c, q);
    at.layer = l;
    timed(c, K_ATTN, 0, 0, [&] {
      at.stamp = c->cur_stamp;
      if (attn_tc) launch_attn_tc(at, n_z, s);
      else launch_attn(c->dtype, at, n_z, s);
      at.stamp = nullptr;
    });
    GemmArgs o = gemm_base(c, m, EPI_RESID, H * hd, c->Xa, H * hd, R);
    o.w[0] = W[W_O]; o.seg_rows[0] = D; o.n_seg = 1; o.n_virtual = D;
    residual_out(o, W[W_FFN_NORM], c->ss_b, false);
    gemm(c, o);
    GemmArgs g = gemm_base(c, m, EPI_SWIGLU, D, c->X1, D, R);
    g.w[0] = W[W_GATE]; g.w[1] = W[W_UP]; g.seg_rows[0] = F; g.seg_rows[1] = F; g.n_seg = 2;
    g.n_virtual = (F + 63) / 64 * 128;
    g.d_ffn = F;
    g.out_act = c->X2; g.ld_act = F;
    normed_input(g, c->ss_b);
    gemm(c, g);
    GemmArgs dn = gemm_base(c, m, EPI_RESID, F, c->X2, F, R);
    dn.w[0] = W[W_DOWN]; dn.seg_rows[0] = D; dn.n_seg = 1; dn.n_virtual = D;
    const bool last = l + 1 == L;
    residual_out(dn, last ? m.final_norm : m.layers[l + 1][W_ATTN_NORM], c->ss_a,
                 last && want_head && c->head_w);
    gemm(c, dn);
  }
  if (lm_rows > 0) {
    GemmArgs lm = gemm_base(c, m, EPI_STORE, D, c->X1, D, lm_rows);
    lm.w[0] = m.lm_head; lm.seg_rows[0] = cfg.vocab; lm.n_seg = 1; lm.n_virtual = cfg.vocab;
    lm.out_f32 = logits; lm.ld_out = cfg.vocab;
    if (gather) {   // prefill: normalize the gathered rows explicitly
      timed(c, K_NORM, 0, 0, [&] {
        launch_rmsnorm(c->dtype, c->h, lm_rows, D, m.final_norm, cfg.norm_eps, c->X1,
                       c->act_plane, gather, nullptr, nullptr, s);
      });
    } else {
      normed_input(lm, c->ss_a);
    }
    gemm(c, lm);
  }
}

void do_lookahead(cdsl_ctx* c) {
  for (int j = 1; j <= c->d; ++j) {
    timed(c, K_STEPLOGIC, 0, 0, [&] { launch_plan_draft(c->st, j, c->dft.spb, c->rows_d, c->stream); });
    const int R = c->B * c->k + (j == 1 ? c->B : 0);
    AttnPass ap;
    ap.rows_per_prompt = c->k + (j == 1 ? 1 : 0);
    ap.n_tchunks = attn_tail_chunks(ap.rows_per_prompt, group_size(c->dcfg), 1, j);
    forward(c, c->dft, c->rows_d, R, c->B * c->k, nullptr, c->logits, false, ap);
    RowStatsArgs a{};
    a.logits = c->logits; a.R = c->B * c->k; a.V = c->V; a.k = c->k;
    a.x_out = c->st.x; a.logq_out = c->st.logq; a.out_stride = c->d; a.out_off = j - 1;
    a.status = c->st.status;
    timed(c, K_ROWSTATS, 0, 0, [&] {
      a.stamp = c->cur_stamp;
      launch_row_stats(a, c->stream);
    });
  }
}

void do_verify(cdsl_ctx* c) {
  timed(c, K_STEPLOGIC, 0, 0, [&] { launch_plan_verify(c->st, c->rows_v, c->stream); });
  AttnPass ap;
  ap.rows_per_prompt = c->k * (c->d + 1);
  ap.n_tchunks = attn_tail_chunks(ap.rows_per_prompt, group_size(c->tcfg), c->d + 1, c->d + 1);
  forward(c, c->tgt, c->rows_v, c->R_v, c->R_v, nullptr, c->logits, c->run.reward_head != 0, ap);
  RowStatsArgs a{};
  a.logits = c->logits; a.R = c->R_v; a.V = c->V; a.k = c->k; a.dp1 = c->d + 1;
  a.next_x = c->st.x; a.amax = c->st.v_amax; a.logp = c->st.v_logp; a.topk = c->st.v_topk;
  a.status = c->st.status;
  if (c->run.reward_head) {
    a.ss = c->ss_a; a.hw = c->ss_hw; a.norm_D = c->tcfg.d_model; a.ld_ss = c->R_pad;
    a.norm_eps = c->tcfg.norm_eps; a.head_out = c->st.v_head;
  }
  timed(c, K_ROWSTATS, 0, 0, [&] {
      a.stamp = c->cur_stamp;
      launch_row_stats(a, c->stream);
    });
}

// Step-1 round 2 (Alg. 1 S2/S3, budget b = 2) for every prompt: d draft calls from
// pfx + c_1 + x' and one target pass over [x', c_1, lh_1..lh_d]; k_select_s1 then keeps the
// Step-2 emission or replaces it with c_1, x'. The round's work is the same every step (the
// graph is static); only prompts whose round 1 failed in S2/S3 use its result.
void do_step1_round(cdsl_ctx* c) {
  const int B = c->B, d = c->d;
  for (int j = 1; j <= d; ++j) {
    timed(c, K_STEPLOGIC, 0, 0, [&] { launch_plan_s1_draft(c->st, j, c->rows_d, c->stream); });
    AttnPass ap;
    ap.rows_per_prompt = j == 1 ? 2 : 1;
    ap.n_tchunks = s1_tail_chunks_d(c->dcfg, c->run, j);
    forward(c, c->dft, c->rows_d, ap.rows_per_prompt * B, B, nullptr, c->logits, false, ap);
    RowStatsArgs a{};
    a.logits = c->logits; a.R = B; a.V = c->V; a.k = c->k;
    a.x_out = c->st.s1_tok; a.logq_out = c->st.s1_logq; a.out_stride = d + 1; a.out_off = j;
    a.status = c->st.status;
    timed(c, K_ROWSTATS, 0, 0, [&] {
      a.stamp = c->cur_stamp;
      launch_row_stats(a, c->stream);
    });
  }
  timed(c, K_STEPLOGIC, 0, 0, [&] { launch_plan_s1_verify(c->st, c->rows_v, c->stream); });
  AttnPass ap;
  ap.rows_per_prompt = d + 2;
  ap.n_tchunks = s1_tail_chunks_t(c->tcfg, c->run);
  forward(c, c->tgt, c->rows_v, c->R_s1, B, nullptr, c->logits, c->run.reward_head != 0, ap);
  RowStatsArgs a{};
  a.logits = c->logits; a.R = B; a.V = c->V; a.k = c->k;
  a.topk = c->st.s1_topk; a.status = c->st.status;
  timed(c, K_ROWSTATS, 0, 0, [&] {
      a.stamp = c->cur_stamp;
      launch_row_stats(a, c->stream);
    });
  timed(c, K_STEPLOGIC, 0, 0, [&] {
    launch_select_s1(c->st, c->tgt.kv, c->dft.kv, c->ss_a, c->ss_hw, c->tcfg.d_model, c->R_pad,
                     c->tcfg.norm_eps, c->stream);
  });
}

void do_select(cdsl_ctx* c) {
  timed(c, K_STEPLOGIC, 0, 0, [&] { launch_select(c->st, c->tgt.kv, c->dft.kv, 1, c->stream); });
  if (c->run.step1_budget >= 2) do_step1_round(c);
  timed(c, K_STEPLOGIC, 0, 0, [&] {
    launch_commit_kv(c->st, c->tgt.kv, c->tgt.spb, 0, c->stream);
    launch_commit_kv(c->st, c->dft.kv, c->dft.spb, 1, c->stream);
    launch_advance(c->st, c->stream);
  });
}

void copy_out(cdsl_ctx* c, void* dst, const void* src, size_t bytes) {
  if (dst) cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, c->stream);
}

void copy_select_outputs(cdsl_ctx* c, int32_t* beam, int32_t* state, int32_t* emitted,
                         int32_t* n_emitted, float* reward) {
  const size_t B = c->B;
  copy_out(c, beam, c->st.beam, B * 4);
  copy_out(c, state, c->st.state, B * 4);
  copy_out(c, emitted, c->st.emitted, B * (c->d + 1) * 4);
  copy_out(c, n_emitted, c->st.n_emit, B * 4);
  copy_out(c, reward, c->st.reward, B * c->k * 2 * 4);
}

int bind_model(ModelW& m, const cdsl_model_cfg& cfg, const void* const* w, const char* name,
               std::string* why) {
  const int n = cdsl_num_weights(&cfg);
  for (int i = 0; i < n; ++i) {
    if (!w[i] || (reinterpret_cast<uintptr_t>(w[i]) & 15)) {
      char buf[160];
      snprintf(buf, sizeof buf, "%s weight %d is NULL or not 16-byte aligned", name, i);
      *why = buf;
      return CDSL_EINVAL;
    }
  }
  m.cfg = cfg;
  m.embed = w[0];
  m.layers.resize(cfg.n_layers);
  for (int l = 0; l < cfg.n_layers; ++l)
    for (int j = 0; j < 9; ++j) m.layers[l][j] = w[1 + 9 * l + j];
  m.final_norm = w[1 + 9 * cfg.n_layers];
  m.lm_head = w[2 + 9 * cfg.n_layers];
  return CDSL_OK;
}

int validate_all(const cdsl_model_cfg* t, const cdsl_model_cfg* dr, const cdsl_run_cfg* r,
                 std::string* why) {
  int e = check_model(t, "target", why);
  if (e) return e;
  if ((e = check_model(dr, "draft", why))) return e;
  if (t->vocab != dr->vocab) { *why = "target and draft vocabularies differ"; return CDSL_EINVAL; }
  if (t->dtype != dr->dtype) { *why = "target and draft dtypes differ"; return CDSL_EINVAL; }
  if ((e = check_run(r, t->vocab, why))) return e;
  if (prefix_chunks(*r) + tail_chunks_max(*t, *dr, *r) > attn_max_chunks()) {
    *why = "run config: max_prompt + max_new and the beam tails exceed the attention chunks";
    return CDSL_EINVAL;
  }
  return CDSL_OK;
}

}  // namespace

void cdsl::set_thread_error(const char* msg) { g_init_error = msg ? msg : ""; }

extern "C" {

int32_t cdsl_num_weights(const cdsl_model_cfg* cfg) {
  if (!cfg || cfg->n_layers < 1) return -1;
  return 3 + 9 * cfg->n_layers;
}

int32_t cdsl_workspace_size(const cdsl_model_cfg* target, const cdsl_model_cfg* draft,
                            const cdsl_run_cfg* run, size_t* bytes) {
  std::string why;
  int e = validate_all(target, draft, run, &why);
  if (e) return fail(nullptr, e, why);
  if (!bytes) return fail(nullptr, CDSL_EINVAL, "bytes is NULL");
  cdsl_ctx tmp;
  tmp.tcfg = *target; tmp.dcfg = *draft; tmp.run = *run;
  derive_dims(&tmp);
  *bytes = carve(&tmp, nullptr);
  return CDSL_OK;
}

int32_t cdsl_init(const cdsl_model_cfg* target, const void* const* h_target_weights,
                  const cdsl_model_cfg* draft, const void* const* h_draft_weights,
                  const cdsl_run_cfg* run, const float* d_reward_head, void* d_workspace,
                  size_t workspace_bytes, void* stream, cdsl_ctx** out) {
  std::string why;
  int e = validate_all(target, draft, run, &why);
  if (e) return fail(nullptr, e, why);
  if (!out) return fail(nullptr, CDSL_EINVAL, "out is NULL");
  *out = nullptr;
  if (!h_target_weights || !h_draft_weights) return fail(nullptr, CDSL_EINVAL, "weights are NULL");
  if (run->reward_head && !d_reward_head)
    return fail(nullptr, CDSL_EINVAL, "reward_head requested but d_reward_head is NULL");
  if (!d_workspace || (reinterpret_cast<uintptr_t>(d_workspace) & 255))
    return fail(nullptr, CDSL_EINVAL, "workspace is NULL or not 256-byte aligned");
  cdsl_ctx* c = new cdsl_ctx();
  c->tcfg = *target; c->dcfg = *draft; c->run = *run;
  c->head_w = d_reward_head;
  c->stream = static_cast<cudaStream_t>(stream);
  derive_dims(c);
  if ((e = bind_model(c->tgt, *target, h_target_weights, "target", &why)) ||
      (e = bind_model(c->dft, *draft, h_draft_weights, "draft", &why))) {
    delete c;
    return fail(nullptr, e, why);
  }
  c->ws_total = carve(c, nullptr);
  if (workspace_bytes < c->ws_total) {
    char buf[160];
    snprintf(buf, sizeof buf, "workspace has %zu bytes, needs %zu", workspace_bytes, c->ws_total);
    delete c;
    return fail(nullptr, CDSL_ENOMEM, buf);
  }
  carve(c, d_workspace);
  cudaGetLastError();
  if (configure_attention()) {
    delete c;
    return fail(nullptr, CDSL_ECUDA, "cannot configure the attention kernel (shared memory)");
  }
  if (c->dtype == CDSL_DTYPE_BF16 && configure_attention_tc()) {
    delete c;
    return fail(nullptr, CDSL_ECUDA, "cannot configure the tensor-core attention (shared memory)");
  }
  if (c->dtype == CDSL_DTYPE_BF16 && configure_gemm_tc()) {
    delete c;
    return fail(nullptr, CDSL_ECUDA, "cannot configure the tensor-core GEMM (shared memory)");
  }
  {  // the large-row GEMM's stream-K grid must be resident at once (one block per SM)
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && sms > 0)
      c->plan_sms = std::min(kPlanSMs, sms);
  }
  cudaMemsetAsync(d_workspace, 0, c->ws_total, c->stream);
  launch_rope_table(c->tgt.rope, c->lrope, target->head_dim, target->rope_theta, c->stream);
  launch_rope_table(c->dft.rope, c->lrope, draft->head_dim, draft->rope_theta, c->stream);
  if ((e = cuda_check(c, "cdsl_init"))) {
    g_init_error = c->err;
    delete c;
    return e;
  }
  c->phase = PH_NEW;
  *out = c;
  return CDSL_OK;
}

int32_t cdsl_prefill(cdsl_ctx* c, const int32_t* d_prompts, const int32_t* h_prompt_lens,
                     const int32_t* d_keywords) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (!d_prompts || !h_prompt_lens || !d_keywords)
    return fail(c, CDSL_EINVAL, "prompts, prompt lengths and keywords are required");
  const int B = c->B, P = 1 << c->page_shift;
  for (int b = 0; b < B; ++b)
    if (h_prompt_lens[b] < 1 || h_prompt_lens[b] > c->run.max_prompt)
      return fail(c, CDSL_EINVAL, "prompt length out of 1..max_prompt");
  cudaStream_t s = c->stream;
  StepState& st = c->st;
  cudaGetLastError();
  // reset the decoding state
  cudaMemsetAsync(st.tokens, 0xff, sizeof(int32_t) * B * c->lcap, s);
  cudaMemsetAsync(st.pend, 0, sizeof(int32_t) * B, s);
  cudaMemsetAsync(st.gen, 0, sizeof(int32_t) * B, s);
  cudaMemsetAsync(st.cov, 0, sizeof(uint32_t) * B, s);
  cudaMemsetAsync(st.status, 0, sizeof(int32_t), s);
  cudaMemsetAsync(st.counters, 0, sizeof(long long) * 8, s);
  cudaMemcpy2DAsync(st.tokens, sizeof(int32_t) * c->lcap, d_prompts,
                    sizeof(int32_t) * c->run.max_prompt, sizeof(int32_t) * c->run.max_prompt, B,
                    cudaMemcpyDeviceToDevice, s);
  cudaMemcpyAsync(st.len, h_prompt_lens, sizeof(int32_t) * B, cudaMemcpyHostToDevice, s);
  cudaMemcpyAsync(st.kw, d_keywords, sizeof(int32_t) * B * c->nk, cudaMemcpyDeviceToDevice, s);
  // pages for the prompts: contiguous runs handed out in prompt order
  std::vector<int32_t> pt((size_t)B * c->max_pages, -1);
  int next = 0;
  for (int b = 0; b < B; ++b)
    for (int p = 0; p < (h_prompt_lens[b] + P - 1) / P; ++p) pt[(size_t)b * c->max_pages + p] = next++;
  int32_t np[2] = {next, next};
  cudaMemcpyAsync(c->tgt.kv.page_table, pt.data(), pt.size() * 4, cudaMemcpyHostToDevice, s);
  cudaMemcpyAsync(c->dft.kv.page_table, pt.data(), pt.size() * 4, cudaMemcpyHostToDevice, s);
  cudaMemcpyAsync(st.next_page, np, sizeof np, cudaMemcpyHostToDevice, s);
  // causal prompt rows, in chunks of at most R_p rows
  std::vector<RowDesc> rows;
  std::vector<int32_t> gather, dst;
  auto flush = [&]() {
    if (rows.empty()) return;
    const int R = (int)rows.size();
    cudaMemcpyAsync(c->rows_p, rows.data(), sizeof(RowDesc) * R, cudaMemcpyHostToDevice, s);
    const int nlm = (int)gather.size();
    if (nlm) {
      cudaMemcpyAsync(c->lm_gather, gather.data(), 4 * nlm, cudaMemcpyHostToDevice, s);
      cudaMemcpyAsync(c->lm_dst, dst.data(), 4 * nlm, cudaMemcpyHostToDevice, s);
    }
    // z maps: each prompt present in the chunk, its rows in query blocks
    std::vector<int> per_prompt(B, 0);
    int maxpos = 0;
    for (const RowDesc& rd : rows) { per_prompt[rd.b]++; maxpos = std::max(maxpos, rd.pos); }
    auto zmap_for = [&](const cdsl_model_cfg& mc) {
      std::vector<int32_t> z;
      const int G = mc.n_heads / mc.n_kv_heads;
      for (int b = 0; b < B; ++b)
        for (int q = 0; q < (per_prompt[b] * G + attn_qblock() - 1) / attn_qblock(); ++q) {
          z.push_back(b);
          z.push_back(q);
        }
      return z;
    };
    const std::vector<int32_t> zt = zmap_for(c->tcfg), zd = zmap_for(c->dcfg);
    AttnPass apt, apd;
    apt.zmap = &zt;
    apd.zmap = &zd;
    apt.n_chunks = apd.n_chunks = (maxpos + attn_chunk()) / attn_chunk();
    forward(c, c->tgt, c->rows_p, R, nlm, c->lm_gather, c->logits, false, apt);
    if (nlm) {
      RowStatsArgs a{};
      a.logits = c->logits; a.R = nlm; a.V = c->V; a.k = c->k;
      a.topk = st.roots; a.dst = c->lm_dst; a.status = st.status;
      launch_row_stats(a, s);
    }
    forward(c, c->dft, c->rows_p, R, 0, nullptr, nullptr, false, apd);
    cudaStreamSynchronize(s);  // host row buffers are reused by the next chunk
    rows.clear(); gather.clear(); dst.clear();
  };
  std::vector<int32_t> host_tokens((size_t)B * c->run.max_prompt);
  cudaMemcpyAsync(host_tokens.data(), d_prompts, host_tokens.size() * 4, cudaMemcpyDeviceToHost, s);
  cudaStreamSynchronize(s);
  for (int b = 0; b < B; ++b) {
    for (int p = 0; p < h_prompt_lens[b]; ++p) {
      const int32_t tok = host_tokens[(size_t)b * c->run.max_prompt + p];
      if (tok < 0 || tok >= c->V) return fail(c, CDSL_EINVAL, "prompt token id out of range");
      RowDesc rd{};
      rd.b = b; rd.pos = p; rd.token = tok; rd.n_prefix = p + 1; rd.tail_base = 0; rd.n_tail = 0;
      rd.kv_dst = KV_PREFIX; rd.out_idx = (p == h_prompt_lens[b] - 1) ? b : -1;
      if (rd.out_idx >= 0) { gather.push_back((int)rows.size()); dst.push_back(b); }
      rows.push_back(rd);
      if ((int)rows.size() == c->R_p) flush();
    }
  }
  flush();
  int e = cuda_check(c, "cdsl_prefill");
  if (e) return e;
  c->phase = PH_READY;
  return CDSL_OK;
}

int32_t cdsl_lookahead(cdsl_ctx* c, int32_t* d_roots, int32_t* d_draft_tok, float* d_logq) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (c->phase != PH_READY) return fail(c, CDSL_ESTATE, "cdsl_lookahead needs a prefilled context");
  cudaGetLastError();
  do_lookahead(c);
  const size_t n = (size_t)c->B * c->k;
  copy_out(c, d_roots, c->st.roots, n * 4);
  copy_out(c, d_draft_tok, c->st.x, n * c->d * 4);
  copy_out(c, d_logq, c->st.logq, n * c->d * 4);
  int e = cuda_check(c, "cdsl_lookahead");
  if (e) return e;
  c->phase = PH_LOOKED;
  return CDSL_OK;
}

int32_t cdsl_verify(cdsl_ctx* c, float* d_logp, int32_t* d_argmax, int32_t* d_n_accept,
                    float* d_logits) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (c->phase != PH_LOOKED) return fail(c, CDSL_ESTATE, "cdsl_verify needs a preceding cdsl_lookahead");
  cudaGetLastError();
  do_verify(c);
  const size_t n = (size_t)c->B * c->k;
  copy_out(c, d_logp, c->st.v_logp, n * c->d * 4);
  copy_out(c, d_argmax, c->st.v_amax, n * (c->d + 1) * 4);
  copy_out(c, d_logits, c->logits, (size_t)c->R_v * c->V * 4);
  if (d_n_accept) {
    // n_b is settled by the decision kernel; run it here without committing anything.
    launch_select(c->st, c->tgt.kv, c->dft.kv, 0, c->stream);
    copy_out(c, d_n_accept, c->st.n_acc, n * 4);
  }
  int e = cuda_check(c, "cdsl_verify");
  if (e) return e;
  c->phase = PH_VERIFIED;
  return CDSL_OK;
}

int32_t cdsl_select(cdsl_ctx* c, int32_t* d_beam, int32_t* d_state, int32_t* d_emitted,
                    int32_t* d_n_emitted, float* d_reward) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (c->phase != PH_VERIFIED) return fail(c, CDSL_ESTATE, "cdsl_select needs a preceding cdsl_verify");
  cudaGetLastError();
  do_select(c);
  copy_select_outputs(c, d_beam, d_state, d_emitted, d_n_emitted, d_reward);
  int e = cuda_check(c, "cdsl_select");
  if (e) return e;
  c->phase = PH_READY;
  return CDSL_OK;
}

}  // extern "C"

namespace {

// Capture one whole step (lookahead, verify, select) into an executable graph.
int capture_step(cdsl_ctx* c, cudaGraphExec_t* out, long long* nodes_out) {
  cudaGraph_t g = nullptr;
  if (cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
    return fail(c, CDSL_ECUDA, "cudaStreamBeginCapture failed");
  do_lookahead(c);
  do_verify(c);
  do_select(c);
  cudaError_t ce = cudaStreamEndCapture(c->stream, &g);
  if (ce != cudaSuccess) return fail(c, CDSL_ECUDA, std::string("capture: ") + cudaGetErrorString(ce));
  size_t nodes = 0;
  cudaGraphGetNodes(g, nullptr, &nodes);
  if (nodes_out) *nodes_out = (long long)nodes;
  ce = cudaGraphInstantiate(out, g, 0);
  cudaGraphDestroy(g);
  if (ce != cudaSuccess) {
    *out = nullptr;
    return fail(c, CDSL_ECUDA, std::string("graph instantiate: ") + cudaGetErrorString(ce));
  }
  return CDSL_OK;
}

// Fold the stamped step's launch records into the per-launch totals. Launches are taken in
// stream order; each is charged from its first block's entry, or from the latest exit of the
// launches before it when it started earlier (programmatic dependent launch overlaps a
// kernel's prologue with its predecessor's tail), to its last block's exit. The charged
// intervals are disjoint, so their sum never exceeds the step's span. Launches without a
// record (the small step kernels) are charged nothing.
int fold_stamps(cdsl_ctx* c) {
  const size_t L = std::min(c->st_recs.size(), (size_t)kStampStride);
  std::vector<unsigned long long> h((size_t)3 * kStampStride);
  for (int w = 0; w < 3; ++w)
    if (cudaMemcpy(h.data() + (size_t)w * kStampStride, c->stamps + (size_t)w * kStampStride,
                   L * sizeof(unsigned long long), cudaMemcpyDeviceToHost) != cudaSuccess)
      return cuda_check(c, "cdsl_step (stamps)");
  c->st_ms.resize(c->st_recs.size(), 0.0);
  c->st_kbytes.resize(c->st_recs.size(), 0.0);
  unsigned long long prev_end = 0, first = ~0ull, last = 0;
  for (size_t i = 0; i < L; ++i) {
    const unsigned long long t0 = h[i], t1 = h[kStampStride + i];
    if (t0 == ~0ull || t1 == 0 || t1 < t0) continue;   // no record written
    first = std::min(first, t0);
    last = std::max(last, t1);
    const unsigned long long from = std::max(t0, prev_end);
    if (t1 > from) c->st_ms[i] += (double)(t1 - from) * 1e-6;
    prev_end = std::max(prev_end, t1);
    c->st_kbytes[i] += (double)h[2 * (size_t)kStampStride + i];
  }
  if (last > first) c->st_span_ms += (double)(last - first) * 1e-6;
  c->st_steps += 1;
  return CDSL_OK;
}

}  // namespace

extern "C" {

int32_t cdsl_step(cdsl_ctx* c, int32_t* d_beam, int32_t* d_state, int32_t* d_emitted,
                  int32_t* d_n_emitted, float* d_reward) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (c->phase != PH_READY) return fail(c, CDSL_ESTATE, "cdsl_step needs a prefilled context");
  cudaGetLastError();
  bool stamped = false;
  if (c->stream == nullptr || c->profiling) {  // legacy stream / event timing: launch directly
    do_lookahead(c);
    do_verify(c);
    do_select(c);
  } else if (c->prof_mode == 2) {             // in-graph timing: the stamped graph
    if (!c->graph_st) {
      c->stamping = true;
      c->st_recs.clear();
      const int e = capture_step(c, &c->graph_st, nullptr);
      c->stamping = false;
      if (e) return e;
    }
    const size_t n = sizeof(unsigned long long) * kStampStride;
    cudaMemsetAsync(c->stamps, 0xff, n, c->stream);
    cudaMemsetAsync(c->stamps + kStampStride, 0, 2 * n, c->stream);
    cudaGraphLaunch(c->graph_st, c->stream);
    stamped = true;
  } else {
    if (!c->graph) {
      const int e = capture_step(c, &c->graph, &c->graph_nodes);
      if (e) return e;
    }
    cudaGraphLaunch(c->graph, c->stream);
  }
  copy_select_outputs(c, d_beam, d_state, d_emitted, d_n_emitted, d_reward);
  int e = cuda_check(c, "cdsl_step");
  if (e || !stamped) return e;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cuda_check(c, "cdsl_step");
  return fold_stamps(c);
}

int32_t cdsl_get_tokens(cdsl_ctx* c, int32_t* d_tokens, int32_t* d_lengths) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  const int W = c->run.max_prompt + c->run.max_new;
  if (d_tokens)
    cudaMemcpy2DAsync(d_tokens, sizeof(int32_t) * W, c->st.tokens, sizeof(int32_t) * c->lcap,
                      sizeof(int32_t) * W, c->B, cudaMemcpyDeviceToDevice, c->stream);
  copy_out(c, d_lengths, c->st.len, sizeof(int32_t) * c->B);
  return cuda_check(c, "cdsl_get_tokens");
}

int32_t cdsl_get_counters(cdsl_ctx* c, int64_t* h_counters) {
  if (!c || !h_counters) return fail(c, CDSL_EINVAL, "ctx or counters is NULL");
  long long tmp[8];
  cudaMemcpyAsync(tmp, c->st.counters, sizeof tmp, cudaMemcpyDeviceToHost, c->stream);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cuda_check(c, "cdsl_get_counters");
  for (int i = 0; i < 6; ++i) h_counters[i] = tmp[i];
  h_counters[6] = c->graph_nodes;
  h_counters[7] = 0;
  return CDSL_OK;
}

int32_t cdsl_profile(cdsl_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (enable < 0 || enable > 2) return fail(c, CDSL_EINVAL, "cdsl_profile: mode must be 0, 1 or 2");
  c->prof_mode = enable;
  c->profiling = enable == 1;
  c->ev_used = 0;
  c->prof.clear();
  std::fill(c->st_ms.begin(), c->st_ms.end(), 0.0);
  std::fill(c->st_kbytes.begin(), c->st_kbytes.end(), 0.0);
  c->st_steps = 0;
  c->st_span_ms = 0;
  return CDSL_OK;
}

int32_t cdsl_get_profile(cdsl_ctx* c, int32_t impl, double* h_out) {
  if (!c || !h_out) return fail(c, CDSL_EINVAL, "ctx or out is NULL");
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return fail(c, CDSL_ECUDA, std::string("cdsl_get_profile: ") + cudaGetErrorString(e));
  double n = 0, ms = 0, by = 0, fl = 0;
  if (c->prof_mode == 2) {
    const double steps = c->st_steps;
    if (impl == K_CLASSES) {   // the stamped steps themselves
      n = steps;
      ms = c->st_span_ms;
    }
    for (size_t i = 0; i < c->st_recs.size() && i < c->st_ms.size(); ++i) {
      const auto& r = c->st_recs[i];
      if (r.impl != impl) continue;
      n += steps; ms += c->st_ms[i];
      by += r.bytes > 0 ? r.bytes * steps : c->st_kbytes[i];
      fl += r.flops * steps;
    }
  } else {
    for (const auto& r : c->prof) {
      if (r.impl != impl) continue;
      float t = 0;
      cudaEventElapsedTime(&t, c->ev_pool[r.ev], c->ev_pool[r.ev + 1]);
      n += 1; ms += t; by += r.bytes; fl += r.flops;
    }
  }
  h_out[0] = n; h_out[1] = ms; h_out[2] = by; h_out[3] = fl;
  return cuda_check(c, "cdsl_get_profile");
}

int32_t cdsl_get_profile_launches(cdsl_ctx* c, double* h_out, int32_t h_capacity) {
  if (!c || !h_out || h_capacity < 0) return -fail(c, CDSL_EINVAL, "ctx or out is NULL");
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess)
    return -fail(c, CDSL_ECUDA, std::string("cdsl_get_profile_launches: ") + cudaGetErrorString(e));
  int32_t n = 0;
  if (c->prof_mode == 2) {   // per launch of the stamped step, averaged over the steps
    const double steps = std::max(1, c->st_steps);
    for (size_t i = 0; i < c->st_recs.size() && i < c->st_ms.size(); ++i) {
      if (n >= h_capacity) break;
      const auto& r = c->st_recs[i];
      h_out[4 * n] = r.impl;
      h_out[4 * n + 1] = c->st_ms[i] / steps;
      h_out[4 * n + 2] = r.bytes > 0 ? r.bytes : c->st_kbytes[i] / steps;
      h_out[4 * n + 3] = r.flops;
      ++n;
    }
    return n;
  }
  for (const auto& r : c->prof) {
    if (n >= h_capacity) break;
    float t = 0;
    cudaEventElapsedTime(&t, c->ev_pool[r.ev], c->ev_pool[r.ev + 1]);
    h_out[4 * n] = r.impl; h_out[4 * n + 1] = t; h_out[4 * n + 2] = r.bytes; h_out[4 * n + 3] = r.flops;
    ++n;
  }
  return n;
}

int32_t cdsl_set_wait_limit(cdsl_ctx* c, uint64_t ns) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cuda_check(c, "cdsl_set_wait_limit");
  c->wait_ns = ns;
  // the step graphs hold the old limit in their kernel arguments: capture them again
  if (c->graph) cudaGraphExecDestroy(c->graph);
  if (c->graph_st) cudaGraphExecDestroy(c->graph_st);
  c->graph = c->graph_st = nullptr;
  return CDSL_OK;
}

int32_t cdsl_get_step1(cdsl_ctx* c, int32_t* d_need, int32_t* d_tokens, float* d_reward) {
  if (!c) return fail(nullptr, CDSL_EINVAL, "ctx is NULL");
  if (c->run.step1_budget < 2) return fail(c, CDSL_EINVAL, "cdsl_get_step1 needs step1_budget 2");
  const size_t B = c->B;
  copy_out(c, d_need, c->st.s1_need, B * 4);
  copy_out(c, d_tokens, c->st.s1_tok, B * (c->d + 1) * 4);
  copy_out(c, d_reward, c->st.s1_reward, B * 4);
  return cuda_check(c, "cdsl_get_step1");
}

int32_t cdsl_get_status(cdsl_ctx* c, int32_t* h_device_status) {
  if (!c || !h_device_status) return fail(c, CDSL_EINVAL, "ctx or status is NULL");
  int32_t v = 0;
  cudaMemcpyAsync(&v, c->st.status, sizeof v, cudaMemcpyDeviceToHost, c->stream);
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return fail(c, CDSL_ECUDA, std::string("cdsl_get_status: ") + cudaGetErrorString(e));
  *h_device_status = v;
  return CDSL_OK;
}

const char* cdsl_last_error(const cdsl_ctx* c) {
  return c ? c->err.c_str() : g_init_error.c_str();
}

void cdsl_destroy(cdsl_ctx* c) {
  if (!c) return;
  if (c->graph) cudaGraphExecDestroy(c->graph);
  if (c->graph_st) cudaGraphExecDestroy(c->graph_st);
  for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
  delete c;
}

}  // extern "C"
