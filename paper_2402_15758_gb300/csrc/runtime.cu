// Host runtime of the C ABI: context, paged KV allocator, static tree, the launch plan
// of one step (captured once into a CUDA graph and replayed), prefill, debug hooks and
// the stateless kernel-level entry points.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <functional>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/chimera.h"
#include "common.cuh"
#include "kernels.h"
#include "step_kernels.h"

using namespace chimera;

namespace {

constexpr int CHUNK = 64;        // prefill rows per sequence per pass (one 64-bit mask)
constexpr int LOG_CAP = 4096;    // per-step accepted-count log
constexpr int MAX_KMAX = 8;
constexpr int CHAIN_BAR_INTS = 16;     // >= CHAIN_MAX_STEPS + 1 counters per chain launch
constexpr int CHAIN_BAR_BLOCKS = 256;  // chain launches with their own counters

struct Lin {
  bool tc = false;
  TcLinearPlan tp;
  int M = 0, N = 0, K = 0, ldx = 0, ldy = 0, epi = 0, out_f32 = 0;
  const void* X = nullptr;
  const void* W = nullptr;
  const void* W2 = nullptr;  // optional second weight: outputs at columns N .. N+N2-1
  int N2 = 0;
  void* Y = nullptr;
  const int* skip = nullptr;  // device flag: nonzero -> the launch does nothing
  double bytes = 0;
};

struct ProfEvent {
  int kind, phase;
  double bytes;
  cudaEvent_t a, b;
};

// Static tree (reading of Section "Inference"): the N-1 rank tuples with the largest
// product of per-head marginal top-k accuracies of Table 4 (Chimera rows).
struct Tree {
  int n = 0, depth_max = 0;
  std::vector<int> depth, parent, rank, child_start, child;
  std::vector<uint64_t> anc;
};

bool build_tree(const int* topk, int K, int N, Tree* t, std::string* err) {
  static const int acc[4][5] = {{66, 78, 83, 87, 90}, {49, 55, 60, 68, 75}, {38, 44, 49, 55, 62},
                                {33, 38, 43, 46, 54}};
  int marg[4][5];
  for (int h = 0; h < 4; ++h)
    for (int r = 0; r < 5; ++r) marg[h][r] = r == 0 ? acc[h][0] : acc[h][r] - acc[h][r - 1];
  if (K > 4) {
    *err = "the static tree covers at most 4 draft heads (Table 4)";
    return false;
  }
  struct Cand {
    long long score;
    std::vector<int> r;
  };
  std::vector<Cand> cands;
  std::vector<int> cur;
  // enumerate every rank tuple of depth 1..K with r_i < min(topk[i], 5)
  std::function<void(int, long long)> rec = [&](int d, long long s) {
    if (d > 0) {
      long long sc = s;
      for (int i = d; i < 4; ++i) sc *= 100;
      cands.push_back({sc, cur});
    }
    if (d == K) return;
    const int lim = std::min(topk[d], 5);
    for (int r = 0; r < lim; ++r) {
      cur.push_back(r);
      rec(d + 1, s * marg[d][r]);
      cur.pop_back();
    }
  };
  rec(0, 1);
  if (static_cast<int>(cands.size()) < N - 1) {
    *err = "tree_nodes exceeds the number of rank tuples allowed by topk";
    return false;
  }
  std::sort(cands.begin(), cands.end(), [](const Cand& a, const Cand& b) {
    if (a.score != b.score) return a.score > b.score;
    if (a.r.size() != b.r.size()) return a.r.size() < b.r.size();
    return a.r < b.r;
  });
  std::vector<std::vector<int>> nodes(1);
  for (int i = 0; i < N - 1; ++i) nodes.push_back(cands[i].r);
  std::sort(nodes.begin() + 1, nodes.end(), [](const std::vector<int>& a, const std::vector<int>& b) {
    if (a.size() != b.size()) return a.size() < b.size();
    return a < b;
  });
  t->n = N;
  t->depth.assign(N, 0);
  t->parent.assign(N, -1);
  t->rank.assign(N, 0);
  t->anc.assign(N, 0);
  t->depth_max = 0;
  for (int i = 1; i < N; ++i) {
    t->depth[i] = static_cast<int>(nodes[i].size());
    t->rank[i] = nodes[i].back();
    std::vector<int> pre(nodes[i].begin(), nodes[i].end() - 1);
    for (int j = 0; j < i; ++j)
      if (nodes[j] == pre) t->parent[i] = j;
    if (t->parent[i] < 0) {
      *err = "static tree is not prefix-closed";
      return false;
    }
    t->depth_max = std::max(t->depth_max, t->depth[i]);
  }
  for (int i = 0; i < N; ++i) {
    uint64_t m = 0;
    for (int j = i; j >= 0; j = t->parent[j]) m |= 1ull << j;
    t->anc[i] = m;
  }
  t->child_start.assign(N + 1, 0);
  t->child.clear();
  for (int i = 0; i < N; ++i) {
    t->child_start[i] = static_cast<int>(t->child.size());
    for (int c = i + 1; c < N; ++c)
      if (t->parent[c] == i) t->child.push_back(c);
  }
  t->child_start[N] = static_cast<int>(t->child.size());
  if (t->child.empty()) t->child.push_back(0);
  return true;
}

}  // namespace

struct chimera_ctx {
  chimera_config cfg;
  int L = 0, d = 0, H = 0, hd = 0, F = 0, V = 0, K = 0, N = 0, KMAX = 0, D1 = 0, Bmax = 0, cap = 0;
  int dtype = 0;
  size_t esz = 4;      // weights / GEMM operands
  int split = 0;       // bf16 GEMM operands kept as hi + lo pairs
  int kv_planes = 2;   // KV planes per (block, head): K, V or K_hi, K_lo, V_hi, V_lo
  size_t kv_esz = 4;   // element size of the KV pools (the model dtype)
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  int num_sms = 1;

  // weights (device pointers, caller-owned)
  const void* embed = nullptr;
  std::vector<chimera_block_weights> layers;
  chimera_block_weights draft{};
  const void* final_norm = nullptr;
  const void* lm_head = nullptr;
  const void* tri_w1 = nullptr;
  const void* tri_w2 = nullptr;
  std::vector<const void*> heads;

  // variants of the method (see chimera_config)
  int draft_mode = 0;   // bit 0: one-pass draft; bit 1: heads without the residual input
  int accept_mode = 0;  // 0: greedy, 1: typical acceptance
  float typ_eps = 0.f, typ_delta = 0.f;
  // trigram cache: keys / LRU stamps / h_tri rows of tc_entries ways (4 per set)
  int tc_entries = 0, tc_nsets = 0;
  unsigned long long* tc_keys = nullptr;
  int *tc_stamp = nullptr, *tc_hit = nullptr, *tc_slot = nullptr, *tc_skip = nullptr, *tc_clock = nullptr;
  int* tc_hit_log = nullptr;     // [K][B] hits of the last step's sub-steps
  float* tc_vals = nullptr;
  float* htri_log = nullptr;     // [K][B][d] h_tri rows of the last step (cache on)
  float* d_stats = nullptr;      // [B*N][3] softmax stats of the verify rows (typical acceptance)
  int* d_parent = nullptr;

  Tree tree;
  std::vector<uint64_t> chain;
  int *d_depth = nullptr, *d_rank = nullptr, *d_child_start = nullptr, *d_child = nullptr;
  unsigned long long *d_anc = nullptr, *d_chain = nullptr;

  // device state
  int *d_n = nullptr, *d_tok = nullptr, *d_node_tok = nullptr, *d_topk = nullptr, *d_amax = nullptr;
  int *d_path = nullptr, *d_L = nullptr, *d_bonus = nullptr, *d_ovr = nullptr, *d_ovr_flag = nullptr;
  int *d_valid = nullptr, *d_last = nullptr, *d_count_log = nullptr, *d_step = nullptr, *d_err = nullptr;
  float* d_topk_val = nullptr;
  int tok_stride = 0;

  // KV
  void* kv = nullptr;
  void* dkv = nullptr;
  long long kv_layer_stride = 0;  // elements
  int NB = 0, max_pages = 0;
  int* d_pt = nullptr;
  int* h_pt = nullptr;  // pinned mirror of the page table
  size_t h_pt_len = 0;
  cudaEvent_t pt_event = nullptr;  // last upload of h_pt
  bool pt_inflight = false;
  std::vector<std::vector<int>> seq_blocks;
  std::vector<int> free_blocks;
  bool pt_dirty = false;
  float2* d_rope = nullptr;
  int max_pos = 0;

  // activations
  int R = 0;
  float* x = nullptr;
  // GEMM operands in the model dtype; *_lo = the bf16 rounding residuals (split mode)
  void *xn = nullptr, *xn_lo = nullptr, *ao = nullptr, *ao_lo = nullptr, *hf = nullptr, *hf_lo = nullptr;
  void *hfin = nullptr, *hfin_lo = nullptr;
  float* hfin32 = nullptr;              // post-final-norm hidden states (H_LLM), fp32
  float* qr = nullptr;                  // rotated queries, fp32
  float *qkv = nullptr, *gu = nullptr;  // fp32 GEMM outputs feeding RoPE / SwiGLU
  float* logits = nullptr;
  void *tbuf = nullptr, *ubuf = nullptr, *ubuf_lo = nullptr, *headin = nullptr, *headin_lo = nullptr;
  float *hfull_log = nullptr, *hsel = nullptr, *kvtmp = nullptr;
  float *dres = nullptr, *hlog = nullptr;
  bool tc_zero = false;  // tensor-core linears clear the next accumulators (see enqueue_layer)

  // scratch of the split kernels
  float* lin_ws = nullptr;
  int* lin_cnt = nullptr;
  float* att_ws = nullptr;
  size_t att_ws_floats = 0;
  int* att_cnt = nullptr;
  float* topk_ws_v = nullptr;
  int* topk_ws_i = nullptr;
  int* topk_cnt = nullptr;

  // plan of the current batch
  int batch = 0;
  std::vector<int> host_n;
  std::vector<Lin> ver, pre, ar;  // 5 per layer: qkv, wo, gate, up, down
  Lin ver_lm, pre_lm, ar_lm, pre_dkv, tri1, tri2, dqkv, dwo, dgate, dup, ddown, commit_kv;
  std::vector<Lin> dhead;
  // persistent chains (bf16 models): the linears and row steps between two attentions
  // in one launch each (chain_tc.cu)
  bool use_chain = false;
  std::vector<ChainPlan> ver_chain, ar_chain, draft_chain_a, draft_chain_b;
  ChainPlan commit_chain;
  int* chain_bars = nullptr;  // [CHAIN_BAR_BLOCKS][CHAIN_BAR_INTS] step counters, zero between launches
  int chain_bar_next = 0;
  int att_splits_ver = 1, att_splits_pre = 1, att_splits_draft = 1, att_splits_ar = 1;
  int plan_keys = 0;  // longest prompt of the batch (sizes the attention splits)
  cudaGraphExec_t graph = nullptr;
  cudaGraphExec_t ar_graph = nullptr;  // one plain autoregressive step (eq. 1)
  int *d_one = nullptr, *d_child_start1 = nullptr, *d_child1 = nullptr;  // a one-node tree
  bool prefilled = false;
  bool ovr_pending = false;

  int* h_stage = nullptr;  // pinned staging
  size_t h_stage_ints = 0;

  // profiling
  bool prof = false;
  std::vector<ProfEvent> prof_ev;
  size_t prof_used = 0;
  cudaGraphExec_t prof_graph = nullptr;  // the step with an event pair around every launch
  size_t prof_count = 0;
  int cur_phase = 0;
  int last_kind = 0;  // kernel class of the latest launch (CHIMERA_KIND_*)
  // graph of the step with an event at each phase boundary (draft | verify | commit)
  cudaGraphExec_t phase_graph = nullptr;
  cudaEvent_t phase_ev[4] = {nullptr, nullptr, nullptr, nullptr};
  bool phase_marks = false;
  // graph of only one kernel class's launches of the step, in step order
  int filter_kind = 0;  // 0: every launch is enqueued
  cudaGraphExec_t class_graph = nullptr;
  int class_graph_kind = 0;
  size_t class_launches = 0;
  double class_bytes = 0;

  std::string err;
  std::vector<void*> allocs;
};

namespace {

chimera_status fail(chimera_ctx* c, chimera_status st, const std::string& msg) {
  if (c) c->err = msg;
  return st;
}

#define CK(call)                                                                     \
  do {                                                                               \
    cudaError_t e_ = (call);                                                         \
    if (e_ != cudaSuccess)                                                           \
      return fail(ctx, CHIMERA_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

template <typename T>
bool dalloc(chimera_ctx* ctx, T** p, size_t count) {
  void* q = nullptr;
  if (count == 0) count = 1;
  if (cudaMalloc(&q, count * sizeof(T)) != cudaSuccess) return false;
  ctx->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return true;
}
bool dalloc_bytes(chimera_ctx* ctx, void** p, size_t bytes) {
  if (bytes == 0) bytes = 16;
  if (cudaMalloc(p, bytes) != cudaSuccess) return false;
  ctx->allocs.push_back(*p);
  return true;
}

// True when a launch of class `kind` is left out of the graph being captured.
bool filtered(const chimera_ctx* ctx, int kind) { return ctx->filter_kind != 0 && ctx->filter_kind != kind; }

// ---------------------------------------------------------------------------
// launch helpers (events around every launch when profiling)
// ---------------------------------------------------------------------------
struct Scope {
  chimera_ctx* c;
  ProfEvent* ev = nullptr;
  Scope(chimera_ctx* ctx, int kind, double bytes) : c(ctx) {
    c->last_kind = kind;
    if (c->filter_kind == kind) {
      ++c->class_launches;
      c->class_bytes += bytes;
    }
    if (!c->prof) return;
    if (c->prof_used == c->prof_ev.size()) {
      ProfEvent e{};
      cudaEventCreate(&e.a);
      cudaEventCreate(&e.b);
      c->prof_ev.push_back(e);
    }
    ev = &c->prof_ev[c->prof_used++];
    ev->kind = kind;
    ev->phase = c->cur_phase;
    ev->bytes = bytes;
    // recorded inside a stream capture: external records become event nodes
    cudaEventRecordWithFlags(ev->a, c->stream, cudaEventRecordExternal);
  }
  ~Scope() {
    if (ev) cudaEventRecordWithFlags(ev->b, c->stream, cudaEventRecordExternal);
  }
};

cudaError_t run_lin(chimera_ctx* ctx, const Lin& l) {
  if (l.N == 0 || filtered(ctx, CHIMERA_KIND_LINEAR)) return cudaSuccess;  // N = 0: folded into the previous site
  Scope sc(ctx, CHIMERA_KIND_LINEAR, l.bytes);
  if (l.tc) return tc_linear_launch(l.tp, ctx->stream);
  cudaError_t e = f32_linear(l.M, l.N, l.K, static_cast<const float*>(l.X), l.ldx, static_cast<const float*>(l.W),
                             static_cast<float*>(l.Y), l.ldy, l.epi, ctx->stream, l.skip);
  if (e != cudaSuccess || !l.W2) return e;
  return f32_linear(l.M, l.N2, l.K, static_cast<const float*>(l.X), l.ldx, static_cast<const float*>(l.W2),
                    static_cast<float*>(l.Y) + l.N, l.ldy, l.epi, ctx->stream, l.skip);
}

bool make_lin(chimera_ctx* ctx, Lin* l, int M, int N, int K, const void* X, const void* X_lo, int ldx,
              const void* W, void* Y, void* Y_lo, int ldy, int epi, int out_f32, const void* W2 = nullptr,
              int N2 = 0, float* zero = nullptr, long long zero_floats = 0, const int* skip = nullptr) {
  l->M = M;
  l->N = N;
  l->K = K;
  l->X = X;
  l->ldx = ldx;
  l->W = W;
  l->Y = Y;
  l->ldy = ldy;
  l->epi = epi;
  l->out_f32 = out_f32;
  l->W2 = W2;
  l->N2 = W2 ? N2 : 0;
  l->bytes = static_cast<double>(N + l->N2) * K * ctx->esz;
  l->skip = skip;
  l->tc = ctx->dtype == 1;
  if (!l->tc) return true;
  char msg[256];
  if (tc_linear_plan(&l->tp, M, N, K, X, X_lo, ldx, W, Y, Y_lo, ldy, epi, out_f32, ctx->lin_ws, ctx->lin_cnt,
                     ctx->d_err, msg, sizeof(msg), W2, N2, zero, zero_floats) != 0) {
    ctx->err = msg;
    return false;
  }
  l->tp.p.wait_ns = kDefaultWaitNs;  // the timeout hook applies to the stateless entry points only
  l->tp.p.skip = skip;
  return true;
}

// KV splits per (sequence, head): enough CTAs to cover the SMs for single-query
// attention (the draft), and about three 64-key tiles per split for tree queries so
// the per-split partials stay few (their merge is latency-bound).
#ifndef CHIMERA_ATT_TILES_PER_CTA
#define CHIMERA_ATT_TILES_PER_CTA 32
#endif
int att_splits(const chimera_ctx* ctx, int B, int nq, int n_keys) {
  if (attn_fuses_rope(ctx->dtype, ctx->hd)) {
    // tensor-core tree attention: one cluster of S CTAs per (b, h).  While the B * H
    // clusters fit on the SMs at once, as many splits as keep them all resident; with
    // more (sequence, head) pairs than SMs the launch runs in waves whatever S is, so
    // long contexts are cut into splits of at most ~CHIMERA_ATT_TILES_PER_CTA 64-key
    // tiles (a CTA that held a whole long context would set the last wave's length;
    // measured on the 7B batch-8 step: 64 tiles 14.97, 32 tiles 13.66, 16 tiles 14.81,
    // 8 tiles 18.89 ms per step, the CTAs' fixed prologue and merge taking over)
    const int tiles = (n_keys + 63) / 64;
    if (B * ctx->H >= ctx->num_sms)
      return std::max(1, std::min(8, (tiles + CHIMERA_ATT_TILES_PER_CTA - 1) / CHIMERA_ATT_TILES_PER_CTA));
    const int want = std::max(1, std::min(ctx->num_sms / (B * ctx->H), tiles));
    return attn_pick_splits(ctx->dtype, ctx->hd, ctx->kv_planes, B, ctx->H, want);
  }
  const int target = 2 * ctx->num_sms;
  int s = (target + B * ctx->H - 1) / (B * ctx->H);
  if (nq > 1) s = std::min(s, (n_keys + 191) / 192);
  return std::max(1, std::min(16, s));
}

// With qkv (models where attn_fuses_rope holds) the kernel also rotates q and the nq
// fresh rows' k (positions n + pos_base + pos_off[i]) and writes their k, v to the pool.
// It then reads n_ctx, the page table and the committed KV rows BEFORE its own
// dependency wait (prewait_kv).  That is only correct when the launch directly before
// it is a tensor-core linear: that kernel lets its dependents launch only after its
// own griddepcontrol.wait, so every earlier kernel has completed by then.  Most row
// kernels trigger before they wait; one of them directly before this launch could
// let it read stale KV rows.  The order is checked here (and by a CPU lint test).
cudaError_t run_attention(chimera_ctx* ctx, bool draft_pool, int layer, int nq, const int* nq_dev, int q_local0,
                          int n_local, const int* n_local_dev, const unsigned long long* anc, int q_rows, int splits,
                          int nq_max, double bytes, const float* qkv = nullptr, int pos_base = 0,
                          const int* pos_off = nullptr) {
  if (filtered(ctx, CHIMERA_KIND_ATTENTION)) return cudaSuccess;
  if (qkv && !ctx->filter_kind &&
      !(ctx->dtype == 1 && (ctx->last_kind == CHIMERA_KIND_LINEAR || ctx->last_kind == CHIMERA_KIND_CHAIN))) {
    ctx->err = "attention with early KV reads must directly follow a tensor-core linear or chain";
    return cudaErrorInvalidValue;
  }
  Scope sc(ctx, CHIMERA_KIND_ATTENTION, bytes);
  AttnParams p{};
  if (qkv) {
    p.qkv = qkv;
    p.ldqkv = 3 * ctx->d;
    p.rope = ctx->d_rope;
    p.max_pos = ctx->max_pos;
    p.pos_base = pos_base;
    p.pos_off = pos_off;
    p.prewait_kv = 1;
  }
  p.err = ctx->d_err;
  p.q = ctx->qr;
  p.ldq = ctx->d;
  p.q_rows = q_rows;
  p.nq = nq;
  p.nq_dev = nq_dev;
  p.q_local0 = q_local0;
  p.n_local = n_local;
  p.n_local_dev = n_local_dev;
  p.anc = anc;
  p.pool = draft_pool ? ctx->dkv : ctx->kv;
  p.planes = ctx->kv_planes;
  p.pool_layer_stride = draft_pool ? 0 : ctx->kv_layer_stride;
  p.pool_rows = static_cast<long long>(draft_pool ? 1 : ctx->L) * ctx->NB * ctx->H * ctx->kv_planes * 16;
  p.layer = draft_pool ? 0 : layer;
  p.page_table = ctx->d_pt;
  p.max_pages = ctx->max_pages;
  p.n_ctx = ctx->d_n;
  p.out = ctx->ao;
  p.out_lo = ctx->ao_lo;
  p.ldo = ctx->d;
  p.B = ctx->batch;
  p.H = ctx->H;
  p.hd = ctx->hd;
  p.scale = 1.0f / std::sqrt(static_cast<float>(ctx->hd));
  p.splits = splits;
  p.ws = ctx->att_ws;
  p.counters = ctx->att_cnt;
  p.nq_max = nq_max;
  if (attn_ws_floats(p.B, p.H, splits, nq_max, p.hd) > ctx->att_ws_floats) return cudaErrorInvalidValue;
  return attention(p, ctx->dtype, ctx->stream);
}

cudaError_t run_rope(chimera_ctx* ctx, bool draft_pool, int layer, const float* src, int ldsrc, int q_col, int k_col,
                     int v_col, int rows_per_seq, const int* valid, int valid_plus, int pos_base, int slot_base,
                     const int* pos_off) {
  if (filtered(ctx, CHIMERA_KIND_ROPE_KV)) return cudaSuccess;
  Scope sc(ctx, CHIMERA_KIND_ROPE_KV, 0);
  RopeKvParams p{};
  p.qkv = src;
  p.ldqkv = ldsrc;
  p.q_col = q_col;
  p.k_col = k_col;
  p.v_col = v_col;
  p.q_out = ctx->qr;
  p.ldq = ctx->d;
  p.pool = draft_pool ? ctx->dkv : ctx->kv;
  p.planes = ctx->kv_planes;
  p.pool_layer_stride = draft_pool ? 0 : ctx->kv_layer_stride;
  p.layer = draft_pool ? 0 : layer;
  p.page_table = ctx->d_pt;
  p.max_pages = ctx->max_pages;
  p.n = ctx->d_n;
  p.rows_per_seq = rows_per_seq;
  p.valid = valid;
  p.valid_plus = valid_plus;
  p.pos_base = pos_base;
  p.slot_base = slot_base;
  p.pos_off = pos_off;
  p.rope = ctx->d_rope;
  p.max_pos = ctx->max_pos;
  p.B = ctx->batch;
  p.H = ctx->H;
  p.hd = ctx->hd;
  p.err = ctx->d_err;
  return rope_kv(p, ctx->dtype, ctx->stream);
}

// RMSNorm of fp32 rows into the GEMM operand buffer xn (+ lo half); zeroes the rows of
// Z (zcols floats, pitch zcols) that the following linear accumulates into.
cudaError_t run_norm(chimera_ctx* ctx, const float* X, const void* g, int rows, float* Z, int zcols) {
  if (filtered(ctx, CHIMERA_KIND_NORM)) return cudaSuccess;
  Scope sc(ctx, CHIMERA_KIND_NORM, 0);
  return rmsnorm(ctx->dtype, X, ctx->d, g, ctx->xn, ctx->xn_lo, nullptr, ctx->d, rows, ctx->d, ctx->cfg.rms_eps, Z,
                 zcols, zcols, ctx->stream);
}

// Final norm: H_LLM rows in fp32 plus the LM-head operand (+ lo half); zeroes the
// logits rows when the LM head follows.
cudaError_t run_final_norm(chimera_ctx* ctx, int rows, bool zero_logits) {
  if (filtered(ctx, CHIMERA_KIND_NORM)) return cudaSuccess;
  Scope sc(ctx, CHIMERA_KIND_NORM, 0);
  return rmsnorm(ctx->dtype, ctx->x, ctx->d, ctx->final_norm, ctx->hfin, ctx->hfin_lo, ctx->hfin32, ctx->d, rows,
                 ctx->d, ctx->cfg.rms_eps, zero_logits ? ctx->logits : nullptr, ctx->V, ctx->V, ctx->stream);
}

#define RUN(call)                                            \
  do {                                                       \
    cudaError_t e_ = (call);                                 \
    if (e_ != cudaSuccess) return e_;                        \
  } while (0)

// One launch of class `kind` (left out when the capture keeps another class only).
#define LAUNCH(kind, bytes, call)                            \
  do {                                                       \
    if (!filtered(ctx, kind)) {                              \
      Scope sc_(ctx, kind, bytes);                           \
      RUN(call);                                             \
    }                                                        \
  } while (0)

// Phase boundary of the step (an event node in the phase-timed graph).
cudaError_t mark_phase(chimera_ctx* ctx, int i) {
  if (!ctx->phase_marks) return cudaSuccess;
  return cudaEventRecordWithFlags(ctx->phase_ev[i], ctx->stream, cudaEventRecordExternal);
}

char* eoff(const chimera_ctx* ctx, void* base, size_t elems) {
  return static_cast<char*>(base) + elems * ctx->esz;
}

cudaError_t run_chain(chimera_ctx* ctx, const ChainPlan& c) {
  if (filtered(ctx, CHIMERA_KIND_CHAIN)) return cudaSuccess;
  Scope sc(ctx, CHIMERA_KIND_CHAIN, c.weight_bytes);
  return chain_launch(c, ctx->stream);
}

// The base layers as chains: chain 0 (RMSNorm + QKV of layer 0), then per layer its
// tree attention and the chain to the next attention (O .. down, the next layer's
// RMSNorm and QKV; after the last layer the final norm and the LM head).
cudaError_t enqueue_layers_chain(chimera_ctx* ctx, const std::vector<ChainPlan>& ch, int rows_per_seq,
                                 const int* valid, const int* pos_off, const unsigned long long* anc, int splits,
                                 double kv_bytes) {
  RUN(run_chain(ctx, ch[0]));
  for (int l = 0; l < ctx->L; ++l) {
    RUN(run_attention(ctx, false, l, rows_per_seq, valid, 0, rows_per_seq, valid, anc, rows_per_seq, splits,
                      rows_per_seq, kv_bytes, ctx->qkv, 0, pos_off));
    RUN(run_chain(ctx, ch[l + 1]));
  }
  return cudaSuccess;
}

// One Llama layer over the rows of `plan` (5 linears), shared by verify and prefill.
cudaError_t enqueue_layer(chimera_ctx* ctx, int l, const Lin* lin, int rows, int rows_per_seq, const int* valid,
                          const int* pos_off, const unsigned long long* anc, int splits, double kv_bytes) {
  const chimera_block_weights& w = ctx->layers[l];
  const int d = ctx->d;
  // the accumulators of the QKV and gate|up linears are cleared by the norms, or (tensor-
  // core linears) by the previous layer's down linear and this layer's O linear
  const bool z = !ctx->tc_zero;
  RUN(run_norm(ctx, ctx->x, w.attn_norm, rows, (z || l == 0) ? ctx->qkv : nullptr, 3 * d));
  RUN(run_lin(ctx, lin[0]));
  if (attn_fuses_rope(ctx->dtype, ctx->hd)) {
    RUN(run_attention(ctx, false, l, rows_per_seq, valid, 0, rows_per_seq, valid, anc, rows_per_seq, splits,
                      rows_per_seq, kv_bytes, ctx->qkv, 0, pos_off));
  } else {
    RUN(run_rope(ctx, false, l, ctx->qkv, 3 * d, 0, d, 2 * d, rows_per_seq, valid, 0, 0, 0, pos_off));
    RUN(run_attention(ctx, false, l, rows_per_seq, valid, 0, rows_per_seq, valid, anc, rows_per_seq, splits,
                      rows_per_seq, kv_bytes));
  }
  RUN(run_lin(ctx, lin[1]));
  RUN(run_norm(ctx, ctx->x, w.ffn_norm, rows, z ? ctx->gu : nullptr, 2 * ctx->F));
  RUN(run_lin(ctx, lin[2]));
  RUN(run_lin(ctx, lin[3]));
  LAUNCH(CHIMERA_KIND_SWIGLU, 0, swiglu(ctx->dtype, ctx->gu, 2 * ctx->F, ctx->F, ctx->hf, ctx->hf_lo, ctx->F, rows, ctx->stream));
  RUN(run_lin(ctx, lin[4]));
  return cudaSuccess;
}

double kv_read_bytes(const chimera_ctx* ctx, int extra_rows, bool draft) {
  double rows = 0;
  for (int b = 0; b < ctx->batch; ++b) rows += ctx->host_n[b] + extra_rows;
  (void)draft;
  return rows * ctx->kv_planes * static_cast<double>(ctx->d) * ctx->kv_esz;
}

// The whole step on the context stream (graph-capturable: every dynamic value is read
// from device memory).
cudaError_t enqueue_step(chimera_ctx* ctx) {
  const int B = ctx->batch, d = ctx->d, K = ctx->K, N = ctx->N, V = ctx->V, F = ctx->F;
  cudaStream_t s = ctx->stream;
  (void)F;
  // ---- draft: K sequential sub-steps ----
  ctx->cur_phase = CHIMERA_PHASE_DRAFT;
  RUN(mark_phase(ctx, 0));
  const bool one_pass = (ctx->draft_mode & 1) != 0;
  for (int k = 0; k < K; ++k) {
    if (k > 0 && one_pass && ctx->use_chain) {  // every head scores h_full_{n+1}
      RUN(run_chain(ctx, ctx->draft_chain_b[k]));
      LAUNCH(CHIMERA_KIND_TOPK, 0, topk_rows(ctx->hlog + static_cast<size_t>(k) * B * V, V, B, ctx->KMAX,
                                             ctx->d_topk + k * ctx->KMAX, ctx->d_topk_val + k * ctx->KMAX, K * ctx->KMAX,
                                             ctx->topk_ws_v, ctx->topk_ws_i, ctx->topk_cnt, s));
      continue;
    }
    if (k > 0 && one_pass) {  // every head scores h_full_{n+1}: only the head k launch below
      LAUNCH(CHIMERA_KIND_OTHER, 0, launch_hfull_store(ctx->dtype, ctx->dres, d, ctx->headin, ctx->headin_lo,
                                 ctx->hfull_log + static_cast<size_t>(k) * B * d, nullptr, V, B, s));
      RUN(run_lin(ctx, ctx->dhead[k]));
      LAUNCH(CHIMERA_KIND_TOPK, 0, topk_rows(ctx->hlog + static_cast<size_t>(k) * B * V, V, B, ctx->KMAX,
                                             ctx->d_topk + k * ctx->KMAX, ctx->d_topk_val + k * ctx->KMAX, K * ctx->KMAX,
                                             ctx->topk_ws_v, ctx->topk_ws_i, ctx->topk_cnt, s));
      continue;
    }
    // sub-step 0 also clears every head's score rows, which the head linears accumulate
    // into (off the chain of the later sub-steps)
    const bool sep_heads = !ctx->use_chain;
    LAUNCH(CHIMERA_KIND_EMBED, 0, launch_trigram_gather(ctx->dtype, ctx->embed, d, V, ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_topk, K,
                                ctx->KMAX, k, ctx->tbuf, B, ctx->d_err, ctx->dres, s,
                                (sep_heads && k == 0) ? ctx->hlog : nullptr, static_cast<long long>(K) * B * V));
    if (ctx->tc_entries)
      LAUNCH(CHIMERA_KIND_OTHER, 0, launch_trigram_lookup(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_topk, K, ctx->KMAX, k,
                                                          B, d, ctx->tc_nsets, ctx->tc_keys, ctx->tc_stamp, ctx->tc_vals,
                                                          ctx->dres, ctx->tc_hit, ctx->tc_slot, ctx->tc_skip,
                                                          ctx->tc_clock, ctx->tc_hit_log, s));
    RUN(run_lin(ctx, ctx->tri1));
    RUN(run_lin(ctx, ctx->tri2));
    if (ctx->tc_entries)
      LAUNCH(CHIMERA_KIND_OTHER, 0, launch_trigram_insert(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_topk, K, ctx->KMAX, k,
                                                          B, d, ctx->tc_keys, ctx->tc_stamp, ctx->tc_vals, ctx->dres,
                                                          ctx->tc_hit, ctx->tc_slot, ctx->tc_clock, ctx->htri_log, s));
    if (ctx->use_chain) {
      RUN(run_chain(ctx, ctx->draft_chain_a[k]));
      RUN(run_attention(ctx, true, 0, 1, nullptr, k, k + 1, nullptr, ctx->d_chain, 1, ctx->att_splits_draft, 1,
                        kv_read_bytes(ctx, k + 1, true), ctx->qkv, k, nullptr));
      RUN(run_chain(ctx, ctx->draft_chain_b[k]));
      LAUNCH(CHIMERA_KIND_TOPK, 0, topk_rows(ctx->hlog + static_cast<size_t>(k) * B * V, V, B, ctx->KMAX,
                                             ctx->d_topk + k * ctx->KMAX, ctx->d_topk_val + k * ctx->KMAX, K * ctx->KMAX,
                                             ctx->topk_ws_v, ctx->topk_ws_i, ctx->topk_cnt, s));
      continue;
    }
    RUN(run_norm(ctx, ctx->dres, ctx->draft.attn_norm, B, ctx->qkv, 3 * d));
    RUN(run_lin(ctx, ctx->dqkv));
    if (attn_fuses_rope(ctx->dtype, ctx->hd)) {
      RUN(run_attention(ctx, true, 0, 1, nullptr, k, k + 1, nullptr, ctx->d_chain, 1, ctx->att_splits_draft, 1,
                        kv_read_bytes(ctx, k + 1, true), ctx->qkv, k, nullptr));
    } else {
      RUN(run_rope(ctx, true, 0, ctx->qkv, 3 * d, 0, d, 2 * d, 1, nullptr, 0, k, k, nullptr));
      RUN(run_attention(ctx, true, 0, 1, nullptr, k, k + 1, nullptr, ctx->d_chain, 1, ctx->att_splits_draft, 1,
                        kv_read_bytes(ctx, k + 1, true)));
    }
    RUN(run_lin(ctx, ctx->dwo));
    RUN(run_norm(ctx, ctx->dres, ctx->draft.ffn_norm, B, ctx->gu, 2 * ctx->F));
    RUN(run_lin(ctx, ctx->dgate));
    RUN(run_lin(ctx, ctx->dup));
    LAUNCH(CHIMERA_KIND_SWIGLU, 0, swiglu(ctx->dtype, ctx->gu, 2 * ctx->F, ctx->F, ctx->hf, ctx->hf_lo, ctx->F, B, s));
    RUN(run_lin(ctx, ctx->ddown));
    LAUNCH(CHIMERA_KIND_OTHER, 0, launch_hfull_store(ctx->dtype, ctx->dres, d, ctx->headin, ctx->headin_lo,
                             ctx->hfull_log + static_cast<size_t>(k) * B * d, nullptr, V, B, s));
    RUN(run_lin(ctx, ctx->dhead[k]));
    LAUNCH(CHIMERA_KIND_TOPK, 0, topk_rows(ctx->hlog + static_cast<size_t>(k) * B * V, V, B, ctx->KMAX, ctx->d_topk + k * ctx->KMAX,
                    ctx->d_topk_val + k * ctx->KMAX, K * ctx->KMAX, ctx->topk_ws_v, ctx->topk_ws_i,
                    ctx->topk_cnt, s));
  }
  // ---- tree ----
  ctx->cur_phase = CHIMERA_PHASE_VERIFY;
  RUN(mark_phase(ctx, 1));
  LAUNCH(CHIMERA_KIND_TREE, 0, launch_tree_expand(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_topk, K, ctx->KMAX, ctx->d_depth, ctx->d_rank,
                           N, ctx->d_ovr_flag, ctx->d_ovr, ctx->d_node_tok, B, s));
  // ---- verify: one base forward over every tree node ----
  LAUNCH(CHIMERA_KIND_EMBED, 0, embed(ctx->dtype, ctx->embed, d, V, ctx->x, B * N, N, ctx->d_node_tok, nullptr, 0, nullptr, nullptr,
              ctx->d_err, s));
  const double kvb = kv_read_bytes(ctx, N, false);
  if (ctx->use_chain) {
    RUN(enqueue_layers_chain(ctx, ctx->ver_chain, N, nullptr, ctx->d_depth, ctx->d_anc, ctx->att_splits_ver, kvb));
  } else {
    for (int l = 0; l < ctx->L; ++l)
      RUN(enqueue_layer(ctx, l, &ctx->ver[5 * l], B * N, N, nullptr, ctx->d_depth, ctx->d_anc, ctx->att_splits_ver,
                        kvb));
    RUN(run_final_norm(ctx, B * N, true));
    RUN(run_lin(ctx, ctx->ver_lm));
  }
  LAUNCH(CHIMERA_KIND_ARGMAX, 0, argmax_rows(ctx->logits, V, B * N, ctx->d_amax, s, ctx->d_stats));
  // ---- accept and commit ----
  ctx->cur_phase = CHIMERA_PHASE_COMMIT;
  RUN(mark_phase(ctx, 2));
  if (ctx->accept_mode == 1)
    LAUNCH(CHIMERA_KIND_ACCEPT, 0, launch_accept_typical(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_node_tok, ctx->d_amax,
                                                         ctx->logits, V, ctx->d_stats, ctx->d_parent, ctx->d_depth, N,
                                                         ctx->D1, ctx->typ_eps, ctx->typ_delta, ctx->d_path, ctx->d_L,
                                                         ctx->d_bonus, B, s));
  else
    LAUNCH(CHIMERA_KIND_ACCEPT, 0, launch_accept(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_node_tok, ctx->d_amax, ctx->d_child_start,
                        ctx->d_child, N, ctx->D1, ctx->d_path, ctx->d_L, ctx->d_bonus, B, s));
  LAUNCH(CHIMERA_KIND_COMPACT, 0, launch_compact(ctx->kv, ctx->kv_layer_stride * static_cast<long long>(ctx->kv_esz), ctx->L, ctx->H,
                       ctx->kv_planes, static_cast<int>(ctx->hd * ctx->kv_esz), ctx->d_n, ctx->d_path, ctx->d_L,
                       ctx->D1, ctx->d_pt, ctx->max_pages, B, s));
  LAUNCH(CHIMERA_KIND_OTHER, 0, launch_gather_hidden(ctx->dtype, ctx->hfin32, d, N, ctx->d_path, ctx->d_L, ctx->D1, ctx->hsel, ctx->headin,
                             ctx->headin_lo, B, s));
  if (ctx->use_chain) {
    RUN(run_chain(ctx, ctx->commit_chain));
  } else {
    RUN(run_norm(ctx, ctx->hsel, ctx->draft.attn_norm, B * ctx->D1, ctx->kvtmp, 2 * d));
    RUN(run_lin(ctx, ctx->commit_kv));
  }
  RUN(run_rope(ctx, true, 0, ctx->kvtmp, 2 * d, -1, 0, d, ctx->D1, ctx->d_L, 1, 0, 0, nullptr));
  LAUNCH(CHIMERA_KIND_OTHER, 0, launch_finalize(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_L, ctx->d_bonus, ctx->d_count_log, LOG_CAP,
                        ctx->d_step, B, s));
  RUN(mark_phase(ctx, 3));
  return cudaSuccess;
}

// One plain autoregressive step (eq. 1 with argmax; the baseline that speculative
// decoding accelerates): the base forward of each sequence's root x[n] at position n
// (one query row attending the committed rows and itself), LM head, argmax -> the next
// root; the root's base KV is written at slot n, its draft-layer KV appended and
// h_LLM_n refreshed, exactly as a draft-and-verify step that accepts nothing.
cudaError_t enqueue_ar_step(chimera_ctx* ctx) {
  const int B = ctx->batch, d = ctx->d, V = ctx->V;
  cudaStream_t s = ctx->stream;
  ctx->cur_phase = CHIMERA_PHASE_VERIFY;
  LAUNCH(CHIMERA_KIND_EMBED, 0, embed(ctx->dtype, ctx->embed, d, V, ctx->x, B, 1, nullptr, ctx->d_tok, ctx->tok_stride,
                                      ctx->d_n, ctx->d_one, ctx->d_err, s));
  const double kvb = kv_read_bytes(ctx, 1, false);
  if (ctx->use_chain) {
    RUN(enqueue_layers_chain(ctx, ctx->ar_chain, 1, nullptr, nullptr, ctx->d_chain, ctx->att_splits_ar, kvb));
  } else {
    for (int l = 0; l < ctx->L; ++l)
      RUN(enqueue_layer(ctx, l, &ctx->ar[5 * l], B, 1, nullptr, nullptr, ctx->d_chain, ctx->att_splits_ar, kvb));
    RUN(run_final_norm(ctx, B, true));
    RUN(run_lin(ctx, ctx->ar_lm));
  }
  LAUNCH(CHIMERA_KIND_ARGMAX, 0, argmax_rows(ctx->logits, V, B, ctx->d_amax, s));
  ctx->cur_phase = CHIMERA_PHASE_COMMIT;
  // a tree of the root alone: the path is [root], the bonus is its argmax
  LAUNCH(CHIMERA_KIND_ACCEPT, 0, launch_accept(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_node_tok, ctx->d_amax,
                                               ctx->d_child_start1, ctx->d_child1, 1, ctx->D1, ctx->d_path, ctx->d_L,
                                               ctx->d_bonus, B, s));
  LAUNCH(CHIMERA_KIND_OTHER, 0, launch_gather_hidden(ctx->dtype, ctx->hfin32, d, 1, ctx->d_path, ctx->d_L, ctx->D1,
                                                     ctx->hsel, ctx->headin, ctx->headin_lo, B, s));
  if (ctx->use_chain) {
    RUN(run_chain(ctx, ctx->commit_chain));
  } else {
    RUN(run_norm(ctx, ctx->hsel, ctx->draft.attn_norm, B * ctx->D1, ctx->kvtmp, 2 * d));
    RUN(run_lin(ctx, ctx->commit_kv));
  }
  RUN(run_rope(ctx, true, 0, ctx->kvtmp, 2 * d, -1, 0, d, ctx->D1, ctx->d_L, 1, 0, 0, nullptr));
  LAUNCH(CHIMERA_KIND_OTHER, 0, launch_finalize(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_L, ctx->d_bonus,
                                                ctx->d_count_log, LOG_CAP, ctx->d_step, B, s));
  return cudaSuccess;
}

// Capture the step into a graph with the given capture-time options.
cudaError_t capture_step(chimera_ctx* ctx, cudaGraphExec_t* out, bool ar = false) {
  cudaGraph_t g = nullptr;
  cudaError_t e = cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return e;
  e = ar ? enqueue_ar_step(ctx) : enqueue_step(ctx);
  cudaError_t e2 = cudaStreamEndCapture(ctx->stream, &g);
  if (e == cudaSuccess) e = e2;
  if (e == cudaSuccess) e = cudaGraphInstantiate(out, g, 0);
  if (g) cudaGraphDestroy(g);
  return e;
}

// ---------------------------------------------------------------------------
// chain plans (bf16 models)
// ---------------------------------------------------------------------------
struct ChainBuilder {
  chimera_ctx* ctx;
  ChainPlan* c;
  bool ok = true;
  char msg[256] = {0};
  ChainBuilder(chimera_ctx* x, ChainPlan* plan, int M) : ctx(x), c(plan) {
    if (chain_plan(c, M, ctx->split, msg, sizeof(msg)) != 0 || ctx->chain_bar_next >= CHAIN_BAR_BLOCKS) {
      fail_msg(msg[0] ? msg : "too many chain launches");
      return;
    }
    c->p.err = ctx->d_err;
    c->p.bars = ctx->chain_bars + static_cast<size_t>(ctx->chain_bar_next++) * CHAIN_BAR_INTS;
  }
  void fail_msg(const char* m) {
    if (ok) ctx->err = m;
    ok = false;
  }
  int gemm(int wait, const void* X, const void* X_lo, int ldx, int K, const void* W, int N, float* Y, int ldy,
           const void* W2 = nullptr, int N2 = 0) {
    if (!ok) return -1;
    const int st = chain_add_gemm(c, wait, X, X_lo, ldx, K, W, N, W2, N2, Y, ldy, msg, sizeof(msg));
    if (st < 0) fail_msg(msg);
    return st;
  }
  int row(int kind, int wait, const ChainRow& r) {
    if (!ok) return -1;
    const int st = chain_add_row(c, kind, wait, r, msg, sizeof(msg));
    if (st < 0) fail_msg(msg);
    return st;
  }
};

ChainRow norm_row(const chimera_ctx* ctx, const float* X, const void* g, void* Y, void* Y_lo, float* Z, int zcols,
                  int rows, float* Y32 = nullptr) {
  ChainRow r{};
  r.X = X;
  r.ldx = ctx->d;
  r.g = g;
  r.Y = Y;
  r.Y_lo = Y_lo;
  r.ldy = ctx->d;
  r.Y32 = Y32;
  r.ld32 = ctx->d;
  r.Z = Z;
  r.ldz = zcols;
  r.zcols = Z ? zcols : 0;
  r.rows = rows;
  r.cols = ctx->d;
  r.eps = ctx->cfg.rms_eps;
  return r;
}

ChainRow swiglu_row(const chimera_ctx* ctx, int rows) {
  ChainRow r{};
  r.X = ctx->gu;
  r.ldx = 2 * ctx->F;
  r.Y = ctx->hf;
  r.Y_lo = ctx->hf_lo;
  r.ldy = ctx->F;
  r.rows = rows;
  r.cols = ctx->F;
  return r;
}

// O projection .. down of layer l (or of the draft block `w`) appended to `b`, the
// residual stream `x` (M rows); returns the step index of the down projection.
int chain_ffn_half(chimera_ctx* ctx, ChainBuilder& b, const chimera_block_weights& w, float* x, int M) {
  const int d = ctx->d, F = ctx->F;
  const int sO = b.gemm(-1, ctx->ao, ctx->ao_lo, d, d, w.wo, d, x, d);
  const int sN = b.row(CH_NORM, sO, norm_row(ctx, x, w.ffn_norm, ctx->xn, ctx->xn_lo, ctx->gu, 2 * F, M));
  const int sG = b.gemm(sN, ctx->xn, ctx->xn_lo, d, d, w.w_gate, F, ctx->gu, 2 * F, w.w_up, F);
  const int sS = b.row(CH_SWIGLU, sG, swiglu_row(ctx, M));
  return b.gemm(sS, ctx->hf, ctx->hf_lo, F, F, w.w_down, d, x, d);
}

bool build_layer_chains(chimera_ctx* ctx, std::vector<ChainPlan>& ch, int M) {
  const int d = ctx->d, V = ctx->V, L = ctx->L;
  ch.assign(L + 1, ChainPlan());
  {
    ChainBuilder b(ctx, &ch[0], M);
    const int sN = b.row(CH_NORM, -1, norm_row(ctx, ctx->x, ctx->layers[0].attn_norm, ctx->xn, ctx->xn_lo, ctx->qkv,
                                               3 * d, M));
    b.gemm(sN, ctx->xn, ctx->xn_lo, d, d, ctx->layers[0].wqkv, 3 * d, ctx->qkv, 3 * d);
    if (!b.ok) return false;
  }
  for (int l = 0; l < L; ++l) {
    ChainBuilder b(ctx, &ch[l + 1], M);
    const int sD = chain_ffn_half(ctx, b, ctx->layers[l], ctx->x, M);
    if (l + 1 < L) {
      const int sN = b.row(CH_NORM, sD, norm_row(ctx, ctx->x, ctx->layers[l + 1].attn_norm, ctx->xn, ctx->xn_lo,
                                                 ctx->qkv, 3 * d, M));
      b.gemm(sN, ctx->xn, ctx->xn_lo, d, d, ctx->layers[l + 1].wqkv, 3 * d, ctx->qkv, 3 * d);
    } else {  // final norm (H_LLM rows, fp32 copy) and the LM head
      const int sF = b.row(CH_NORM, sD, norm_row(ctx, ctx->x, ctx->final_norm, ctx->hfin, ctx->hfin_lo, ctx->logits, V,
                                                 M, ctx->hfin32));
      b.gemm(sF, ctx->hfin, ctx->hfin_lo, d, d, ctx->lm_head, V, ctx->logits, V);
    }
    if (!b.ok) return false;
  }
  return true;
}

bool build_chains(chimera_ctx* ctx, int B) {
  const int d = ctx->d, V = ctx->V, K = ctx->K, N = ctx->N;
  ctx->chain_bar_next = 0;
  if (!build_layer_chains(ctx, ctx->ver_chain, B * N)) return false;
  if (!build_layer_chains(ctx, ctx->ar_chain, B)) return false;
  const chimera_block_weights& w = ctx->draft;
  const bool no_resid = (ctx->draft_mode & 2) != 0;
  const int hk = no_resid ? d : 2 * d;
  const void* hx = no_resid ? eoff(ctx, ctx->headin, d) : ctx->headin;
  const void* hx_lo = ctx->headin_lo ? (no_resid ? eoff(ctx, ctx->headin_lo, d) : ctx->headin_lo) : nullptr;
  ctx->draft_chain_a.assign(K, ChainPlan());
  ctx->draft_chain_b.assign(K, ChainPlan());
  for (int k = 0; k < K; ++k) {
    const bool head_only = k > 0 && (ctx->draft_mode & 1);
    if (!head_only) {
      ChainBuilder a(ctx, &ctx->draft_chain_a[k], B);
      const int sN = a.row(CH_NORM, -1, norm_row(ctx, ctx->dres, w.attn_norm, ctx->xn, ctx->xn_lo, ctx->qkv, 3 * d, B));
      a.gemm(sN, ctx->xn, ctx->xn_lo, d, d, w.wqkv, 3 * d, ctx->qkv, 3 * d);
      if (!a.ok) return false;
    }
    ChainBuilder b(ctx, &ctx->draft_chain_b[k], B);
    const int sD = head_only ? -1 : chain_ffn_half(ctx, b, w, ctx->dres, B);
    // h_full (the block output) into the head input [h_LLM_n ; h_full] and the per-head
    // log; the head's score rows cleared
    ChainRow cp{};
    cp.X = ctx->dres;
    cp.ldx = d;
    cp.Y = eoff(ctx, ctx->headin, d);
    cp.Y_lo = ctx->headin_lo ? eoff(ctx, ctx->headin_lo, d) : nullptr;
    cp.ldy = 2 * d;
    cp.Y32 = ctx->hfull_log + static_cast<size_t>(k) * B * d;
    cp.ld32 = d;
    cp.Z = ctx->hlog + static_cast<size_t>(k) * B * V;
    cp.ldz = V;
    cp.zcols = V;
    cp.rows = B;
    cp.cols = d;
    const int sC = b.row(CH_COPY, sD, cp);
    b.gemm(sC, hx, hx_lo, 2 * d, hk, ctx->heads[k], V, ctx->hlog + static_cast<size_t>(k) * B * V, V);
    if (!b.ok) return false;
  }
  {
    ChainBuilder c(ctx, &ctx->commit_chain, B * ctx->D1);
    const int sN = c.row(CH_NORM, -1, norm_row(ctx, ctx->hsel, w.attn_norm, ctx->xn, ctx->xn_lo, ctx->kvtmp, 2 * d,
                                               B * ctx->D1));
    const void* dl_kv = eoff(ctx, const_cast<void*>(w.wqkv), static_cast<size_t>(d) * d);
    c.gemm(sN, ctx->xn, ctx->xn_lo, d, d, dl_kv, 2 * d, ctx->kvtmp, 2 * d);
    if (!c.ok) return false;
  }
  return true;
}

// (Re)build every linear call site for `batch` sequences.
bool build_plans(chimera_ctx* ctx, int B) {
  const int d = ctx->d, F = ctx->F, V = ctx->V, N = ctx->N;
  const int f32 = 1, tb = ctx->dtype == 0 ? 1 : 0;  // bf16 storage -> out_f32 = 0
  ctx->ver.assign(5 * ctx->L, Lin());
  ctx->pre.assign(5 * ctx->L, Lin());
  ctx->ar.assign(5 * ctx->L, Lin());
  // fp32 outputs accumulate (split-K partials added atomically) into buffers that the
  // preceding kernel zeroed, or into the residual stream itself
  constexpr int ACC = EPI_RESID;
  void *xn = ctx->xn, *xl = ctx->xn_lo, *ao = ctx->ao, *al = ctx->ao_lo, *hf = ctx->hf, *hl = ctx->hf_lo;
  auto layer_plans = [&](std::vector<Lin>& v, int M) {
    for (int l = 0; l < ctx->L; ++l) {
      const chimera_block_weights& w = ctx->layers[l];
      Lin* p = &v[5 * l];
      if (!make_lin(ctx, &p[0], M, 3 * d, d, xn, xl, d, w.wqkv, ctx->qkv, nullptr, 3 * d, ACC, f32)) return false;
      // the O linear clears the gate|up accumulator of this layer, the down linear the
      // QKV accumulator of the next one (their epilogue warps, off the critical path)
      if (!make_lin(ctx, &p[1], M, d, d, ao, al, d, w.wo, ctx->x, nullptr, d, ACC, f32, nullptr, 0,
                    ctx->tc_zero ? ctx->gu : nullptr, static_cast<long long>(M) * 2 * F))
        return false;
      // gate and up: one launch writing gu[:, 0:F] and gu[:, F:2F]
      if (!make_lin(ctx, &p[2], M, F, d, xn, xl, d, w.w_gate, ctx->gu, nullptr, 2 * F, ACC, f32, w.w_up, F))
        return false;
      p[3] = Lin();  // N = 0: nothing to launch
      if (!make_lin(ctx, &p[4], M, d, F, hf, hl, F, w.w_down, ctx->x, nullptr, d, ACC, f32, nullptr, 0,
                    ctx->tc_zero ? ctx->qkv : nullptr, static_cast<long long>(M) * 3 * d))
        return false;
    }
    return true;
  };
  if (!layer_plans(ctx->ver, B * N)) return false;
  if (!layer_plans(ctx->ar, B)) return false;
  if (!make_lin(ctx, &ctx->ar_lm, B, V, d, ctx->hfin, ctx->hfin_lo, d, ctx->lm_head, ctx->logits, nullptr, V, ACC,
                f32))
    return false;
  if (!layer_plans(ctx->pre, B * CHUNK)) return false;
  if (!make_lin(ctx, &ctx->ver_lm, B * N, V, d, ctx->hfin, ctx->hfin_lo, d, ctx->lm_head, ctx->logits, nullptr, V,
                ACC, f32))
    return false;
  if (!make_lin(ctx, &ctx->pre_lm, B, V, d, ctx->headin, ctx->headin_lo, 2 * d, ctx->lm_head, ctx->logits, nullptr, V,
                ACC, f32))
    return false;
  const void* dl_kv = eoff(ctx, const_cast<void*>(ctx->draft.wqkv), static_cast<size_t>(d) * d);
  if (!make_lin(ctx, &ctx->pre_dkv, B * CHUNK, 2 * d, d, xn, xl, d, dl_kv, ctx->kvtmp, nullptr, 2 * d, ACC, f32))
    return false;
  if (!make_lin(ctx, &ctx->commit_kv, B * ctx->D1, 2 * d, d, xn, xl, d, dl_kv, ctx->kvtmp, nullptr, 2 * d, ACC,
                f32))
    return false;
  // draft (M = B rows); the trigram input is a gather of bf16 embeddings: exact, no lo half
  // W2 stores h_tri (partials summed in a fixed order): the same trigram always gives
  // the same row, so a cached row equals a recomputed one bit for bit
  if (!make_lin(ctx, &ctx->tri1, B, d, 3 * d, ctx->tbuf, nullptr, 3 * d, ctx->tri_w1, ctx->ubuf, ctx->ubuf_lo, d,
                EPI_SILU, tb, nullptr, 0, nullptr, 0, ctx->tc_skip))
    return false;
  if (!make_lin(ctx, &ctx->tri2, B, d, d, ctx->ubuf, ctx->ubuf_lo, d, ctx->tri_w2, ctx->dres, nullptr, d, EPI_STORE,
                f32, nullptr, 0, nullptr, 0, ctx->tc_skip))
    return false;
  const chimera_block_weights& w = ctx->draft;
  if (!make_lin(ctx, &ctx->dqkv, B, 3 * d, d, xn, xl, d, w.wqkv, ctx->qkv, nullptr, 3 * d, ACC, f32)) return false;
  if (!make_lin(ctx, &ctx->dwo, B, d, d, ao, al, d, w.wo, ctx->dres, nullptr, d, ACC, f32)) return false;
  if (!make_lin(ctx, &ctx->dgate, B, F, d, xn, xl, d, w.w_gate, ctx->gu, nullptr, 2 * F, ACC, f32, w.w_up, F))
    return false;
  ctx->dup = Lin();
  if (!make_lin(ctx, &ctx->ddown, B, d, F, hf, hl, F, w.w_down, ctx->dres, nullptr, d, ACC, f32)) return false;
  ctx->dhead.assign(ctx->K, Lin());
  // residual heads read [h_LLM_n ; h_full] (2d); heads without the residual h_full alone
  const bool no_resid = (ctx->draft_mode & 2) != 0;
  const int hk = no_resid ? d : 2 * d;
  const void* hx = no_resid ? eoff(ctx, ctx->headin, d) : ctx->headin;
  const void* hx_lo = ctx->headin_lo ? (no_resid ? eoff(ctx, ctx->headin_lo, d) : ctx->headin_lo) : nullptr;
  for (int k = 0; k < ctx->K; ++k)
    if (!make_lin(ctx, &ctx->dhead[k], B, V, hk, hx, hx_lo, 2 * d, ctx->heads[k],
                  ctx->hlog + static_cast<size_t>(k) * B * V, nullptr, V, ACC, f32))
      return false;
  ctx->att_splits_ver = att_splits(ctx, B, N, ctx->plan_keys + N);
  ctx->att_splits_pre = att_splits(ctx, B, CHUNK, ctx->plan_keys);
  ctx->att_splits_draft = att_splits(ctx, B, 1, ctx->plan_keys);
  ctx->att_splits_ar = att_splits(ctx, B, 1, ctx->plan_keys + 1);
  if (ctx->use_chain && !build_chains(ctx, B)) return false;
  return true;
}

// The pinned mirror may still be read by the last upload: wait for it before editing.
void pt_wait(chimera_ctx* ctx) {
  if (ctx->pt_inflight) {
    cudaEventSynchronize(ctx->pt_event);
    ctx->pt_inflight = false;
  }
}

chimera_status ensure_blocks(chimera_ctx* ctx, int b, int slots) {
  pt_wait(ctx);
  if (slots > ctx->cap)
    return fail(ctx, CHIMERA_ECAPACITY, "sequence " + std::to_string(b) + " needs " + std::to_string(slots) +
                                            " KV slots > max_seq_len " + std::to_string(ctx->cap));
  auto& blocks = ctx->seq_blocks[b];
  while (static_cast<int>(blocks.size()) * 16 < slots) {
    if (ctx->free_blocks.empty()) return fail(ctx, CHIMERA_ECAPACITY, "KV block pool exhausted");
    const int blk = ctx->free_blocks.back();
    ctx->free_blocks.pop_back();
    ctx->h_pt[b * ctx->max_pages + blocks.size()] = blk;
    blocks.push_back(blk);
    ctx->pt_dirty = true;
  }
  return CHIMERA_OK;
}

chimera_status flush_page_table(chimera_ctx* ctx) {
  if (!ctx->pt_dirty) return CHIMERA_OK;
  CK(cudaMemcpyAsync(ctx->d_pt, ctx->h_pt, ctx->h_pt_len * sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaEventRecord(ctx->pt_event, ctx->stream));
  ctx->pt_inflight = true;
  ctx->pt_dirty = false;
  return CHIMERA_OK;
}

chimera_status check_err(chimera_ctx* ctx) {
  int e = 0;
  CK(cudaMemcpyAsync(&ctx->h_stage[0], ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  e = ctx->h_stage[0];
  if (e == 0) return CHIMERA_OK;
  CK(cudaMemsetAsync(ctx->d_err, 0, sizeof(int), ctx->stream));
  if ((e & ERR_TIMEOUT) && ctx->chain_bars)  // an aborted chain can leave step counters raised
    CK(cudaMemsetAsync(ctx->chain_bars, 0, static_cast<size_t>(CHAIN_BAR_BLOCKS) * CHAIN_BAR_INTS * sizeof(int),
                       ctx->stream));
  if (e & ERR_TIMEOUT) return fail(ctx, CHIMERA_ETIMEDOUT, "a bounded device wait timed out");
  if (e & ERR_CAPACITY) return fail(ctx, CHIMERA_ECAPACITY, "a kernel hit the KV capacity bound");
  return fail(ctx, CHIMERA_EINVAL, "a kernel saw an out-of-range token id or index");
}

chimera_status steps_prepare(chimera_ctx* ctx, int n_steps) {
  if (!ctx->prefilled) return fail(ctx, CHIMERA_ESTATE, "step before prefill");
  const int need = std::max(ctx->N, ctx->K) + 1;
  for (int b = 0; b < ctx->batch; ++b) {
    const long long slots = static_cast<long long>(ctx->host_n[b]) + static_cast<long long>(n_steps - 1) * ctx->D1 + need +
                            ctx->D1;
    if (slots > ctx->cap)
      return fail(ctx, CHIMERA_ECAPACITY, "sequence " + std::to_string(b) + " would exceed max_seq_len");
    chimera_status st = ensure_blocks(ctx, b, static_cast<int>(slots));
    if (st != CHIMERA_OK) return st;
  }
  return flush_page_table(ctx);
}

chimera_status launch_steps(chimera_ctx* ctx, int n_steps) {
  if (!ctx->graph) {
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
    cudaError_t e = enqueue_step(ctx);
    cudaError_t e2 = cudaStreamEndCapture(ctx->stream, &g);
    if (e != cudaSuccess || e2 != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      return fail(ctx, CHIMERA_ECUDA, std::string("capturing the step: ") + cudaGetErrorString(e != cudaSuccess ? e : e2));
    }
    e = cudaGraphInstantiate(&ctx->graph, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) return fail(ctx, CHIMERA_ECUDA, std::string("instantiating the step graph: ") + cudaGetErrorString(e));
  }
  if (ctx->ovr_pending) {
    const int one = 1;
    CK(cudaMemcpyAsync(ctx->d_ovr_flag, &one, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  }
  for (int i = 0; i < n_steps; ++i) {
    CK(cudaGraphLaunch(ctx->graph, ctx->stream));
    if (i == 0 && ctx->ovr_pending) {
      CK(cudaMemsetAsync(ctx->d_ovr_flag, 0, sizeof(int), ctx->stream));
      ctx->ovr_pending = false;
    }
  }
  return CHIMERA_OK;
}

chimera_status read_new_tokens(chimera_ctx* ctx, int32_t* out_tokens, int per_seq, int32_t* out_count) {
  const int B = ctx->batch;
  std::vector<int> n_new(B);
  CK(cudaMemcpyAsync(n_new.data(), ctx->d_n, B * sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  chimera_status st = check_err(ctx);
  if (st != CHIMERA_OK) return st;
  for (int b = 0; b < B; ++b) {
    const int cnt = n_new[b] - ctx->host_n[b];
    if (cnt < 1 || cnt > per_seq) return fail(ctx, CHIMERA_ECUDA, "inconsistent committed length after a step");
    CK(cudaMemcpyAsync(out_tokens + static_cast<size_t>(b) * per_seq,
                       ctx->d_tok + static_cast<size_t>(b) * ctx->tok_stride + ctx->host_n[b], cnt * sizeof(int),
                       cudaMemcpyDeviceToHost, ctx->stream));
    out_count[b] = cnt;
  }
  CK(cudaStreamSynchronize(ctx->stream));
  for (int b = 0; b < B; ++b) ctx->host_n[b] = n_new[b];
  return CHIMERA_OK;
}

void free_ctx(chimera_ctx* ctx) {
  if (!ctx) return;
  if (ctx->graph) cudaGraphExecDestroy(ctx->graph);
  if (ctx->prof_graph) cudaGraphExecDestroy(ctx->prof_graph);
  if (ctx->phase_graph) cudaGraphExecDestroy(ctx->phase_graph);
  if (ctx->class_graph) cudaGraphExecDestroy(ctx->class_graph);
  if (ctx->ar_graph) cudaGraphExecDestroy(ctx->ar_graph);
  for (auto& e : ctx->phase_ev)
    if (e) cudaEventDestroy(e);
  for (auto& e : ctx->prof_ev) {
    cudaEventDestroy(e.a);
    cudaEventDestroy(e.b);
  }
  for (void* p : ctx->allocs) cudaFree(p);
  if (ctx->h_stage) cudaFreeHost(ctx->h_stage);
  if (ctx->h_pt) cudaFreeHost(ctx->h_pt);
  if (ctx->pt_event) cudaEventDestroy(ctx->pt_event);
  if (ctx->own_stream && ctx->stream) cudaStreamDestroy(ctx->stream);
  delete ctx;
}

bool valid_block(const chimera_block_weights& b) {
  return b.attn_norm && b.wqkv && b.wo && b.ffn_norm && b.w_gate && b.w_up && b.w_down;
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================
extern "C" {

chimera_status chimera_init(const chimera_config* cfg, const chimera_weights* w, void* cuda_stream,
                            chimera_ctx** out) {
  if (!out) return CHIMERA_EINVAL;
  *out = nullptr;
  if (!cfg || !w) return CHIMERA_EINVAL;
  const chimera_config& c = *cfg;
  if (c.n_layers < 1 || c.d_model < 32 || c.n_heads < 1 || c.head_dim * c.n_heads != c.d_model ||
      (c.head_dim != 64 && c.head_dim != 128) || c.ffn_dim < 8 || c.vocab < 8 || (c.dtype != 0 && c.dtype != 1) ||
      c.n_draft_heads < 1 || c.n_draft_heads > 4 || c.tree_nodes < 2 || c.tree_nodes > 64 || c.max_batch < 1 ||
      c.max_batch > 64 || c.kv_block != 16 || c.max_seq_len < 32 || !(c.rms_eps > 0) || !(c.rope_theta > 0) ||
      (c.precision != 0 && c.precision != 1))
    return CHIMERA_EINVAL;
  if (c.dtype == 1 && (c.d_model % 64 != 0 || c.ffn_dim % 128 != 0)) return CHIMERA_EINVAL;
  if (c.draft_mode < 0 || c.draft_mode > 3 || (c.accept_mode != 0 && c.accept_mode != 1) ||
      (c.fused_chain != 0 && c.fused_chain != 1))
    return CHIMERA_EINVAL;
  if (c.accept_mode == 1 && (!(c.typical_eps >= 0.f) || !(c.typical_delta >= 0.f))) return CHIMERA_EINVAL;
  if (c.trigram_cache < 0 || c.trigram_cache > 65536 ||
      (c.trigram_cache && (c.trigram_cache % 4 || ((c.trigram_cache / 4) & (c.trigram_cache / 4 - 1)))))
    return CHIMERA_EINVAL;
  // row kernels read 16-byte vectors; the top-k covers at most 64 slices of 2048 scores
  if ((c.d_model & 3) || (c.ffn_dim & 3) || (c.vocab & 3) || c.vocab > TOPK_MAX_BLOCKS * 2048) return CHIMERA_EINVAL;
  for (int k = 0; k < c.n_draft_heads; ++k)
    if (c.topk[k] < 1 || c.topk[k] > MAX_KMAX) return CHIMERA_EINVAL;
  if (!w->embed || !w->layers || !w->final_norm || !w->lm_head || !w->tri_w1 || !w->tri_w2 || !w->heads ||
      !valid_block(w->draft))
    return CHIMERA_EINVAL;
  for (int l = 0; l < c.n_layers; ++l)
    if (!valid_block(w->layers[l])) return CHIMERA_EINVAL;
  for (int k = 0; k < c.n_draft_heads; ++k)
    if (!w->heads[k]) return CHIMERA_EINVAL;

  chimera_ctx* ctx = new chimera_ctx();
  ctx->cfg = c;
  ctx->L = c.n_layers;
  ctx->d = c.d_model;
  ctx->H = c.n_heads;
  ctx->hd = c.head_dim;
  ctx->F = c.ffn_dim;
  ctx->V = c.vocab;
  ctx->K = c.n_draft_heads;
  ctx->N = c.tree_nodes;
  ctx->dtype = c.dtype;
  ctx->esz = c.dtype == 0 ? 4 : 2;
  ctx->split = (c.dtype == 1 && c.precision == 1) ? 1 : 0;
  ctx->kv_planes = ctx->split ? 4 : 2;
  ctx->kv_esz = ctx->esz;
  ctx->Bmax = c.max_batch;
  ctx->cap = c.max_seq_len;
  ctx->KMAX = 1;
  for (int k = 0; k < ctx->K; ++k) ctx->KMAX = std::max(ctx->KMAX, c.topk[k]);
  std::string terr;
  if (!build_tree(c.topk, ctx->K, ctx->N, &ctx->tree, &terr)) {
    ctx->err = terr;
    free_ctx(ctx);
    return CHIMERA_EINVAL;
  }
  ctx->D1 = ctx->tree.depth_max + 1;
  ctx->draft_mode = c.draft_mode;
  ctx->accept_mode = c.accept_mode;
  ctx->typ_eps = c.typical_eps;
  ctx->typ_delta = c.typical_delta;
  ctx->tc_entries = c.trigram_cache;
  ctx->tc_nsets = c.trigram_cache / 4;
  ctx->embed = w->embed;
  ctx->layers.assign(w->layers, w->layers + c.n_layers);
  ctx->draft = w->draft;
  ctx->final_norm = w->final_norm;
  ctx->lm_head = w->lm_head;
  ctx->tri_w1 = w->tri_w1;
  ctx->tri_w2 = w->tri_w2;
  ctx->heads.assign(w->heads, w->heads + c.n_draft_heads);
  ctx->num_sms = tc_num_sms();
  // the weights may have been written on any stream (an own stream is not ordered after
  // them): let every earlier piece of device work finish before this context reads them
  if (cudaDeviceSynchronize() != cudaSuccess) {
    free_ctx(ctx);
    return CHIMERA_ECUDA;
  }

  if (cuda_stream) {
    ctx->stream = static_cast<cudaStream_t>(cuda_stream);
  } else {
    if (cudaStreamCreateWithFlags(&ctx->stream, cudaStreamNonBlocking) != cudaSuccess) {
      free_ctx(ctx);
      return CHIMERA_ECUDA;
    }
    ctx->own_stream = true;
  }

  const int B = ctx->Bmax, d = ctx->d, F = ctx->F, V = ctx->V, N = ctx->N, K = ctx->K;
  ctx->tok_stride = ctx->cap + 1;
  ctx->max_pages = (ctx->cap + 15) / 16;
  ctx->NB = B * ctx->max_pages;
  ctx->kv_layer_stride = static_cast<long long>(ctx->NB) * ctx->H * ctx->kv_planes * 16 * ctx->hd;
  ctx->max_pos = ctx->cap + 64;
  ctx->R = B * std::max(N, CHUNK);
  const int Rc = B * std::max(CHUNK, ctx->D1);
  bool ok = true;
  const size_t Rx = static_cast<size_t>(std::max(ctx->R, Rc));
  const bool sp = ctx->split != 0;
  ok = ok && dalloc_bytes(ctx, &ctx->kv, static_cast<size_t>(ctx->kv_layer_stride) * ctx->L * ctx->kv_esz);
  ok = ok && dalloc_bytes(ctx, &ctx->dkv, static_cast<size_t>(ctx->kv_layer_stride) * ctx->kv_esz);
  ok = ok && dalloc(ctx, &ctx->d_pt, static_cast<size_t>(B) * ctx->max_pages);
  ok = ok && dalloc(ctx, &ctx->d_rope, static_cast<size_t>(ctx->max_pos) * (ctx->hd / 2));
  ok = ok && dalloc(ctx, &ctx->x, static_cast<size_t>(ctx->R) * d);
  ok = ok && dalloc_bytes(ctx, &ctx->xn, Rx * d * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->xn_lo, Rx * d * ctx->esz);
  ok = ok && dalloc(ctx, &ctx->qkv, static_cast<size_t>(ctx->R) * 3 * d);
  ctx->tc_zero = ctx->dtype == 1;
  ok = ok && dalloc(ctx, &ctx->qr, static_cast<size_t>(ctx->R) * d);
  ok = ok && dalloc_bytes(ctx, &ctx->ao, static_cast<size_t>(ctx->R) * d * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->ao_lo, static_cast<size_t>(ctx->R) * d * ctx->esz);
  ok = ok && dalloc(ctx, &ctx->gu, static_cast<size_t>(ctx->R) * 2 * F);
  ok = ok && dalloc_bytes(ctx, &ctx->hf, static_cast<size_t>(ctx->R) * F * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->hf_lo, static_cast<size_t>(ctx->R) * F * ctx->esz);
  ok = ok && dalloc_bytes(ctx, &ctx->hfin, static_cast<size_t>(ctx->R) * d * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->hfin_lo, static_cast<size_t>(ctx->R) * d * ctx->esz);
  ok = ok && dalloc(ctx, &ctx->hfin32, static_cast<size_t>(ctx->R) * d);
  ok = ok && dalloc(ctx, &ctx->logits, static_cast<size_t>(B) * N * V);
  ok = ok && dalloc_bytes(ctx, &ctx->tbuf, static_cast<size_t>(B) * 3 * d * ctx->esz);
  ok = ok && dalloc_bytes(ctx, &ctx->ubuf, static_cast<size_t>(B) * d * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->ubuf_lo, static_cast<size_t>(B) * d * ctx->esz);
  ok = ok && dalloc(ctx, &ctx->dres, static_cast<size_t>(B) * d);
  ok = ok && dalloc_bytes(ctx, &ctx->headin, static_cast<size_t>(B) * 2 * d * ctx->esz);
  if (sp) ok = ok && dalloc_bytes(ctx, &ctx->headin_lo, static_cast<size_t>(B) * 2 * d * ctx->esz);
  ok = ok && dalloc(ctx, &ctx->hfull_log, static_cast<size_t>(K) * B * d);
  ok = ok && dalloc(ctx, &ctx->hlog, static_cast<size_t>(K) * B * V);
  ok = ok && dalloc(ctx, &ctx->hsel, static_cast<size_t>(B) * ctx->D1 * d);
  ok = ok && dalloc(ctx, &ctx->kvtmp, static_cast<size_t>(Rc) * 2 * d);
  ok = ok && dalloc(ctx, &ctx->d_n, B);
  ok = ok && dalloc(ctx, &ctx->d_tok, static_cast<size_t>(B) * ctx->tok_stride);
  ok = ok && dalloc(ctx, &ctx->d_node_tok, static_cast<size_t>(B) * N);
  ok = ok && dalloc(ctx, &ctx->d_topk, static_cast<size_t>(B) * K * ctx->KMAX);
  ok = ok && dalloc(ctx, &ctx->d_topk_val, static_cast<size_t>(B) * K * ctx->KMAX);
  ok = ok && dalloc(ctx, &ctx->d_amax, static_cast<size_t>(std::max(B * N, B)));
  ok = ok && dalloc(ctx, &ctx->d_path, static_cast<size_t>(B) * ctx->D1);
  ok = ok && dalloc(ctx, &ctx->d_L, B);
  ok = ok && dalloc(ctx, &ctx->d_bonus, B);
  ok = ok && dalloc(ctx, &ctx->d_ovr, static_cast<size_t>(B) * N);
  ok = ok && dalloc(ctx, &ctx->d_ovr_flag, 1);
  ok = ok && dalloc(ctx, &ctx->d_valid, B);
  ok = ok && dalloc(ctx, &ctx->d_last, B);
  ok = ok && dalloc(ctx, &ctx->d_count_log, static_cast<size_t>(B) * LOG_CAP);
  ok = ok && dalloc(ctx, &ctx->d_step, 1);
  ok = ok && dalloc(ctx, &ctx->d_err, 1);
  ok = ok && dalloc(ctx, &ctx->d_depth, N);
  ok = ok && dalloc(ctx, &ctx->d_rank, N);
  ok = ok && dalloc(ctx, &ctx->d_anc, N);
  ok = ok && dalloc(ctx, &ctx->d_chain, 64);
  ok = ok && dalloc(ctx, &ctx->d_child_start, N + 1);
  ok = ok && dalloc(ctx, &ctx->d_child, ctx->tree.child.size());
  ok = ok && dalloc(ctx, &ctx->d_one, B);
  ok = ok && dalloc(ctx, &ctx->d_parent, N);
  if (ctx->accept_mode == 1) ok = ok && dalloc(ctx, &ctx->d_stats, static_cast<size_t>(B) * N * 3);
  if (ctx->tc_entries) {
    ok = ok && dalloc(ctx, &ctx->tc_keys, ctx->tc_entries);
    ok = ok && dalloc(ctx, &ctx->tc_stamp, ctx->tc_entries);
    ok = ok && dalloc(ctx, &ctx->tc_vals, static_cast<size_t>(ctx->tc_entries) * d);
    ok = ok && dalloc(ctx, &ctx->tc_hit, B);
    ok = ok && dalloc(ctx, &ctx->tc_slot, B);
    ok = ok && dalloc(ctx, &ctx->tc_skip, 1);
    ok = ok && dalloc(ctx, &ctx->tc_clock, 1);
    ok = ok && dalloc(ctx, &ctx->tc_hit_log, static_cast<size_t>(K) * B);
    ok = ok && dalloc(ctx, &ctx->htri_log, static_cast<size_t>(K) * B * d);
  }
  ok = ok && dalloc(ctx, &ctx->d_child_start1, 2);
  ok = ok && dalloc(ctx, &ctx->d_child1, 1);
  // bf16 models with fused_chain run the linears and row steps between two attentions
  // as one persistent chain launch; otherwise every linear and row kernel is launched
  // on its own (the default: faster on this GPU, see the chain kernel's notes)
  ctx->use_chain = ctx->dtype == 1 && c.fused_chain == 1;
  if (ctx->use_chain) ok = ok && dalloc(ctx, &ctx->chain_bars, static_cast<size_t>(CHAIN_BAR_BLOCKS) * CHAIN_BAR_INTS);
  if (ctx->dtype == 1) {
    ok = ok && dalloc(ctx, &ctx->lin_ws, tc_ws_floats(256));
    ok = ok && dalloc(ctx, &ctx->lin_cnt, static_cast<size_t>(tc_max_tiles()));
  }
  ctx->att_ws_floats = attn_ws_floats(B, ctx->H, 16, std::max(N, CHUNK), ctx->hd);
  ok = ok && dalloc(ctx, &ctx->att_ws, ctx->att_ws_floats);
  ok = ok && dalloc(ctx, &ctx->att_cnt, static_cast<size_t>(B) * ctx->H);
  ok = ok && dalloc(ctx, &ctx->topk_ws_v, static_cast<size_t>(B) * TOPK_MAX_BLOCKS * 8);
  ok = ok && dalloc(ctx, &ctx->topk_ws_i, static_cast<size_t>(B) * TOPK_MAX_BLOCKS * 8);
  ok = ok && dalloc(ctx, &ctx->topk_cnt, static_cast<size_t>(B));
  if (ok && cudaMallocHost(reinterpret_cast<void**>(&ctx->h_stage), 4096 * sizeof(int)) != cudaSuccess) ok = false;
  ctx->h_pt_len = static_cast<size_t>(B) * ctx->max_pages;
  if (ok && cudaMallocHost(reinterpret_cast<void**>(&ctx->h_pt), ctx->h_pt_len * sizeof(int)) != cudaSuccess) ok = false;
  if (ok && cudaEventCreateWithFlags(&ctx->pt_event, cudaEventDisableTiming) != cudaSuccess) ok = false;
  if (!ok) {
    free_ctx(ctx);
    return CHIMERA_ENOMEM;
  }
  ctx->h_stage_ints = 4096;

  // zero-initialised state and scratch
  cudaStream_t s = ctx->stream;
  bool zok = true;
  zok = zok && cudaMemsetAsync(ctx->kv, 0, static_cast<size_t>(ctx->kv_layer_stride) * ctx->L * ctx->kv_esz, s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->dkv, 0, static_cast<size_t>(ctx->kv_layer_stride) * ctx->kv_esz, s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->att_cnt, 0, static_cast<size_t>(B) * ctx->H * sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->topk_cnt, 0, static_cast<size_t>(B) * sizeof(int), s) == cudaSuccess;
  if (ctx->lin_cnt)
    zok = zok && cudaMemsetAsync(ctx->lin_cnt, 0, static_cast<size_t>(tc_max_tiles()) * sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_err, 0, sizeof(int), s) == cudaSuccess;
  if (ctx->chain_bars)
    zok = zok && cudaMemsetAsync(ctx->chain_bars, 0, static_cast<size_t>(CHAIN_BAR_BLOCKS) * CHAIN_BAR_INTS * sizeof(int),
                                 s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_ovr_flag, 0, sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_step, 0, sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_topk, 0, static_cast<size_t>(B) * K * ctx->KMAX * sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->headin, 0, static_cast<size_t>(B) * 2 * d * ctx->esz, s) == cudaSuccess;
  if (ctx->headin_lo)
    zok = zok && cudaMemsetAsync(ctx->headin_lo, 0, static_cast<size_t>(B) * 2 * d * ctx->esz, s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->x, 0, static_cast<size_t>(ctx->R) * d * sizeof(float), s) == cudaSuccess;

  // tree, chain masks and the RoPE table (fp64 on the host, rounded to fp32)
  std::vector<unsigned long long> chain(64);
  for (int i = 0; i < 64; ++i) chain[i] = i == 63 ? ~0ull : ((1ull << (i + 1)) - 1);
  const int half = ctx->hd / 2;
  std::vector<float2> rope(static_cast<size_t>(ctx->max_pos) * half);
  for (int p = 0; p < ctx->max_pos; ++p)
    for (int j = 0; j < half; ++j) {
      const double inv = std::pow(static_cast<double>(c.rope_theta), -2.0 * j / ctx->hd);
      const double a = static_cast<double>(p) * inv;
      rope[static_cast<size_t>(p) * half + j] = make_float2(static_cast<float>(std::cos(a)), static_cast<float>(std::sin(a)));
    }
  const Tree& t = ctx->tree;
  std::vector<unsigned long long> anc(t.anc.begin(), t.anc.end());
  zok = zok && cudaMemcpyAsync(ctx->d_depth, t.depth.data(), N * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_rank, t.rank.data(), N * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_anc, anc.data(), N * sizeof(unsigned long long), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_chain, chain.data(), 64 * sizeof(unsigned long long), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_child_start, t.child_start.data(), (N + 1) * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_child, t.child.data(), t.child.size() * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice, s) == cudaSuccess;
  const std::vector<int> ones(B, 1);
  zok = zok && cudaMemcpyAsync(ctx->d_one, ones.data(), B * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_child_start1, 0, 2 * sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemsetAsync(ctx->d_child1, 0, sizeof(int), s) == cudaSuccess;
  zok = zok && cudaMemcpyAsync(ctx->d_parent, t.parent.data(), N * sizeof(int), cudaMemcpyHostToDevice, s) == cudaSuccess;
  if (ctx->tc_entries) {
    zok = zok && cudaMemsetAsync(ctx->tc_keys, 0, ctx->tc_entries * sizeof(unsigned long long), s) == cudaSuccess;
    zok = zok && cudaMemsetAsync(ctx->tc_stamp, 0, ctx->tc_entries * sizeof(int), s) == cudaSuccess;
    zok = zok && cudaMemsetAsync(ctx->tc_clock, 0, sizeof(int), s) == cudaSuccess;
    zok = zok && cudaMemsetAsync(ctx->tc_hit_log, 0, static_cast<size_t>(K) * B * sizeof(int), s) == cudaSuccess;
  }
  zok = zok && cudaStreamSynchronize(s) == cudaSuccess;
  if (!zok) {
    free_ctx(ctx);
    return CHIMERA_ECUDA;
  }
  std::fill(ctx->h_pt, ctx->h_pt + ctx->h_pt_len, 0);
  ctx->seq_blocks.assign(B, {});
  ctx->free_blocks.clear();
  for (int i = ctx->NB - 1; i >= 0; --i) ctx->free_blocks.push_back(i);
  *out = ctx;
  return CHIMERA_OK;
}

chimera_status chimera_prefill(chimera_ctx* ctx, int batch, const int32_t* tokens, const int32_t* lens) {
  if (!ctx) return CHIMERA_EINVAL;
  if (batch < 1 || batch > ctx->Bmax || !tokens || !lens) return fail(ctx, CHIMERA_EINVAL, "bad batch or NULL input");
  long long total = 0;
  int max_len = 0;
  for (int b = 0; b < batch; ++b) {
    if (lens[b] < 1) return fail(ctx, CHIMERA_EINVAL, "empty prompt");
    total += lens[b];
    max_len = std::max(max_len, static_cast<int>(lens[b]));
  }
  for (long long i = 0; i < total; ++i)
    if (tokens[i] < 0 || tokens[i] >= ctx->V) return fail(ctx, CHIMERA_EINVAL, "token id out of range");
  const int need = std::max(ctx->N, ctx->K) + 1 + ctx->D1;
  for (int b = 0; b < batch; ++b)
    if (lens[b] + need > ctx->cap) return fail(ctx, CHIMERA_ECAPACITY, "prompt too long for max_seq_len");

  // reset: free every block, rebuild plans for this batch, drop the step graph
  ctx->prefilled = false;
  pt_wait(ctx);
  for (auto& blocks : ctx->seq_blocks) {
    for (int blk : blocks) ctx->free_blocks.push_back(blk);
    blocks.clear();
  }
  std::fill(ctx->h_pt, ctx->h_pt + ctx->h_pt_len, 0);
  ctx->pt_dirty = true;
  if (ctx->graph) {
    cudaGraphExecDestroy(ctx->graph);
    ctx->graph = nullptr;
  }
  if (ctx->prof_graph) {
    cudaGraphExecDestroy(ctx->prof_graph);
    ctx->prof_graph = nullptr;
  }
  if (ctx->phase_graph) {
    cudaGraphExecDestroy(ctx->phase_graph);
    ctx->phase_graph = nullptr;
  }
  if (ctx->class_graph) {
    cudaGraphExecDestroy(ctx->class_graph);
    ctx->class_graph = nullptr;
  }
  if (ctx->ar_graph) {
    cudaGraphExecDestroy(ctx->ar_graph);
    ctx->ar_graph = nullptr;
  }
  ctx->batch = batch;
  ctx->plan_keys = max_len;
  if (!build_plans(ctx, batch)) return CHIMERA_EINVAL;
  for (int b = 0; b < batch; ++b) {
    chimera_status st = ensure_blocks(ctx, b, lens[b] + need);
    if (st != CHIMERA_OK) return st;
  }
  chimera_status st = flush_page_table(ctx);
  if (st != CHIMERA_OK) return st;

  cudaStream_t s = ctx->stream;
  CK(cudaMemsetAsync(ctx->d_n, 0, ctx->Bmax * sizeof(int), s));
  CK(cudaMemsetAsync(ctx->d_tok, 0, static_cast<size_t>(ctx->Bmax) * ctx->tok_stride * sizeof(int), s));
  CK(cudaMemsetAsync(ctx->d_step, 0, sizeof(int), s));
  CK(cudaMemsetAsync(ctx->d_ovr_flag, 0, sizeof(int), s));
  ctx->ovr_pending = false;
  {
    long long off = 0;
    for (int b = 0; b < batch; ++b) {
      CK(cudaMemcpyAsync(ctx->d_tok + static_cast<size_t>(b) * ctx->tok_stride, tokens + off, lens[b] * sizeof(int),
                         cudaMemcpyHostToDevice, s));
      off += lens[b];
    }
    CK(cudaStreamSynchronize(s));
  }
  ctx->host_n.assign(batch, 0);
  const int d = ctx->d, B = batch;
  const int chunks = (max_len + CHUNK - 1) / CHUNK;
  const void* dl_norm = ctx->draft.attn_norm;
  for (int cidx = 0; cidx < chunks; ++cidx) {
    int* hv = ctx->h_stage;
    for (int b = 0; b < B; ++b) {
      const int v = std::max(0, std::min(CHUNK, lens[b] - cidx * CHUNK));
      hv[b] = v;
      const int li = lens[b] - 1 - cidx * CHUNK;
      hv[64 + b] = (li >= 0 && li < CHUNK) ? li : -1;
    }
    CK(cudaMemcpyAsync(ctx->d_valid, hv, B * sizeof(int), cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(ctx->d_last, hv + 64, B * sizeof(int), cudaMemcpyHostToDevice, s));
    CK(embed(ctx->dtype, ctx->embed, d, ctx->V, ctx->x, B * CHUNK, CHUNK, nullptr, ctx->d_tok, ctx->tok_stride, ctx->d_n,
             ctx->d_valid, ctx->d_err, s));
    for (int l = 0; l < ctx->L; ++l)
      CK(enqueue_layer(ctx, l, &ctx->pre[5 * l], B * CHUNK, CHUNK, ctx->d_valid, nullptr, ctx->d_chain,
                       ctx->att_splits_pre, 0));
    CK(run_final_norm(ctx, B * CHUNK, false));
    // draft-layer K/V of the chunk's H_LLM rows
    CK(run_norm(ctx, ctx->hfin32, dl_norm, B * CHUNK, ctx->kvtmp, 2 * d));
    CK(run_lin(ctx, ctx->pre_dkv));
    CK(run_rope(ctx, true, 0, ctx->kvtmp, 2 * d, -1, 0, d, CHUNK, ctx->d_valid, 0, 0, 0, nullptr));
    CK(launch_prefill_advance(ctx->dtype, ctx->hfin32, d, CHUNK, ctx->d_valid, ctx->d_last, ctx->d_n, ctx->headin,
                              ctx->headin_lo, B, s));
    CK(cudaStreamSynchronize(s));  // the staging buffer is reused by the next chunk
  }
  // root = greedy next token of each prompt (eq. 1)
  CK(cudaMemsetAsync(ctx->logits, 0, static_cast<size_t>(B) * ctx->V * sizeof(float), s));
  CK(run_lin(ctx, ctx->pre_lm));
  CK(argmax_rows(ctx->logits, ctx->V, B, ctx->d_amax, s));
  CK(launch_set_root(ctx->d_n, ctx->d_tok, ctx->tok_stride, ctx->d_amax, B, s));
  CK(cudaStreamSynchronize(s));
  st = check_err(ctx);
  if (st != CHIMERA_OK) return st;
  for (int b = 0; b < B; ++b) ctx->host_n[b] = lens[b];
  ctx->prefilled = true;
  return CHIMERA_OK;
}

chimera_status chimera_step(chimera_ctx* ctx, int32_t* out_tokens, int32_t* out_count) {
  if (!ctx) return CHIMERA_EINVAL;
  if (!out_tokens || !out_count) return fail(ctx, CHIMERA_EINVAL, "NULL output");
  chimera_status st = steps_prepare(ctx, 1);
  if (st != CHIMERA_OK) return st;
  st = launch_steps(ctx, 1);
  if (st != CHIMERA_OK) return st;
  return read_new_tokens(ctx, out_tokens, ctx->D1, out_count);
}

chimera_status chimera_generate(chimera_ctx* ctx, int n_steps, int32_t* out_tokens, int32_t* out_count) {
  if (!ctx) return CHIMERA_EINVAL;
  if (n_steps < 1 || !out_tokens || !out_count) return fail(ctx, CHIMERA_EINVAL, "bad arguments");
  chimera_status st = steps_prepare(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  st = launch_steps(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  return read_new_tokens(ctx, out_tokens, n_steps * ctx->D1, out_count);
}

chimera_status chimera_step_async(chimera_ctx* ctx, int n_steps) {
  if (!ctx) return CHIMERA_EINVAL;
  if (n_steps < 1) return fail(ctx, CHIMERA_EINVAL, "n_steps < 1");
  chimera_status st = steps_prepare(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  st = launch_steps(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  // host_n is refreshed by chimera_sync
  return CHIMERA_OK;
}

chimera_status chimera_ar_generate(chimera_ctx* ctx, int n_steps, int32_t* out_tokens, int32_t* out_count) {
  if (!ctx) return CHIMERA_EINVAL;
  if (n_steps < 1) return fail(ctx, CHIMERA_EINVAL, "n_steps < 1");
  chimera_status st = steps_prepare(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  if (!ctx->ar_graph) {
    cudaError_t e = capture_step(ctx, &ctx->ar_graph, true);
    if (e != cudaSuccess) {
      ctx->ar_graph = nullptr;
      return fail(ctx, CHIMERA_ECUDA, std::string("capturing the autoregressive step: ") + cudaGetErrorString(e));
    }
  }
  for (int i = 0; i < n_steps; ++i) CK(cudaGraphLaunch(ctx->ar_graph, ctx->stream));
  if (!out_tokens) return CHIMERA_OK;  // timing: no host output, no synchronisation
  if (!out_count) return fail(ctx, CHIMERA_EINVAL, "NULL count");
  return read_new_tokens(ctx, out_tokens, n_steps, out_count);
}

chimera_status chimera_sync(chimera_ctx* ctx) {
  if (!ctx) return CHIMERA_EINVAL;
  CK(cudaStreamSynchronize(ctx->stream));
  if (ctx->batch > 0) {
    CK(cudaMemcpy(ctx->host_n.data(), ctx->d_n, ctx->batch * sizeof(int), cudaMemcpyDeviceToHost));
  }
  return check_err(ctx);
}

void chimera_free(chimera_ctx* ctx) {
  if (ctx && ctx->stream) cudaStreamSynchronize(ctx->stream);
  free_ctx(ctx);
}

const char* chimera_last_error(const chimera_ctx* ctx) { return ctx ? ctx->err.c_str() : "NULL context"; }

chimera_status chimera_tree(const chimera_ctx* ctx, int32_t* depth, int32_t* parent, int32_t* rank, uint64_t* anc) {
  if (!ctx) return CHIMERA_EINVAL;
  for (int i = 0; i < ctx->N; ++i) {
    if (depth) depth[i] = ctx->tree.depth[i];
    if (parent) parent[i] = ctx->tree.parent[i];
    if (rank) rank[i] = ctx->tree.rank[i];
    if (anc) anc[i] = ctx->tree.anc[i];
  }
  return CHIMERA_OK;
}

chimera_status chimera_static_tree(const int32_t* topk, int n_heads, int n_nodes, int32_t* depth,
                                   int32_t* parent, int32_t* rank, uint64_t* anc) {
  if (!topk || n_heads < 1 || n_heads > 4 || n_nodes < 2 || n_nodes > 64) return CHIMERA_EINVAL;
  int lim[4];
  for (int k = 0; k < n_heads; ++k) {
    if (topk[k] < 1 || topk[k] > MAX_KMAX) return CHIMERA_EINVAL;
    lim[k] = topk[k];
  }
  Tree t;
  std::string err;
  if (!build_tree(lim, n_heads, n_nodes, &t, &err)) return CHIMERA_EINVAL;
  for (int i = 0; i < n_nodes; ++i) {
    if (depth) depth[i] = t.depth[i];
    if (parent) parent[i] = t.parent[i];
    if (rank) rank[i] = t.rank[i];
    if (anc) anc[i] = t.anc[i];
  }
  return CHIMERA_OK;
}

chimera_status chimera_profile_step(chimera_ctx* ctx, int max, int32_t* kinds, int32_t* phases, float* ms,
                                    double* bytes, int32_t* count) {
  if (!ctx) return CHIMERA_EINVAL;
  if (!count) return fail(ctx, CHIMERA_EINVAL, "NULL count");
  chimera_status st = steps_prepare(ctx, 1);
  if (st != CHIMERA_OK) return st;
  if (!ctx->prof_graph) {
    ctx->prof_ev.reserve(8192);
    ctx->prof = true;
    ctx->prof_used = 0;
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
    cudaError_t e = enqueue_step(ctx);
    cudaError_t e2 = cudaStreamEndCapture(ctx->stream, &g);
    ctx->prof = false;
    if (e != cudaSuccess || e2 != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      return fail(ctx, CHIMERA_ECUDA, std::string("capturing the profiled step: ") +
                                          cudaGetErrorString(e != cudaSuccess ? e : e2));
    }
    e = cudaGraphInstantiate(&ctx->prof_graph, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) return fail(ctx, CHIMERA_ECUDA, std::string("instantiating: ") + cudaGetErrorString(e));
    ctx->prof_count = ctx->prof_used;
  }
  if (ctx->ovr_pending) {
    const int one = 1;
    CK(cudaMemcpyAsync(ctx->d_ovr_flag, &one, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  }
  CK(cudaGraphLaunch(ctx->prof_graph, ctx->stream));
  if (ctx->ovr_pending) {
    CK(cudaMemsetAsync(ctx->d_ovr_flag, 0, sizeof(int), ctx->stream));
    ctx->ovr_pending = false;
  }
  CK(cudaStreamSynchronize(ctx->stream));
  const int n = static_cast<int>(ctx->prof_count);
  for (int i = 0; i < n && i < max; ++i) {
    float t = 0;
    cudaEventElapsedTime(&t, ctx->prof_ev[i].a, ctx->prof_ev[i].b);
    if (kinds) kinds[i] = ctx->prof_ev[i].kind;
    if (phases) phases[i] = ctx->prof_ev[i].phase;
    if (ms) ms[i] = t;
    if (bytes) bytes[i] = ctx->prof_ev[i].bytes;
  }
  *count = n;
  CK(cudaMemcpy(ctx->host_n.data(), ctx->d_n, ctx->batch * sizeof(int), cudaMemcpyDeviceToHost));
  return check_err(ctx);
}

chimera_status chimera_profile_phases(chimera_ctx* ctx, int n_steps, float* draft_ms, float* verify_ms,
                                      float* commit_ms) {
  if (!ctx) return CHIMERA_EINVAL;
  if (n_steps < 1) return fail(ctx, CHIMERA_EINVAL, "n_steps < 1");
  chimera_status st = steps_prepare(ctx, n_steps);
  if (st != CHIMERA_OK) return st;
  if (!ctx->phase_graph) {
    for (auto& e : ctx->phase_ev)
      if (!e) CK(cudaEventCreate(&e));
    ctx->phase_marks = true;
    cudaError_t e = capture_step(ctx, &ctx->phase_graph);
    ctx->phase_marks = false;
    if (e != cudaSuccess) {
      ctx->phase_graph = nullptr;
      return fail(ctx, CHIMERA_ECUDA, std::string("capturing the phase-timed step: ") + cudaGetErrorString(e));
    }
  }
  if (ctx->ovr_pending) {
    const int one = 1;
    CK(cudaMemcpyAsync(ctx->d_ovr_flag, &one, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  }
  for (int i = 0; i < n_steps; ++i) {
    CK(cudaGraphLaunch(ctx->phase_graph, ctx->stream));
    if (i == 0 && ctx->ovr_pending) {
      CK(cudaMemsetAsync(ctx->d_ovr_flag, 0, sizeof(int), ctx->stream));
      ctx->ovr_pending = false;
    }
    CK(cudaStreamSynchronize(ctx->stream));
    float t[3] = {0, 0, 0};
    for (int p = 0; p < 3; ++p) CK(cudaEventElapsedTime(&t[p], ctx->phase_ev[p], ctx->phase_ev[p + 1]));
    if (draft_ms) draft_ms[i] = t[0];
    if (verify_ms) verify_ms[i] = t[1];
    if (commit_ms) commit_ms[i] = t[2];
  }
  CK(cudaMemcpy(ctx->host_n.data(), ctx->d_n, ctx->batch * sizeof(int), cudaMemcpyDeviceToHost));
  return check_err(ctx);
}

chimera_status chimera_profile_kind(chimera_ctx* ctx, int kind, int n_reps, float* ms, int32_t* launches,
                                    double* bytes) {
  if (!ctx) return CHIMERA_EINVAL;
  // classes whose kernels write only step scratch (never n, the token history or
  // committed KV rows), so the replays leave the committed state intact
  const bool allowed = kind == CHIMERA_KIND_LINEAR || kind == CHIMERA_KIND_ATTENTION || kind == CHIMERA_KIND_NORM ||
                       kind == CHIMERA_KIND_SWIGLU || kind == CHIMERA_KIND_EMBED || kind == CHIMERA_KIND_TOPK ||
                       kind == CHIMERA_KIND_ARGMAX || kind == CHIMERA_KIND_ROPE_KV || kind == CHIMERA_KIND_CHAIN;
  if (!allowed || n_reps < 1 || !ms) return fail(ctx, CHIMERA_EINVAL, "bad kernel class or repetition count");
  chimera_status st = steps_prepare(ctx, 1);
  if (st != CHIMERA_OK) return st;
  if (ctx->class_graph && ctx->class_graph_kind != kind) {
    CK(cudaGraphExecDestroy(ctx->class_graph));
    ctx->class_graph = nullptr;
  }
  if (!ctx->class_graph) {
    ctx->filter_kind = kind;
    ctx->class_launches = 0;
    ctx->class_bytes = 0;
    cudaError_t e = capture_step(ctx, &ctx->class_graph);
    ctx->filter_kind = 0;
    if (e != cudaSuccess) {
      ctx->class_graph = nullptr;
      return fail(ctx, CHIMERA_ECUDA, std::string("capturing the kernel-class graph: ") + cudaGetErrorString(e));
    }
    ctx->class_graph_kind = kind;
  }
  cudaEvent_t a, b;
  CK(cudaEventCreate(&a));
  CK(cudaEventCreate(&b));
  CK(cudaGraphLaunch(ctx->class_graph, ctx->stream));  // warm-up
  CK(cudaEventRecord(a, ctx->stream));
  for (int i = 0; i < n_reps; ++i) CK(cudaGraphLaunch(ctx->class_graph, ctx->stream));
  CK(cudaEventRecord(b, ctx->stream));
  CK(cudaEventSynchronize(b));
  float t = 0;
  CK(cudaEventElapsedTime(&t, a, b));
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  *ms = t / n_reps;
  if (launches) *launches = static_cast<int32_t>(ctx->class_launches);
  if (bytes) *bytes = ctx->class_bytes;
  return check_err(ctx);
}

chimera_status chimera_debug_override_tree(chimera_ctx* ctx, const int32_t* node_tokens) {
  if (!ctx) return CHIMERA_EINVAL;
  if (!ctx->prefilled) return fail(ctx, CHIMERA_ESTATE, "override before prefill");
  if (!node_tokens) return fail(ctx, CHIMERA_EINVAL, "NULL tokens");
  const size_t n = static_cast<size_t>(ctx->batch) * ctx->N;
  for (size_t i = 0; i < n; ++i)
    if (i % ctx->N != 0 && (node_tokens[i] < 0 || node_tokens[i] >= ctx->V))
      return fail(ctx, CHIMERA_EINVAL, "override token out of range");
  CK(cudaMemcpy(ctx->d_ovr, node_tokens, n * sizeof(int), cudaMemcpyHostToDevice));
  ctx->ovr_pending = true;
  return CHIMERA_OK;
}

chimera_status chimera_debug_set_root(chimera_ctx* ctx, const int32_t* roots) {
  if (!ctx) return CHIMERA_EINVAL;
  if (!ctx->prefilled) return fail(ctx, CHIMERA_ESTATE, "set_root before prefill");
  for (int b = 0; b < ctx->batch; ++b) {
    if (roots[b] < 0 || roots[b] >= ctx->V) return fail(ctx, CHIMERA_EINVAL, "root out of range");
    CK(cudaMemcpy(ctx->d_tok + static_cast<size_t>(b) * ctx->tok_stride + ctx->host_n[b], &roots[b], sizeof(int),
                  cudaMemcpyHostToDevice));
  }
  return CHIMERA_OK;
}

chimera_status chimera_debug_read(chimera_ctx* ctx, int what, void* dst, size_t bytes) {
  if (!ctx) return CHIMERA_EINVAL;
  if (!dst) return fail(ctx, CHIMERA_EINVAL, "NULL destination");
  const size_t B = ctx->batch ? ctx->batch : 1, N = ctx->N, V = ctx->V, d = ctx->d, K = ctx->K;
  const void* src = nullptr;
  size_t need = 0;
  switch (what) {
    case CHIMERA_DBG_NODE_TOKENS: src = ctx->d_node_tok; need = B * N * 4; break;
    case CHIMERA_DBG_VERIFY_LOGITS: src = ctx->logits; need = B * N * V * 4; break;
    case CHIMERA_DBG_VERIFY_HIDDEN: src = ctx->hfin32; need = B * N * d * 4; break;
    case CHIMERA_DBG_ARGMAX: src = ctx->d_amax; need = B * N * 4; break;
    case CHIMERA_DBG_PATH: src = ctx->d_path; need = B * ctx->D1 * 4; break;
    case CHIMERA_DBG_ACCEPT_LEN: src = ctx->d_L; need = B * 4; break;
    case CHIMERA_DBG_DRAFT_LOGITS: src = ctx->hlog; need = K * B * V * 4; break;
    case CHIMERA_DBG_TOPK: src = ctx->d_topk; need = B * K * ctx->KMAX * 4; break;
    case CHIMERA_DBG_HFULL: src = ctx->hfull_log; need = K * B * d * 4; break;
    case CHIMERA_DBG_N: src = ctx->d_n; need = B * 4; break;
    case CHIMERA_DBG_TOKENS: src = ctx->d_tok; need = B * ctx->tok_stride * 4; break;
    case CHIMERA_DBG_PREFILL_LOGITS: src = ctx->logits; need = B * V * 4; break;
    case CHIMERA_DBG_TRIGRAM_HITS: src = ctx->tc_hit_log; need = K * B * 4; break;
    case CHIMERA_DBG_HTRI: src = ctx->htri_log; need = K * B * d * 4; break;
    default: return fail(ctx, CHIMERA_EINVAL, "unknown debug buffer");
  }
  if (!src) return fail(ctx, CHIMERA_EINVAL, "debug buffer not kept in this configuration");
  if (bytes != need)
    return fail(ctx, CHIMERA_EINVAL, "debug read: expected " + std::to_string(need) + " bytes, got " + std::to_string(bytes));
  CK(cudaStreamSynchronize(ctx->stream));
  CK(cudaMemcpy(dst, src, need, cudaMemcpyDeviceToHost));
  return CHIMERA_OK;
}

chimera_status chimera_debug_read_kv(chimera_ctx* ctx, int layer, int seq, int pos0, int count, void* k_dst,
                                     void* v_dst) {
  if (!ctx) return CHIMERA_EINVAL;
  if (layer < -1 || layer >= ctx->L || seq < 0 || seq >= ctx->batch || pos0 < 0 || count < 0 ||
      pos0 + count > static_cast<int>(ctx->seq_blocks[seq].size()) * 16 || !k_dst || !v_dst)
    return fail(ctx, CHIMERA_EINVAL, "bad KV read");
  CK(cudaStreamSynchronize(ctx->stream));
  const int P = ctx->kv_planes, hd = ctx->hd;
  const size_t row = static_cast<size_t>(hd) * ctx->kv_esz;
  const char* pool = static_cast<const char*>(layer < 0 ? ctx->dkv : ctx->kv) +
                     (layer < 0 ? 0 : static_cast<size_t>(layer) * ctx->kv_layer_stride * ctx->kv_esz);
  std::vector<uint16_t> tmp(static_cast<size_t>(P) * hd);
  for (int i = 0; i < count; ++i) {
    const int slot = pos0 + i;
    const int page = ctx->h_pt[seq * ctx->max_pages + slot / 16];
    for (int h = 0; h < ctx->H; ++h) {
      const char* base = pool + ((static_cast<size_t>(page) * ctx->H + h) * P) * 16 * row + (slot % 16) * row;
      const size_t o = (static_cast<size_t>(i) * ctx->H + h);
      if (P == 2) {
        CK(cudaMemcpy(static_cast<char*>(k_dst) + o * row, base, row, cudaMemcpyDeviceToHost));
        CK(cudaMemcpy(static_cast<char*>(v_dst) + o * row, base + 16 * row, row, cudaMemcpyDeviceToHost));
      } else {  // split planes: return hi + lo as fp32
        for (int pl = 0; pl < 4; ++pl)
          CK(cudaMemcpy(tmp.data() + pl * hd, base + pl * 16 * row, row, cudaMemcpyDeviceToHost));
        float* kd = static_cast<float*>(k_dst) + o * hd;
        float* vd = static_cast<float*>(v_dst) + o * hd;
        auto bf = [](uint16_t u) {
          uint32_t x = static_cast<uint32_t>(u) << 16;
          float f;
          memcpy(&f, &x, 4);
          return f;
        };
        for (int j = 0; j < hd; ++j) {
          kd[j] = bf(tmp[j]) + bf(tmp[hd + j]);
          vd[j] = bf(tmp[2 * hd + j]) + bf(tmp[3 * hd + j]);
        }
      }
    }
  }
  return CHIMERA_OK;
}

// ---------------------------------------------------------------------------
// stateless kernel-level entry points
// ---------------------------------------------------------------------------
namespace {
// Scratch of the stateless entry points, one set per device (allocated on the first
// call made with that device current and kept until exit).
struct OpScratch {
  bool ready = false;
  float* lin_ws = nullptr;
  int* lin_cnt = nullptr;
  int* err = nullptr;
  float* att_ws = nullptr;
  size_t att_floats = 0;
  int* att_cnt = nullptr;
};
constexpr int OP_MAX_DEVICES = 64;
constexpr int OP_ATT_COUNTERS = 64 * 256;
std::mutex g_op_mu;
OpScratch g_op_dev[OP_MAX_DEVICES];

// The current device's scratch (nullptr on failure).  Caller holds g_op_mu.
OpScratch* op_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= OP_MAX_DEVICES) return nullptr;
  OpScratch& s = g_op_dev[dev];
  if (s.ready) return &s;
  OpScratch n;
  n.att_floats = static_cast<size_t>(16) << 20;
  bool ok = cudaMalloc(&n.lin_ws, tc_ws_floats(256) * sizeof(float)) == cudaSuccess;
  ok = ok && cudaMalloc(&n.lin_cnt, tc_max_tiles() * sizeof(int)) == cudaSuccess;
  ok = ok && cudaMalloc(&n.err, sizeof(int)) == cudaSuccess;
  ok = ok && cudaMalloc(&n.att_ws, n.att_floats * sizeof(float)) == cudaSuccess;
  ok = ok && cudaMalloc(&n.att_cnt, OP_ATT_COUNTERS * sizeof(int)) == cudaSuccess;
  ok = ok && cudaMemset(n.lin_cnt, 0, tc_max_tiles() * sizeof(int)) == cudaSuccess;
  ok = ok && cudaMemset(n.err, 0, sizeof(int)) == cudaSuccess;
  ok = ok && cudaMemset(n.att_cnt, 0, OP_ATT_COUNTERS * sizeof(int)) == cudaSuccess;
  ok = ok && cudaDeviceSynchronize() == cudaSuccess;
  if (!ok) {
    cudaFree(n.lin_ws);
    cudaFree(n.lin_cnt);
    cudaFree(n.err);
    cudaFree(n.att_ws);
    cudaFree(n.att_cnt);
    return nullptr;
  }
  n.ready = true;
  s = n;
  return &s;
}
}  // namespace

chimera_status chimera_op_linear(int dtype, int epi, int out_f32, int M, int N, int K, const void* X,
                                 const void* X_lo, int ldx, const void* W, void* Y, int ldy, void* cuda_stream) {
  if ((dtype != 0 && dtype != 1) || epi < 0 || epi > 2 || M < 1 || N < 1 || K < 1 || !X || !W || !Y || ldx < K ||
      ldy < N)
    return CHIMERA_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  if (dtype == 0) return f32_linear(M, N, K, static_cast<const float*>(X), ldx, static_cast<const float*>(W),
                                    static_cast<float*>(Y), ldy, epi, s) == cudaSuccess
                             ? CHIMERA_OK
                             : CHIMERA_ECUDA;
  std::lock_guard<std::mutex> lk(g_op_mu);
  OpScratch* sc = op_scratch();
  if (!sc) return CHIMERA_ENOMEM;
  TcLinearPlan plan;
  char msg[256];
  if (tc_linear_plan(&plan, M, N, K, X, X_lo, ldx, W, Y, nullptr, ldy, epi, epi == EPI_RESID ? 1 : out_f32, sc->lin_ws,
                     sc->lin_cnt, sc->err, msg, sizeof(msg)) != 0)
    return CHIMERA_EINVAL;
  return tc_linear_launch(plan, s) == cudaSuccess ? CHIMERA_OK : CHIMERA_ECUDA;
}

chimera_status chimera_op_attention(int dtype, int kv_split, int batch, int n_heads, int head_dim, int nq, int q_local0,
                                    int n_local, const float* q, int ldq, int q_rows, const void* pool, int n_blocks,
                                    const int32_t* page_table, int max_pages, const int32_t* n_ctx, const uint64_t* anc,
                                    void* out, void* out_lo, int ldo, int splits, void* cuda_stream) {
  if ((dtype != 0 && dtype != 1) || batch < 1 || n_heads < 1 || (head_dim != 64 && head_dim != 128) || nq < 1 ||
      nq > 64 || n_local < 0 || n_local > 64 || q_local0 < 0 || !q || !pool || !page_table || !n_ctx || !anc || !out ||
      splits < 1 || splits > 16 || (dtype == 1 && head_dim == 128 && splits > 8) || batch * n_heads > 64 * 256 ||
      n_blocks < 1)
    return CHIMERA_EINVAL;
  std::lock_guard<std::mutex> lk(g_op_mu);
  OpScratch* sc = op_scratch();
  if (!sc) return CHIMERA_ENOMEM;
  AttnParams p{};
  p.q = q;
  p.ldq = ldq;
  p.q_rows = q_rows;
  p.nq = nq;
  p.q_local0 = q_local0;
  p.n_local = n_local;
  p.anc = reinterpret_cast<const unsigned long long*>(anc);
  p.pool = pool;
  p.planes = (dtype == 1 && kv_split) ? 4 : 2;
  p.pool_rows = static_cast<long long>(n_blocks) * n_heads * p.planes * 16;
  p.page_table = page_table;
  p.max_pages = max_pages;
  p.n_ctx = n_ctx;
  p.out = out;
  p.out_lo = out_lo;
  p.ldo = ldo;
  p.B = batch;
  p.H = n_heads;
  p.hd = head_dim;
  p.scale = 1.0f / std::sqrt(static_cast<float>(head_dim));
  p.splits = splits;
  p.ws = sc->att_ws;
  p.counters = sc->att_cnt;
  p.err = sc->err;
  p.nq_max = nq;
  if (attn_ws_floats(batch, n_heads, splits, nq, head_dim) > sc->att_floats) return CHIMERA_EINVAL;
  return attention(p, dtype, static_cast<cudaStream_t>(cuda_stream)) == cudaSuccess
             ? CHIMERA_OK
             : CHIMERA_ECUDA;
}

chimera_status chimera_op_sync(void* cuda_stream) {
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return CHIMERA_ECUDA;
  int word = 0;
  {
    std::lock_guard<std::mutex> lk(g_op_mu);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= OP_MAX_DEVICES) return CHIMERA_ECUDA;
    OpScratch& sc = g_op_dev[dev];
    if (sc.ready) {
      int e = 0;
      if (cudaMemcpy(&e, sc.err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return CHIMERA_ECUDA;
      if (e) {
        // a launch that gave up can leave split-K or split-merge counters raised
        if (cudaMemset(sc.err, 0, sizeof(int)) != cudaSuccess ||
            cudaMemset(sc.lin_cnt, 0, tc_max_tiles() * sizeof(int)) != cudaSuccess ||
            cudaMemset(sc.att_cnt, 0, OP_ATT_COUNTERS * sizeof(int)) != cudaSuccess ||
            cudaDeviceSynchronize() != cudaSuccess)
          return CHIMERA_ECUDA;
      }
      word |= e;
    }
  }
  int na = 0;
  if (noalloc_take_error(&na) != 0) return CHIMERA_ECUDA;
  word |= na;
  if (word & ERR_TIMEOUT) return CHIMERA_ETIMEDOUT;
  if (word & ERR_CAPACITY) return CHIMERA_ECAPACITY;
  if (word) return CHIMERA_EINVAL;
  return CHIMERA_OK;
}

chimera_status chimera_debug_set_wait_limit(uint64_t ns) {
  if (ns == 0) ns = kDefaultWaitNs;
  g_lin_wait_ns.store(ns);
  return CHIMERA_OK;
}

}  // extern "C"
