/*
 * chimera.h — C ABI of one Chimera draft-and-verify step on one GB300 (sm_103a).
 *
 * Chimera (arXiv 2402.15758) speeds up greedy decoding of a Llama-style LLM without
 * changing its output.  Each step:
 *   1. drafts K tokens with the lightweight draft model: a trigram encoder
 *      (eq. "trigram_calculations"), a full-context Transformer block over the base
 *      model's last hidden states and the trigram states (eq.
 *      "fullcontext_calculations"), and K residual decoding heads (eq. "residual
 *      decoding head"), head k predicting word n+2+k from [h_LLM_n ; h_full_{n+1+k}];
 *   2. expands the per-head top-k tokens into a static candidate tree (Section
 *      "Inference");
 *   3. verifies every tree node in one tree-masked forward of the base model
 *      (Section "Verification");
 *   4. greedily accepts the longest path whose tokens equal the base model's argmax,
 *      and compacts the accepted nodes' KV entries into the cache.
 * The emitted stream equals plain greedy autoregressive decoding (eq. 1, argmax).
 *
 * Conventions
 *   - Every call returns a chimera_status; the message of the last failure is in
 *     chimera_last_error().  Calls on one context are not thread-safe.
 *   - Weights are caller-owned DEVICE memory that must outlive the context.
 *     Matrices are row-major [out][in] (one output feature per row, y = W x).
 *     dtype 0 = fp32 everywhere; dtype 1 = bf16 weights, fp32 accumulation, an fp32
 *     residual stream and fp32 projection outputs; `precision` selects how the
 *     activations that feed the tensor cores and the KV caches are stored.
 *   - The context owns the paged KV caches (blocks of 16 positions), the draft KV
 *     cache, all scratch and the captured CUDA graph of the step.
 *   - Host buffers are caller-owned host memory.  chimera_step / chimera_generate /
 *     chimera_prefill return after their work on the context's stream is done.
 *   - Positions are 0-based.  After prefill of a prompt x[0..n-1] the state is
 *     (x[0..n], n) where x[n] — the "root" — is the base model's own next token.
 *     A step emits the root plus the L accepted drafted tokens (1..depth+1 tokens);
 *     the bonus token (base argmax after the accepted path) becomes the next root.
 */
#ifndef CHIMERA_H
#define CHIMERA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct chimera_ctx chimera_ctx;

typedef enum {
  CHIMERA_OK = 0,
  CHIMERA_EINVAL = -1,     /* bad argument (shape, pointer, token id, batch) */
  CHIMERA_ENOMEM = -2,     /* device allocation failed */
  CHIMERA_ECAPACITY = -3,  /* a sequence would exceed max_seq_len KV slots */
  CHIMERA_ECUDA = -4,      /* a CUDA call or kernel failed */
  CHIMERA_ETIMEDOUT = -5,  /* a bounded device-side wait gave up */
  CHIMERA_ESTATE = -6      /* call out of order (e.g. step before prefill) */
} chimera_status;

/* Model and decoding shapes.  Table 1 of the paper gives layers / hidden size /
 * heads of the backbones; the draft has one full-context block of the same shape
 * and n_draft_heads residual heads of shape [vocab][2*d_model]. */
typedef struct {
  int n_layers, d_model, n_heads, head_dim, ffn_dim, vocab;
  int dtype;            /* 0 = fp32, 1 = bf16 */
  float rms_eps;        /* RMSNorm epsilon (1e-6) */
  float rope_theta;     /* RoPE base (10000) */
  int n_draft_heads;    /* K, 1..4 */
  int tree_nodes;       /* N including the root, 2..64 */
  int topk[8];          /* rank limit per head (1..8); the tree draws ranks < topk[k] */
  int max_batch;        /* sequences per context, 1..64 */
  int max_seq_len;      /* KV slots per sequence (prompt + generated + N tree slots) */
  int kv_block;         /* must be 16 */
  int precision;        /* bf16 models only.  1: every activation that feeds a tensor core
                           (GEMM operands, attention queries and probabilities) and every
                           KV-cache entry is kept as a hi + lo pair of bf16 values, products
                           taken term by term with fp32 accumulation (~fp32 accuracy);
                           0: activations and KV entries rounded once to bf16.
                           fp32 models ignore it. */
  int draft_mode;       /* 0: the draft of the method (K sequential sub-steps, residual heads).
                           Ablation variants (Section "Residual decoding heads" and its
                           ablation): bit 0 = one-pass draft (the trigram encoder and the
                           full-context block run once, every head scores h_full_{n+1});
                           bit 1 = heads without the residual input (Theta_k is
                           [vocab][d_model] on h_full alone). */
  int accept_mode;      /* 0: greedy acceptance (lossless); 1: typical acceptance at temperature
                           1 (Section "Verification"): node c is acceptable when its parent is
                           and p_parent(token_c) > min(typical_eps, typical_delta * exp(-H)),
                           H the entropy of the parent's distribution; the path ends at the
                           deepest acceptable node (smallest index among the deepest) and the
                           bonus token is the base argmax there.  Not lossless. */
  float typical_eps;    /* typical acceptance: hard threshold (e.g. 0.09) */
  float typical_delta;  /* typical acceptance: entropy factor (e.g. 0.3) */
  int trigram_cache;    /* entries of the device trigram cache (Section "Trigram encoder",
                           lookup table): 0 = off; else a multiple of 4 with a power-of-two
                           number of 4-way sets, <= 65536.  Each entry keeps one h_tri row
                           (d_model fp32 values) keyed by its three token ids; the least
                           recently used way of a set is replaced.  A sub-step whose trigrams
                           all hit skips the encoder's two linears; results are unchanged. */
  int fused_chain;      /* bf16 models: 1 runs the linears and row steps between two attentions
                           (O, RMSNorm, gate|up, SwiGLU, down, the next RMSNorm and QKV; the
                           draft block and head; the commit projection) as one persistent
                           launch with grid-wide step counters; 0 (default) launches each
                           linear and row kernel separately.  Same results either way. */
} chimera_config;

/* One Llama block: RMSNorm gains [d]; wqkv [3d][d] (rows q, then k, then v; head h
 * at rows h*hd..h*hd+hd-1 of each part); wo [d][d]; w_gate, w_up [F][d]; w_down [d][F]. */
typedef struct {
  const void* attn_norm;
  const void* wqkv;
  const void* wo;
  const void* ffn_norm;
  const void* w_gate;
  const void* w_up;
  const void* w_down;
} chimera_block_weights;

typedef struct {
  const void* embed;                   /* [V][d] */
  const chimera_block_weights* layers; /* host array [n_layers] of device pointers */
  const void* final_norm;              /* [d] */
  const void* lm_head;                 /* [V][d] */
  const void* tri_w1;                  /* [d][3d]: W1 of the trigram encoder, input
                                          [x_{i-2}; x_{i-1}; x_i] */
  const void* tri_w2;                  /* [d][d]: W2 */
  chimera_block_weights draft;         /* full-context encoder block */
  const void* const* heads;            /* host array [K] of [V][2d]: Theta_k, input
                                          [h_LLM_n ; h_full_{n+1+k}] */
} chimera_weights;

/* Create a context.  `cuda_stream` is a cudaStream_t (NULL: the context creates its
 * own non-blocking stream).  Validates shapes, records the weight pointers and
 * allocates the KV pools (max_batch * max_seq_len slots), scratch and the tree.
 * It synchronizes the device first, so weights written by earlier work on any stream
 * are complete before the context reads them; the weights must not change while the
 * context lives.  EINVAL on bad shapes or a NULL weight, ENOMEM on allocation failure,
 * ECUDA when the device reports an earlier error. */
chimera_status chimera_init(const chimera_config* cfg, const chimera_weights* w,
                            void* cuda_stream, chimera_ctx** out);

/* Prefill `batch` prompts (host int32, concatenated; lens[b] >= 1 tokens each, ids in
 * [0, vocab)) with the causal base forward, fill the base and draft KV caches and
 * set each root to the base model's greedy next token (eq. 1).  Resets any previous
 * state of the context.  EINVAL / ECAPACITY on bad input. */
chimera_status chimera_prefill(chimera_ctx* ctx, int batch, const int32_t* tokens,
                               const int32_t* lens);

/* One draft-and-verify step for every sequence.  out_tokens: host int32
 * [batch][depth+1] (depth = number of draft heads) receives the emitted tokens of
 * each sequence (root first); out_count: host int32 [batch] their number (1..depth+1).
 * ESTATE before prefill, ECAPACITY when n + N + depth + 1 > max_seq_len. */
chimera_status chimera_step(chimera_ctx* ctx, int32_t* out_tokens, int32_t* out_count);

/* n_steps steps back to back on the device (one synchronisation at the end).
 * out_tokens: host int32 [batch][n_steps * (depth+1)], each sequence's emitted
 * tokens packed in order; out_count: host int32 [batch] total emitted per sequence.
 * Capacity is checked up front for the worst case (every step accepts depth tokens). */
chimera_status chimera_generate(chimera_ctx* ctx, int n_steps, int32_t* out_tokens,
                                int32_t* out_count);

/* Enqueue n_steps steps on the context stream and return without synchronising
 * (no host output; capacity checked for the worst case).  For timing. */
chimera_status chimera_step_async(chimera_ctx* ctx, int n_steps);

/* n_steps plain autoregressive steps (eq. 1 with argmax: one base forward per token),
 * the baseline that speculative decoding accelerates.  Each step runs the base model
 * on every sequence's root x[n] at position n, emits that root, writes its KV at slot n,
 * appends its draft-layer KV and makes the argmax the next root: the same state update
 * as a draft-and-verify step that accepts no drafted token, so the two kinds of step
 * can be mixed and produce the same stream.  out_tokens: host int32 [batch][n_steps]
 * (NULL: enqueue only, for timing; then out_count is ignored and chimera_sync
 * completes the steps); out_count: host int32 [batch] (= n_steps). */
chimera_status chimera_ar_generate(chimera_ctx* ctx, int n_steps, int32_t* out_tokens, int32_t* out_count);

/* Block until the context stream is idle and report device-side errors. */
chimera_status chimera_sync(chimera_ctx* ctx);

void chimera_free(chimera_ctx* ctx);
const char* chimera_last_error(const chimera_ctx* ctx);

/* Static tree descriptor (reading of Section "Inference" with Table 4 marginals):
 * depth[N], parent[N] (-1 for the root), rank[N] (rank drawn from head depth-1),
 * anc[N] (bit j set iff node j is an ancestor-or-self).  Host outputs of size N. */
chimera_status chimera_tree(const chimera_ctx* ctx, int32_t* depth, int32_t* parent,
                            int32_t* rank, uint64_t* anc);

/* The same static tree from the configuration alone, on the host, with no context and
 * no GPU: topk host int32 [n_heads], each 1..8 (ranks past the five of Table 4 have no
 * marginal and never enter the tree), 1 <= n_heads <= 4, 2 <= n_nodes <= 64.  Outputs
 * as chimera_tree, host arrays of n_nodes; any may be NULL.  CHIMERA_EINVAL for an
 * argument out of range or when n_nodes - 1 exceeds the rank tuples the limits allow. */
chimera_status chimera_static_tree(const int32_t* topk, int n_heads, int n_nodes, int32_t* depth,
                                   int32_t* parent, int32_t* rank, uint64_t* anc);

/* Per-kernel timing of one step, launched eagerly with CUDA events around every
 * launch (test and benchmark hook).  kinds: host int32 [max] kernel class (see
 * CHIMERA_KIND_*), ms: host float [max], bytes: host double [max] algorithmic HBM
 * bytes of the launch.  *count receives the number of launches. */
enum {
  CHIMERA_KIND_LINEAR = 1,
  CHIMERA_KIND_ATTENTION = 2,
  CHIMERA_KIND_NORM = 3,
  CHIMERA_KIND_ROPE_KV = 4,
  CHIMERA_KIND_SWIGLU = 5,
  CHIMERA_KIND_EMBED = 6,
  CHIMERA_KIND_TOPK = 7,
  CHIMERA_KIND_ARGMAX = 8,
  CHIMERA_KIND_TREE = 9,
  CHIMERA_KIND_ACCEPT = 10,
  CHIMERA_KIND_COMPACT = 11,
  CHIMERA_KIND_OTHER = 12,
  CHIMERA_KIND_CHAIN = 13  /* a persistent chain of linears and row steps (bf16 models) */
};
enum { CHIMERA_PHASE_DRAFT = 0, CHIMERA_PHASE_VERIFY = 1, CHIMERA_PHASE_COMMIT = 2 };
chimera_status chimera_profile_step(chimera_ctx* ctx, int max, int32_t* kinds, int32_t* phases,
                                    float* ms, double* bytes, int32_t* count);

/* Phase-timed steps (benchmark hook): n_steps steps replayed from a graph that records
 * an event at each phase boundary (draft | tree + verify forward + LM head + argmax |
 * acceptance + compaction + draft-KV append), with a synchronisation after each step.
 * draft_ms / verify_ms / commit_ms: host float [n_steps] (any may be NULL).  The steps
 * advance the state like chimera_step_async. */
chimera_status chimera_profile_phases(chimera_ctx* ctx, int n_steps, float* draft_ms, float* verify_ms,
                                      float* commit_ms);

/* One kernel class in isolation (benchmark hook): a graph holding only the launches of
 * class `kind` of one step, in step order and with the step's launch attributes, is
 * replayed n_reps times back to back between two events.  *ms: mean time of one
 * replay; *launches, *bytes (may be NULL): launches per replay and their algorithmic
 * HBM bytes.  The launches read whatever their inputs hold and overwrite only step
 * scratch, which the next step recomputes; classes that update the committed state
 * (acceptance, compaction, the state update) are refused with EINVAL. */
chimera_status chimera_profile_kind(chimera_ctx* ctx, int kind, int n_reps, float* ms, int32_t* launches,
                                    double* bytes);

/* ---- test hooks (part of the library; used by the parity tests) ---- */

/* Replace the drafted tokens of tree nodes 1..N-1 for the NEXT step only
 * (node_tokens: host int32 [batch][N], entry 0 ignored; ids in [0, vocab)). */
chimera_status chimera_debug_override_tree(chimera_ctx* ctx, const int32_t* node_tokens);

/* Replace the root token x[n] of every sequence (host int32 [batch]). */
chimera_status chimera_debug_set_root(chimera_ctx* ctx, const int32_t* roots);

enum {
  CHIMERA_DBG_NODE_TOKENS = 1,    /* int32 [batch][N] tree tokens of the last step */
  CHIMERA_DBG_VERIFY_LOGITS = 2,  /* f32 [batch][N][V] */
  CHIMERA_DBG_VERIFY_HIDDEN = 3,  /* f32 [batch][N][d] post final norm (H_LLM rows) */
  CHIMERA_DBG_ARGMAX = 4,         /* int32 [batch][N] */
  CHIMERA_DBG_PATH = 5,           /* int32 [batch][depth+1] accepted node indices */
  CHIMERA_DBG_ACCEPT_LEN = 6,     /* int32 [batch] L (drafted tokens accepted) */
  CHIMERA_DBG_DRAFT_LOGITS = 7,   /* f32 [K][batch][V] residual-head scores */
  CHIMERA_DBG_TOPK = 8,           /* int32 [batch][K][kmax] */
  CHIMERA_DBG_HFULL = 9,          /* f32 [K][batch][d] full-context outputs */
  CHIMERA_DBG_N = 10,             /* int32 [batch] committed length n */
  CHIMERA_DBG_TOKENS = 11,        /* int32 [batch][max_seq_len + 1] token history */
  CHIMERA_DBG_PREFILL_LOGITS = 12, /* f32 [batch][V] LM-head scores of the last prompt row
                                      (until the first step; after chimera_ar_generate: the
                                      scores of its last step's rows) */
  CHIMERA_DBG_TRIGRAM_HITS = 13,  /* int32 [K][batch] 1 where the last step's sub-step hit the
                                     trigram cache (trigram_cache > 0 only) */
  CHIMERA_DBG_HTRI = 14           /* f32 [K][batch][d] the last step's h_tri rows (trigram_cache
                                     > 0 only) */
};
/* Copy a device buffer of the context to host memory; `bytes` must equal its size. */
chimera_status chimera_debug_read(chimera_ctx* ctx, int what, void* host_dst, size_t bytes);

/* Gather KV rows [pos0, pos0+count) of sequence `seq` from the paged cache of base
 * layer `layer` (layer = -1: the draft block's cache) into host buffers
 * k_dst / v_dst of shape [count][H][hd]: fp32 for fp32 models and for bf16 models with
 * precision 1 (hi + lo), bf16 for precision 0. */
chimera_status chimera_debug_read_kv(chimera_ctx* ctx, int layer, int seq, int pos0, int count,
                                     void* k_dst, void* v_dst);

/* ---- kernel-level entry points (stateless; for per-kernel parity tests) ---- */

/* Y[M][N] (epilogue)= (X + X_lo)[M][K] . W[N][K]^T on the given stream (NULL: default).
 * dtype 1: X, X_lo (optional, NULL = none), W bf16 (K, ldx multiples of 8; 16-byte
 * aligned), tcgen05 kernel; dtype 0: everything fp32, X_lo ignored.  epi 0: Y = acc,
 * 1: Y = SiLU(acc), 2: Y(fp32) += acc.  out_f32 selects an fp32 Y for epi 0/1 with
 * dtype 1.  Device pointers.  Uses a workspace per device, allocated on the first call
 * made with that device current.  Asynchronous: the status covers the arguments and
 * the launch; what the kernel flags on the device (a bounded wait that gave up) is
 * reported by chimera_op_sync. */
chimera_status chimera_op_linear(int dtype, int epi, int out_f32, int M, int N, int K,
                                 const void* X, const void* X_lo, int ldx, const void* W, void* Y,
                                 int ldy, void* cuda_stream);

/* Tree-masked attention over a paged KV pool [blocks][H][planes][16][hd] (device):
 * dtype 0: fp32 planes K, V; dtype 1: bf16 planes K, V, or with kv_split the two-term
 * split K_hi, K_lo, V_hi, V_lo; n_blocks = blocks in the pool (every page-table entry
 * of a visible key must be below it).  q fp32 [batch*q_rows][ldq] rotated queries,
 * query i of sequence b at row b*q_rows+i;
 * n_ctx (device int32 [batch]) committed rows visible to all; n_local rows follow at
 * slots n_ctx..; query i sees local row j iff bit j of anc[q_local0+i] (device
 * uint64); page_table device int32 [batch][max_pages]; out [batch*q_rows][ldo] in the
 * model dtype, out_lo (optional, bf16 only) its lo half.  nq <= 64, n_local <= 64,
 * hd in {64, 128}.  `splits` cuts each sequence's keys into that many contiguous
 * ranges: at most 16, and at most 8 for dtype 1 with hd 128 (the ranges of one
 * (sequence, head) run as one thread-block cluster); EINVAL beyond. */
chimera_status chimera_op_attention(int dtype, int kv_split, int batch, int n_heads, int head_dim,
                                    int nq, int q_local0, int n_local, const float* q, int ldq,
                                    int q_rows, const void* pool, int n_blocks, const int32_t* page_table,
                                    int max_pages, const int32_t* n_ctx, const uint64_t* anc,
                                    void* out, void* out_lo, int ldo, int splits, void* cuda_stream);

/* Wait until `cuda_stream` (NULL: the default stream) is idle, then read and clear the
 * device error words of the stateless entry points (chimera_op_linear,
 * chimera_op_attention, chimera_op_linear_noalloc) on the current device: everything
 * their kernels flagged since the previous chimera_op_sync.  CHIMERA_ETIMEDOUT when a
 * bounded wait gave up (the outputs of those calls are undefined; the split counters
 * of the workspaces are reset, so later calls compute correctly again),
 * CHIMERA_ECAPACITY / CHIMERA_EINVAL for an out-of-range slot or index, CHIMERA_ECUDA
 * when a CUDA call fails, else CHIMERA_OK. */
chimera_status chimera_op_sync(void* cuda_stream);

/* Test hook: limit (ns) of every bounded wait of the tensor-core linear launched by the
 * stateless entry points from now on (0 restores the default of 2 s).  Contexts always
 * use the default.  A limit of a few ns makes the waits give up, which exercises the
 * kernel's clean exit (in-flight copies and MMAs drained, tensor memory freed) and the
 * CHIMERA_ETIMEDOUT report of chimera_op_sync without any fault. */
chimera_status chimera_debug_set_wait_limit(uint64_t ns);

/* Same computation as chimera_op_linear with dtype 1 (bf16, tcgen05), but it allocates
 * nothing: for callers that cannot allocate device memory when they call (code running
 * under a fixed per-process memory budget, inside host callbacks or allocator hooks,
 * or on memory owned by another allocator).  Its split-K scratch lives in arrays that
 * the library defines at file scope (5.2 MB on every GPU that loads the library, held
 * until the process exits).  The paper has no counterpart; it is a service of this
 * library.  Limits: M <= 32, at most 4096 output tiles of 128 columns; larger sizes
 * return CHIMERA_EINVAL with a message on stderr.  The first call on a device looks up
 * the arrays' device addresses (make that first call outside any stream capture).
 * Every call shares the arrays and keeps the last call's contents; the call clears
 * what must start at zero.  Calls that overlap on the GPU race on the scratch: the
 * caller serialises them (one stream, or explicit synchronisation).  A bounded wait
 * that gives up inside the kernel is reported by the next chimera_op_sync. */
chimera_status chimera_op_linear_noalloc(int epi, int out_f32, int M, int N, int K, const void* X,
                                         const void* X_lo, int ldx, const void* W, void* Y, int ldy,
                                         void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* CHIMERA_H */
