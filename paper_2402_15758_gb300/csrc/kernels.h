// Host-side launchers of the sm_103a kernels (internal to the library).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace chimera {

// ----------------------------------------------------------------------------
// bf16 linear on tcgen05: Y[M][N] (epilogue) = X[M][K] . W[N][K]^T
// ----------------------------------------------------------------------------
struct TcLinearParams {
  CUtensorMap tmA;   // W: [N][K] bf16, box 128 x 64, 128-byte swizzle
  CUtensorMap tmA2;  // optional second weight W2 [N2][K]: output columns N .. N+N2-1
  CUtensorMap tmB;   // X: [M][K] bf16 (row pitch ldx), box BN x 64, 128-byte swizzle
  CUtensorMap tmB2;  // X_lo (same shape) when the activation is a hi + lo split
  int has_lo;        // 1: two MMAs per K slice, W.X_hi + W.X_lo into one accumulator
  int ft_split;      // feature tiles taken from W (the rest from W2); = feat_tiles without W2
  int M, N, K;       // N = total output columns (N of W plus N2 of W2)
  int BN;            // token tile = UMMA N (multiple of 16, <= 256)
  int tok_tiles, feat_tiles, kblocks;
  long long units;   // feat_tiles * tok_tiles * kblocks
  int stages;        // smem pipeline depth
  int vec_red;       // EPI_RESID through float4 reductions
  int epi;           // EPI_*
  int out_f32;       // Y is fp32 (else bf16) for EPI_STORE / EPI_SILU
  void* Y;
  void* Y2;          // optional bf16 lo half of Y (EPI_STORE / EPI_SILU, bf16 Y)
  int ldy;
  float* ws;         // split partials: [grid][2][128 * BN] fp32
  int* counters;     // [feat_tiles * tok_tiles], all zero between launches
  int* err;          // device error word
  unsigned long long wait_ns;  // limit of every bounded wait of the launch (ns)
  const int* skip;   // optional device flag: nonzero at run time -> the launch does nothing
  uint32_t tmem_cols;
  uint32_t acc_stride;  // TMEM column distance between the two accumulators
  // optional: [zero, zero + zero_floats) cleared by the epilogue warps after the
  // dependency wait, spread over the CTAs (a later linear's fp32 accumulator)
  float* zero;
  long long zero_floats;
};

struct TcLinearPlan {
  TcLinearParams p;
  int grid = 0;
  size_t smem = 0;
  double weight_bytes = 0;  // algorithmic bytes streamed per launch (W once)
};

// Limit of the linear kernel's bounded waits, taken by every plan encoded afterwards
// (default 2 s; lowered only by the timeout test hook of the stateless entry points).
constexpr unsigned long long kDefaultWaitNs = 2000000000ull;
extern std::atomic<unsigned long long> g_lin_wait_ns;

// Largest grid of the linear kernel (one CTA per SM) and the workspace it needs.
int tc_num_sms();
size_t tc_ws_floats(int max_bn);
int tc_max_tiles();

// Encode the plan for one call site.  X/W/Y are device pointers; ws/counters are
// scratch owned by the caller (sizes from tc_ws_floats / tc_max_tiles).
// Returns 0 on success, otherwise a negative code and a message in `msg`.
// W2 (optional, N2 rows): a second weight matrix whose outputs follow W's in Y (one
// launch for two projections of the same input, e.g. SwiGLU gate and up); needs N % 128 == 0.
int tc_linear_plan(TcLinearPlan* plan, int M, int N, int K, const void* X, const void* X_lo, int ldx,
                   const void* W, void* Y, void* Y_lo, int ldy, int epi, int out_f32, float* ws,
                   int* counters, int* err, char* msg, size_t msg_len, const void* W2 = nullptr, int N2 = 0,
                   float* zero = nullptr, long long zero_floats = 0);
cudaError_t tc_linear_launch(const TcLinearPlan& plan, cudaStream_t s);

// Error word of the allocation-free linear's static scratch on the current device:
// read into *word and cleared.  0 on success, -1 when a CUDA call failed.
int noalloc_take_error(int* word);

// ----------------------------------------------------------------------------
// Persistent chain of bf16 linears and row steps in one launch (chain_tc.cu)
// ----------------------------------------------------------------------------
constexpr int CHAIN_MAX_GEMM = 4;
constexpr int CHAIN_MAX_ROW = 4;
constexpr int CHAIN_MAX_STEPS = 8;
enum : int { CH_GEMM = 0, CH_NORM = 1, CH_SWIGLU = 2, CH_COPY = 3 };

// One linear of a chain: Y[M][N] (fp32) += X[M][K] . W[N][K]^T (X bf16, optional lo half).
struct ChainGemm {
  CUtensorMap tmA, tmA2, tmB, tmB2;  // W, optional W2 (outputs N1..), X, X_lo
  int N, K, ft_split, feat_tiles, kblocks;
  uint32_t units;                    // feat_tiles * tok_tiles * kblocks
  float* Y;
  int ldy;
};
// One row step: CH_NORM  y = RMSNorm(X row; gains g, eps) -> Y (+ Y_lo), Y32; Z row cleared
//               CH_SWIGLU y = SiLU(X[:, :cols]) * X[:, cols:2 cols] -> Y (+ Y_lo)
//               CH_COPY  y = X row -> Y (+ Y_lo), Y32; Z row cleared
struct ChainRow {
  const float* X;
  int ldx;
  const void* g;
  void* Y;
  void* Y_lo;
  int ldy;
  float* Y32;
  int ld32;
  float* Z;
  int ldz, zcols;
  int rows, cols;
  float eps;
};
struct ChainParams {
  ChainGemm gemm[CHAIN_MAX_GEMM];
  ChainRow row[CHAIN_MAX_ROW];
  int n_steps, n_gemm, n_row;
  int kind[CHAIN_MAX_STEPS];       // CH_*
  int idx[CHAIN_MAX_STEPS];        // index into gemm[] or row[]
  int wait[CHAIN_MAX_STEPS];       // step whose completion the step's input needs (-1: none)
  int gemm_step[CHAIN_MAX_GEMM];   // step of each linear
  int M, BN, tok_tiles, has_lo, stages;
  int* bars;                       // [CHAIN_MAX_STEPS + 1] counters, all zero between launches
  int* err;
  unsigned long long wait_ns;
  uint32_t tmem_cols, acc_stride;
};
struct ChainPlan {
  ChainParams p;
  int grid = 0;
  size_t smem = 0;
  double weight_bytes = 0;
};
// Start a plan for M token rows (has_lo: the activations are hi + lo bf16 pairs).
int chain_plan(ChainPlan* plan, int M, int has_lo, char* msg, size_t msg_len);
// Append a linear / a row step that waits for step `wait` (-1: none); returns the new
// step's index, or -1 with a message.
int chain_add_gemm(ChainPlan* plan, int wait, const void* X, const void* X_lo, int ldx, int K, const void* W, int N,
                   const void* W2, int N2, float* Y, int ldy, char* msg, size_t msg_len);
int chain_add_row(ChainPlan* plan, int kind, int wait, const ChainRow& row, char* msg, size_t msg_len);
cudaError_t chain_launch(const ChainPlan& plan, cudaStream_t s);

// ----------------------------------------------------------------------------
// fp32 linear (SIMT, exact fp32 FMA order per output)
// ----------------------------------------------------------------------------
// skip (optional, device): when *skip != 0 at run time the launch does nothing (its
// output was provided another way, e.g. by the trigram cache).
cudaError_t f32_linear(int M, int N, int K, const float* X, int ldx, const float* W, float* Y,
                       int ldy, int epi, cudaStream_t s, const int* skip = nullptr);

// ----------------------------------------------------------------------------
// attention over the paged KV cache with a per-query ancestor bitmask
// ----------------------------------------------------------------------------
struct AttnParams {
  const float* q;         // rotated fp32 queries, row (b * q_rows + i), head h at col h*hd
  int ldq, q_rows;
  int nq;                 // queries per sequence
  const int* nq_dev;      // optional per-sequence query count (overrides nq when set)
  int q_local0;           // local row index of query 0 (mask lookup: anc[q_local0 + i])
  int n_local;            // local rows at slots n..n+n_local-1
  const int* n_local_dev; // optional per-sequence local count
  const unsigned long long* anc;  // [q_local0 + nq] ancestor-or-self masks over local rows
  const void* pool;       // [blocks][H][planes][16][hd], element type of the model
  long long pool_rows;    // 16-row page rows in the whole allocation (layers x blocks x H x planes x 16)
  int planes;             // 2: K, V;  4: K_hi, K_lo, V_hi, V_lo (bf16 two-term split)
  long long pool_layer_stride;  // elements between layers (0 for the draft pool)
  int layer;
  const int* page_table;  // [B][max_pages]
  int max_pages;
  const int* n_ctx;       // [B] committed rows (all visible)
  void* out;              // [b * q_rows + i][H * hd] (model dtype)
  void* out_lo;           // optional lo half (bf16 split activations)
  int ldo;
  int B, H, hd;
  float scale;
  int splits;             // KV splits per (b, h)
  float* ws;              // [B][H][splits][nq_max][hd + 4] (output, max, sum, pad)
  int* counters;          // [B][H], zero between launches
  int nq_max;
  // Fused RoPE + KV write (bf16 models, head_dim 128).  With qkv set, the queries and
  // the nq fresh local rows come from the fp32 projections: row (b * q_rows + i) holds
  // q at column h*hd, k at H*hd + h*hd, v at 2*H*hd + h*hd.  Query / fresh row i sits at
  // position n_ctx + pos_base + (pos_off ? pos_off[i] : i) and at local row q_local0 + i
  // (slot n_ctx + q_local0 + i); the kernel rotates q and k and writes k and v of its
  // key range into the pool before reading it.
  const float* qkv;
  int ldqkv;
  const float2* rope;     // [max_pos][hd / 2] (cos, sin)
  int max_pos;
  int pos_base;
  const int* pos_off;
  // 1: the preceding kernel in the stream lets its dependents launch only after its
  // own griddepcontrol.wait, so every kernel before it is complete and committed KV
  // rows (slots < n_ctx) may be read before this kernel's own wait
  int prewait_kv;
  int* err;
};
// dtype: 0 fp32 model (fp32 KV), 1 bf16 model (bf16 KV planes).
cudaError_t attention(const AttnParams& p, int dtype, cudaStream_t s);
size_t attn_ws_floats(int B, int H, int splits, int nq_max, int hd);
// Splits per (b, h) for the tensor-core tree attention (bf16, head_dim 128): at most
// `want` and 8 (one thread-block cluster per (b, h)), reduced until all B * H clusters
// are resident at once.  Other paths return `want` unchanged.
int attn_pick_splits(int dtype, int hd, int planes, int B, int H, int want);
// 2D bf16 tensor map (128-byte swizzle, zero fill out of bounds) of a row-major matrix
// [outer][pitch_elems] with an inner extent of `inner` elements; 0 on success.
int encode_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_elems,
                   uint32_t box_inner, uint32_t box_outer);
// Tensor-core tree attention (bf16 planes, head_dim 128; splits <= 8 form one cluster).
cudaError_t attention_tc(const AttnParams& p, cudaStream_t s);
int attention_tc_splits(int planes, int BH, int want);
// True when attention() fuses RoPE and the KV write (qkv given) for this model.
bool attn_fuses_rope(int dtype, int hd);

// ----------------------------------------------------------------------------
// row-wise / small kernels
// ----------------------------------------------------------------------------
// Y (model dtype, plus the optional lo half) and an optional fp32 copy Y32; also zeroes
// rows [0, rows) x [0, zcols) of Z when given (zcols, ldz multiples of 4).
cudaError_t rmsnorm(int dtype, const float* X, int ldx, const void* g, void* Y, void* Y_lo, float* Y32,
                    int ldy, int rows, int d, float eps, float* Z, int ldz, int zcols, cudaStream_t s);

struct RopeKvParams {
  const float* qkv;  // [rows][ldqkv] fp32 projections
  int ldqkv;
  int q_col, k_col, v_col;  // column offsets (q_col < 0: no query output)
  float* q_out;      // [rows][H*hd] fp32
  int ldq;
  void* pool;          // [blocks][H][planes][16][hd]
  int planes;          // 2 or 4 (split hi/lo planes, bf16 models)
  long long pool_layer_stride;
  int layer;
  const int* page_table;
  int max_pages;
  const int* n;        // [B]
  int rows_per_seq;
  const int* valid;    // optional [B] rows written to the cache
  int valid_plus;      // valid[b] + valid_plus rows are written (accept length -> path length)
  int pos_base, slot_base;
  const int* pos_off;  // optional [rows_per_seq]
  const float2* rope;  // [max_pos][hd/2] (cos, sin)
  int max_pos;
  int B, H, hd;
  int* err;
};
cudaError_t rope_kv(const RopeKvParams& p, int dtype, cudaStream_t s);

cudaError_t swiglu(int dtype, const float* gu, int ldgu, int F, void* h, void* h_lo, int ldh, int rows,
                   cudaStream_t s);

// x[r][:] = E[tok(r)] with tok(r) = tokens[r] (mode 0) or tok_hist[b][n[b]+i] for
// i < valid[b] and 0 otherwise (mode 1, prefill chunks).
cudaError_t embed(int dtype, const void* E, int d, int V, float* x, int rows, int rows_per_seq,
                  const int* tokens, const int* tok_hist, int hist_stride, const int* n,
                  const int* valid, int* err, cudaStream_t s);

// Argmax of each row (larger value first, then smaller index); with `stats` also the
// row's max m, log sum exp(z - m) and entropy of softmax(z) in nats: stats[row][3].
cudaError_t argmax_rows(const float* logits, int V, int rows, int* out, cudaStream_t s, float* stats = nullptr);
// Top-k (k <= 8) of each row, larger score first, then smaller index.  Scratch:
// ws_v / ws_i [rows][TOPK_MAX_BLOCKS][8], counters [rows] (zero between launches).
constexpr int TOPK_MAX_BLOCKS = 64;  // V <= 64 * 2048
cudaError_t topk_rows(const float* logits, int V, int rows, int k, int* idx, float* val, int out_stride,
                      float* ws_v, int* ws_i, int* counters, cudaStream_t s);

}  // namespace chimera
