// Small kernels that stitch the step together: trigram gather, tree expansion,
// greedy acceptance, KV compaction, hidden-state gathers and state update.
#include "common.cuh"
#include "launch.cuh"
#include "step_kernels.h"

namespace chimera {
namespace {

// Trigram input of draft sub-step k (eq. trigram_calculations): the embeddings of
// x[n-2+k], x[n-1+k], x[n+k], where x[n] is the root and x[n+1+j] is head j's top-1.
// A position before the start of the sequence contributes a zero block.
// Also zeroes row b of `zero` (d floats): the draft residual that W2 accumulates into.
template <typename T>
__global__ void trigram_gather_kernel(const T* E, int d, int V, const int* n_arr,
                                      const int* tok, int tok_stride, const int* topk, int K,
                                      int KMAX, int k, T* out, int* err, float* zero, float* zero2,
                                      long long zero2_floats) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  // blockIdx.y = t < 3: block t of the trigram; t = 3: the residual row; t > 3: a share
  // of zero2 (the CTAs run side by side, so the three dependent gathers overlap)
  const int b = blockIdx.x, t = blockIdx.y;
  if (t > 3) {
    const long long n4 = zero2_floats / 4, nz = static_cast<long long>(gridDim.x) * (gridDim.y - 4);
    const long long per = (n4 + nz - 1) / nz, z0 = (static_cast<long long>(t - 4) * gridDim.x + b) * per;
    float4* z = reinterpret_cast<float4*>(zero2);
    for (long long i = z0 + threadIdx.x; i < min(n4, z0 + per); i += blockDim.x) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  if (t == 3) {
    for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4)
      *reinterpret_cast<float4*>(zero + static_cast<size_t>(b) * d + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  const int n = n_arr[b];
  const int i = n - 2 + k + t;
  int id = -1;
  if (i >= 0) id = i <= n ? tok[static_cast<size_t>(b) * tok_stride + i] : topk[(b * K + (i - n - 1)) * KMAX];
  if (id >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERR_BAD_INDEX);
    id = 0;
  }
  T* o = out + static_cast<size_t>(b) * 3 * d + t * d;
  const T* e = E + static_cast<size_t>(id < 0 ? 0 : id) * d;
  // 16-byte chunks (d * sizeof(T) is a multiple of 16)
  constexpr int PER = 16 / sizeof(T);
  for (int c = threadIdx.x * PER; c < d; c += blockDim.x * PER)
    *reinterpret_cast<uint4*>(o + c) = id < 0 ? make_uint4(0, 0, 0, 0) : *reinterpret_cast<const uint4*>(e + c);
}

// headin[b][d..2d) = h_full (the draft block output), kept per head for debugging;
// with `zero`, also zeroes row b of the head's score buffer (V floats) that its linear
// accumulates into.
template <typename T>
__global__ void hfull_store_kernel(const float* dres, int d, T* headin,
                                   T* headin_lo, float* hlog,
                                   float* zero, int V) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x;
  if (zero)
    for (int c = threadIdx.x * 4; c < V; c += blockDim.x * 4)
      *reinterpret_cast<float4*>(zero + static_cast<size_t>(b) * V + c) = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(dres + static_cast<size_t>(b) * d + c);
    const size_t o = static_cast<size_t>(b) * 2 * d + d + c;
    store_act4(headin, headin_lo, o, v);
    *reinterpret_cast<float4*>(hlog + static_cast<size_t>(b) * d + c) = v;
  }
}

// Node tokens of the static tree: the root is x[n]; node i at depth >= 1 takes the
// rank_i-th token of head depth_i - 1 (Section "Inference").
__global__ void tree_expand_kernel(const int* n_arr, const int* tok, int tok_stride, const int* topk,
                                   int K, int KMAX, const int* depth, const int* rank, int N,
                                   const int* ovr_flag, const int* ovr, int* node_tok) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x, i = threadIdx.x;
  if (i >= N) return;
  int t;
  if (i == 0)
    t = tok[static_cast<size_t>(b) * tok_stride + n_arr[b]];
  else if (*ovr_flag)
    t = ovr[b * N + i];
  else
    t = topk[(b * K + depth[i] - 1) * KMAX + rank[i]];
  node_tok[b * N + i] = t;
}

// Greedy acceptance (Section "Verification"): from the root, move to the child whose
// token equals the base argmax of the current node; the argmax after the last
// accepted node is the bonus token.  Writes the path and the accepted tokens into
// the token history at x[n..n+L].
__global__ void accept_kernel(const int* n_arr, int* tok, int tok_stride, const int* node_tok,
                              const int* amax, const int* child_start, const int* child, int N,
                              int D1, int* path, int* Lacc, int* bonus) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x;
  if (threadIdx.x != 0) return;
  const int n = n_arr[b];
  int cur = 0, L = 0;
  path[b * D1] = 0;
  while (true) {
    const int p = amax[b * N + cur];
    int nxt = -1;
    for (int c = child_start[cur]; c < child_start[cur + 1]; ++c)
      if (node_tok[b * N + child[c]] == p) {
        nxt = child[c];
        break;
      }
    if (nxt < 0 || L + 1 >= D1) break;
    cur = nxt;
    ++L;
    path[b * D1 + L] = cur;
    tok[static_cast<size_t>(b) * tok_stride + n + L] = node_tok[b * N + cur];
  }
  for (int j = L + 1; j < D1; ++j) path[b * D1 + j] = path[b * D1 + L];
  Lacc[b] = L;
  bonus[b] = amax[b * N + cur];
}

// Move the accepted nodes' K/V rows from tree slot n+path[j] to slot n+j (j = 1..L)
// in every layer.  All source rows are loaded before any store: a destination slot
// can be the source of another path entry.
__global__ void compact_kernel(char* pool, long long layer_stride_bytes, int H, int planes, int row_bytes,
                               const int* n_arr, const int* path, const int* Lacc, int D1,
                               const int* page_table, int max_pages) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.y;
  const int L = Lacc[b];
  if (L == 0) return;
  const int layer = blockIdx.x / (planes * H);
  const int kv = (blockIdx.x / H) % planes;  // plane index
  const int h = blockIdx.x % H;
  const int n = n_arr[b];
  const int chunks = row_bytes / 16;
  const int j = 1 + threadIdx.x / chunks;
  const int c = threadIdx.x % chunks;
  char* base = pool + layer * layer_stride_bytes;
  auto row_ptr = [&](int slot) {
    const int page = page_table[b * max_pages + (slot >> 4)];
    return reinterpret_cast<uint4*>(base + ((static_cast<size_t>(page) * H + h) * planes + kv) * 16 * row_bytes +
                                    static_cast<size_t>(slot & 15) * row_bytes) + c;
  };
  uint4 v = make_uint4(0, 0, 0, 0);
  const bool active = j <= L && j < D1;
  if (active) v = *row_ptr(n + path[b * D1 + j]);
  __syncthreads();
  if (active) *row_ptr(n + j) = v;
}

// hsel[b][j] = verify hidden (fp32) of path node j (j <= L; later rows repeat the
// last); headin[b][0..d) = hidden of the last accepted node (h_LLM of the new prefix end).
template <typename T>
__global__ void gather_hidden_kernel(const float* hfin, int d, int N, const int* path,
                                     const int* Lacc, int D1, float* hsel,
                                     T* headin, T* headin_lo) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x, j = blockIdx.y;
  const int L = Lacc[b];
  const int node = path[b * D1 + (j <= L ? j : L)];
  const float* src = hfin + static_cast<size_t>(b * N + node) * d;
  float* dst = hsel + static_cast<size_t>(b * D1 + j) * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = src[c];
    dst[c] = v;
    if (j == L) store_act(headin, headin_lo, static_cast<size_t>(b) * 2 * d + c, v);
  }
}

// Commit: x[n+L+1] = bonus (the next root), n += L + 1, per-step count log.
__global__ void finalize_kernel(int* n_arr, int* tok, int tok_stride, const int* Lacc,
                                const int* bonus, int* count_log, int log_cap, int* step, int B) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = threadIdx.x;
  const int s = *step;
  __syncthreads();
  if (b < B) {
    const int L = Lacc[b];
    const int n = n_arr[b];
    tok[static_cast<size_t>(b) * tok_stride + n + L + 1] = bonus[b];
    n_arr[b] = n + L + 1;
    count_log[b * log_cap + (s % log_cap)] = L + 1;
  }
  __syncthreads();
  if (threadIdx.x == 0) *step = s + 1;
}

// Prefill chunk bookkeeping: keep h_LLM of the last prompt row, advance n.
template <typename T>
__global__ void prefill_advance_kernel(const float* hfin, int d, int rows_per_seq,
                                       const int* valid, const int* last, int* n_arr,
                                       T* headin, T* headin_lo) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x;
  const int li = last[b];
  if (li >= 0) {
    const float* src = hfin + static_cast<size_t>(b * rows_per_seq + li) * d;
    for (int c = threadIdx.x; c < d; c += blockDim.x)
      store_act(headin, headin_lo, static_cast<size_t>(b) * 2 * d + c, src[c]);
  }
  if (threadIdx.x == 0) n_arr[b] += valid[b];
}

__global__ void set_root_kernel(const int* n_arr, int* tok, int tok_stride, const int* amax, int B) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = threadIdx.x;
  if (b < B) tok[static_cast<size_t>(b) * tok_stride + n_arr[b]] = amax[b];
}

// ---------------------------------------------------------------------------
// Trigram cache (the lookup table of the trigram encoder's outputs): a 4-way set-
// associative table of h_tri rows keyed by the three token ids, least recently used
// way replaced.  Key = (x_{i-2}+1) << 42 | (x_{i-1}+1) << 21 | x_i (a missing leading
// token is -1, so its field is 0); 0 marks an empty way.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int trigram_id(const int* tok, int tok_stride, const int* topk, int K, int KMAX, int b,
                                          int n, int i) {
  if (i < 0) return -1;
  return i <= n ? tok[static_cast<size_t>(b) * tok_stride + i] : topk[(b * K + (i - n - 1)) * KMAX];
}

__device__ __forceinline__ unsigned long long trigram_key(int a, int b, int c) {
  return (static_cast<unsigned long long>(a + 1) << 42) | (static_cast<unsigned long long>(b + 1) << 21) |
         static_cast<unsigned long long>(c);
}

// One block for the batch.  For sequence b: the trigram of sub-step k; on a hit its
// row is copied into dres[b] (the h_tri the encoder would produce) and its stamp
// refreshed; on a miss the way to replace is recorded.  skip = every sequence hit
// (the encoder's two linears then do nothing).
__global__ void trigram_lookup_kernel(const int* n_arr, const int* tok, int tok_stride, const int* topk, int K,
                                      int KMAX, int k, int B, int d, int nsets,
                                      const unsigned long long* keys, int* stamp, const float* vals,
                                      float* dres, int* hit, int* slot, int* skip, int* clock, int* hit_log) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  __shared__ int s_all;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  if (threadIdx.x == 0) s_all = 1;
  __syncthreads();
  const int now = *clock;
  for (int b = warp; b < B; b += nw) {
    const int n = n_arr[b];
    const int x0 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n - 2 + k);
    const int x1 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n - 1 + k);
    const int x2 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n + k);
    const unsigned long long key = trigram_key(x0, x1, x2);
    const int set = static_cast<int>((key * 0x9E3779B97F4A7C15ull) >> 40) & (nsets - 1);
    int found = -1, victim = 0, oldest = 0x7fffffff;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int e = set * 4 + w;
      const unsigned long long kk = keys[e];
      if (kk == key && found < 0) found = e;
      const int age = kk == 0ull ? -1 : stamp[e];  // an empty way is replaced first
      if (age < oldest) {
        oldest = age;
        victim = e;
      }
    }
    if (found >= 0) {
      const float4* src = reinterpret_cast<const float4*>(vals + static_cast<size_t>(found) * d);
      float4* dst = reinterpret_cast<float4*>(dres + static_cast<size_t>(b) * d);
      for (int c = lane; c < d / 4; c += 32) dst[c] = src[c];
    }
    if (lane == 0) {
      hit[b] = found >= 0 ? 1 : 0;
      slot[b] = found >= 0 ? found : victim;
      if (found >= 0) stamp[found] = now;
      else s_all = 0;
      if (hit_log) hit_log[k * B + b] = found >= 0 ? 1 : 0;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    *skip = s_all;
    *clock = now + 1;
  }
}

// After the encoder ran: store each missed sequence's h_tri row (dres[b]) in the way
// chosen by the lookup.  Sequences are taken in order, so two of them that picked the
// same way leave one consistent entry.  Also logs every h_tri row of the sub-step.
__global__ void trigram_insert_kernel(const int* n_arr, const int* tok, int tok_stride, const int* topk, int K,
                                      int KMAX, int k, int B, int d, unsigned long long* keys, int* stamp,
                                      float* vals, const float* dres, const int* hit, const int* slot,
                                      const int* clock, float* htri_log) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int now = *clock - 1;
  for (int b = 0; b < B; ++b) {
    const float4* src = reinterpret_cast<const float4*>(dres + static_cast<size_t>(b) * d);
    if (htri_log) {
      float4* lg = reinterpret_cast<float4*>(htri_log + (static_cast<size_t>(k) * B + b) * d);
      for (int c = threadIdx.x; c < d / 4; c += blockDim.x) lg[c] = src[c];
    }
    if (hit[b]) continue;
    const int e = slot[b];
    float4* dst = reinterpret_cast<float4*>(vals + static_cast<size_t>(e) * d);
    for (int c = threadIdx.x; c < d / 4; c += blockDim.x) dst[c] = src[c];
    if (threadIdx.x == 0) {
      const int n = n_arr[b];
      const int x0 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n - 2 + k);
      const int x1 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n - 1 + k);
      const int x2 = trigram_id(tok, tok_stride, topk, K, KMAX, b, n, n + k);
      keys[e] = trigram_key(x0, x1, x2);
      stamp[e] = now;
    }
    __syncthreads();
  }
}

// Typical acceptance (Section "Verification", temperature 1): node c is acceptable
// when its parent is and p_parent(token_c) > min(eps, delta exp(-H_parent)), p the
// softmax of the parent's logits and H its entropy (stats from the argmax kernel:
// max, log-sum-exp, entropy).  The path ends at the deepest acceptable node (the
// smallest index among the deepest); the bonus is the base argmax there.  Writes the
// path and the accepted tokens into the token history at x[n+1..n+L].
__global__ void accept_typical_kernel(const int* n_arr, int* tok, int tok_stride, const int* node_tok,
                                      const int* amax, const float* logits, int V, const float* stats,
                                      const int* parent, const int* depth, int N, int D1, float eps, float delta,
                                      int* path, int* Lacc, int* bonus) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int b = blockIdx.x;
  __shared__ int s_ok[64];
  // thread c decides node c against its parent's distribution
  const int c = threadIdx.x;
  int pass = 0;
  if (c < N) {
    if (c == 0) {
      pass = 1;
    } else {
      const int par = parent[c];
      const size_t row = static_cast<size_t>(b) * N + par;
      const float m = stats[3 * row], lse = stats[3 * row + 1], H = stats[3 * row + 2];
      const int t = node_tok[b * N + c];
      const float p = expf(logits[row * V + t] - m - lse);
      const float thr = fminf(eps, delta * expf(-H));
      pass = p > thr ? 1 : 0;
    }
    s_ok[c] = pass;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  // parents precede children: fold the ancestors' decisions in node order
  for (int i = 1; i < N; ++i) s_ok[i] = s_ok[i] && s_ok[parent[i]];
  int best = 0;
  for (int i = 1; i < N; ++i)
    if (s_ok[i] && depth[i] > depth[best]) best = i;
  const int L = depth[best];
  const int n = n_arr[b];
  for (int j = L, i = best; j >= 0; --j, i = parent[i]) {
    path[b * D1 + j] = i;
    if (j >= 1) tok[static_cast<size_t>(b) * tok_stride + n + j] = node_tok[b * N + i];
  }
  for (int j = L + 1; j < D1; ++j) path[b * D1 + j] = best;
  Lacc[b] = L;
  bonus[b] = amax[b * N + best];
}

}  // namespace

cudaError_t launch_trigram_gather(int dtype, const void* E, int d, int V, const int* n, const int* tok,
                                  int tok_stride, const int* topk, int K, int KMAX, int k, void* out,
                                  int B, int* err, float* zero, cudaStream_t s, float* zero2, long long zero2_floats) {
  if (zero2 && ((zero2_floats & 3) || (reinterpret_cast<uintptr_t>(zero2) & 15))) return cudaErrorInvalidValue;
  const int zy = zero2 ? 16 : 0;  // CTAs per sequence that clear zero2
  if (dtype == 0)
    launch_pdl(trigram_gather_kernel<float>, dim3(B, 4 + zy), dim3(256), 0, s, static_cast<const float*>(E), d, V, n, tok,
               tok_stride, topk, K, KMAX, k, static_cast<float*>(out), err, zero, zero2, zero2_floats);
  else
    launch_pdl(trigram_gather_kernel<bf16>, dim3(B, 4 + zy), dim3(256), 0, s, static_cast<const bf16*>(E), d, V, n, tok,
               tok_stride, topk, K, KMAX, k, static_cast<bf16*>(out), err, zero, zero2, zero2_floats);
  return cudaGetLastError();
}

cudaError_t launch_hfull_store(int dtype, const float* dres, int d, void* headin, void* headin_lo, float* hlog,
                               float* zero, int V, int B, cudaStream_t s) {
  if (dtype == 0)
    launch_pdl(hfull_store_kernel<float>, dim3(B), dim3(256), 0, s, dres, d, static_cast<float*>(headin), nullptr, hlog, zero, V);
  else
    launch_pdl(hfull_store_kernel<bf16>, dim3(B), dim3(256), 0, s, dres, d, static_cast<bf16*>(headin), static_cast<bf16*>(headin_lo),
                                               hlog, zero, V);
  return cudaGetLastError();
}

cudaError_t launch_tree_expand(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX,
                               const int* depth, const int* rank, int N, const int* ovr_flag, const int* ovr,
                               int* node_tok, int B, cudaStream_t s) {
  launch_pdl(tree_expand_kernel, dim3(B), dim3(64), 0, s, n, tok, tok_stride, topk, K, KMAX, depth, rank, N, ovr_flag, ovr, node_tok);
  return cudaGetLastError();
}

cudaError_t launch_accept(const int* n, int* tok, int tok_stride, const int* node_tok, const int* amax,
                          const int* child_start, const int* child, int N, int D1, int* path, int* Lacc,
                          int* bonus, int B, cudaStream_t s) {
  launch_pdl(accept_kernel, dim3(B), dim3(32), 0, s, n, tok, tok_stride, node_tok, amax, child_start, child, N, D1, path, Lacc,
                                 bonus);
  return cudaGetLastError();
}

cudaError_t launch_trigram_lookup(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX, int k,
                                  int B, int d, int nsets, const unsigned long long* keys, int* stamp,
                                  const float* vals, float* dres, int* hit, int* slot, int* skip, int* clock,
                                  int* hit_log, cudaStream_t s) {
  launch_pdl(trigram_lookup_kernel, dim3(1), dim3(256), 0, s, n, tok, tok_stride, topk, K, KMAX, k, B, d, nsets, keys,
             stamp, vals, dres, hit, slot, skip, clock, hit_log);
  return cudaGetLastError();
}

cudaError_t launch_trigram_insert(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX, int k,
                                  int B, int d, unsigned long long* keys, int* stamp, float* vals, const float* dres,
                                  const int* hit, const int* slot, const int* clock, float* htri_log, cudaStream_t s) {
  launch_pdl(trigram_insert_kernel, dim3(1), dim3(256), 0, s, n, tok, tok_stride, topk, K, KMAX, k, B, d, keys, stamp,
             vals, dres, hit, slot, clock, htri_log);
  return cudaGetLastError();
}

cudaError_t launch_accept_typical(const int* n, int* tok, int tok_stride, const int* node_tok, const int* amax,
                                  const float* logits, int V, const float* stats, const int* parent, const int* depth,
                                  int N, int D1, float eps, float delta, int* path, int* Lacc, int* bonus, int B,
                                  cudaStream_t s) {
  if (N > 64) return cudaErrorInvalidValue;
  launch_pdl(accept_typical_kernel, dim3(B), dim3(64), 0, s, n, tok, tok_stride, node_tok, amax, logits, V, stats, parent,
             depth, N, D1, eps, delta, path, Lacc, bonus);
  return cudaGetLastError();
}

cudaError_t launch_compact(void* pool, long long layer_stride_bytes, int n_layers, int H, int planes, int row_bytes,
                           const int* n, const int* path, const int* Lacc, int D1, const int* page_table,
                           int max_pages, int B, cudaStream_t s) {
  const int threads = (row_bytes / 16) * (D1 - 1);
  if (threads <= 0) return cudaSuccess;
  dim3 grid(n_layers * planes * H, B);
  launch_pdl(compact_kernel, dim3(grid), dim3(threads), 0, s, static_cast<char*>(pool), layer_stride_bytes, H, planes, row_bytes, n,
                                          path, Lacc, D1, page_table, max_pages);
  return cudaGetLastError();
}

cudaError_t launch_gather_hidden(int dtype, const float* hfin, int d, int N, const int* path, const int* Lacc,
                                 int D1, float* hsel, void* headin, void* headin_lo, int B, cudaStream_t s) {
  dim3 grid(B, D1);
  if (dtype == 0)
    launch_pdl(gather_hidden_kernel<float>, dim3(grid), dim3(256), 0, s, hfin, d, N, path, Lacc, D1, hsel, static_cast<float*>(headin),
                                                     nullptr);
  else
    launch_pdl(gather_hidden_kernel<bf16>, dim3(grid), dim3(256), 0, s, hfin, d, N, path, Lacc, D1, hsel, static_cast<bf16*>(headin),
                                                    static_cast<bf16*>(headin_lo));
  return cudaGetLastError();
}

cudaError_t launch_finalize(int* n, int* tok, int tok_stride, const int* Lacc, const int* bonus, int* count_log,
                            int log_cap, int* step, int B, cudaStream_t s) {
  launch_pdl(finalize_kernel, dim3(1), dim3(((B + 31) / 32) * 32), 0, s, n, tok, tok_stride, Lacc, bonus, count_log, log_cap, step, B);
  return cudaGetLastError();
}

cudaError_t launch_prefill_advance(int dtype, const float* hfin, int d, int rows_per_seq, const int* valid,
                                   const int* last, int* n, void* headin, void* headin_lo, int B, cudaStream_t s) {
  if (dtype == 0)
    launch_pdl(prefill_advance_kernel<float>, dim3(B), dim3(256), 0, s, hfin, d, rows_per_seq, valid, last, n,
                                                    static_cast<float*>(headin), nullptr);
  else
    launch_pdl(prefill_advance_kernel<bf16>, dim3(B), dim3(256), 0, s, hfin, d, rows_per_seq, valid, last, n,
                                                   static_cast<bf16*>(headin), static_cast<bf16*>(headin_lo));
  return cudaGetLastError();
}

cudaError_t launch_set_root(const int* n, int* tok, int tok_stride, const int* amax, int B, cudaStream_t s) {
  launch_pdl(set_root_kernel, dim3(1), dim3(((B + 31) / 32) * 32), 0, s, n, tok, tok_stride, amax, B);
  return cudaGetLastError();
}

}  // namespace chimera
