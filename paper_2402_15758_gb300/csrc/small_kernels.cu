// Row-wise kernels of the step: RMSNorm, RoPE + paged KV write, SwiGLU, embedding
// gather, argmax and top-k over the vocabulary.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "launch.cuh"
#include "kernels.h"

namespace chimera {
namespace {

// Deterministic block sum (fixed tree order), blockDim.x multiple of 32, <= 1024.
__device__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  float t = lane < nw ? red[lane] : 0.f;
  if (warp == 0) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) red[32] = t;
  }
  __syncthreads();
  const float r = red[32];
  __syncthreads();
  return r;
}

// RMSNorm (Llama): y = x / sqrt(mean(x^2) + eps) * g, from the fp32 residual stream.
// Writes the GEMM operand (model dtype, optional lo half) and an optional fp32 copy.
// Side job: zero row r of Z (the fp32 output that the next linear accumulates into).
constexpr int NORM_THREADS = 256;
constexpr int NORM_VEC = 8;  // float4 per thread: d <= 8192

template <typename T>
__device__ __forceinline__ float4 load_g4(const T* g, int i);
template <>
__device__ __forceinline__ float4 load_g4<float>(const float* g, int i) {
  return *reinterpret_cast<const float4*>(g + i);
}
template <>
__device__ __forceinline__ float4 load_g4<bf16>(const bf16* g, int i) {
  const uint2 u = *reinterpret_cast<const uint2*>(g + i);
  const bf16* h = reinterpret_cast<const bf16*>(&u);
  return make_float4(__bfloat162float(h[0]), __bfloat162float(h[1]), __bfloat162float(h[2]), __bfloat162float(h[3]));
}

// One block per row; every thread loads its (<= NORM_VEC) float4 of the row at once.
template <typename T>
__global__ void __launch_bounds__(NORM_THREADS) rmsnorm_kernel(const float* X, int ldx,
                                                               const T* g, T* Y,
                                                               T* Y_lo, float* Y32,
                                                               int ldy, int d, float eps, float* Z,
                                                               int ldz, int zcols) {
  pdl_trigger();  // the next kernel may start its prologue
  // the gains are weights (never written by a kernel): load them before the wait
  float4 gg[NORM_VEC];
#pragma unroll
  for (int k = 0; k < NORM_VEC; ++k) {
    const int i = (threadIdx.x + k * NORM_THREADS) * 4;
    gg[k] = i < d ? load_g4(g, i) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  pdl_wait();     // inputs of this kernel are complete
  __shared__ float red[33];
  const float* x = X + static_cast<size_t>(blockIdx.x) * ldx;
  float4 v[NORM_VEC];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < NORM_VEC; ++k) {
    const int i = (threadIdx.x + k * NORM_THREADS) * 4;
    v[k] = i < d ? *reinterpret_cast<const float4*>(x + i) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
#pragma unroll
  for (int k = 0; k < NORM_VEC; ++k) ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
  if (Z) {
    float4* z = reinterpret_cast<float4*>(Z + static_cast<size_t>(blockIdx.x) * ldz);
    for (int i = threadIdx.x; i < zcols / 4; i += NORM_THREADS) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  const size_t row = static_cast<size_t>(blockIdx.x) * ldy;
#pragma unroll
  for (int k = 0; k < NORM_VEC; ++k) {
    const int i = (threadIdx.x + k * NORM_THREADS) * 4;
    if (i < d) {
      const float4 y = make_float4(v[k].x * r * gg[k].x, v[k].y * r * gg[k].y, v[k].z * r * gg[k].z,
                                   v[k].w * r * gg[k].w);
      store_act4(Y, Y_lo, row + i, y);
      if (Y32) *reinterpret_cast<float4*>(Y32 + row + i) = y;
    }
  }
}

// Rotate-half RoPE of q and k, plus the write of k and v into the paged cache
// (T = element type of the cache).  One block per row; an item is 4 consecutive
// pair indices j..j+3 of one head (pairs (j, j + hd/2)).

template <typename T>
__global__ void rope_kv_kernel(const RopeKvParams p) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int row = blockIdx.x;
  const int b = row / p.rows_per_seq, i = row % p.rows_per_seq;
  const int n = p.n[b];
  int pos = n + p.pos_base + (p.pos_off ? p.pos_off[i] : i);
  const int slot = n + p.slot_base + i;
  const int nvalid = p.valid ? p.valid[b] + p.valid_plus : p.rows_per_seq;
  const bool write_kv = i < nvalid;
  const int half = p.hd / 2;
  if (pos < 0 || pos >= p.max_pos) {
    if (threadIdx.x == 0) atomicOr(p.err, ERR_CAPACITY);
    pos = 0;
  }
  int page = -1;
  if (write_kv) {
    const int pi = slot >> 4;
    if (slot < 0 || pi >= p.max_pages) {
      if (threadIdx.x == 0) atomicOr(p.err, ERR_CAPACITY);
    } else {
      page = p.page_table[b * p.max_pages + pi];
    }
  }
  const float* src = p.qkv + static_cast<size_t>(row) * p.ldqkv;
  T* pool = static_cast<T*>(p.pool) + static_cast<size_t>(p.layer) * p.pool_layer_stride;
  const float2* tab = p.rope + static_cast<size_t>(pos) * half;
  const int per_head = half / 4;
  for (int it = threadIdx.x; it < p.H * per_head; it += blockDim.x) {
    const int h = it / per_head, j = (it % per_head) * 4;
    const float4 cs01 = *reinterpret_cast<const float4*>(tab + j);
    const float4 cs23 = *reinterpret_cast<const float4*>(tab + j + 2);
    const float4 c = make_float4(cs01.x, cs01.z, cs23.x, cs23.z);
    const float4 sn = make_float4(cs01.y, cs01.w, cs23.y, cs23.w);
    const int hb = h * p.hd + j;
    float4 q1, q2, k1, k2, v1, v2;
    if (p.q_col >= 0) {
      q1 = *reinterpret_cast<const float4*>(src + p.q_col + hb);
      q2 = *reinterpret_cast<const float4*>(src + p.q_col + hb + half);
    }
    if (page >= 0) {
      k1 = *reinterpret_cast<const float4*>(src + p.k_col + hb);
      k2 = *reinterpret_cast<const float4*>(src + p.k_col + hb + half);
      v1 = *reinterpret_cast<const float4*>(src + p.v_col + hb);
      v2 = *reinterpret_cast<const float4*>(src + p.v_col + hb + half);
    }
    if (p.q_col >= 0) {
      float* qo = p.q_out + static_cast<size_t>(row) * p.ldq + hb;
      *reinterpret_cast<float4*>(qo) = rot_lo(q1, q2, c, sn);
      *reinterpret_cast<float4*>(qo + half) = rot_hi(q1, q2, c, sn);
    }
    if (page >= 0) {
      T* base = pool + (static_cast<size_t>(page) * p.H + h) * p.planes * 16 * p.hd + (slot & 15) * p.hd + j;
      const size_t plane = 16 * static_cast<size_t>(p.hd);
      const float4 ka = rot_lo(k1, k2, c, sn), kb = rot_hi(k1, k2, c, sn);
      if (p.planes == 4) {  // K_hi, K_lo, V_hi, V_lo
        store4_split(base, base + plane, ka);
        store4_split(base + half, base + plane + half, kb);
        store4_split(base + 2 * plane, base + 3 * plane, v1);
        store4_split(base + 2 * plane + half, base + 3 * plane + half, v2);
      } else {
        store4<T>(base, ka);
        store4<T>(base + half, kb);
        store4<T>(base + plane, v1);
        store4<T>(base + plane + half, v2);
      }
    }
  }
}

// SwiGLU: h = SiLU(gate) * up, gate in columns [0, F), up in [F, 2F).
// A whole number of waves of CTAs (the tree verify: two per SM, next to a resident linear
// CTA), each taking an equal contiguous share of the float4 items: every SM gets the
// same work, so no SM holds up the next kernel.  A thread takes at most SWIGLU_IT
// items of its CTA's share, all loads issued before any store.
constexpr int SWIGLU_THREADS = 256;
constexpr int SWIGLU_IT = 4;
template <typename T>
__global__ void __launch_bounds__(SWIGLU_THREADS) swiglu_kernel(const float* gu, int ldgu, int F, T* h,
                                                                T* h_lo, int ldh, int rows, int per_cta) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int per_row = F / 4;
  const long long total = static_cast<long long>(rows) * per_row;
  const long long c0 = static_cast<long long>(blockIdx.x) * per_cta;
  const long long c1 = min(total, c0 + per_cta);
  float4 a[SWIGLU_IT], u[SWIGLU_IT];
#pragma unroll
  for (int k = 0; k < SWIGLU_IT; ++k) {
    const long long it = c0 + threadIdx.x + static_cast<long long>(k) * SWIGLU_THREADS;
    if (it < c1) {
      const float* g = gu + (it / per_row) * ldgu + (it % per_row) * 4;
      a[k] = *reinterpret_cast<const float4*>(g);
      u[k] = *reinterpret_cast<const float4*>(g + F);
    }
  }
#pragma unroll
  for (int k = 0; k < SWIGLU_IT; ++k) {
    const long long it = c0 + threadIdx.x + static_cast<long long>(k) * SWIGLU_THREADS;
    if (it < c1)
      store_act4(h, h_lo, static_cast<size_t>((it / per_row) * ldh + (it % per_row) * 4),
                 make_float4(silu_f(a[k].x) * u[k].x, silu_f(a[k].y) * u[k].y, silu_f(a[k].z) * u[k].z,
                             silu_f(a[k].w) * u[k].w));
  }
}

template <typename T>
__global__ void embed_kernel(const T* E, int d, int V, float* x,
                             int rows_per_seq, const int* tokens, const int* tok_hist,
                             int hist_stride, const int* n, const int* valid, int* err) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  const int r = blockIdx.x;
  int tok;
  if (tokens) {
    tok = tokens[r];
  } else {
    const int b = r / rows_per_seq, i = r % rows_per_seq;
    tok = i < valid[b] ? tok_hist[static_cast<size_t>(b) * hist_stride + n[b] + i] : 0;
  }
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERR_BAD_INDEX);
    tok = 0;
  }
  const T* e = E + static_cast<size_t>(tok) * d;
  float* y = x + static_cast<size_t>(r) * d;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) *reinterpret_cast<float4*>(y + i) = load_g4(e, i);
}

// (value, index) order of the method: larger value first, then smaller index.
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

__global__ void __launch_bounds__(512) argmax_kernel(const float* logits, int V, int* out, float* stats) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  __shared__ float sv[32];
  __shared__ int si[32];
  const float* z = logits + static_cast<size_t>(blockIdx.x) * V;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  const int V4 = V / 4;
  for (int base = threadIdx.x; base < V4; base += 4 * blockDim.x) {
    float4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i4 = base + u * blockDim.x;
      v[u] = i4 < V4 ? *reinterpret_cast<const float4*>(z + 4 * i4) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (base + u * static_cast<int>(blockDim.x) >= V4) break;
      const int i = 4 * (base + u * blockDim.x);
      if (better(v[u].x, i, bv, bi)) { bv = v[u].x; bi = i; }
      if (better(v[u].y, i + 1, bv, bi)) { bv = v[u].y; bi = i + 1; }
      if (better(v[u].z, i + 2, bv, bi)) { bv = v[u].z; bi = i + 2; }
      if (better(v[u].w, i + 3, bv, bi)) { bv = v[u].w; bi = i + 3; }
    }
  }
  for (int i = 4 * V4 + threadIdx.x; i < V; i += blockDim.x)
    if (better(z[i], i, bv, bi)) { bv = z[i]; bi = i; }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (better(ov, oi, bv, bi)) {
      bv = ov;
      bi = oi;
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) {
    sv[warp] = bv;
    si[warp] = bi;
  }
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    bv = lane < nw ? sv[lane] : -INFINITY;
    bi = lane < nw ? si[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (better(ov, oi, bv, bi)) {
        bv = ov;
        bi = oi;
      }
    }
    if (lane == 0) {
      out[blockIdx.x] = bi < V ? bi : 0;
      sv[0] = bv;
    }
  }
  if (!stats) return;
  // softmax statistics of the row at temperature 1: with e_i = exp(z_i - m),
  // S = sum e_i, A = sum e_i (z_i - m): log S and the entropy H = log S - A / S
  __syncthreads();
  const float m = sv[0];
  float S = 0.f, A = 0.f;
  for (int i4 = threadIdx.x; i4 < V4; i4 += blockDim.x) {
    const float4 v = *reinterpret_cast<const float4*>(z + 4 * i4);
    const float a = v.x - m, b = v.y - m, c = v.z - m, d = v.w - m;
    const float ea = expf(a), eb = expf(b), ec = expf(c), ed = expf(d);
    S += (ea + eb) + (ec + ed);
    A += (ea * a + eb * b) + (ec * c + ed * d);
  }
  for (int i = 4 * V4 + threadIdx.x; i < V; i += blockDim.x) {
    const float a = z[i] - m, ea = expf(a);
    S += ea;
    A += ea * a;
  }
  __shared__ float red[2][33];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    S += __shfl_xor_sync(0xffffffffu, S, o);
    A += __shfl_xor_sync(0xffffffffu, A, o);
  }
  if (lane == 0) {
    red[0][warp] = S;
    red[1][warp] = A;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s2 = 0.f, a2 = 0.f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) {
      s2 += red[0][w];
      a2 += red[1][w];
    }
    const float lse = logf(s2);
    stats[3 * blockIdx.x] = m;
    stats[3 * blockIdx.x + 1] = lse;
    stats[3 * blockIdx.x + 2] = lse - a2 / s2;
  }
}

constexpr int TOPK_MAX = 8;

// Top-k of a row in two levels: each block selects the top-k of a 2048-score slice
// (every thread keeps a sorted register list of its 8 scores, then k rounds of a
// block-wide arg-best), writes its k candidates, and the last block of the row to
// finish merges the candidates (counter per row, reset by the merger).
constexpr int TOPK_THREADS = 256;
constexpr int TOPK_SLICE = TOPK_THREADS * 8;

__device__ __forceinline__ void topk_insert(float (&lv)[TOPK_MAX], int (&li)[TOPK_MAX], int k, float v, int ii) {
#pragma unroll
  for (int j = 0; j < TOPK_MAX; ++j) {
    if (j < k && better(v, ii, lv[j], li[j])) {
      const float sv2 = lv[j];
      const int si2 = li[j];
      lv[j] = v;
      li[j] = ii;
      v = sv2;
      ii = si2;
    }
  }
}

// k rounds of block-wide arg-best over the heads of the per-thread sorted lists;
// round r's winner is written to (out_v[r], out_i[r]) by thread 0.
__device__ void topk_block_select(float (&lv)[TOPK_MAX], int (&li)[TOPK_MAX], int k, float* out_v, int* out_i) {
  __shared__ float sv[32];
  __shared__ int si[32];
  __shared__ int s_win;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int head = 0;
  for (int r = 0; r < k; ++r) {
    float bv = -INFINITY;
    int bi = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < TOPK_MAX; ++j)
      if (j == head) {
        bv = lv[j];
        bi = li[j];
      }
    float cv = bv;
    int ci = bi;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, cv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, ci, o);
      if (better(ov, oi, cv, ci)) {
        cv = ov;
        ci = oi;
      }
    }
    if (lane == 0) {
      sv[warp] = cv;
      si[warp] = ci;
    }
    __syncthreads();
    if (warp == 0) {
      const int nw = blockDim.x >> 5;
      cv = lane < nw ? sv[lane] : -INFINITY;
      ci = lane < nw ? si[lane] : 0x7fffffff;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, cv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, ci, o);
        if (better(ov, oi, cv, ci)) {
          cv = ov;
          ci = oi;
        }
      }
      if (lane == 0) {
        s_win = ci;
        out_v[r] = cv;
        out_i[r] = ci;
      }
    }
    __syncthreads();
    if (bi == s_win && bi != 0x7fffffff) ++head;  // indices are unique: one owner
    __syncthreads();
  }
}

__global__ void __launch_bounds__(TOPK_THREADS) topk_kernel(const float* logits, int V, int k,
                                                            int* idx, float* val,
                                                            int out_stride, float* ws_v,
                                                            int* ws_i, int* counters) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  __shared__ float s_bv[TOPK_MAX];
  __shared__ int s_bi[TOPK_MAX];
  __shared__ int s_last;
  const int row = blockIdx.y, blk = blockIdx.x, nblk = gridDim.x;
  const float* z = logits + static_cast<size_t>(row) * V;
  float lv[TOPK_MAX];
  int li[TOPK_MAX];
#pragma unroll
  for (int j = 0; j < TOPK_MAX; ++j) {
    lv[j] = -INFINITY;
    li[j] = 0x7fffffff;
  }
  // this thread's 8 scores: two float4 of the slice (V is a multiple of 4)
  const int s0 = blk * TOPK_SLICE;
  float4 v[2];
  int i0[2];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    i0[u] = s0 + (threadIdx.x + u * TOPK_THREADS) * 4;
    v[u] = i0[u] < V ? *reinterpret_cast<const float4*>(z + i0[u]) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    if (i0[u] >= V) continue;
    topk_insert(lv, li, k, v[u].x, i0[u]);
    topk_insert(lv, li, k, v[u].y, i0[u] + 1);
    topk_insert(lv, li, k, v[u].z, i0[u] + 2);
    topk_insert(lv, li, k, v[u].w, i0[u] + 3);
  }
  const size_t wbase = (static_cast<size_t>(row) * nblk + blk) * TOPK_MAX;
  if (nblk == 1) {
    topk_block_select(lv, li, k, s_bv, s_bi);
  } else {
    topk_block_select(lv, li, k, ws_v + wbase, ws_i + wbase);
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      const int old = atomicAdd(&counters[row], 1);
      s_last = (old == nblk - 1) ? 1 : 0;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // merge: thread t holds candidates t, t + 256, ... of the nblk * k list
#pragma unroll
    for (int j = 0; j < TOPK_MAX; ++j) {
      lv[j] = -INFINITY;
      li[j] = 0x7fffffff;
    }
    const int ncand = nblk * k;
    for (int c = threadIdx.x; c < ncand; c += TOPK_THREADS) {
      const size_t o = static_cast<size_t>(row) * nblk * TOPK_MAX + (c / k) * TOPK_MAX + (c % k);
      topk_insert(lv, li, k, __ldcg(ws_v + o), __ldcg(ws_i + o));
    }
    topk_block_select(lv, li, k, s_bv, s_bi);
    if (threadIdx.x == 0) counters[row] = 0;
  }
  if (threadIdx.x < k) {
    const int ci = s_bi[threadIdx.x];
    idx[static_cast<size_t>(row) * out_stride + threadIdx.x] = ci < V ? ci : 0;
    if (val) val[static_cast<size_t>(row) * out_stride + threadIdx.x] = s_bv[threadIdx.x];
  }
}

}  // namespace

cudaError_t rmsnorm(int dtype, const float* X, int ldx, const void* g, void* Y, void* Y_lo, float* Y32,
                    int ldy, int rows, int d, float eps, float* Z, int ldz, int zcols, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (Z && ((zcols & 3) || (ldz & 3) || (reinterpret_cast<uintptr_t>(Z) & 15))) return cudaErrorInvalidValue;
  if ((d & 3) || (ldx & 3) || (ldy & 3) || d > NORM_THREADS * NORM_VEC * 4) return cudaErrorInvalidValue;
  if (dtype == 0)
    launch_pdl(rmsnorm_kernel<float>, dim3(rows), dim3(NORM_THREADS), 0, s, X, ldx, static_cast<const float*>(g), static_cast<float*>(Y),
                                               nullptr, Y32, ldy, d, eps, Z, ldz, zcols);
  else
    launch_pdl(rmsnorm_kernel<bf16>, dim3(rows), dim3(NORM_THREADS), 0, s, X, ldx, static_cast<const bf16*>(g), static_cast<bf16*>(Y),
                                              static_cast<bf16*>(Y_lo), Y32, ldy, d, eps, Z, ldz, zcols);
  return cudaGetLastError();
}

cudaError_t rope_kv(const RopeKvParams& p, int dtype, cudaStream_t s) {
  const int rows = p.B * p.rows_per_seq;
  if (rows <= 0) return cudaSuccess;
  if ((p.hd & 15) || (p.ldqkv & 3) || (p.ldq & 3) || (p.q_col >= 0 && (p.q_col & 3)) || (p.k_col & 3) ||
      (p.v_col & 3))
    return cudaErrorInvalidValue;
  if (p.planes != 2 && !(p.planes == 4 && dtype == 1)) return cudaErrorInvalidValue;
  if (dtype == 0)
    launch_pdl(rope_kv_kernel<float>, dim3(rows), dim3(256), 0, s, p);
  else
    launch_pdl(rope_kv_kernel<bf16>, dim3(rows), dim3(256), 0, s, p);
  return cudaGetLastError();
}

cudaError_t swiglu(int dtype, const float* gu, int ldgu, int F, void* h, void* h_lo, int ldh, int rows,
                   cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if ((F & 3) || (ldh & 3) || (ldgu & 3)) return cudaErrorInvalidValue;
  const long long items = static_cast<long long>(rows) * (F / 4);
  const long long cap = SWIGLU_THREADS * SWIGLU_IT;  // items one CTA can take
  const int sms = tc_num_sms();
  long long grid = (items + cap - 1) / cap;
  if (grid > sms) grid = ((grid + sms - 1) / sms) * sms;  // whole waves of equal shares
  const int per_cta = static_cast<int>((items + grid - 1) / grid);  // <= cap
  if (dtype == 0)
    launch_pdl(swiglu_kernel<float>, dim3(static_cast<unsigned>(grid)), dim3(SWIGLU_THREADS), 0, s, gu, ldgu, F,
               static_cast<float*>(h), nullptr, ldh, rows, per_cta);
  else
    launch_pdl(swiglu_kernel<bf16>, dim3(static_cast<unsigned>(grid)), dim3(SWIGLU_THREADS), 0, s, gu, ldgu, F,
               static_cast<bf16*>(h), static_cast<bf16*>(h_lo), ldh, rows, per_cta);
  return cudaGetLastError();
}

cudaError_t embed(int dtype, const void* E, int d, int V, float* x, int rows, int rows_per_seq,
                  const int* tokens, const int* tok_hist, int hist_stride, const int* n,
                  const int* valid, int* err, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (dtype == 0)
    launch_pdl(embed_kernel<float>, dim3(rows), dim3(256), 0, s, static_cast<const float*>(E), d, V, x, rows_per_seq,
                                             tokens, tok_hist, hist_stride, n, valid, err);
  else
    launch_pdl(embed_kernel<bf16>, dim3(rows), dim3(256), 0, s, static_cast<const bf16*>(E), d, V, x, rows_per_seq,
                                            tokens, tok_hist, hist_stride, n, valid, err);
  return cudaGetLastError();
}

cudaError_t argmax_rows(const float* logits, int V, int rows, int* out, cudaStream_t s, float* stats) {
  if (rows <= 0) return cudaSuccess;
  if (V & 3) return cudaErrorInvalidValue;  // rows are read as float4
  launch_pdl(argmax_kernel, dim3(rows), dim3(512), 0, s, logits, V, out, stats);
  return cudaGetLastError();
}

cudaError_t topk_rows(const float* logits, int V, int rows, int k, int* idx, float* val, int out_stride,
                      float* ws_v, int* ws_i, int* counters, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (k < 1 || k > TOPK_MAX || (V & 3)) return cudaErrorInvalidValue;
  const int nblk = (V + TOPK_SLICE - 1) / TOPK_SLICE;
  if (nblk > TOPK_MAX_BLOCKS) return cudaErrorInvalidValue;
  dim3 grid(nblk, rows);
  launch_pdl(topk_kernel, dim3(grid), dim3(TOPK_THREADS), 0, s, logits, V, k, idx, val, out_stride, ws_v, ws_i, counters);
  return cudaGetLastError();
}

}  // namespace chimera
