// Row-wise kernels of the step: RMSNorm, RoPE + paged KV write, SwiGLU, embedding
// gather, argmax and top-k over the vocabulary.
#include <cmath>

#include "common.cuh"
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
template <typename T>
__global__ void rmsnorm_kernel(const float* __restrict__ X, int ldx, const T* __restrict__ g,
                               T* __restrict__ Y, T* __restrict__ Y_lo, float* __restrict__ Y32,
                               int ldy, int d, float eps) {
  __shared__ float red[33];
  const float* x = X + static_cast<size_t>(blockIdx.x) * ldx;
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) ss = fmaf(x[i], x[i], ss);
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  const size_t row = static_cast<size_t>(blockIdx.x) * ldy;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float v = x[i] * r * to_f(g[i]);
    store_act(Y, Y_lo, row + i, v);
    if (Y32) Y32[row + i] = v;
  }
}

// Rotate-half RoPE of q and k, plus the write of k and v into the paged cache
// (T = element type of the cache).
template <typename T>
__global__ void rope_kv_kernel(const RopeKvParams p) {
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
  for (int idx = threadIdx.x; idx < p.H * half; idx += blockDim.x) {
    const int h = idx / half, j = idx % half;
    const float2 cs = p.rope[static_cast<size_t>(pos) * half + j];
    if (p.q_col >= 0) {
      const float x1 = src[p.q_col + h * p.hd + j];
      const float x2 = src[p.q_col + h * p.hd + j + half];
      float* qo = p.q_out + static_cast<size_t>(row) * p.ldq + h * p.hd;
      qo[j] = x1 * cs.x - x2 * cs.y;
      qo[j + half] = x2 * cs.x + x1 * cs.y;
    }
    if (page >= 0) {
      T* base = pool + (static_cast<size_t>(page) * p.H + h) * 2 * 16 * p.hd + (slot & 15) * p.hd;
      const float k1 = src[p.k_col + h * p.hd + j];
      const float k2 = src[p.k_col + h * p.hd + j + half];
      base[j] = from_f<T>(k1 * cs.x - k2 * cs.y);
      base[j + half] = from_f<T>(k2 * cs.x + k1 * cs.y);
      base[16 * p.hd + j] = from_f<T>(src[p.v_col + h * p.hd + j]);
      base[16 * p.hd + j + half] = from_f<T>(src[p.v_col + h * p.hd + j + half]);
    }
  }
}

// SwiGLU: h = SiLU(gate) * up, gate in columns [0, F), up in [F, 2F).
template <typename T>
__global__ void swiglu_kernel(const float* __restrict__ gu, int ldgu, int F, T* __restrict__ h,
                              T* __restrict__ h_lo, int ldh) {
  const float* g = gu + static_cast<size_t>(blockIdx.y) * ldgu;
  const size_t row = static_cast<size_t>(blockIdx.y) * ldh;
  for (int f = blockIdx.x * blockDim.x + threadIdx.x; f < F; f += gridDim.x * blockDim.x)
    store_act(h, h_lo, row + f, silu_f(g[f]) * g[F + f]);
}

template <typename T>
__global__ void embed_kernel(const T* __restrict__ E, int d, int V, float* __restrict__ x,
                             int rows_per_seq, const int* tokens, const int* tok_hist,
                             int hist_stride, const int* n, const int* valid, int* err) {
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
  for (int i = threadIdx.x; i < d; i += blockDim.x) y[i] = to_f(e[i]);
}

// (value, index) order of the method: larger value first, then smaller index.
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

__global__ void argmax_kernel(const float* __restrict__ logits, int V, int* __restrict__ out) {
  __shared__ float sv[32];
  __shared__ int si[32];
  const float* z = logits + static_cast<size_t>(blockIdx.x) * V;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int i = threadIdx.x; i < V; i += blockDim.x) {
    const float v = z[i];
    if (better(v, i, bv, bi)) {
      bv = v;
      bi = i;
    }
  }
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
    if (lane == 0) out[blockIdx.x] = bi < V ? bi : 0;
  }
}

constexpr int TOPK_MAX = 8;

// Top-k of a row: every thread keeps a sorted list of its strided elements; then k
// rounds of a block-wide arg-best over the list heads.
__global__ void topk_kernel(const float* __restrict__ logits, int V, int k, int* __restrict__ idx,
                            float* __restrict__ val, int out_stride) {
  __shared__ float sv[32];
  __shared__ int si[32];
  __shared__ int s_win;
  const float* z = logits + static_cast<size_t>(blockIdx.x) * V;
  float lv[TOPK_MAX];
  int li[TOPK_MAX];
#pragma unroll
  for (int j = 0; j < TOPK_MAX; ++j) {
    lv[j] = -INFINITY;
    li[j] = 0x7fffffff;
  }
  for (int i = threadIdx.x; i < V; i += blockDim.x) {
    float v = z[i];
    int ii = i;
    if (!better(v, ii, lv[k - 1], li[k - 1])) continue;
#pragma unroll
    for (int j = 0; j < TOPK_MAX; ++j) {
      if (j < k && better(v, ii, lv[j], li[j])) {
        const float tv = lv[j];
        const int ti = li[j];
        lv[j] = v;
        li[j] = ii;
        v = tv;
        ii = ti;
      }
    }
  }
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
        idx[static_cast<size_t>(blockIdx.x) * out_stride + r] = ci < V ? ci : 0;
        if (val) val[static_cast<size_t>(blockIdx.x) * out_stride + r] = cv;
      }
    }
    __syncthreads();
    if (bi == s_win && bi != 0x7fffffff) ++head;  // indices are unique: one owner
    __syncthreads();
  }
}

}  // namespace

cudaError_t rmsnorm(int dtype, const float* X, int ldx, const void* g, void* Y, void* Y_lo, float* Y32,
                    int ldy, int rows, int d, float eps, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (dtype == 0)
    rmsnorm_kernel<float><<<rows, 256, 0, s>>>(X, ldx, static_cast<const float*>(g), static_cast<float*>(Y),
                                               nullptr, Y32, ldy, d, eps);
  else
    rmsnorm_kernel<bf16><<<rows, 256, 0, s>>>(X, ldx, static_cast<const bf16*>(g), static_cast<bf16*>(Y),
                                              static_cast<bf16*>(Y_lo), Y32, ldy, d, eps);
  return cudaGetLastError();
}

cudaError_t rope_kv(const RopeKvParams& p, int kv_f32, cudaStream_t s) {
  const int rows = p.B * p.rows_per_seq;
  if (rows <= 0) return cudaSuccess;
  if (kv_f32)
    rope_kv_kernel<float><<<rows, 256, 0, s>>>(p);
  else
    rope_kv_kernel<bf16><<<rows, 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t swiglu(int dtype, const float* gu, int ldgu, int F, void* h, void* h_lo, int ldh, int rows,
                   cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  dim3 grid((F + 255) / 256, rows);
  if (dtype == 0)
    swiglu_kernel<float><<<grid, 256, 0, s>>>(gu, ldgu, F, static_cast<float*>(h), nullptr, ldh);
  else
    swiglu_kernel<bf16><<<grid, 256, 0, s>>>(gu, ldgu, F, static_cast<bf16*>(h), static_cast<bf16*>(h_lo), ldh);
  return cudaGetLastError();
}

cudaError_t embed(int dtype, const void* E, int d, int V, float* x, int rows, int rows_per_seq,
                  const int* tokens, const int* tok_hist, int hist_stride, const int* n,
                  const int* valid, int* err, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (dtype == 0)
    embed_kernel<float><<<rows, 256, 0, s>>>(static_cast<const float*>(E), d, V, x, rows_per_seq,
                                             tokens, tok_hist, hist_stride, n, valid, err);
  else
    embed_kernel<bf16><<<rows, 256, 0, s>>>(static_cast<const bf16*>(E), d, V, x, rows_per_seq,
                                            tokens, tok_hist, hist_stride, n, valid, err);
  return cudaGetLastError();
}

cudaError_t argmax_rows(const float* logits, int V, int rows, int* out, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  argmax_kernel<<<rows, 512, 0, s>>>(logits, V, out);
  return cudaGetLastError();
}

cudaError_t topk_rows(const float* logits, int V, int rows, int k, int* idx, float* val,
                      int out_stride, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (k < 1 || k > TOPK_MAX) return cudaErrorInvalidValue;
  topk_kernel<<<rows, 512, 0, s>>>(logits, V, k, idx, val, out_stride);
  return cudaGetLastError();
}

}  // namespace chimera
