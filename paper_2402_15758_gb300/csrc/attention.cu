// Tree-masked attention over the paged KV cache (tree verification, prefill chunks
// and the draft's full-context layer).
//
// Keys of sequence b: the n_ctx[b] committed rows (visible to every query) followed by
// n_local rows at slots n_ctx..n_ctx+n_local-1; query i sees local row j iff bit j of
// anc[q_local0 + i] is set (a tree node's ancestors-or-self, or a causal chain).
// KV layout: pool[layer][block][head][K|V][16 rows][hd], page_table[b][slot / 16].
//
// Grid (splits, heads, batch).  Each CTA loads every KV tile of its key range once
// into shared memory for all the sequence's queries; online softmax in fp32.  With
// several splits, every CTA writes (unnormalised output, running max, running sum)
// and the last CTA of the (b, h) pair merges them in split order.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace chimera {
namespace {

constexpr int KT = 32;      // keys per tile
constexpr int WARPS = 8;
constexpr int QPW = 8;      // queries per warp (nq <= 64)

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename TKV, typename T, int HD>
__global__ void __launch_bounds__(WARPS * 32) attn_kernel(const AttnParams p) {
  constexpr int DPL = HD / 32;
  extern __shared__ float sm[];
  float* Ks = sm;                   // [KT][HD + 1]
  float* Vs = Ks + KT * (HD + 1);   // [KT][HD]
  float* Qs = Vs + KT * HD;         // [nq][HD]
  __shared__ int s_last;

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nctx = p.n_ctx[b];
  const int nloc = p.n_local_dev ? p.n_local_dev[b] : p.n_local;
  const int nq = p.nq_dev ? p.nq_dev[b] : p.nq;
  const int total = nctx + nloc;
  const int ntiles = (total + KT - 1) / KT;
  const int tps = (ntiles + p.splits - 1) / p.splits;
  const int t0 = s * tps;
  const int t1 = min(ntiles, t0 + tps);
  const float* q = p.q;
  const TKV* pool = static_cast<const TKV*>(p.pool) + static_cast<size_t>(p.layer) * p.pool_layer_stride;

  for (int idx = threadIdx.x; idx < nq * HD; idx += blockDim.x) {
    const int i = idx / HD, dd = idx % HD;
    Qs[idx] = q[static_cast<size_t>(b * p.q_rows + i) * p.ldq + h * HD + dd];
  }

  float m[QPW], l[QPW], acc[QPW][DPL];
  unsigned long long msk[QPW];
#pragma unroll
  for (int qq = 0; qq < QPW; ++qq) {
    m[qq] = -INFINITY;
    l[qq] = 0.f;
    const int qi = warp + WARPS * qq;
    msk[qq] = qi < nq ? p.anc[p.q_local0 + qi] : 0ull;
#pragma unroll
    for (int r = 0; r < DPL; ++r) acc[qq][r] = 0.f;
  }

  for (int t = t0; t < t1; ++t) {
    __syncthreads();
    for (int idx = threadIdx.x; idx < KT * HD; idx += blockDim.x) {
      const int j = idx / HD, dd = idx % HD;
      const int key = t * KT + j;
      float kv = 0.f, vv = 0.f;
      if (key < total) {
        const int page = p.page_table[b * p.max_pages + (key >> 4)];
        const TKV* base = pool + (static_cast<size_t>(page) * p.H + h) * 2 * 16 * HD;
        kv = to_f(base[(key & 15) * HD + dd]);
        vv = to_f(base[16 * HD + (key & 15) * HD + dd]);
      }
      Ks[j * (HD + 1) + dd] = kv;
      Vs[j * HD + dd] = vv;
    }
    __syncthreads();
    const int key = t * KT + lane;
#pragma unroll
    for (int qq = 0; qq < QPW; ++qq) {
      const int qi = warp + WARPS * qq;
      if (qi < nq) {
        const bool vis = key < nctx || (key < total && ((msk[qq] >> (key - nctx)) & 1ull));
        float sc = -INFINITY;
        if (vis) {
          float d = 0.f;
#pragma unroll 16
          for (int dd = 0; dd < HD; ++dd) d = fmaf(Qs[qi * HD + dd], Ks[lane * (HD + 1) + dd], d);
          sc = d * p.scale;
        }
        const float mnew = fmaxf(m[qq], warp_max(sc));
        if (mnew != -INFINITY) {
          const float pj = vis ? expf(sc - mnew) : 0.f;
          const float corr = expf(m[qq] - mnew);
          l[qq] = l[qq] * corr + warp_sum(pj);
#pragma unroll
          for (int r = 0; r < DPL; ++r) acc[qq][r] *= corr;
          for (int j = 0; j < KT; ++j) {
            const float pjj = __shfl_sync(0xffffffffu, pj, j);
#pragma unroll
            for (int r = 0; r < DPL; ++r) acc[qq][r] = fmaf(pjj, Vs[j * HD + lane + 32 * r], acc[qq][r]);
          }
          m[qq] = mnew;
        }
      }
    }
  }

  T* out = static_cast<T*>(p.out);
  T* out_lo = static_cast<T*>(p.out_lo);
  if (p.splits == 1) {
#pragma unroll
    for (int qq = 0; qq < QPW; ++qq) {
      const int qi = warp + WARPS * qq;
      if (qi < nq) {
        const float inv = l[qq] > 0.f ? 1.f / l[qq] : 0.f;
#pragma unroll
        for (int r = 0; r < DPL; ++r)
          store_act(out, out_lo, static_cast<size_t>(b * p.q_rows + qi) * p.ldo + h * HD + lane + 32 * r,
                    acc[qq][r] * inv);
      }
    }
    return;
  }

  const size_t rec = HD + 2;
  float* wsb = p.ws + (static_cast<size_t>(b * p.H + h) * p.splits) * p.nq_max * rec;
#pragma unroll
  for (int qq = 0; qq < QPW; ++qq) {
    const int qi = warp + WARPS * qq;
    if (qi < nq) {
      float* w = wsb + (static_cast<size_t>(s) * p.nq_max + qi) * rec;
#pragma unroll
      for (int r = 0; r < DPL; ++r) __stcg(&w[lane + 32 * r], acc[qq][r]);
      if (lane == 0) {
        __stcg(&w[HD], m[qq]);
        __stcg(&w[HD + 1], l[qq]);
      }
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int old = atomicAdd(&p.counters[b * p.H + h], 1);
    s_last = (old == p.splits - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int qi = warp; qi < nq; qi += WARPS) {
    float M = -INFINITY;
    for (int sp = 0; sp < p.splits; ++sp)
      M = fmaxf(M, __ldcg(&wsb[(static_cast<size_t>(sp) * p.nq_max + qi) * rec + HD]));
    float L = 0.f, o[DPL];
#pragma unroll
    for (int r = 0; r < DPL; ++r) o[r] = 0.f;
    if (M != -INFINITY) {
      for (int sp = 0; sp < p.splits; ++sp) {
        const float* w = wsb + (static_cast<size_t>(sp) * p.nq_max + qi) * rec;
        const float ms = __ldcg(&w[HD]);
        if (ms == -INFINITY) continue;
        const float e = expf(ms - M);
        L += e * __ldcg(&w[HD + 1]);
#pragma unroll
        for (int r = 0; r < DPL; ++r) o[r] += e * __ldcg(&w[lane + 32 * r]);
      }
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int r = 0; r < DPL; ++r)
      store_act(out, out_lo, static_cast<size_t>(b * p.q_rows + qi) * p.ldo + h * HD + lane + 32 * r, o[r] * inv);
  }
  if (threadIdx.x == 0) p.counters[b * p.H + h] = 0;
}

template <typename TKV, typename T, int HD>
cudaError_t launch(const AttnParams& p, cudaStream_t s) {
  const size_t smem = (KT * (HD + 1) + KT * HD + static_cast<size_t>(p.nq_max) * HD) * sizeof(float);
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(attn_kernel<TKV, T, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    attr = true;
  }
  dim3 grid(p.splits, p.H, p.B);
  attn_kernel<TKV, T, HD><<<grid, WARPS * 32, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

size_t attn_ws_floats(int B, int H, int splits, int nq_max, int hd) {
  return static_cast<size_t>(B) * H * splits * nq_max * (hd + 2);
}

cudaError_t attention(const AttnParams& p, int dtype, int kv_f32, cudaStream_t s) {
  if (p.nq_max > WARPS * QPW || p.n_local > 64) return cudaErrorInvalidValue;
  if (dtype == 0) {
    if (p.hd == 64) return launch<float, float, 64>(p, s);
    if (p.hd == 128) return launch<float, float, 128>(p, s);
  } else if (kv_f32) {
    if (p.hd == 64) return launch<float, bf16, 64>(p, s);
    if (p.hd == 128) return launch<float, bf16, 128>(p, s);
  } else {
    if (p.hd == 64) return launch<bf16, bf16, 64>(p, s);
    if (p.hd == 128) return launch<bf16, bf16, 128>(p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace chimera
